// BF16 GEMM for GB300 (sm_103a): C = A B, the third kernel the paper evaluates (GEMM,
// Sec. 4), with tile width and ring depth from the analytic model (Eq. 6-9).
//
// Persistent CTAs walk the output tiles (BM = 128 rows x BN columns) in groups of 8 tile
// rows, so that CTAs working at the same time share A rows and B columns in L2:
//
//   warp 8 (loader, 1 thread)   A tile 128 x 64 and B tile 64 x BN per K stage into an
//                               NSTAGE-deep ring of 128B-swizzled slots (TMA, full/empty
//                               mbarriers)
//   warp 9 (MMA, whole warp,    tcgen05.mma kind::f16, M = 128, N = BN, K = 16: A K-major,
//     one elected lane issues)
//                               B MN-major (rows of B are contiguous in N), fp32 into one of
//                               two TMEM accumulators
//   warps 0-7 (epilogue)        warp w reads TMEM lanes 32 (w mod 4) .. + 31 (its 32 rows
//                               of the tile) and every other 64-column chunk from w div 4:
//                               fp32 -> bf16, staged per warp in shared memory and stored
//                               with TMA; the accumulator is released as soon as it is in
//                               registers, so the next-but-one tile may reuse it.
//
// TMEM: [0, BN) accumulator 0 | [BN, 2 BN) accumulator 1.
#include <cuda.h>
#include <cuda_bf16.h>

#include <atomic>
#include <mutex>

#include "gemm.h"
#include "gemm_model.h"
#include "kernels.h"
#include "ptx.cuh"

namespace loom {
namespace {

// NS other than 0 overrides the model's ring depth (the neighbours measured by the
// block-size ablation).
template <int BN, int NS = 0>
struct GemmCfg {
  static constexpr model::GemmPlan kPlan = model::gemm_plan_variant(BN);
  static_assert(kPlan.feasible, "no feasible GEMM plan for this tile width");
  static constexpr int BM = 128, BK = 64;
  static constexpr int NSTAGE = NS ? NS : kPlan.stages;
  static constexpr int THREADS = 320;                       // 8 epilogue warps, loader, MMA
  static constexpr int SPLIT_THREADS = 192;                 // split-K: 4 epilogue warps, loader, MMA
  static constexpr int NB = BN / 64;                        // 64-column boxes of a B stage
  static constexpr uint32_t A_BYTES = BM * BK * 2;          // one 128B-swizzled box
  static constexpr uint32_t B_BOX_BYTES = BK * 64 * 2;      // 64 K-rows x 64 N-columns
  static constexpr uint32_t STAGE_BYTES = A_BYTES + NB * B_BOX_BYTES;
  static constexpr uint32_t STG_OFF = NSTAGE * STAGE_BYTES;  // epilogue staging
  static constexpr uint32_t STG_WARP = 32 * 128;             // one 32-row x 128 B block per warp
  static constexpr uint32_t BAR_OFF = STG_OFF + 8 * STG_WARP;
  // barriers: full[NSTAGE], empty[NSTAGE], acc_full[2], acc_empty[2], drain
  static constexpr int NBAR = 2 * NSTAGE + 5;
  static constexpr uint32_t TMEM_PTR_OFF = BAR_OFF + NBAR * 8;
  static constexpr uint32_t ABORT_OFF = TMEM_PTR_OFF + 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16 + 1024;  // + alignment slack
  static constexpr uint32_t TMEM_COLS = 2 * BN <= 32 ? 32 : 2 * BN <= 64 ? 64 : 2 * BN <= 128 ? 128
                                        : 2 * BN <= 256 ? 256 : 512;
  static_assert(STG_WARP * 8 == model::kGemmStagingBytes, "staging layout matches the model");
  static_assert(BYTES <= 227 * 1024, "shared memory budget");
};

struct GemmParams {
  __nv_bfloat16* c;
  int M, N, K;
  int tiles_m, tiles_n, k_iters;
  int splits;  // split-K kernel: CTAs per cluster (= per tile)
  int group;   // tile rows per group of the tile order
  int k_alt;   // CTA-pair kernel: 1 walks K backwards in every other round of tiles
  int b_blocks;  // B [K, N]: 1 when tm_b views B as 64-column blocks (a stage's B in one box)
  int narrow_from;  // CTA-pair kernel: units from here on are 256 x 128 halves of the last tiles
  int n_units;      // CTA-pair kernel: work units (whole tiles, then the narrow halves)
  KernelCtl ctl;
};

// Tile t -> (tm, tn): groups of p.group tile rows, column-major inside a group (CTAs
// working at the same time share A rows and B columns in L2).
__device__ __forceinline__ void tile_coords(const GemmParams& p, int t, int& tm, int& tn) {
  const int group = p.group;
  const int per_group = group * p.tiles_n;
  const int g = t / per_group;
  const int first = g * group;
  const int rows = min(group, p.tiles_m - first);
  const int in = t - g * per_group;
  tm = first + in % rows;
  tn = in / rows;
}

// One epilogue warp's share of a finished accumulator: its 32 TMEM lanes (rows row0 ..
// row0 + 31 of C) and the 64-column chunks c = h, h + 2, ... < NB of the accumulator at
// `acc`.  Once its last chunk is in registers the warp arrives on `release` (the even
// CTA's barrier, over the cluster, when `remote`), so the MMA warp may reuse the
// accumulator while the stores drain.  A chunk goes through the warp's 4 KB staging block
// (128B-swizzled like the TMA box) and leaves with a TMA store; chunks wholly outside C
// are not stored.
template <int NB>
__device__ __forceinline__ void epilogue_warp(const CUtensorMap* tm_c, uint32_t acc, uint32_t stg, int h, int col0,
                                              int row0, int M, int N, uint32_t release, bool remote) {
  const int lane = threadIdx.x & 31;
  bool released = false;
#pragma unroll 1
  for (int c = h; c < NB; c += 2) {
    uint32_t r0[32], r1[32];
    tmem_ld32(acc + c * 64, r0);
    tmem_ld32(acc + c * 64 + 32, r1);
    tmem_wait_ld();
    reg_fence32(r0);
    reg_fence32(r1);
    if (c + 2 >= NB) {
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (remote) mbar_arrive_cluster(release);
        else mbar_arrive(release);
      }
      released = true;
    }
    if (col0 + c * 64 >= N || row0 >= M) continue;
    uint32_t w[32];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      w[i] = pack_bf16x2(__uint_as_float(r0[2 * i]), __uint_as_float(r0[2 * i + 1]));
      w[16 + i] = pack_bf16x2(__uint_as_float(r1[2 * i]), __uint_as_float(r1[2 * i + 1]));
    }
    if (lane == 0) bulk_wait_group_read0();  // this warp's previous store has read the block
    __syncwarp();
    const uint32_t row = stg + static_cast<uint32_t>(lane) * 128u;
#pragma unroll
    for (int q = 0; q < 8; ++q)
      st_shared_v4(row + (static_cast<uint32_t>(q ^ (lane & 7)) << 4), w[4 * q], w[4 * q + 1], w[4 * q + 2],
                   w[4 * q + 3]);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_3d(tm_c, stg, col0 + c * 64, row0, 0);
      bulk_commit_group();
    }
  }
  if (!released) {  // no chunk for this warp (a 64-column tile): nothing read, release at once
    __syncwarp();
    if (lane == 0) {
      if (remote) mbar_arrive_cluster(release);
      else mbar_arrive(release);
    }
  }
}

// BK_MAJOR: B given [N, K] (C = A B^T), its tiles K-major like A's; else B [K, N].
template <int BN, bool BK_MAJOR, int NS = 0>
__global__ void __launch_bounds__(GemmCfg<BN, NS>::THREADS, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                const __grid_constant__ CUtensorMap tm_c, const GemmParams p) {
  using C = GemmCfg<BN, NS>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_base = smem_u32(smem_raw);
  const uint32_t sbase = (raw_base + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (sbase - raw_base);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const uint32_t bar_full = sbase + C::BAR_OFF;         // [NSTAGE] stage loaded
  const uint32_t bar_empty = bar_full + 8 * C::NSTAGE;  // [NSTAGE] stage read by the MMAs
  const uint32_t bar_acc = bar_empty + 8 * C::NSTAGE;   // [2] accumulator b complete
  const uint32_t bar_acce = bar_acc + 16;               // [2] accumulator b read out
  const uint32_t bar_drain = bar_acce + 16;
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::TMEM_PTR_OFF);
  Abort ab{reinterpret_cast<volatile int*>(smem + C::ABORT_OFF)};
  const int tiles = p.tiles_m * p.tiles_n;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar_acc + 8 * b, 1);
      mbar_init(bar_acce + 8 * b, 8);  // one arrive per epilogue warp
    }
    mbar_init(bar_drain, 1);
    *ab.flag = 0;
    *(ab.flag + 1) = 0;
    fence_barrier_init();
  }
  if (warp == 9) tmem_alloc(smem_u32(tmem_ptr), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_ptr;
  // Launched as a programmatic dependent of the previous kernel in the stream: the set-up
  // above touches no global memory; from here on that kernel's writes must be complete
  // and visible, and the next launch may start its own set-up on SMs this grid frees.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;");

  if (warp == 8) {
    // ------------------------------------------------------------------ loader
    if (lane == 0) {
      prefetch_tensormap(&tm_a);
      prefetch_tensormap(&tm_b);
      int it = 0, issued = 0, skipped = -1;
      bool ok = true;
      for (int t = blockIdx.x; ok && t < tiles; t += gridDim.x) {
        int tm, tn;
        tile_coords(p, t, tm, tn);
        for (int ks = 0; ks < p.k_iters; ++ks, ++it) {
          const int s = it % C::NSTAGE;
          if (!(ok = mbar_wait(bar_empty + 8 * s, ((it / C::NSTAGE) & 1) ^ 1, p.ctl, ab))) break;
          issued = it + 1;
          if (p.ctl.inject == 3 && it == 2) {  // test hook: never load this stage
            skipped = it;
            continue;
          }
          const uint32_t dst = sbase + s * C::STAGE_BYTES;
          mbar_expect_tx(bar_full + 8 * s, C::STAGE_BYTES);
          tma_load_3d(dst, &tm_a, ks * C::BK, tm * C::BM, 0, bar_full + 8 * s);
          if constexpr (BK_MAJOR) {  // BN rows of B [N, K], 64 K-columns: one box
            tma_load_3d(dst + C::A_BYTES, &tm_b, ks * C::BK, tn * BN, 0, bar_full + 8 * s);
          } else if (p.b_blocks) {  // the tile's NB 64-column blocks of B [K, N]: one box
            tma_load_3d(dst + C::A_BYTES, &tm_b, 0, ks * C::BK, tn * C::NB, bar_full + 8 * s);
          } else {
#pragma unroll
            for (int x = 0; x < C::NB; ++x)
              tma_load_3d(dst + C::A_BYTES + x * C::B_BOX_BYTES, &tm_b, tn * BN + x * 64, ks * C::BK, 0,
                          bar_full + 8 * s);
          }
        }
      }
      Abort no_abort{ab.flag + 1};
      for (int i = max(0, issued - C::NSTAGE); i < issued; ++i)
        if (i != skipped) mbar_wait(bar_full + 8 * (i % C::NSTAGE), (i / C::NSTAGE) & 1, p.ctl, no_abort);
    }
  } else if (warp == 9) {
    // ------------------------------------------------------------------ MMA issuer
    {  // the whole warp runs this role; one elected lane issues
      // A: K-major, 8-row groups 1024 B apart, K-step +32 B inside the swizzle row.
      // B [K, N]: MN-major, 64-column boxes B_BOX_BYTES apart (LBO), 8 K-rows 1024 B apart
      //    (SBO), K-step +16 rows = +2048 B.  B [N, K]: K-major like A.
      constexpr uint32_t idesc = idesc_bf16(C::BM, BN, 0, BK_MAJOR ? 0 : 1);
      constexpr uint32_t kstep_b = BK_MAJOR ? 2u : 128u;
      const uint64_t da0 = sdesc_sw128(sbase, 16, 1024);
      const uint64_t db0 = sdesc_sw128(sbase + C::A_BYTES, BK_MAJOR ? 16u : C::B_BOX_BYTES, 1024);
      constexpr uint32_t kStage16 = C::STAGE_BYTES >> 4;
      int it = 0, lt = 0;
      bool ok = true;
      for (int t = blockIdx.x; ok && t < tiles; t += gridDim.x, ++lt) {
        const int b = lt & 1, use = lt >> 1;
        // the epilogue has read this accumulator's previous tile out
        if (lt >= 2 && !(ok = mbar_wait_warp(bar_acce + 8 * b, (use - 1) & 1, p.ctl, ab))) break;
        tc_fence_after();
        const uint32_t d = tmem + static_cast<uint32_t>(b * BN);
        for (int ks = 0; ks < p.k_iters; ++ks, ++it) {
          const int s = it % C::NSTAGE;
          if (!(ok = mbar_wait_warp(bar_full + 8 * s, (it / C::NSTAGE) & 1, p.ctl, ab))) break;
          tc_fence_after();
          const uint64_t da = da0 + s * kStage16, db = db0 + s * kStage16;
#pragma unroll
          for (int kk = 0; kk < C::BK / 16; ++kk)
            mma_ss_el(d, da + kk * 2, db + kk * kstep_b, idesc, (ks > 0 || kk > 0) ? 1u : 0u);
          tc_commit_el(bar_empty + 8 * s);
        }
        if (!ok) break;
        tc_commit_el(bar_acc + 8 * b);  // the tile's accumulator is complete
      }
      Abort no_abort{ab.flag + 1};
      tc_commit_el(bar_drain);
      mbar_wait_warp(bar_drain, 0, p.ctl, no_abort);
    }
  } else {
    // ------------------------------------------------------------------ epilogue (warps 0-7)
    const int quarter = warp & 3, half = warp >> 2;
    const uint32_t lane_addr = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t stg = sbase + C::STG_OFF + static_cast<uint32_t>(warp) * C::STG_WARP;
    int lt = 0;
    bool ok = true;
    for (int t = blockIdx.x; ok && t < tiles; t += gridDim.x, ++lt) {
      int tm, tn;
      tile_coords(p, t, tm, tn);
      const int b = lt & 1, use = lt >> 1;
      if (!(ok = mbar_wait_warp(bar_acc + 8 * b, use & 1, p.ctl, ab))) break;
      tc_fence_after();
      epilogue_warp<C::NB>(&tm_c, tmem + lane_addr + static_cast<uint32_t>(b * BN), stg, half, tn * BN,
                           tm * C::BM + quarter * 32, p.M, p.N, bar_acce + 8 * b, false);
    }
    if (lane == 0) bulk_wait_group0();  // the C stores have completed before the CTA exits
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------- split-K clusters
// One cluster of S = p.splits CTAs per C tile; CTA r of the cluster multiplies the K
// stages [r k_iters / S, (r + 1) k_iters / S) into its TMEM accumulator with the same
// loader / MMA roles as above.  The epilogue warps then park the fp32 partial tile in the
// CTA's own shared memory (over the ring, which is idle by then), rows 128 B-swizzled in
// 16-byte chunks; after a cluster barrier CTA r sums rows [r 128 / S, (r + 1) 128 / S)
// over the S partials in the order s = 0 .. S - 1, reading its peers' shared memory,
// and stores them as bf16.  A second cluster barrier keeps every partial alive until all
// peers have read it.  The summation order does not depend on timing, so the result is
// deterministic for a given S.
template <int BN, bool BK_MAJOR>
__global__ void __launch_bounds__(GemmCfg<BN>::SPLIT_THREADS, 1)
    gemm_splitk_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                       const GemmParams p) {
  using C = GemmCfg<BN>;
  constexpr uint32_t kCols = BN <= 64 ? 64 : BN <= 128 ? 128 : 256;  // one accumulator
  constexpr uint32_t kRowBytes = BN * 4;                                // fp32 partial row
  static_assert(C::BM * kRowBytes <= C::STG_OFF, "the partial tile fits in the ring");
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_base = smem_u32(smem_raw);
  const uint32_t sbase = (raw_base + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (sbase - raw_base);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const uint32_t bar_full = sbase + C::BAR_OFF;
  const uint32_t bar_empty = bar_full + 8 * C::NSTAGE;
  const uint32_t bar_acc = bar_empty + 8 * C::NSTAGE;  // accumulator complete
  const uint32_t bar_drain = bar_acc + 32;
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::TMEM_PTR_OFF);
  Abort ab{reinterpret_cast<volatile int*>(smem + C::ABORT_OFF)};

  const int S = p.splits;
  const uint32_t rank = cluster_ctarank();
  const int tile = static_cast<int>(blockIdx.x) / S;
  int tm, tn;
  tile_coords(p, tile, tm, tn);
  const int k0 = static_cast<int>(static_cast<long long>(p.k_iters) * rank / S);
  const int k1 = static_cast<int>(static_cast<long long>(p.k_iters) * (rank + 1) / S);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    mbar_init(bar_acc, 1);
    mbar_init(bar_drain, 1);
    *ab.flag = 0;
    *(ab.flag + 1) = 0;
    fence_barrier_init();
  }
  if (warp == 5) tmem_alloc(smem_u32(tmem_ptr), kCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_ptr;
  // Launched as a programmatic dependent of the previous kernel in the stream: the set-up
  // above touches no global memory; from here on that kernel's writes must be complete
  // and visible, and the next launch may start its own set-up.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;");

  if (warp == 4) {
    // ------------------------------------------------------------------ loader
    if (lane == 0) {
      prefetch_tensormap(&tm_a);
      prefetch_tensormap(&tm_b);
      int issued = 0, skipped = -1;
      for (int ks = k0, it = 0; ks < k1; ++ks, ++it) {
        const int s = it % C::NSTAGE;
        if (!mbar_wait(bar_empty + 8 * s, ((it / C::NSTAGE) & 1) ^ 1, p.ctl, ab)) break;
        issued = it + 1;
        if (p.ctl.inject == 3 && it == 2) {  // test hook: never load this stage
          skipped = it;
          continue;
        }
        const uint32_t dst = sbase + s * C::STAGE_BYTES;
        mbar_expect_tx(bar_full + 8 * s, C::STAGE_BYTES);
        tma_load_3d(dst, &tm_a, ks * C::BK, tm * C::BM, 0, bar_full + 8 * s);
        if constexpr (BK_MAJOR) {
          tma_load_3d(dst + C::A_BYTES, &tm_b, ks * C::BK, tn * BN, 0, bar_full + 8 * s);
        } else if (p.b_blocks) {
          tma_load_3d(dst + C::A_BYTES, &tm_b, 0, ks * C::BK, tn * C::NB, bar_full + 8 * s);
        } else {
#pragma unroll
          for (int x = 0; x < C::NB; ++x)
            tma_load_3d(dst + C::A_BYTES + x * C::B_BOX_BYTES, &tm_b, tn * BN + x * 64, ks * C::BK, 0,
                        bar_full + 8 * s);
        }
      }
      Abort no_abort{ab.flag + 1};
      for (int i = max(0, issued - C::NSTAGE); i < issued; ++i)
        if (i != skipped) mbar_wait(bar_full + 8 * (i % C::NSTAGE), (i / C::NSTAGE) & 1, p.ctl, no_abort);
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------------ MMA issuer
    {  // the whole warp runs this role; one elected lane issues
      constexpr uint32_t idesc = idesc_bf16(C::BM, BN, 0, BK_MAJOR ? 0 : 1);
      constexpr uint32_t kstep_b = BK_MAJOR ? 2u : 128u;
      const uint64_t da0 = sdesc_sw128(sbase, 16, 1024);
      const uint64_t db0 = sdesc_sw128(sbase + C::A_BYTES, BK_MAJOR ? 16u : C::B_BOX_BYTES, 1024);
      constexpr uint32_t kStage16 = C::STAGE_BYTES >> 4;
      bool ok = true;
      for (int ks = k0, it = 0; ks < k1; ++ks, ++it) {
        const int s = it % C::NSTAGE;
        if (!(ok = mbar_wait_warp(bar_full + 8 * s, (it / C::NSTAGE) & 1, p.ctl, ab))) break;
        tc_fence_after();
        const uint64_t da = da0 + s * kStage16, db = db0 + s * kStage16;
#pragma unroll
        for (int kk = 0; kk < C::BK / 16; ++kk)
          mma_ss_el(tmem, da + kk * 2, db + kk * kstep_b, idesc, (it > 0 || kk > 0) ? 1u : 0u);
        tc_commit_el(bar_empty + 8 * s);
      }
      if (ok) tc_commit_el(bar_acc);  // with no stages at all this arrives at once
      Abort no_abort{ab.flag + 1};
      tc_commit_el(bar_drain);
      mbar_wait_warp(bar_drain, 0, p.ctl, no_abort);
    }
  } else {
    // ------------------------------------------------------------------ partial tile -> smem
    const int row = warp * 32 + lane;
    const uint32_t prow = sbase + static_cast<uint32_t>(row) * kRowBytes;
    if (mbar_wait_warp(bar_acc, 0, p.ctl, ab)) {
      tc_fence_after();
      fence_proxy_async_smem();  // the ring's last TMA writes and MMA reads are complete
      const uint32_t src = tmem + (static_cast<uint32_t>(warp * 32) << 16);
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        uint32_t r[32];
        if (k1 > k0) {
          tmem_ld32(src + c * 32, r);
          tmem_wait_ld();
          reg_fence32(r);
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) r[i] = 0u;
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const uint32_t chunk = static_cast<uint32_t>(c * 8 + q) ^ static_cast<uint32_t>(row & 7);
          st_shared_v4(prow + chunk * 16u, r[4 * q], r[4 * q + 1], r[4 * q + 2], r[4 * q + 3]);
        }
      }
    }
  }

  __syncwarp();
  cluster_sync_all();  // every partial tile is in its CTA's shared memory

  if (warp < 4 && !ab.raised()) {
    // ------------------------------------------------------------------ reduce rows, store
    const int rows = C::BM / S;
    constexpr int kChunks = BN / 4;  // 16-byte chunks of a partial row
    const int r_first = static_cast<int>(rank) * rows;
    for (int i = threadIdx.x; i < rows * kChunks; i += 128) {
      const int r = r_first + i / kChunks, j = i % kChunks;
      const uint32_t off = static_cast<uint32_t>(r) * kRowBytes + ((static_cast<uint32_t>(j) ^ (r & 7)) << 4);
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int s = 0; s < S; ++s) {
        const float4 v = ld_dsmem_f4(map_shared_rank(sbase + off, static_cast<uint32_t>(s)));
        acc.x += v.x;
        acc.y += v.y;
        acc.z += v.z;
        acc.w += v.w;
      }
      const int grow = tm * C::BM + r, gcol = tn * BN + j * 4;
      if (grow < p.M && gcol < p.N) {  // N % 8 == 0: the 4 columns are all inside C
        uint2 w;
        w.x = pack_bf16x2(acc.x, acc.y);
        w.y = pack_bf16x2(acc.z, acc.w);
        *reinterpret_cast<uint2*>(p.c + static_cast<size_t>(grow) * p.N + gcol) = w;
      }
    }
  }

  __syncwarp();
  cluster_sync_all();  // no CTA leaves while a peer may still read its partial
  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    tmem_dealloc(tmem, kCols);
  }
}

// ---------------------------------------------------------------- CTA-pair tiles
// A cluster of two CTAs (a CTA pair) computes 256 x 256 tiles of C with
// tcgen05.mma.cta_group::2 (M = 256, N = 256, issued by the even CTA): each CTA holds its
// own 128 rows of A and one half (128 columns) of B per K stage, and its TMEM receives
// its 128 rows x 256 columns of the accumulator.  Per K stage an SM thus loads 32 KB
// instead of the 48 KB of a 128 x 256 single-CTA tile, and six stages fit.  Both CTAs'
// copies complete on the even CTA's full barrier (armed once for 64 KB); the even CTA's
// commits signal stage-free and accumulator-ready on both CTAs at once; each CTA's eight
// epilogue warps tell the even CTA that an accumulator has been read (16 arrivals).
template <int NS = 6>
struct GemmPairCfgT {
  static constexpr int BM = 128, BN = 256, BK = 64;   // per CTA: 128 rows x 256 columns of C
  static constexpr int NSTAGE = NS;                    // 6: the model's depth (the deepest that fits)
  static constexpr int THREADS = 320;                  // 8 epilogue warps, loader, MMA
  static constexpr int NBH = 2;                        // 64-column boxes of this CTA's half of B
  static constexpr uint32_t A_BYTES = BM * BK * 2;
  static constexpr uint32_t B_BOX_BYTES = BK * 64 * 2;
  static constexpr uint32_t STAGE_BYTES = A_BYTES + NBH * B_BOX_BYTES;  // 32 KB
  static constexpr uint32_t STG_OFF = NSTAGE * STAGE_BYTES;
  static constexpr uint32_t STG_WARP = 32 * 128;
  static constexpr uint32_t BAR_OFF = STG_OFF + 8 * STG_WARP;
  static constexpr int NBAR = 2 * NSTAGE + 5;  // full, empty, acc_full[2], acc_empty[2], drain
  static constexpr uint32_t TMEM_PTR_OFF = BAR_OFF + NBAR * 8;
  static constexpr uint32_t ABORT_OFF = TMEM_PTR_OFF + 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16 + 1024;
  static constexpr uint32_t TMEM_COLS = 512;  // two accumulators of 256 columns
  static_assert(BYTES <= 227 * 1024, "shared memory budget");
};
using GemmPairCfg = GemmPairCfgT<6>;

__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst, uint32_t ncols) {
  // one warp of each CTA of the pair, together: the same columns in both SMs
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// 3-D TMA load into this CTA's shared memory completing on `bar`, which may be the peer
// CTA's barrier (a shared::cluster address).
__device__ __forceinline__ void tma_load_3d_pair(uint32_t dst, const CUtensorMap* map, int x, int y, int z,
                                                 uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, "
      "{%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar)
      : "memory");
}
// The pair MMA and its commits, executed by the whole issuing warp with one elected lane
// issuing (see mma_ss_el).
__device__ __forceinline__ void mma_ss_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p, e;\n\tsetp.ne.b32 p, %4, 0;\n\telect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on the barrier at the same offset in both CTAs of the pair once the MMAs issued
// so far have completed.
__device__ __forceinline__ void tc_commit_pair_both(uint32_t bar) {
  asm volatile(
      "{\n\t.reg .pred e;\n\telect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;\n\t}" ::"r"(bar),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}
__device__ __forceinline__ void tc_commit_pair(uint32_t bar) {
  asm volatile(
      "{\n\t.reg .pred e;\n\telect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(bar)
      : "memory");
}

// Work unit u of the pair kernel: a whole 256 x 256 tile, or (u >= p.narrow_from) one
// 256 x 128 half of one of the tiles of the last, thinly filled round.  Its tiles are then
// halved along N, so twice as many pairs take them and the round takes about half as long
// (no partial sums to combine: the halves are different columns of C).
struct PairUnit {
  int tm, col0;  // 256-row tile index, first column of C
  bool narrow;
};
__device__ __forceinline__ PairUnit pair_unit(const GemmParams& p, int u) {
  PairUnit w;
  int t = u, half = 0;
  w.narrow = u >= p.narrow_from;
  if (w.narrow) {
    const int v = u - p.narrow_from;
    t = p.narrow_from + (v >> 1);
    half = v & 1;
  }
  int tn;
  tile_coords(p, t, w.tm, tn);
  w.col0 = tn * 256 + half * 128;
  return w;
}

// tm_bn: B for a narrow unit's stage, this CTA's 64 columns (K-major: 64 rows of B [N, K];
// B [K, N] as 64-column blocks: one block; otherwise tm_b's own 64 x 64 box).
template <bool BK_MAJOR, int NS = 6>
__global__ void __launch_bounds__(GemmPairCfgT<NS>::THREADS, 1)
    gemm_pair_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                     const __grid_constant__ CUtensorMap tm_c, const __grid_constant__ CUtensorMap tm_bn,
                     const GemmParams p) {
  using C = GemmPairCfgT<NS>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_base = smem_u32(smem_raw);
  const uint32_t sbase = (raw_base + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (sbase - raw_base);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();  // 0: issues the MMAs; 1: its peer
  const int pair = static_cast<int>(blockIdx.x) >> 1, n_pairs = static_cast<int>(gridDim.x) >> 1;

  const uint32_t bar_full = sbase + C::BAR_OFF;
  const uint32_t bar_empty = bar_full + 8 * C::NSTAGE;
  const uint32_t bar_acc = bar_empty + 8 * C::NSTAGE;
  const uint32_t bar_acce = bar_acc + 16;
  const uint32_t bar_drain = bar_acce + 16;
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::TMEM_PTR_OFF);
  Abort ab{reinterpret_cast<volatile int*>(smem + C::ABORT_OFF)};
  const int units = p.n_units;  // whole tiles, then narrow halves

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar_acc + 8 * b, 1);
      mbar_init(bar_acce + 8 * b, 16);  // 8 epilogue warps x 2 CTAs
    }
    mbar_init(bar_drain, 1);
    *ab.flag = 0;
    *(ab.flag + 1) = 0;
    fence_barrier_init();
  }
  if (warp == 9) tmem_alloc_pair(smem_u32(tmem_ptr), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers initialised, TMEM allocated in both
  tc_fence_after();
  const uint32_t tmem = *tmem_ptr;
  // Launched as a programmatic dependent of the previous kernel in the stream: the set-up
  // above touches no global memory; from here on that kernel's writes must be complete
  // and visible, and the next launch may start its own set-up on SMs this grid frees.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;");

  if (warp == 8) {
    // ------------------------------------------------------------------ loader (both CTAs)
    if (lane == 0) {
      prefetch_tensormap(&tm_a);
      prefetch_tensormap(&tm_b);
      prefetch_tensormap(&tm_bn);
      int it = 0, issued = 0, skipped = -1, lt = 0;
      bool ok = true;
      for (int t = pair; ok && t < units; t += n_pairs, ++lt) {
        const PairUnit w = pair_unit(p, t);
        const int tm = w.tm;
        const int bcol = w.col0 + static_cast<int>(rank) * (w.narrow ? 64 : 128);  // this CTA's B columns
        const bool back = p.k_alt && (lt & 1);
        for (int kq = 0; kq < p.k_iters; ++kq, ++it) {
          const int ks = back ? p.k_iters - 1 - kq : kq;
          const int s = it % C::NSTAGE;
          if (!(ok = mbar_wait(bar_empty + 8 * s, ((it / C::NSTAGE) & 1) ^ 1, p.ctl, ab))) break;
          issued = it + 1;
          if (p.ctl.inject == 3 && it == 2 && rank == 0) {  // test hook: never arm this stage
            skipped = it;
            continue;
          }
          const uint32_t full0 = map_shared_rank(bar_full + 8 * s, 0);  // the even CTA's barrier
          if (rank == 0)
            mbar_expect_tx(bar_full + 8 * s, 2 * (w.narrow ? C::A_BYTES + C::B_BOX_BYTES : C::STAGE_BYTES));
          const uint32_t dst = sbase + s * C::STAGE_BYTES;
          tma_load_3d_pair(dst, &tm_a, ks * C::BK, tm * 256 + static_cast<int>(rank) * C::BM, 0, full0);
          if (w.narrow) {  // this CTA's 64 columns of B: one box
            if constexpr (BK_MAJOR) {
              tma_load_3d_pair(dst + C::A_BYTES, &tm_bn, ks * C::BK, bcol, 0, full0);
            } else if (p.b_blocks) {
              tma_load_3d_pair(dst + C::A_BYTES, &tm_bn, 0, ks * C::BK, bcol / 64, full0);
            } else {
              tma_load_3d_pair(dst + C::A_BYTES, &tm_bn, bcol, ks * C::BK, 0, full0);
            }
          } else if constexpr (BK_MAJOR) {  // this CTA's 128 rows of B [N, K], 64 K-columns: one box
            tma_load_3d_pair(dst + C::A_BYTES, &tm_b, ks * C::BK, bcol, 0, full0);
          } else if (p.b_blocks) {  // both 64-column blocks of this CTA's half in one box
            tma_load_3d_pair(dst + C::A_BYTES, &tm_b, 0, ks * C::BK, bcol / 64, full0);
          } else {
#pragma unroll
            for (int x = 0; x < C::NBH; ++x)
              tma_load_3d_pair(dst + C::A_BYTES + x * C::B_BOX_BYTES, &tm_b, bcol + x * 64, ks * C::BK, 0, full0);
          }
        }
      }
      if (rank == 0) {  // the even CTA's barriers count both CTAs' copies
        Abort no_abort{ab.flag + 1};
        for (int i = max(0, issued - C::NSTAGE); i < issued; ++i)
          if (i != skipped) mbar_wait(bar_full + 8 * (i % C::NSTAGE), (i / C::NSTAGE) & 1, p.ctl, no_abort);
      }
    }
  } else if (warp == 9) {
    // ------------------------------------------------------------------ MMA issuer (even CTA)
    if (rank == 0) {  // the whole warp; one elected lane issues
      constexpr uint32_t idesc = idesc_bf16(256, C::BN, 0, BK_MAJOR ? 0 : 1);
      constexpr uint32_t idesc_n = idesc_bf16(256, C::BN / 2, 0, BK_MAJOR ? 0 : 1);  // narrow units
      constexpr uint32_t kstep_b = BK_MAJOR ? 2u : 128u;
      const uint64_t da0 = sdesc_sw128(sbase, 16, 1024);
      const uint64_t db0 = sdesc_sw128(sbase + C::A_BYTES, BK_MAJOR ? 16u : C::B_BOX_BYTES, 1024);
      constexpr uint32_t kStage16 = C::STAGE_BYTES >> 4;
      int it = 0, lt = 0;
      bool ok = true;
      for (int t = pair; ok && t < units; t += n_pairs, ++lt) {
        const int b = lt & 1, use = lt >> 1;
        const uint32_t id = t >= p.narrow_from ? idesc_n : idesc;
        if (lt >= 2 && !(ok = mbar_wait_cluster_warp(bar_acce + 8 * b, (use - 1) & 1, p.ctl, ab))) break;
        tc_fence_after();
        const uint32_t d = tmem + static_cast<uint32_t>(b * C::BN);
        for (int ks = 0; ks < p.k_iters; ++ks, ++it) {
          const int s = it % C::NSTAGE;
          if (!(ok = mbar_wait_warp(bar_full + 8 * s, (it / C::NSTAGE) & 1, p.ctl, ab))) break;
          tc_fence_after();
          const uint64_t da = da0 + s * kStage16, db = db0 + s * kStage16;
#pragma unroll
          for (int kk = 0; kk < C::BK / 16; ++kk)
            mma_ss_pair(d, da + kk * 2, db + kk * kstep_b, id, (ks > 0 || kk > 0) ? 1u : 0u);
          tc_commit_pair_both(bar_empty + 8 * s);
        }
        if (!ok) break;
        tc_commit_pair_both(bar_acc + 8 * b);
      }
      Abort no_abort{ab.flag + 1};
      tc_commit_pair(bar_drain);
      mbar_wait_warp(bar_drain, 0, p.ctl, no_abort);
    }
  } else {
    // ------------------------------------------------------------------ epilogue (both CTAs, warps 0-7)
    const int quarter = warp & 3, half = warp >> 2;
    const uint32_t lane_addr = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t stg = sbase + C::STG_OFF + static_cast<uint32_t>(warp) * C::STG_WARP;
    int lt = 0;
    bool ok = true;
    for (int t = pair; ok && t < units; t += n_pairs, ++lt) {
      const PairUnit w = pair_unit(p, t);
      const int b = lt & 1, use = lt >> 1;
      if (!(ok = mbar_wait_warp(bar_acc + 8 * b, use & 1, p.ctl, ab))) break;
      tc_fence_after();
      const uint32_t acc = tmem + lane_addr + static_cast<uint32_t>(b * C::BN);
      const int row0 = w.tm * 256 + static_cast<int>(rank) * C::BM + quarter * 32;
      const uint32_t release = map_shared_rank(bar_acce + 8 * b, 0);
      if (w.narrow)
        epilogue_warp<C::BN / 128>(&tm_c, acc, stg, half, w.col0, row0, p.M, p.N, release, true);
      else
        epilogue_warp<C::BN / 64>(&tm_c, acc, stg, half, w.col0, row0, p.M, p.N, release, true);
    }
    if (lane == 0) bulk_wait_group0();
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // the pair's MMAs, copies and TMEM reads are over in both CTAs
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------- host side
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult qres;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &qres) ==
            cudaSuccess &&
        qres == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

// 2-D row-major bf16 matrix [rows, cols] as a 3-D tensor with a unit third dimension.
bool matrix_map(CUtensorMap* map, const void* base, int rows, int cols, int box_cols, int box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows), 1};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(cols) * 2, static_cast<cuuint64_t>(cols) * 2 * rows};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(box_cols), static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Devices whose cluster occupancy answers are cached (others query on every call).
constexpr int kSlotCacheDevices = 64;

template <int BN, int NS = 0>
bool set_smem_attr(const void* fn, PerDeviceOnce& done, int dev) {
  // one opt-in per kernel and device (the flags are per template instance)
  return done.run(dev, [fn] {
    return cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, GemmCfg<BN, NS>::BYTES) ==
           cudaSuccess;
  });
}

// B [K, N] with N % 64 == 0 as a 3-D tensor of 64-column blocks: (column in block, K row,
// block), strides 2 B, 2N B and 128 B; a box of `blocks` blocks x 64 K-rows lands in shared
// memory as `blocks` consecutive 8 KB (64 x 64, 128B-swizzled) blocks.
bool b_blocks_map(CUtensorMap* map, const void* base, int K, int N, int blocks) {
  EncodeTiledFn enc = encode_fn();
  if (!enc || N % 64 != 0) return false;
  cuuint64_t dims[3] = {64, static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(N / 64)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(N) * 2, 128};
  cuuint32_t box[3] = {64, 64, static_cast<cuuint32_t>(blocks)};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// B's box: 64 columns x 64 K-rows of B [K, N], or 64 K-columns x b_rows rows of B [N, K].
bool make_maps(const GemmArgs& a, int bm, int b_rows, CUtensorMap* ma, CUtensorMap* mb, CUtensorMap* mc) {
  const bool b_ok = a.b_kmajor ? matrix_map(mb, a.b, a.N, a.K, 64, b_rows) : matrix_map(mb, a.b, a.K, a.N, 64, 64);
  return matrix_map(ma, a.a, a.M, a.K, 64, bm) && b_ok && (mc == nullptr || matrix_map(mc, a.c, a.M, a.N, 64, 32));
}

GemmParams make_params(const GemmArgs& a, const KernelCtl& ctl, int bn, int splits) {
  GemmParams p;
  p.c = static_cast<__nv_bfloat16*>(a.c);
  p.M = a.M;
  p.N = a.N;
  p.K = a.K;
  p.tiles_m = (a.M + 127) / 128;
  p.tiles_n = (a.N + bn - 1) / bn;
  p.k_iters = (a.K + 63) / 64;
  p.splits = splits;
  p.group = a.group > 0 ? a.group : 8;
  p.k_alt = 0;
  p.b_blocks = 0;
  p.narrow_from = 0x7fffffff;
  p.n_units = 0;
  p.ctl = ctl;
  return p;
}

// B [K, N] with N % 64 == 0: one TMA box per stage for all of a stage's 64-column blocks of
// B instead of one box per block.  Measured on GB300 (CTA pair, 8192^3): 1699 against 1550
// TFLOP/s with two boxes, level with B given [N, K] (1690), whose stage is one box too.
void use_b_blocks(const GemmArgs& a, int blocks, CUtensorMap* mb, GemmParams* p) {
  CUtensorMap m;
  if (!a.b_kmajor && b_blocks_map(&m, a.b, a.K, a.N, blocks)) {
    *mb = m;
    p->b_blocks = 1;
  }
}

template <int BN, bool BKM, int NS = 0>
cudaError_t launch_bn(const GemmArgs& a, const KernelCtl& ctl, cudaStream_t stream, int dev, int sms) {
  using C = GemmCfg<BN, NS>;
  static PerDeviceOnce configured;
  if (!set_smem_attr<BN, NS>(reinterpret_cast<const void*>(gemm_kernel<BN, BKM, NS>), configured, dev))
    return cudaErrorInvalidValue;
  CUtensorMap ma, mb, mc;
  if (!make_maps(a, C::BM, BN, &ma, &mb, &mc)) return cudaErrorInvalidValue;
  GemmParams p = make_params(a, ctl, BN, 1);
  use_b_blocks(a, C::NB, &mb, &p);
  const long long tiles = static_cast<long long>(p.tiles_m) * p.tiles_n;
  if (tiles > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  const int grid = static_cast<int>(tiles < sms ? tiles : sms);
  // a programmatic dependent of the previous kernel (the kernel waits for it after its set-up)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(C::THREADS);
  cfg.dynamicSmemBytes = C::BYTES;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gemm_kernel<BN, BKM, NS>, ma, mb, mc, p);
}

template <int BN>
cudaLaunchConfig_t splitk_config(int grid, int S, cudaStream_t stream, cudaLaunchAttribute* attr,
                                 bool dependent = false) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
  cfg.blockDim = dim3(GemmCfg<BN>::SPLIT_THREADS, 1, 1);
  cfg.dynamicSmemBytes = GemmCfg<BN>::BYTES;
  cfg.stream = stream;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(S);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (dependent) {  // a programmatic dependent of the previous kernel (attr holds two entries)
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.numAttrs = 2;
  }
  return cfg;
}

template <int BN, bool BKM>
bool prepare_splitk(int dev) {
  static PerDeviceOnce configured, nonportable;
  const void* fn = reinterpret_cast<const void*>(gemm_splitk_kernel<BN, BKM>);
  if (!set_smem_attr<BN>(fn, configured, dev)) return false;
  return nonportable.run(dev, [fn] {
    return cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess;
  });
}

// CTAs of clusters of S that fit on the device at once (0: none, or cannot be queried); both
// B layouts have the same resources, so the [K, N] instance answers for both.
template <int BN>
int splitk_slots(int dev, int S) {
  static std::atomic<int> cache[kSlotCacheDevices][5];  // [device][log2 S], value + 1 once known
  int lg = 0;
  while ((1 << lg) < S) ++lg;
  if (dev < 0 || lg > 4 || (1 << lg) != S) return 0;
  const bool cached = dev < kSlotCacheDevices;
  if (cached) {
    const int c = cache[dev][lg].load(std::memory_order_relaxed);
    if (c != 0) return c - 1;
  }
  int clusters = 0;
  if (prepare_splitk<BN, false>(dev)) {
    cudaLaunchAttribute attr[1];
    cudaLaunchConfig_t cfg = splitk_config<BN>(S * 64, S, nullptr, attr);
    if (cudaOccupancyMaxActiveClusters(&clusters, gemm_splitk_kernel<BN, false>, &cfg) != cudaSuccess) {
      cudaGetLastError();
      clusters = 0;
    }
  }
  if (cached) cache[dev][lg].store(clusters * S + 1, std::memory_order_relaxed);
  return clusters * S;
}

int splitk_slots_any(int dev, int bn, int S) {
  switch (bn) {
    case 64: return splitk_slots<64>(dev, S);
    case 128: return splitk_slots<128>(dev, S);
    case 192: return splitk_slots<192>(dev, S);
    default: return splitk_slots<256>(dev, S);
  }
}

template <int BN, bool BKM>
cudaError_t launch_splitk(const GemmArgs& a, const KernelCtl& ctl, cudaStream_t stream, int dev, int S) {
  if (!prepare_splitk<BN, BKM>(dev)) return cudaErrorInvalidValue;
  CUtensorMap ma, mb;
  if (!make_maps(a, GemmCfg<BN>::BM, BN, &ma, &mb, nullptr)) return cudaErrorInvalidValue;
  GemmParams p = make_params(a, ctl, BN, S);
  use_b_blocks(a, GemmCfg<BN>::NB, &mb, &p);
  const long long ctas = static_cast<long long>(p.tiles_m) * p.tiles_n * S;
  if (ctas > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = splitk_config<BN>(static_cast<int>(ctas), S, stream, attr, true);
  return cudaLaunchKernelEx(&cfg, gemm_splitk_kernel<BN, BKM>, ma, mb, p);
}

template <bool BKM, int NS = 6>
bool prepare_pair(int dev) {
  static PerDeviceOnce configured;
  const void* fn = reinterpret_cast<const void*>(gemm_pair_kernel<BKM, NS>);
  return configured.run(dev, [fn] {
    return cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, GemmPairCfgT<NS>::BYTES) ==
           cudaSuccess;
  });
}

template <int NS = 6>
cudaLaunchConfig_t pair_config(int grid, cudaStream_t stream, cudaLaunchAttribute* attr, bool dependent = false) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
  cfg.blockDim = dim3(GemmPairCfgT<NS>::THREADS, 1, 1);
  cfg.dynamicSmemBytes = GemmPairCfgT<NS>::BYTES;
  cfg.stream = stream;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (dependent) {  // a programmatic dependent of the previous kernel (attr holds two entries)
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.numAttrs = 2;
  }
  return cfg;
}

// CTAs of CTA pairs that fit on the device at once (0: none, or cannot be queried).
int pair_slots(int dev) {
  static std::atomic<int> cache[kSlotCacheDevices];  // value + 1 once known
  if (dev < 0) return 0;
  const bool cached = dev < kSlotCacheDevices;
  if (cached) {
    const int c = cache[dev].load(std::memory_order_relaxed);
    if (c != 0) return c - 1;
  }
  int clusters = 0;
  if (prepare_pair<false>(dev)) {
    cudaLaunchAttribute attr[1];
    cudaLaunchConfig_t cfg = pair_config(128, nullptr, attr);
    if (cudaOccupancyMaxActiveClusters(&clusters, gemm_pair_kernel<false>, &cfg) != cudaSuccess) {
      cudaGetLastError();
      clusters = 0;
    }
  }
  if (cached) cache[dev].store(2 * clusters + 1, std::memory_order_relaxed);
  return 2 * clusters;
}

template <bool BKM, int NS = 6>
cudaError_t launch_pair(const GemmArgs& a, const KernelCtl& ctl, cudaStream_t stream, int dev) {
  const int slots = pair_slots(dev);
  if (slots < 2 || !prepare_pair<BKM, NS>(dev)) return cudaErrorInvalidConfiguration;
  CUtensorMap ma, mb, mc;
  if (!make_maps(a, GemmPairCfg::BM, 128, &ma, &mb, &mc)) return cudaErrorInvalidValue;
  GemmParams p = make_params(a, ctl, GemmPairCfg::BN, 1);
  p.tiles_m = (a.M + 255) / 256;  // 256-row tiles of the pair
  // 76 pairs in flight cover 12 tile rows x 6-7 tile columns; with every other round
  // walking K backwards, a round starts on the K slices of A the previous round (same rows)
  // read last.  GB300, 8192^3: 812 MB read from DRAM against 1064 MB in groups of 8 rows
  // walked forwards (A + B: 268 MB; cuBLAS 1005-1020 MB), time within 1 %.
  if (a.group <= 0) p.group = 12;
  p.k_alt = a.k_alt >= 0 ? 1 : 0;
  use_b_blocks(a, GemmPairCfg::NBH, &mb, &p);
  const long long tiles = static_cast<long long>(p.tiles_m) * p.tiles_n;
  if (tiles > 0x3fffffffLL) return cudaErrorInvalidConfiguration;
  // The last round's tiles become two 256 x 128 units each when that round would keep at
  // most a quarter of the pairs busy.  GB300, same-box A/B: 2304^2 x 8192 (5 of 76 pairs in
  // the last round) 941 -> 1066-1081 TFLOP/s; with a third or more of the pairs busy the
  // halves lost 1-3 % (4096^3: 28 pairs, 8192^3: 36): a wide tile in a thinly filled round
  // runs faster than in a full one.
  const long long avail = slots / 2;
  const long long rest = tiles % avail;
  p.narrow_from = static_cast<int>(tiles);
  p.n_units = static_cast<int>(tiles);
  CUtensorMap mbn = mb;  // narrow units' B: one 64-column box per CTA
  if (rest > 0 && 4 * rest <= avail) {
    bool ok = true;
    if (BKM) ok = matrix_map(&mbn, a.b, a.N, a.K, 64, 64);
    else if (p.b_blocks) ok = b_blocks_map(&mbn, a.b, a.K, a.N, 1);
    if (ok) {
      p.narrow_from = static_cast<int>(tiles - rest);
      p.n_units = static_cast<int>(tiles + rest);
    }
  }
  const long long pairs = p.n_units < avail ? p.n_units : avail;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = pair_config<NS>(static_cast<int>(2 * pairs), stream, attr, true);
  return cudaLaunchKernelEx(&cfg, gemm_pair_kernel<BKM, NS>, ma, mb, mc, mbn, p);
}

// Ring depths compiled beside the model's for the block-size ablation ([K, N] B only): the
// CTA pair with 5 stages (model: 6), persistent 256-wide tiles with 3 (model: 4), 128-wide
// tiles with 5 (model: 6); the deeper neighbours do not fit in shared memory.
bool gemm_stages_compiled(const GemmChoice& c, int stages) {
  if (c.pair == 1) return stages == 5;
  if (c.splits > 1) return false;
  return (c.tile_n == 256 && stages == 3) || (c.tile_n == 128 && stages == 5);
}

cudaError_t launch_ablation(const GemmArgs& a, const GemmChoice& c, const KernelCtl& ctl, cudaStream_t stream,
                            int dev, int sms) {
  if (c.pair == 1) return launch_pair<false, 5>(a, ctl, stream, dev);
  if (c.tile_n == 256) return launch_bn<256, false, 3>(a, ctl, stream, dev, sms);
  return launch_bn<128, false, 5>(a, ctl, stream, dev, sms);
}

template <bool BKM>
cudaError_t launch_choice(const GemmArgs& a, const GemmChoice& c, const KernelCtl& ctl, cudaStream_t stream, int dev,
                          int sms) {
  if (c.pair == 1) return launch_pair<BKM>(a, ctl, stream, dev);
  if (c.splits > 1) {
    switch (c.tile_n) {
      case 64: return launch_splitk<64, BKM>(a, ctl, stream, dev, c.splits);
      case 128: return launch_splitk<128, BKM>(a, ctl, stream, dev, c.splits);
      case 192: return launch_splitk<192, BKM>(a, ctl, stream, dev, c.splits);
      default: return launch_splitk<256, BKM>(a, ctl, stream, dev, c.splits);
    }
  }
  switch (c.tile_n) {
    case 64: return launch_bn<64, BKM>(a, ctl, stream, dev, sms);
    case 128: return launch_bn<128, BKM>(a, ctl, stream, dev, sms);
    case 192: return launch_bn<192, BKM>(a, ctl, stream, dev, sms);
    default: return launch_bn<256, BKM>(a, ctl, stream, dev, sms);
  }
}

bool device_sms(int* dev, int* sms) {
  if (cudaGetDevice(dev) != cudaSuccess) return false;
  return cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, *dev) == cudaSuccess && *sms > 0;
}

}  // namespace

GemmChoice gemm_choice(int M, int N, int K, GemmChoice forced) {
  int dev = 0, sms = 0;
  if (!device_sms(&dev, &sms)) return {0, 0};
  const model::GemmChoiceModel c = model::gemm_choose(
      M, N, K, sms, [dev](int bn, int S) { return splitk_slots_any(dev, bn, S); }, model::kGb300, forced.tile_n,
      forced.splits, forced.pair >= 0 ? pair_slots(dev) : 0, forced.pair);
  return {c.bn, c.splits, c.pair ? 1 : 0};
}

cudaError_t launch_gemm(const GemmArgs& a, const KernelCtl& ctl, cudaStream_t stream) {
  int dev = 0, sms = 0;
  if (!device_sms(&dev, &sms)) return cudaErrorNoDevice;
  const GemmChoice c = gemm_choice(a.M, a.N, a.K, {a.tile_n, a.splits, a.pair});
  if (c.tile_n == 0) return cudaErrorInvalidConfiguration;
  if (a.stages > 0 && !a.b_kmajor && gemm_stages_compiled(c, a.stages))
    return launch_ablation(a, c, ctl, stream, dev, sms);
  return a.b_kmajor ? launch_choice<true>(a, c, ctl, stream, dev, sms)
                    : launch_choice<false>(a, c, ctl, stream, dev, sms);
}

}  // namespace loom
