// Flash Decode for GB300: split-KV partial attention + log-sum-exp merge.
//
// Paper: Sec. 2.6 (the Flash Decode HEG is a sequential composition of a local
// softmax loop, a gather of partial results, a global softmax and a final scaling) and
// Sec. 3.2.3 (the sequence axis, the reduction axis, is split across cores).
//
// Kernel 1, decode_split_kernel -- one CTA per (split, kv head, head group, batch):
//   * a loader warp streams the split's K and V rows with 1-D bulk copies
//     (cp.async.bulk, 16 KB per tile) into an NSTAGE-deep shared-memory ring guarded by
//     full/empty mbarriers, so that 2 CTAs x 3 stages x 32 KB are in flight per SM;
//     with a paged cache it reads the sequence's block table 32 entries at a time (one
//     per lane) and lane j copies the stage's j-th page piece with a 3-D TMA load of
//     the cache viewed as [keys of all pages, Hkv, D];
//   * 8 compute warps each take T/8 tokens of every stage; they read K rows with
//     128-bit shared loads, form the scores of all GT query heads of the kv head at
//     once (fp32 FMA), reduce them across lanes with a transposing butterfly, run an
//     online softmax in base 2 with a lazily rescaled running max, and accumulate P.V;
//   * the 8 warps' states are merged in shared memory into the split's normalised
//     partial O_i (fp32) and lse_i (natural log) in the workspace.
// Kernel 2, decode_merge_kernel -- one CTA per (batch, query head): L = max_i lse_i,
//   w_i = exp(lse_i - L), O = sum w_i O_i / sum w_i -> bf16, lse = L + ln sum w_i.
//   It is launched with programmatic dependent launch so its launch overlaps the
//   split kernel's tail.
// Single-kernel form (FUSED instantiation of kernel 1, at most 16 splits): the splits of
// one (batch, kv head, head group) are one thread-block cluster.  Each CTA keeps its
// partial (O_i, lse_i) in its own shared memory; after a cluster barrier CTA r gathers
// outputs [r n / splits, (r + 1) n / splits) of the unit's n = heads x D outputs from
// all the cluster's CTAs over distributed shared memory (in the order i = 0 .. splits-1,
// so the result does not depend on timing), applies the global softmax and the final
// scaling, and writes O (bf16) and LSE; a second cluster barrier keeps every partial
// alive until all peers have read it.  No workspace, no second launch.
#include <cuda.h>
#include <cuda_bf16.h>

#include <atomic>
#include <cmath>
#include <cstring>
#include <mutex>

#include "kernels.h"
#include "model.h"
#include "paged.h"
#include "ptx.cuh"

namespace loom {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
// Lazy rescaling: the running max of a head is only moved when the new tile max
// exceeds it by more than this many base-2 units; P stays <= 2^8, exact in fp32.
constexpr float kRescaleThreshold = 8.0f;

// Stage constants: the analytic model's choice for this head dimension.
template <int D>
struct DecodeCfg {
  static constexpr model::DecodeStagePlan kPlan = model::decode_stage_plan(D);
  static_assert(kPlan.feasible, "no feasible decode stage plan");
  static constexpr int T = kPlan.tokens;           // tokens per stage
  static constexpr int NSTAGE = kPlan.stages;
  static constexpr int CTAS_PER_SM = kPlan.ctas_per_sm;
  static constexpr int NCW = 8;                    // compute warps
  static constexpr int THREADS = (NCW + 1) * 32;   // + loader warp
  static constexpr int TW = T / NCW;               // tokens per warp per stage
  static constexpr int KL = D / 8;                 // lanes per K row (8 dims = 16 B each)
  static constexpr int TPR = 32 / KL;              // tokens per 128-bit load round
  static constexpr int KROUNDS = TW / TPR;
  static constexpr int VD = D / 32;                // dims per lane in the P.V phase
  static constexpr uint32_t TILE_BYTES = T * D * 2;
  static constexpr uint32_t STAGE_BYTES = 2 * TILE_BYTES;
  static constexpr uint32_t RING_BYTES = NSTAGE * STAGE_BYTES;
  static_assert(TW % TPR == 0, "whole 128-bit load rounds per warp");
};

template <int D, int GT, bool FUSED = false>
struct DecodeSmem {
  using C = DecodeCfg<D>;
  // ring first (16-byte aligned bulk-copy destinations), then the small arrays
  static constexpr uint32_t P_OFF = C::RING_BYTES;                      // [NCW][TW][GT] f32
  static constexpr uint32_t ALPHA_OFF = P_OFF + C::NCW * C::TW * GT * 4;  // [NCW][GT] f32
  static constexpr uint32_t WM_OFF = ALPHA_OFF + C::NCW * GT * 4;       // [NCW][GT] f32
  static constexpr uint32_t WL_OFF = WM_OFF + C::NCW * GT * 4;          // [NCW][GT] f32
  // single-kernel form: the CTA's partial, read by the cluster's CTAs over DSMEM
  static constexpr uint32_t PART_O_OFF = (WL_OFF + C::NCW * GT * 4 + 15) / 16 * 16;  // [GT][D] f32
  static constexpr uint32_t PART_L_OFF = PART_O_OFF + (FUSED ? GT * D * 4 : 0);      // [GT] f32
  static constexpr uint32_t BAR_OFF = ((PART_L_OFF + (FUSED ? GT * 4 : 0)) + 7) / 8 * 8;
  static constexpr uint32_t ABORT_OFF = BAR_OFF + 2 * C::NSTAGE * 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16;
  // the cross-warp merge reuses the ring: [NCW][GT][D] f32
  static_assert(C::NCW * GT * D * 4 <= C::RING_BYTES, "merge buffer must fit in the ring");
};

// Sum over the KL lanes of a K row of the GT per-head partial dot products.  Each
// butterfly level halves the number of live values (the "transposing" levels) until
// one is left, so lane l ends up holding the full sum for head head_of_lane(l).
template <int KL, int GT>
__device__ __forceinline__ float transpose_reduce(float (&acc)[GT], int lane) {
  static_assert(GT <= KL, "more heads than lanes per row");
#pragma unroll
  for (int off = KL / 2, n = GT; off >= 1; off >>= 1) {
    if (n > 1) {
      const int half = n >> 1;
      const bool upper = (lane & off) != 0;
#pragma unroll
      for (int i = 0; i < GT / 2; ++i) {
        if (i < half) {
          const float send = upper ? acc[i] : acc[i + half];
          const float keep = upper ? acc[i + half] : acc[i];
          acc[i] = keep + __shfl_xor_sync(0xffffffffu, send, off);
        }
      }
      n = half;
    } else {
      acc[0] += __shfl_xor_sync(0xffffffffu, acc[0], off);
    }
  }
  return acc[0];
}

template <int KL, int GT>
__device__ __forceinline__ int head_of_lane(int lane) {
  int h = 0;
#pragma unroll
  for (int off = KL / 2, n = GT; off >= 1 && n > 1; off >>= 1, n >>= 1)
    if (lane & off) h += n >> 1;
  return h;
}

// Where a paged split kernel finds its keys (unused by the contiguous instantiation).
struct PagedView {
  const int32_t* block_table;
  int page_size, max_pages;
  int num_pages;
  int hnd;  // 1: [num_pages, Hkv, page_size, D]; 0: [num_pages, page_size, Hkv, D]
};

// Gather, global softmax and final scaling of one unit's partials across its cluster (the
// single-kernel form), run by every thread of every CTA of the cluster: the partials
// (part_o [GT][D], part_l [GT] at these shared-memory offsets) of all `splits` CTAs are
// complete after the first barrier; CTA r combines its share of the nh x D outputs, reading
// each split i = 0 .. splits-1 in order; the second barrier keeps the partials alive until
// every peer has read them.  o_row0 = row of O (and index of LSE) of the unit's first head.
template <int D>
__device__ __forceinline__ void cluster_gather(uint32_t part_o, uint32_t part_l, int nh, int splits,
                                               __nv_bfloat16* __restrict__ o, float* __restrict__ lse,
                                               size_t o_row0) {
  cluster_sync_all();
  const int total = nh * D;
  const int per = (total + splits - 1) / splits;
  const int e0 = static_cast<int>(cluster_ctarank()) * per;
  const int e1 = min(total, e0 + per);
  for (int e = e0 + static_cast<int>(threadIdx.x); e < e1; e += static_cast<int>(blockDim.x)) {
    const int h = e / D, d = e % D;
    float l[model::kMaxFusedSplits];
    float M = -INFINITY;
#pragma unroll
    for (int i = 0; i < model::kMaxFusedSplits; ++i) {
      l[i] = i < splits ? ld_dsmem_f32(map_shared_rank(part_l + 4u * h, i)) : -INFINITY;
      M = fmaxf(M, l[i]);
    }
    float W = 0.f, acc = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int i = 0; i < model::kMaxFusedSplits; ++i) {
        if (i < splits) {
          const float w = ex2((l[i] - M) * kLog2e);  // 0 for empty splits
          W += w;
          acc = fmaf(w, ld_dsmem_f32(map_shared_rank(part_o + 4u * e, i)), acc);
        }
      }
    }
    const bool any = W > 0.f;
    o[(o_row0 + h) * D + d] = __float2bfloat16_rn(any ? acc / W : 0.f);
    if (lse && d == 0) lse[o_row0 + h] = any ? M + log2f(W) * kLn2 : -INFINITY;
  }
  cluster_sync_all();
}

template <int D, int GT, bool PAGED, bool FUSED>
__global__ void __launch_bounds__(DecodeCfg<D>::THREADS, DecodeCfg<D>::CTAS_PER_SM)
    decode_split_kernel(const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ k,
                        const __nv_bfloat16* __restrict__ v, const int32_t* __restrict__ seqlens,
                        float* __restrict__ o_part, float* __restrict__ lse_part, int Hq, int Hkv,
                        int Skv, int splits, int n_groups, float c, KernelCtl ctl,
                        const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                        PagedView pv, __nv_bfloat16* __restrict__ o_out, float* __restrict__ lse_out) {
  using C = DecodeCfg<D>;
  using L = DecodeSmem<D, GT, FUSED>;
  extern __shared__ __align__(128) uint8_t smem[];

  // Let the merge grid launch as soon as every split CTA is resident.
  if constexpr (!FUSED) asm volatile("griddepcontrol.launch_dependents;");

  const int split = blockIdx.x;
  const int hk = blockIdx.y / n_groups, grp = blockIdx.y % n_groups;
  const int b = blockIdx.z;
  const int G = Hq / Hkv;
  const int h0 = hk * G + grp * GT;
  const int nh = min(GT, G - grp * GT);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  int len = seqlens ? seqlens[b] : Skv;
  len = max(0, min(len, Skv));
  int chunk = (len + splits - 1) / splits;
  chunk = (chunk + kDecodeChunkAlign - 1) / kDecodeChunkAlign * kDecodeChunkAlign;
  const int t_begin = min(split * chunk, len);
  const int t_end = min(t_begin + chunk, len);
  const size_t row0 = (static_cast<size_t>(b) * Hq + h0) * splits + split;  // head h0's partial
  const uint32_t part_o = smem_u32(smem) + L::PART_O_OFF, part_l = smem_u32(smem) + L::PART_L_OFF;
  const size_t o_row0 = static_cast<size_t>(b) * Hq + h0;  // single-kernel form: first output row

  if (t_begin >= t_end) {  // empty split: contributes nothing to the merge
    if constexpr (FUSED) {
      float* po = reinterpret_cast<float*>(smem + L::PART_O_OFF);
      for (int i = threadIdx.x; i < nh * D; i += blockDim.x) po[i] = 0.f;
      if (threadIdx.x < nh) reinterpret_cast<float*>(smem + L::PART_L_OFF)[threadIdx.x] = -INFINITY;
      cluster_gather<D>(part_o, part_l, nh, splits, o_out, lse_out, o_row0);
    } else {
      for (int i = threadIdx.x; i < nh * D; i += blockDim.x)
        o_part[(row0 + static_cast<size_t>(i / D) * splits) * D + i % D] = 0.f;
      if (threadIdx.x < nh) lse_part[row0 + static_cast<size_t>(threadIdx.x) * splits] = -INFINITY;
    }
    return;
  }
  const int n_stages = (t_end - t_begin + C::T - 1) / C::T;

  const uint32_t s_base = smem_u32(smem);
  const uint32_t bar_full = s_base + L::BAR_OFF;
  const uint32_t bar_empty = bar_full + C::NSTAGE * 8;
  Abort ab{reinterpret_cast<volatile int*>(smem + L::ABORT_OFF)};
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, C::NCW);
    }
    *ab.flag = 0;
    fence_barrier_init();
  }
  __syncthreads();

  const size_t kv_row0 = (static_cast<size_t>(b) * Hkv + hk) * Skv;

  if (warp == C::NCW) {
    // ------------------------------------------------------------ loader warp
    if constexpr (PAGED) {
      static_assert(C::T % kDecodeChunkAlign == 0, "stages start on a copy boundary");
      // Copies of `rows` keys: a 64-key piece of one page (page_size a multiple of 64) or
      // one whole page (page_size 8, 16 or 32).  Stages start on a multiple of 64 keys, so
      // no copy crosses a page; a stage takes at most T / 8 copies.
      const int P = pv.page_size;
      const int rows = P < kDecodeChunkAlign ? P : kDecodeChunkAlign;
      const uint32_t copy_bytes = static_cast<uint32_t>(rows) * D * 2;
      const int32_t* tbl = pv.block_table + static_cast<size_t>(b) * pv.max_pages;
      int win = 0, entry = 0;
      bool have = false;
      int issued = 0, skipped = -1;
      for (int it = 0; it < n_stages; ++it) {
        const int slot = it % C::NSTAGE, round = it / C::NSTAGE;
        if (!mbar_wait_warp(bar_empty + 8 * slot, (round & 1) ^ 1, ctl, ab)) break;
        const int tok0 = t_begin + it * C::T;
        const int ncopy = (min(C::T, t_end - tok0) + rows - 1) / rows;
        const int lp_first = tok0 / P, lp_last = (tok0 + (ncopy - 1) * rows) / P;
        if (!have || lp_first < win || lp_last >= win + 32) {  // refill the table window
          win = lp_first;
          entry = (win + lane < pv.max_pages) ? tbl[win + lane] : 0;
          have = true;
        }
        issued = it + 1;
        if (ctl.inject == 1 && it == 1) {  // test hook: never fill this stage
          skipped = it;
          continue;
        }
        const uint32_t dst = s_base + slot * C::STAGE_BYTES;
        if (lane == 0) mbar_expect_tx(bar_full + 8 * slot, 2u * ncopy * copy_bytes);
        __syncwarp();
        const int t = tok0 + lane * rows;
        const int page = __shfl_sync(0xffffffffu, entry, (t / P - win) & 31);
        if (lane < ncopy) {
          // An out-of-range page (a caller error) is sent past the end of the cache, where
          // the copy engine reads zeros.  NHD view [keys of all pages, Hkv, D]: (0, hk, key);
          // HND view [pages x Hkv, page_size, D]: (0, row in page, page x Hkv + hk).
          const bool bad = page < 0 || page >= pv.num_pages;
          int y, z;
          if (pv.hnd) {
            y = t % P;
            z = bad ? pv.num_pages * Hkv : page * Hkv + hk;
          } else {
            y = hk;
            z = bad ? pv.num_pages * P : page * P + t % P;
          }
          tma_load_3d(dst + lane * copy_bytes, &tm_k, 0, y, z, bar_full + 8 * slot);
          tma_load_3d(dst + C::TILE_BYTES + lane * copy_bytes, &tm_v, 0, y, z, bar_full + 8 * slot);
        }
      }
      if (lane == 0) {
        Abort no_abort{reinterpret_cast<volatile int*>(smem + L::ABORT_OFF + 4)};
        *no_abort.flag = 0;
        for (int it = max(0, issued - C::NSTAGE); it < issued; ++it) {
          if (it == skipped) continue;
          mbar_wait(bar_full + 8 * (it % C::NSTAGE), (it / C::NSTAGE) & 1, ctl, no_abort);
        }
      }
    } else if (lane == 0) {
      int issued = 0, skipped = -1;
      for (int it = 0; it < n_stages; ++it) {
        const int slot = it % C::NSTAGE, round = it / C::NSTAGE;
        if (!mbar_wait(bar_empty + 8 * slot, (round & 1) ^ 1, ctl, ab)) break;
        const int tok0 = t_begin + it * C::T;
        const uint32_t bytes = static_cast<uint32_t>(min(C::T, t_end - tok0)) * D * 2;
        issued = it + 1;
        if (ctl.inject == 1 && it == 1) {  // test hook: never fill this stage
          skipped = it;
          continue;
        }
        const uint32_t dst = s_base + slot * C::STAGE_BYTES;
        mbar_expect_tx(bar_full + 8 * slot, 2 * bytes);
        bulk_g2s(dst, k + (kv_row0 + tok0) * D, bytes, bar_full + 8 * slot);
        bulk_g2s(dst + C::TILE_BYTES, v + (kv_row0 + tok0) * D, bytes, bar_full + 8 * slot);
      }
      // Drain: never leave the CTA with copies still landing in its shared memory.
      Abort no_abort{reinterpret_cast<volatile int*>(smem + L::ABORT_OFF + 4)};
      *no_abort.flag = 0;
      for (int it = max(0, issued - C::NSTAGE); it < issued; ++it) {
        if (it == skipped) continue;
        mbar_wait(bar_full + 8 * (it % C::NSTAGE), (it / C::NSTAGE) & 1, ctl, no_abort);
      }
    }
    if constexpr (FUSED) {  // the loader warp takes its share of the cluster gather
      __syncwarp();
      cluster_gather<D>(part_o, part_l, nh, splits, o_out, lse_out, o_row0);
    }
    return;
  }

  // -------------------------------------------------------------- compute warps
  const int kl = lane % C::KL;   // 16-byte column of the K row this lane reads
  const int tg = lane / C::KL;   // token within a load round
  const int hl = head_of_lane<C::KL, GT>(lane);
  const bool primary = ((lane % C::KL) & (C::KL / GT - 1)) == 0;  // one lane per (token, head)

  // q of the GT heads, pre-multiplied by scale*log2(e) so scores come out in base 2
  float qf[GT][8];
#pragma unroll
  for (int h = 0; h < GT; ++h) {
    if (h < nh) {
      const uint4 raw = *reinterpret_cast<const uint4*>(
          q + (static_cast<size_t>(b) * Hq + h0 + h) * D + kl * 8);
      const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        qf[h][2 * i] = bf16lo(w[i]) * c;
        qf[h][2 * i + 1] = bf16hi(w[i]) * c;
      }
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) qf[h][i] = 0.f;
    }
  }

  float m_run = -INFINITY, l_run = 0.f;
  float acc_o[GT][C::VD];
#pragma unroll
  for (int h = 0; h < GT; ++h)
#pragma unroll
    for (int d = 0; d < C::VD; ++d) acc_o[h][d] = 0.f;

  float* ps = reinterpret_cast<float*>(smem + L::P_OFF) + warp * C::TW * GT;
  float* alpha_s = reinterpret_cast<float*>(smem + L::ALPHA_OFF) + warp * GT;

  for (int it = 0; it < n_stages; ++it) {
    const int slot = it % C::NSTAGE;
    if (!mbar_wait_warp(bar_full + 8 * slot, (it / C::NSTAGE) & 1, ctl, ab)) break;
    const int ntok = min(C::T, t_end - (t_begin + it * C::T));
    const uint8_t* ks = smem + slot * C::STAGE_BYTES;
    const uint8_t* vs = ks + C::TILE_BYTES;

    // scores of this warp's TW tokens, in base-2 units
    float sc[C::KROUNDS];
#pragma unroll
    for (int r = 0; r < C::KROUNDS; ++r) {
      const int tl = warp * C::TW + r * C::TPR + tg;
      const uint4 raw = *reinterpret_cast<const uint4*>(ks + tl * (D * 2) + kl * 16);
      const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
      float kf[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        kf[2 * i] = bf16lo(w[i]);
        kf[2 * i + 1] = bf16hi(w[i]);
      }
      float acc[GT];
#pragma unroll
      for (int h = 0; h < GT; ++h) {
        float s = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) s = fmaf(qf[h][i], kf[i], s);
        acc[h] = s;
      }
      const float s = transpose_reduce<C::KL, GT>(acc, lane);
      sc[r] = (tl < ntok) ? s : -INFINITY;
    }

    // online softmax (per head, over this warp's tokens)
    float mx = sc[0];
#pragma unroll
    for (int r = 1; r < C::KROUNDS; ++r) mx = fmaxf(mx, sc[r]);
#pragma unroll
    for (int off = C::KL; off < 32; off <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    const float m_new = fmaxf(m_run, mx);
    const bool need = m_new > m_run + kRescaleThreshold;
    const float alpha = need ? ex2(m_run - m_new) : 1.f;
    if (need) m_run = m_new;
    const float ms = (m_run == -INFINITY) ? 0.f : m_run;
    float psum = 0.f;
    __syncwarp();
#pragma unroll
    for (int r = 0; r < C::KROUNDS; ++r) {
      const float p = ex2(sc[r] - ms);
      psum += p;
      if (primary) ps[(r * C::TPR + tg) * GT + hl] = p;
    }
    l_run = l_run * alpha + psum;
    if (primary && tg == 0) alpha_s[hl] = alpha;
    __syncwarp();

    if (__any_sync(0xffffffffu, need)) {
#pragma unroll
      for (int h = 0; h < GT; ++h) {
        const float a = alpha_s[h];
#pragma unroll
        for (int d = 0; d < C::VD; ++d) acc_o[h][d] *= a;
      }
    }

    // P.V over this warp's tokens; lane owns dims [lane*VD, lane*VD + VD)
    const int nmine = min(C::TW, ntok - warp * C::TW);
#pragma unroll 4
    for (int tt = 0; tt < nmine; ++tt) {
      const int tl = warp * C::TW + tt;
      float vf[C::VD];
      if constexpr (C::VD == 4) {
        const uint2 raw = *reinterpret_cast<const uint2*>(vs + tl * (D * 2) + lane * 8);
        vf[0] = bf16lo(raw.x);
        vf[1] = bf16hi(raw.x);
        vf[2] = bf16lo(raw.y);
        vf[3] = bf16hi(raw.y);
      } else {
        const uint32_t raw = *reinterpret_cast<const uint32_t*>(vs + tl * (D * 2) + lane * 4);
        vf[0] = bf16lo(raw);
        vf[1] = bf16hi(raw);
      }
      float pv[GT];
      if constexpr (GT % 4 == 0) {
#pragma unroll
        for (int h = 0; h < GT; h += 4) {
          const float4 p4 = *reinterpret_cast<const float4*>(ps + tt * GT + h);
          pv[h] = p4.x;
          pv[h + 1] = p4.y;
          pv[h + 2] = p4.z;
          pv[h + 3] = p4.w;
        }
      } else {
#pragma unroll
        for (int h = 0; h < GT; ++h) pv[h] = ps[tt * GT + h];
      }
#pragma unroll
      for (int h = 0; h < GT; ++h)
#pragma unroll
        for (int d = 0; d < C::VD; ++d) acc_o[h][d] = fmaf(pv[h], vf[d], acc_o[h][d]);
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_empty + 8 * slot);
  }

  // ---------------------------------------------------------------- merge the 8 warps
#pragma unroll
  for (int off = C::KL; off < 32; off <<= 1) l_run += __shfl_xor_sync(0xffffffffu, l_run, off);
  asm volatile("bar.sync 1, %0;" ::"n"(C::NCW * 32) : "memory");  // ring no longer read
  float* wm = reinterpret_cast<float*>(smem + L::WM_OFF);
  float* wl = reinterpret_cast<float*>(smem + L::WL_OFF);
  float* wo = reinterpret_cast<float*>(smem);  // [NCW][GT][D], reuses the ring
  if (primary && tg == 0) {
    wm[warp * GT + hl] = m_run;
    wl[warp * GT + hl] = l_run;
  }
#pragma unroll
  for (int h = 0; h < GT; ++h)
#pragma unroll
    for (int d = 0; d < C::VD; ++d) wo[(warp * GT + h) * D + lane * C::VD + d] = acc_o[h][d];
  asm volatile("bar.sync 1, %0;" ::"n"(C::NCW * 32) : "memory");

  for (int idx = threadIdx.x; idx < nh * D; idx += C::NCW * 32) {
    const int h = idx / D, d = idx % D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < C::NCW; ++w) M = fmaxf(M, wm[w * GT + h]);
    float lsum = 0.f, osum = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < C::NCW; ++w) {
        const float a = ex2(wm[w * GT + h] - M);  // 0 for warps that saw no key
        lsum = fmaf(a, wl[w * GT + h], lsum);
        osum = fmaf(a, wo[(w * GT + h) * D + d], osum);
      }
    }
    const bool any = lsum > 0.f;
    if constexpr (FUSED) {
      reinterpret_cast<float*>(smem + L::PART_O_OFF)[idx] = any ? osum / lsum : 0.f;
      if (d == 0) reinterpret_cast<float*>(smem + L::PART_L_OFF)[h] = any ? (M + log2f(lsum)) * kLn2 : -INFINITY;
    } else {
      const size_t row = row0 + static_cast<size_t>(h) * splits;
      o_part[row * D + d] = any ? osum / lsum : 0.f;
      if (d == 0) lse_part[row] = any ? (M + log2f(lsum)) * kLn2 : -INFINITY;
    }
  }
  if constexpr (FUSED) cluster_gather<D>(part_o, part_l, nh, splits, o_out, lse_out, o_row0);
}

// One CTA (D threads) per (batch, query head).  The split log-sum-exps are read in
// parallel (one per thread), reduced, turned into weights in shared memory, and the
// partial rows are streamed with 8 independent loads in flight per thread.
template <int D>
__global__ void __launch_bounds__(D) decode_merge_kernel(const float* __restrict__ o_part,
                                                         const float* __restrict__ lse_part,
                                                         __nv_bfloat16* __restrict__ o,
                                                         float* __restrict__ lse, int splits) {
  constexpr int NW = D / 32;
  __shared__ float w_s[kMaxDecodeSplits];
  __shared__ float red[NW];
  // Wait until the split kernel's partials are complete and visible.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int bh = blockIdx.x, d = threadIdx.x, lane = d & 31, wid = d >> 5;
  const float* lp = lse_part + static_cast<size_t>(bh) * splits;

  float m = -INFINITY;
  for (int i = d; i < splits; i += D) m = fmaxf(m, lp[i]);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
  if (lane == 0) red[wid] = m;
  __syncthreads();
  float M = red[0];
#pragma unroll
  for (int w = 1; w < NW; ++w) M = fmaxf(M, red[w]);
  __syncthreads();

  float ws = 0.f;
  for (int i = d; i < splits; i += D) {
    const float w = (M == -INFINITY) ? 0.f : ex2((lp[i] - M) * kLog2e);  // 0 for empty splits
    w_s[i] = w;
    ws += w;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) ws += __shfl_xor_sync(0xffffffffu, ws, off);
  if (lane == 0) red[wid] = ws;
  __syncthreads();
  float W = 0.f;
#pragma unroll
  for (int w = 0; w < NW; ++w) W += red[w];

  const float* op = o_part + static_cast<size_t>(bh) * splits * D + d;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  int i = 0;
  for (; i + 8 <= splits; i += 8) {
#pragma unroll
    for (int u = 0; u < 8; ++u) acc[u] = fmaf(w_s[i + u], op[static_cast<size_t>(i + u) * D], acc[u]);
  }
  for (; i < splits; ++i) acc[0] = fmaf(w_s[i], op[static_cast<size_t>(i) * D], acc[0]);
  const float sum = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
  const bool any = W > 0.f;
  o[static_cast<size_t>(bh) * D + d] = __float2bfloat16_rn(any ? sum / W : 0.f);
  if (lse && d == 0) lse[bh] = any ? M + log2f(W) * kLn2 : -INFINITY;
}

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

// A paged cache as a 3-D tensor whose box is `rows` keys of one kv head, landing in
// shared memory as rows x D contiguous bf16:
//   NHD [num_pages, page_size, Hkv, D] -> [num_pages * page_size keys, Hkv, D], box D x 1 x rows
//   HND [num_pages, Hkv, page_size, D] -> [num_pages * Hkv, page_size, D],      box D x rows x 1
bool paged_map(CUtensorMap* map, const void* cache, const PagedKV& pk, int Hkv, int D, int rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  const bool hnd = pk.layout == kPagedHND;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D),
                        static_cast<cuuint64_t>(hnd ? pk.page_size : Hkv),
                        static_cast<cuuint64_t>(pk.num_pages) * (hnd ? Hkv : pk.page_size)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2,
                           static_cast<cuuint64_t>(hnd ? pk.page_size : Hkv) * D * 2};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(D), static_cast<cuuint32_t>(hnd ? rows : 1),
                       static_cast<cuuint32_t>(hnd ? 1 : rows)};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(cache), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Per-device set-up of one kernel instance: the shared-memory opt-in and, for the cluster
// form, clusters of up to 16 CTAs (beyond the portable 8).
template <int D, int GT, bool PAGED, bool FUSED>
bool prepare_split() {
  static PerDeviceOnce configured;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  return configured.run(dev, [] {
    const void* fn = reinterpret_cast<const void*>(decode_split_kernel<D, GT, PAGED, FUSED>);
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, DecodeSmem<D, GT, FUSED>::BYTES) !=
        cudaSuccess)
      return false;
    if constexpr (FUSED) return cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess;
    return true;
  });
}

template <int D, int GT, bool FUSED>
cudaLaunchConfig_t split_config(dim3 grid, int cluster, cudaStream_t stream, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(DecodeCfg<D>::THREADS);
  cfg.dynamicSmemBytes = DecodeSmem<D, GT, FUSED>::BYTES;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 0;
  if (FUSED) {
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(cluster);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.numAttrs = 1;
  }
  return cfg;
}

// CTA slots of the cluster form with clusters of `splits` CTAs on the current device: whole
// clusters that fit at once (cudaOccupancyMaxActiveClusters) x splits; 0 if none fit or the
// device cannot be asked.  Cached per device and cluster size.
template <int D, int GT, bool PAGED>
int cluster_slots(int splits) {
  static std::atomic<int> cache[64][model::kMaxFusedSplits + 1];  // value + 1 once known
  int dev = 0;
  if (splits < 1 || splits > model::kMaxFusedSplits || cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 0;
  if (dev < 64) {
    const int c = cache[dev][splits].load(std::memory_order_relaxed);
    if (c != 0) return c - 1;
  }
  int clusters = 0;
  if (prepare_split<D, GT, PAGED, true>()) {
    cudaLaunchAttribute attr[1];
    const cudaLaunchConfig_t cfg = split_config<D, GT, true>(dim3(splits, 64, 1), splits, nullptr, attr);
    if (cudaOccupancyMaxActiveClusters(&clusters, decode_split_kernel<D, GT, PAGED, true>, &cfg) != cudaSuccess) {
      cudaGetLastError();
      clusters = 0;
    }
  }
  if (dev < 64) cache[dev][splits].store(clusters * splits + 1, std::memory_order_relaxed);
  return clusters * splits;
}

template <int D, int GT, bool PAGED, bool FUSED>
cudaError_t launch_split(const DecodeArgs& a, const PagedKV* pk, const KernelCtl& ctl, cudaStream_t stream) {
  if (!prepare_split<D, GT, PAGED, FUSED>()) return cudaErrorInvalidValue;
  CUtensorMap tk, tv;
  PagedView view{nullptr, 0, 0, 0, 0};
  if constexpr (PAGED) {
    const int rows = pk->page_size < kDecodeChunkAlign ? pk->page_size : kDecodeChunkAlign;
    if (!paged_map(&tk, a.k, *pk, a.Hkv, D, rows) || !paged_map(&tv, a.v, *pk, a.Hkv, D, rows))
      return cudaErrorInvalidValue;
    view = PagedView{pk->block_table, pk->page_size, pk->max_pages, pk->num_pages, pk->layout == kPagedHND ? 1 : 0};
  } else {
    (void)pk;
    memset(&tk, 0, sizeof(tk));
    memset(&tv, 0, sizeof(tv));
  }
  const int G = a.Hq / a.Hkv;
  const int n_groups = (G + GT - 1) / GT;
  cudaLaunchAttribute attr[1];
  const cudaLaunchConfig_t cfg =
      split_config<D, GT, FUSED>(dim3(a.splits, a.Hkv * n_groups, a.B), a.splits, stream, attr);
  return cudaLaunchKernelEx(&cfg, decode_split_kernel<D, GT, PAGED, FUSED>, static_cast<const __nv_bfloat16*>(a.q),
                            static_cast<const __nv_bfloat16*>(a.k), static_cast<const __nv_bfloat16*>(a.v),
                            a.seqlens, a.o_part, a.lse_part, a.Hq, a.Hkv, a.Skv, a.splits, n_groups,
                            a.scale * kLog2e, ctl, tk, tv, view, static_cast<__nv_bfloat16*>(a.o), a.lse);
}

template <int D>
cudaError_t launch_merge(const DecodeArgs& a, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.B * a.Hq);
  cfg.blockDim = dim3(D);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decode_merge_kernel<D>, static_cast<const float*>(a.o_part),
                            static_cast<const float*>(a.lse_part),
                            static_cast<__nv_bfloat16*>(a.o), a.lse, a.splits);
}

// Which form runs: the cluster form when it is forced (a.fused = 1) or the model prefers
// it (a.fused = 0), provided the split count is a cluster size and such clusters fit.
template <int D, int GT, bool PAGED>
bool use_cluster_form(const DecodeArgs& a) {
  if (a.fused < 0 || a.splits > model::kMaxFusedSplits) return false;
  const int slots = cluster_slots<D, GT, PAGED>(a.splits);
  if (slots < a.splits) return false;
  if (a.fused == 1) return true;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                cudaSuccess)
    return false;
  return model::decode_fused_wins(a.splits, a.B, a.Hq, a.Hkv, a.Skv, D, sms, slots);
}

template <int D, int GT, bool PAGED>
cudaError_t launch_form(const DecodeArgs& a, const PagedKV* pk, const KernelCtl& ctl, cudaStream_t stream) {
  if (use_cluster_form<D, GT, PAGED>(a)) return launch_split<D, GT, PAGED, true>(a, pk, ctl, stream);
  const cudaError_t e = launch_split<D, GT, PAGED, false>(a, pk, ctl, stream);
  if (e != cudaSuccess) return e;
  return launch_merge<D>(a, stream);
}

template <int D, bool PAGED>
cudaError_t launch_decode_d(const DecodeArgs& a, const PagedKV* pk, const KernelCtl& ctl, cudaStream_t stream) {
  const int G = a.Hq / a.Hkv;
  if (G >= 8) return launch_form<D, 8, PAGED>(a, pk, ctl, stream);
  if (G >= 4) return launch_form<D, 4, PAGED>(a, pk, ctl, stream);
  if (G >= 2) return launch_form<D, 2, PAGED>(a, pk, ctl, stream);
  return launch_form<D, 1, PAGED>(a, pk, ctl, stream);
}

template <int D, bool PAGED>
bool cluster_form_d(const DecodeArgs& a) {
  const int G = a.Hq / a.Hkv;
  if (G >= 8) return use_cluster_form<D, 8, PAGED>(a);
  if (G >= 4) return use_cluster_form<D, 4, PAGED>(a);
  if (G >= 2) return use_cluster_form<D, 2, PAGED>(a);
  return use_cluster_form<D, 1, PAGED>(a);
}

template <int D>
int cluster_slots_d(int G, int splits) {
  if (G >= 8) return cluster_slots<D, 8, false>(splits);
  if (G >= 4) return cluster_slots<D, 4, false>(splits);
  if (G >= 2) return cluster_slots<D, 2, false>(splits);
  return cluster_slots<D, 1, false>(splits);
}

}  // namespace

cudaError_t launch_decode(const DecodeArgs& a, const KernelCtl& ctl, cudaStream_t stream) {
  if (a.D == 128) return launch_decode_d<128, false>(a, nullptr, ctl, stream);
  return launch_decode_d<64, false>(a, nullptr, ctl, stream);
}

cudaError_t launch_decode_paged(const DecodeArgs& a, const PagedKV& pk, const KernelCtl& ctl, cudaStream_t stream) {
  if (!paged_page_size_ok(pk.page_size) || !a.seqlens || !pk.block_table ||
      (pk.layout != kPagedNHD && pk.layout != kPagedHND))
    return cudaErrorInvalidValue;
  if (a.D == 128) return launch_decode_d<128, true>(a, &pk, ctl, stream);
  return launch_decode_d<64, true>(a, &pk, ctl, stream);
}

bool decode_cluster_form(const DecodeArgs& a, bool paged) {
  if (a.D == 128) return paged ? cluster_form_d<128, true>(a) : cluster_form_d<128, false>(a);
  return paged ? cluster_form_d<64, true>(a) : cluster_form_d<64, false>(a);
}

int decode_cluster_slots(int D, int G, int splits) {
  return D == 128 ? cluster_slots_d<128>(G, splits) : cluster_slots_d<64>(G, splits);
}

}  // namespace loom
