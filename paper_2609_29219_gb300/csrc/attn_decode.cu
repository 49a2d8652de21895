// Flash Decode for GB300: split-KV partial attention + log-sum-exp merge, in two forms.
//
// Paper: Sec. 2.6 (the Flash Decode HEG is a sequential composition of a local
// softmax loop, a gather of partial results, a global softmax and a final scaling) and
// Sec. 3.2.3 (the sequence axis, the reduction axis, is split across cores).
//
// Split + merge form.
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
//
// Single-kernel (cluster) form, decode_persistent_kernel<.., true> -- persistent clusters of CS CTAs
// (CS divides the split count, CS <= 16).  A unit is one (batch, kv head, head group);
// each cluster walks its units (dealt in a snake order over the units sorted by
// sequence length), and for every unit CTA r of the cluster streams the unit's splits
// r, r + CS, ... with the same loader ring and compute warps as kernel 1, without a
// break between units: the loader fetches the next unit's q and first K/V stages while
// the compute warps finish the current one.  At a unit's end the compute warps merge
// their states in the ring slot of the unit's last stage into the CTA's partial
// (O_r, lse_r), kept in shared memory; once every CTA of the cluster has signalled its
// partial (a remote mbarrier arrive), CTA r gathers outputs [r n / CS, (r + 1) n / CS)
// of the unit's n = heads x D outputs from the CS partials over distributed shared
// memory (in rank order, so the result does not depend on timing), applies the global
// softmax and the final scaling, writes O (bf16) and LSE, and signals that it has read
// the partials, so that their owners may overwrite them with the next unit's.  No
// workspace and no second launch.
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

// Stage constants: the analytic model's choice for this head dimension.  Non-zero T_,
// NSTAGE_, CTAS_ override it (the neighbours measured by the block-size ablation).
template <int D, int T_ = 0, int NSTAGE_ = 0, int CTAS_ = 0>
struct DecodeCfg {
  static constexpr model::DecodeStagePlan kPlan = model::decode_stage_plan(D);
  static_assert(kPlan.feasible, "no feasible decode stage plan");
  static constexpr int DIM = D;
  static constexpr int T = T_ ? T_ : kPlan.tokens;  // tokens per stage
  static constexpr int NSTAGE = NSTAGE_ ? NSTAGE_ : kPlan.stages;
  static constexpr int CTAS_PER_SM = CTAS_ ? CTAS_ : kPlan.ctas_per_sm;
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

template <class C, int GT>
struct DecodeSmem {
  // ring first (16-byte aligned bulk-copy destinations), then the small arrays
  static constexpr uint32_t P_OFF = C::RING_BYTES;                      // [NCW][TW][GT] f32
  static constexpr uint32_t ALPHA_OFF = P_OFF + C::NCW * C::TW * GT * 4;  // [NCW][GT] f32
  static constexpr uint32_t WM_OFF = ALPHA_OFF + C::NCW * GT * 4;       // [NCW][GT] f32
  static constexpr uint32_t WL_OFF = WM_OFF + C::NCW * GT * 4;          // [NCW][GT] f32
  static constexpr uint32_t BAR_OFF = ((WL_OFF + C::NCW * GT * 4) + 7) / 8 * 8;
  static constexpr uint32_t ABORT_OFF = BAR_OFF + 2 * C::NSTAGE * 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16;
  // the cross-warp merge reuses the ring: [NCW][GT][D] f32
  static_assert(C::NCW * GT * C::DIM * 4 <= C::RING_BYTES, "merge buffer must fit in the ring");
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

// Compute-warp lane roles of one stage: lane = (token within a load round, 16-byte column
// of the K row); one primary lane per (token, head) keeps the head's probability.
template <int D, int GT>
struct LaneRole {
  using C = DecodeCfg<D>;
  int kl, tg, hl;
  bool primary;
  __device__ __forceinline__ explicit LaneRole(int lane)
      : kl(lane % C::KL), tg(lane / C::KL), hl(head_of_lane<C::KL, GT>(lane)),
        primary(((lane % C::KL) & (C::KL / GT - 1)) == 0) {}
};

// q of the GT heads at q_rows (row h = head h0 + h; rows >= nh are zero), pre-multiplied by
// scale * log2(e) so that scores come out in base 2.  q_rows may be global or shared.
template <int D, int GT>
__device__ __forceinline__ void load_q(const __nv_bfloat16* q_rows, int nh, int kl, float c, float (&qf)[GT][8]) {
#pragma unroll
  for (int h = 0; h < GT; ++h) {
    if (h < nh) {
      const uint4 raw = *reinterpret_cast<const uint4*>(q_rows + static_cast<size_t>(h) * D + kl * 8);
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
}

// One compute warp's work on one stage of the ring (K tile ks, V tile vs, ntok valid
// keys): the scores of its TW tokens for the GT heads (base 2), the online softmax per
// head with a lazily moved running max (m_run, l_run), and P.V into acc_o.  ps and alpha_s
// are this warp's shared-memory P [TW][GT] and rescale factors [GT].
template <class C, int GT>
__device__ __forceinline__ void decode_stage(const uint8_t* ks, const uint8_t* vs, int ntok, int warp, int lane,
                                             const LaneRole<C::DIM, GT>& lr, const float (&qf)[GT][8],
                                             float& m_run, float& l_run, float (&acc_o)[GT][C::VD], float* ps,
                                             float* alpha_s) {
  constexpr int D = C::DIM;
  // scores of this warp's TW tokens, in base-2 units
  float sc[C::KROUNDS];
#pragma unroll
  for (int r = 0; r < C::KROUNDS; ++r) {
    const int tl = warp * C::TW + r * C::TPR + lr.tg;
    const uint4 raw = *reinterpret_cast<const uint4*>(ks + tl * (D * 2) + lr.kl * 16);
    const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
    float2 kf[4];  // dims (2i, 2i + 1) of this lane's 8
#pragma unroll
    for (int i = 0; i < 4; ++i) kf[i] = make_float2(bf16lo(w[i]), bf16hi(w[i]));
    // two-wide fp32 FMAs (one instruction per pair of dims): even and odd dims summed
    // apart, then added
    float acc[GT];
#pragma unroll
    for (int h = 0; h < GT; ++h) {
      float2 s = __fmul2_rn(make_float2(qf[h][0], qf[h][1]), kf[0]);
#pragma unroll
      for (int i = 1; i < 4; ++i) s = __ffma2_rn(make_float2(qf[h][2 * i], qf[h][2 * i + 1]), kf[i], s);
      acc[h] = s.x + s.y;
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
    if (lr.primary) ps[(r * C::TPR + lr.tg) * GT + lr.hl] = p;
  }
  l_run = l_run * alpha + psum;
  if (lr.primary && lr.tg == 0) alpha_s[lr.hl] = alpha;
  __syncwarp();

  if (__any_sync(0xffffffffu, need)) {
#pragma unroll
    for (int h = 0; h < GT; ++h) {
      const float2 a = make_float2(alpha_s[h], alpha_s[h]);
#pragma unroll
      for (int d = 0; d < C::VD; d += 2) {
        const float2 r = __fmul2_rn(make_float2(acc_o[h][d], acc_o[h][d + 1]), a);
        acc_o[h][d] = r.x;
        acc_o[h][d + 1] = r.y;
      }
    }
  }

  // P.V over this warp's tokens; lane owns dims [lane*VD, lane*VD + VD)
  const int nmine = min(C::TW, ntok - warp * C::TW);
#pragma unroll 4
  for (int tt = 0; tt < nmine; ++tt) {
    const int tl = warp * C::TW + tt;
    float2 vf[C::VD / 2];  // dims (2j, 2j + 1) of this lane's VD
    if constexpr (C::VD == 4) {
      const uint2 raw = *reinterpret_cast<const uint2*>(vs + tl * (D * 2) + lane * 8);
      vf[0] = make_float2(bf16lo(raw.x), bf16hi(raw.x));
      vf[1] = make_float2(bf16lo(raw.y), bf16hi(raw.y));
    } else {
      const uint32_t raw = *reinterpret_cast<const uint32_t*>(vs + tl * (D * 2) + lane * 4);
      vf[0] = make_float2(bf16lo(raw), bf16hi(raw));
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
    for (int h = 0; h < GT; ++h) {
      const float2 p2 = make_float2(pv[h], pv[h]);
#pragma unroll
      for (int j = 0; j < C::VD / 2; ++j) {
        const float2 r = __ffma2_rn(p2, vf[j], make_float2(acc_o[h][2 * j], acc_o[h][2 * j + 1]));
        acc_o[h][2 * j] = r.x;
        acc_o[h][2 * j + 1] = r.y;
      }
    }
  }
}

// Merge of the NCW compute warps' states (run by all of them) into one partial per
// (head, dim): wo is an [NCW][GT][D] fp32 scratch that no warp reads any more when this is
// called, wm / wl [NCW][GT].  emit(idx = h * D + d, h, d, O value, LSE (natural log; valid
// where d == 0)) receives each of the nh x D results.
template <int D, int GT, class Emit>
__device__ __forceinline__ void merge_warps(float* wo, float* wm, float* wl, int nh, int warp, int lane,
                                            const LaneRole<D, GT>& lr, float m_run, float l_run,
                                            const float (&acc_o)[GT][DecodeCfg<D>::VD], Emit emit) {
  using C = DecodeCfg<D>;
#pragma unroll
  for (int off = C::KL; off < 32; off <<= 1) l_run += __shfl_xor_sync(0xffffffffu, l_run, off);
  asm volatile("bar.sync 1, %0;" ::"n"(C::NCW * 32) : "memory");  // the scratch is no longer read
  if (lr.primary && lr.tg == 0) {
    wm[warp * GT + lr.hl] = m_run;
    wl[warp * GT + lr.hl] = l_run;
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
    emit(idx, h, d, any ? osum / lsum : 0.f, any ? (M + log2f(lsum)) * kLn2 : -INFINITY);
  }
}

// Loader of a paged cache for one kv head of one sequence: the block table is read 32
// entries at a time (one per lane) and lane j issues the stage's j-th copy pair.  Copies
// hold `rows` keys: a 64-key piece of one page (page_size a multiple of 64) or one whole
// page (page_size 8, 16 or 32).  Stages start on a multiple of 64 keys, so no copy
// crosses a page.  Run by the whole loader warp.
struct PagedLoader {
  int win = 0, entry = 0;
  bool have = false;
  __device__ __forceinline__ void reset() { have = false; }
  template <int D>
  __device__ __forceinline__ void stage(const PagedView& pv, const int32_t* tbl, int Hkv, int hk, int tok0, int ntok,
                                        uint32_t dst, uint32_t bar, uint32_t tile_bytes, const CUtensorMap* tm_k,
                                        const CUtensorMap* tm_v, int lane) {
    const int P = pv.page_size;
    const int rows = P < kDecodeChunkAlign ? P : kDecodeChunkAlign;
    const uint32_t copy_bytes = static_cast<uint32_t>(rows) * D * 2;
    const int ncopy = (ntok + rows - 1) / rows;
    const int lp_first = tok0 / P, lp_last = (tok0 + (ncopy - 1) * rows) / P;
    if (!have || lp_first < win || lp_last >= win + 32) {  // refill the table window
      win = lp_first;
      entry = (win + lane < pv.max_pages) ? tbl[win + lane] : 0;
      have = true;
    }
    if (lane == 0) mbar_expect_tx(bar, 2u * ncopy * copy_bytes);
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
      tma_load_3d(dst + lane * copy_bytes, tm_k, 0, y, z, bar);
      tma_load_3d(dst + tile_bytes + lane * copy_bytes, tm_v, 0, y, z, bar);
    }
  }
};

template <int D, int GT, bool PAGED, class C = DecodeCfg<D>>
__global__ void __launch_bounds__(C::THREADS, C::CTAS_PER_SM)
    decode_split_kernel(const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ k,
                        const __nv_bfloat16* __restrict__ v, const int32_t* __restrict__ seqlens,
                        float* __restrict__ o_part, float* __restrict__ lse_part, int Hq, int Hkv,
                        int Skv, int splits, int n_groups, float c, KernelCtl ctl,
                        const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                        PagedView pv) {
  static_assert(C::DIM == D, "configuration of this head dimension");
  using L = DecodeSmem<C, GT>;
  extern __shared__ __align__(128) uint8_t smem[];

  // Let the merge grid launch as soon as every split CTA is resident.
  asm volatile("griddepcontrol.launch_dependents;");

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

  if (t_begin >= t_end) {  // empty split: contributes nothing to the merge
    for (int i = threadIdx.x; i < nh * D; i += blockDim.x)
      o_part[(row0 + static_cast<size_t>(i / D) * splits) * D + i % D] = 0.f;
    if (threadIdx.x < nh) lse_part[row0 + static_cast<size_t>(threadIdx.x) * splits] = -INFINITY;
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
      const int32_t* tbl = pv.block_table + static_cast<size_t>(b) * pv.max_pages;
      PagedLoader pl;
      int issued = 0, skipped = -1;
      for (int it = 0; it < n_stages; ++it) {
        const int slot = it % C::NSTAGE, round = it / C::NSTAGE;
        if (!mbar_wait_warp(bar_empty + 8 * slot, (round & 1) ^ 1, ctl, ab)) break;
        issued = it + 1;
        if (ctl.inject == 1 && it == 1) {  // test hook: never fill this stage
          skipped = it;
          continue;
        }
        const int tok0 = t_begin + it * C::T;
        pl.stage<D>(pv, tbl, Hkv, hk, tok0, min(C::T, t_end - tok0), s_base + slot * C::STAGE_BYTES,
                    bar_full + 8 * slot, C::TILE_BYTES, &tm_k, &tm_v, lane);
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
    return;
  }

  // -------------------------------------------------------------- compute warps
  const LaneRole<D, GT> lr(lane);
  float qf[GT][8];
  load_q<D, GT>(q + (static_cast<size_t>(b) * Hq + h0) * D, nh, lr.kl, c, qf);

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
    const uint8_t* ks = smem + slot * C::STAGE_BYTES;
    decode_stage<C, GT>(ks, ks + C::TILE_BYTES, min(C::T, t_end - (t_begin + it * C::T)), warp, lane, lr, qf, m_run,
                        l_run, acc_o, ps, alpha_s);
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_empty + 8 * slot);
  }

  // the 8 warps' states -> the split's partial in the workspace (the drained ring is the scratch)
  merge_warps<D, GT>(reinterpret_cast<float*>(smem), reinterpret_cast<float*>(smem + L::WM_OFF),
                     reinterpret_cast<float*>(smem + L::WL_OFF), nh, warp, lane, lr, m_run, l_run, acc_o,
                     [&](int, int h, int d, float ov, float lv) {
                       const size_t row = row0 + static_cast<size_t>(h) * splits;
                       o_part[row * D + d] = ov;
                       if (d == 0) lse_part[row] = lv;
                     });
}

// ---------------------------------------------------------------- tensor-core split kernel
// The split kernel of the split + merge form with the dot products on the tensor cores
// (Sec. 2.6 Flash Decode HEG, local softmax loop).  The query heads of one kv head are the
// rows of a 128-row tile held in TMEM (rows 0..G-1; the rest are zero and their results
// unused): per stage of T keys (64; 128 at D = 64) S = Q K^T is one M = 128 MMA with A in
// TMEM and the 128B-swizzled K tile as B, one warp (lane = query head) turns S into P =
// 2^(S c - m) in place as bf16, and O += P V is a second MMA with P in TMEM and V as an
// MN-major B.  The padded rows cost nothing that matters here -- the stage's MMAs take a
// fraction of the time its bytes take to arrive -- while the CUDA cores are left with T
// exponentials per head and stage instead of every product of the dot products.
//   warps: 0 query rows (Q into TMEM, softmax, epilogue; TMEM lanes 0-31), 1 loader
//   (TMA, lane 0), 2 MMA issuer (whole warp, one elected lane)
//   TMEM: [0, D/2) Q as bf16 pairs | [64, 64 + T) S, then P over its first T/2 columns |
//         [64 + T, 64 + T + D) O
template <int D>
struct DecodeTcCfg {
  // keys per stage: 64 at D = 128; 128 at D = 64, where a 64-key stage's bytes arrive
  // faster than its S -> softmax -> P.V chain runs and the TMEM columns allow the wider S
  static constexpr int T = model::decode_tc_stage_keys(D);
  // ring depth: 3 stages of 32 KB, so that exactly two CTAs share an SM (their 2 x 256
  // TMEM columns are the SM's 512)
  static constexpr int NSTAGE = 3;
  static constexpr int NBOX = D / 64;                     // 128-byte swizzle atoms along D
  static constexpr uint32_t BOX_BYTES = T * 128;          // 64 keys x 64 dims
  static constexpr uint32_t TILE_BYTES = NBOX * BOX_BYTES;  // one K or V tile
  static constexpr uint32_t STAGE_BYTES = 2 * TILE_BYTES;   // K, then V
  static constexpr uint32_t BAR_OFF = NSTAGE * STAGE_BYTES;
  // barriers: full[NSTAGE], empty[NSTAGE], q, s, p, o, drain
  static constexpr int NBAR = 2 * NSTAGE + 5;
  static constexpr uint32_t TMEM_PTR_OFF = BAR_OFF + NBAR * 8;
  static constexpr uint32_t ABORT_OFF = TMEM_PTR_OFF + 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16 + 1024;  // + 1024-byte alignment slack
  static constexpr uint32_t Q_COL = 0;
  static constexpr uint32_t S_COL = 64;
  static constexpr uint32_t O_COL = S_COL + T;
  static constexpr uint32_t TMEM_COLS = 256;  // a power of two: 2 CTAs per SM
  static constexpr int THREADS = 96;
  static constexpr int MAX_G = kDecodeTcMaxGroup;  // query heads per kv head: TMEM lanes of warp 0
  static_assert(O_COL + D <= TMEM_COLS, "TMEM budget");
  static_assert(Q_COL + D / 2 <= S_COL && S_COL + T <= O_COL && O_COL + D <= TMEM_COLS, "TMEM regions");
  static_assert(T % 64 == 0 && T % kDecodeChunkAlign == 0, "stages of whole 64-key score halves");
  static_assert(2 * (BYTES + 1024) <= 228 * 1024 && 3 * (BYTES + 1024) > 228 * 1024, "exactly two CTAs per SM");
};

// 64 scores of this lane's row from TMEM column `taddr` on, keys at or past `nvalid` (of
// these 64) masked to -inf.
__device__ __forceinline__ void decode_tc_scores64(uint32_t taddr, uint32_t* s, int nvalid) {
  tmem_ld32(taddr, s);
  tmem_ld32(taddr + 32, s + 32);
  tmem_wait_ld();
  reg_fence32(s);
  reg_fence32(s + 32);
  if (nvalid < 64) {
#pragma unroll
    for (int i = 0; i < 64; ++i)
      if (i >= nvalid) s[i] = __float_as_uint(-INFINITY);
  }
}

__device__ __forceinline__ float decode_tc_max64(const uint32_t* s) {
  float mm[8];
#pragma unroll
  for (int g = 0; g < 8; ++g) mm[g] = __uint_as_float(s[g]);
#pragma unroll
  for (int i = 8; i + 16 <= 64; i += 16)
#pragma unroll
    for (int g = 0; g < 8; ++g) mm[g] = max3(mm[g], __uint_as_float(s[i + g]), __uint_as_float(s[i + 8 + g]));
#pragma unroll
  for (int g = 0; g < 8; ++g) mm[g] = fmaxf(mm[g], __uint_as_float(s[56 + g]));
  return fmaxf(max3(mm[0], mm[1], mm[2]), max3(max3(mm[3], mm[4], mm[5]), mm[6], mm[7]));
}

// One stage's softmax on warp 0 of a tensor-core split kernel (lane = a query head's row):
// the stage's T scores are read from TMEM in 64-key halves (twice when T = 128: once for
// the maximum, once for the exponentials, so that 64 scores are live at a time), keys at
// or past ntok are masked, the running maximum (base 2, scaled by c) moves only when it
// grows by more than kRescaleThreshold, and P goes back over S as bf16 pairs (a half's 64
// keys in 32 columns).  Returns the row sum of P; *alpha is the factor O needs, *need
// whether the maximum moved.
template <class C>
__device__ __forceinline__ float decode_tc_softmax(uint32_t tmem, int ntok, float c, float* m_run, float* alpha,
                                                   bool* need) {
  constexpr int NH = C::T / 64;
  uint32_t s[64];
  float mx = -INFINITY;
#pragma unroll
  for (int h = 0; h < NH; ++h) {
    decode_tc_scores64(tmem + C::S_COL + 64 * h, s, ntok - 64 * h);
    mx = fmaxf(mx, decode_tc_max64(s));
  }
  const float m_new = fmaxf(*m_run, mx * c);
  *need = m_new > *m_run + kRescaleThreshold;
  *alpha = *need ? ex2(*m_run - m_new) : 1.f;
  if (*need) *m_run = m_new;
  const float ms = (*m_run == -INFINITY) ? 0.f : *m_run;
  const uint64_t c2 = f2(c, c);
  const uint64_t nms2 = f2(-ms, -ms);
  uint64_t acc[4] = {0, 0, 0, 0};
#pragma unroll
  for (int h = 0; h < NH; ++h) {
    if (NH > 1) decode_tc_scores64(tmem + C::S_COL + 64 * h, s, ntok - 64 * h);  // (one half: still in s)
    uint32_t pk[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const uint64_t x = fma2(f2(__uint_as_float(s[2 * i]), __uint_as_float(s[2 * i + 1])), c2, nms2);
      const float p0 = ex2(f2lo(x));
      const float p1 = ex2(f2hi(x));
      acc[i & 3] = add2(acc[i & 3], f2(p0, p1));
      pk[i] = pack_bf16x2(p0, p1);
    }
    // P of keys [64h, 64h + 64) over S columns [32h, 32h + 32): S of those columns was read
    tmem_st32(tmem + C::S_COL + 32 * h, pk);
  }
  tmem_wait_st();
  const uint64_t a01 = add2(add2(acc[0], acc[1]), add2(acc[2], acc[3]));
  return f2lo(a01) + f2hi(a01);
}

// O += P V over one stage: P (bf16, TMEM, T/2 columns) x the stage's V tile (MN-major), in
// groups of 64 keys (four K = 16 steps each).
template <class C>
__device__ __forceinline__ void decode_tc_issue_pv(uint32_t tmem, uint32_t vtile, uint32_t idesc_pv, bool accumulate) {
#pragma unroll
  for (int g = 0; g < C::T / 64; ++g)
    mma_ts_k64_el(tmem + C::O_COL, tmem + C::S_COL + 32 * g, sdesc_sw128(vtile + g * 64 * 128, C::BOX_BYTES, 1024),
                  idesc_pv, (accumulate || g > 0) ? 1u : 0u);
}

// Warp 0 of decode_tc_split_kernel: lane h is query head h0 + h (lanes >= G carry zero rows).
// Q goes into TMEM as bf16 pairs (its memory order); per stage the lane runs
// decode_tc_softmax over its T scores (keys past the split's end masked, P written over
// S), rescales O in TMEM after the previous P.V when the running max moved, zeroes the V
// rows past the split's end, and arrives on bar_p; at the end O / l and the log-sum-exp
// go to the split's partial.
template <int D>
__device__ __forceinline__ void decode_tc_rows(const __nv_bfloat16* __restrict__ q, float* __restrict__ o_part,
                                               float* __restrict__ lse_part, uint32_t tmem, int b, int h0, int G,
                                               int Hq, int splits, size_t row0, int t_begin, int t_end, int n_st,
                                               float c, uint8_t* smem, uint32_t bar_full, uint32_t bar_q,
                                               uint32_t bar_s, uint32_t bar_p, uint32_t bar_o, const KernelCtl& ctl,
                                               const Abort& ab) {
  using C = DecodeTcCfg<D>;
  const int lane = threadIdx.x & 31;
  const bool real = lane < G;
  {
    uint32_t w[32];
    const uint4* src = reinterpret_cast<const uint4*>(q + (static_cast<size_t>(b) * Hq + h0 + (real ? lane : 0)) * D);
#pragma unroll
    for (int half = 0; half < D / 64; ++half) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const uint4 v = real ? src[half * 8 + i] : make_uint4(0u, 0u, 0u, 0u);
        w[4 * i] = v.x;
        w[4 * i + 1] = v.y;
        w[4 * i + 2] = v.z;
        w[4 * i + 3] = v.w;
      }
      tmem_st32(tmem + C::Q_COL + half * 32, w);
    }
    tmem_wait_st();
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_q);
  }
  float m_run = -INFINITY, l_run = 0.f;
  bool ok = true;
  for (int it = 0; it < n_st; ++it) {
    if (!(ok = mbar_wait_warp(bar_s, it & 1, ctl, ab))) break;
    tc_fence_after();
    const int ntok = min(C::T, t_end - (t_begin + it * C::T));
    float alpha;
    bool need;
    const float psum = decode_tc_softmax<C>(tmem, ntok, c, &m_run, &alpha, &need);
    if (ntok < C::T) {
      // V rows past the split's end may hold anything (a cache past a sequence's length
      // is never written): zero them so that their P = 0 adds exactly nothing to P.V
      const int slot = it % C::NSTAGE;
      if (!(ok = mbar_wait_warp(bar_full + 8 * slot, (it / C::NSTAGE) & 1, ctl, ab))) break;
      uint4* vt = reinterpret_cast<uint4*>(smem + slot * C::STAGE_BYTES + C::TILE_BYTES);
#pragma unroll
      for (int x = 0; x < C::NBOX; ++x)
        for (int i = lane; i < (C::T - ntok) * 8; i += 32)
          vt[x * (C::BOX_BYTES / 16) + ntok * 8 + i] = make_uint4(0u, 0u, 0u, 0u);
      fence_proxy_async_smem();
    }
    // O must hold the previous P.V before it is rescaled (it has: S of this stage was
    // committed after it), and be rescaled before this stage's P.V
    if (it > 0 && __any_sync(0xffffffffu, need)) {
      if (!(ok = mbar_wait_warp(bar_o, (it - 1) & 1, ctl, ab))) break;
      tc_fence_after();
      const uint64_t a2 = f2(alpha, alpha);
#pragma unroll 1
      for (int ch = 0; ch < D / 32; ++ch) {
        uint32_t rr[32];
        tmem_ld32(tmem + C::O_COL + ch * 32, rr);
        tmem_wait_ld();
        reg_fence32(rr);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const uint64_t x = mul2(f2(__uint_as_float(rr[2 * i]), __uint_as_float(rr[2 * i + 1])), a2);
          rr[2 * i] = __float_as_uint(f2lo(x));
          rr[2 * i + 1] = __float_as_uint(f2hi(x));
        }
        tmem_st32(tmem + C::O_COL + ch * 32, rr);
      }
      tmem_wait_st();
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_p);
    l_run = l_run * alpha + psum;
  }
  if (!ok) return;
  // epilogue: the last P.V, then O / l and the log-sum-exp of each real row
  if (!mbar_wait_warp(bar_o, (n_st - 1) & 1, ctl, ab)) return;
  tc_fence_after();
  const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
  float* dst = o_part + (row0 + static_cast<size_t>(real ? lane : 0) * splits) * D;
#pragma unroll 1
  for (int ch = 0; ch < D / 32; ++ch) {
    uint32_t rr[32];
    tmem_ld32(tmem + C::O_COL + ch * 32, rr);
    tmem_wait_ld();
    reg_fence32(rr);
    if (real) {
#pragma unroll
      for (int i = 0; i < 8; ++i)
        reinterpret_cast<float4*>(dst + ch * 32)[i] =
            make_float4(__uint_as_float(rr[4 * i]) * inv_l, __uint_as_float(rr[4 * i + 1]) * inv_l,
                        __uint_as_float(rr[4 * i + 2]) * inv_l, __uint_as_float(rr[4 * i + 3]) * inv_l);
    }
  }
  if (real) lse_part[row0 + static_cast<size_t>(lane) * splits] = l_run > 0.f ? (m_run + log2f(l_run)) * kLn2 : -INFINITY;
}

template <int D>
__global__ void __launch_bounds__(DecodeTcCfg<D>::THREADS, 2)
    decode_tc_split_kernel(const __nv_bfloat16* __restrict__ q, const int32_t* __restrict__ seqlens,
                           float* __restrict__ o_part, float* __restrict__ lse_part, int Hq, int Hkv, int Skv,
                           int splits, float c, KernelCtl ctl, const __grid_constant__ CUtensorMap tm_k,
                           const __grid_constant__ CUtensorMap tm_v) {
  using C = DecodeTcCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  // Let the merge grid launch as soon as every split CTA is resident.
  asm volatile("griddepcontrol.launch_dependents;");
  const uint32_t raw_base = smem_u32(smem_raw);
  const uint32_t sbase = (raw_base + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (sbase - raw_base);
  const int split = blockIdx.x, hk = blockIdx.y, b = blockIdx.z;
  const int G = Hq / Hkv, h0 = hk * G;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  int len = seqlens ? seqlens[b] : Skv;
  len = max(0, min(len, Skv));
  int chunk = (len + splits - 1) / splits;
  chunk = (chunk + kDecodeChunkAlign - 1) / kDecodeChunkAlign * kDecodeChunkAlign;
  const int t_begin = min(split * chunk, len);
  const int t_end = min(t_begin + chunk, len);
  const size_t row0 = (static_cast<size_t>(b) * Hq + h0) * splits + split;  // head h0's partial
  if (t_begin >= t_end) {  // empty split: contributes nothing to the merge
    for (int i = threadIdx.x; i < G * D; i += blockDim.x)
      o_part[(row0 + static_cast<size_t>(i / D) * splits) * D + i % D] = 0.f;
    if (static_cast<int>(threadIdx.x) < G) lse_part[row0 + static_cast<size_t>(threadIdx.x) * splits] = -INFINITY;
    return;
  }
  const int n_st = (t_end - t_begin + C::T - 1) / C::T;
  const int kv_z = b * Hkv + hk;

  const uint32_t bar_full = sbase + C::BAR_OFF;
  const uint32_t bar_empty = bar_full + 8 * C::NSTAGE;
  const uint32_t bar_q = bar_empty + 8 * C::NSTAGE;  // Q is in TMEM
  const uint32_t bar_s = bar_q + 8;                  // S of the stage is in TMEM
  const uint32_t bar_p = bar_s + 8;                  // P of the stage is in TMEM (O rescaled)
  const uint32_t bar_o = bar_p + 8;                  // the stage's P.V is done
  const uint32_t bar_drain = bar_o + 8;
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::TMEM_PTR_OFF);
  Abort ab{reinterpret_cast<volatile int*>(smem + C::ABORT_OFF)};
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    mbar_init(bar_q, 1);
    mbar_init(bar_s, 1);
    mbar_init(bar_p, 1);
    mbar_init(bar_o, 1);
    mbar_init(bar_drain, 1);
    *ab.flag = 0;
    *(ab.flag + 1) = 0;
    fence_barrier_init();
  }
  if (warp == 2) tmem_alloc(smem_u32(tmem_ptr), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_ptr;

  if (warp == 1) {
    // ------------------------------------------------------------ loader (lane 0)
    if (lane == 0) {
      prefetch_tensormap(&tm_k);
      prefetch_tensormap(&tm_v);
      int issued = 0, skipped = -1;
      for (int it = 0; it < n_st; ++it) {
        const int s = it % C::NSTAGE;
        if (!mbar_wait(bar_empty + 8 * s, ((it / C::NSTAGE) & 1) ^ 1, ctl, ab)) break;
        issued = it + 1;
        if (ctl.inject == 1 && it == 1) {  // test hook: never fill this stage
          skipped = it;
          continue;
        }
        // keys [tok0, tok0 + 64) of this kv head; rows past Skv read as zeros and every
        // key past the split's end is masked by the softmax
        const int tok0 = t_begin + it * C::T;
        const uint32_t dst = sbase + s * C::STAGE_BYTES;
        mbar_expect_tx(bar_full + 8 * s, C::STAGE_BYTES);
#pragma unroll
        for (int x = 0; x < C::NBOX; ++x) {
          tma_load_3d(dst + x * C::BOX_BYTES, &tm_k, x * 64, tok0, kv_z, bar_full + 8 * s);
          tma_load_3d(dst + C::TILE_BYTES + x * C::BOX_BYTES, &tm_v, x * 64, tok0, kv_z, bar_full + 8 * s);
        }
      }
      // Drain: never leave the CTA with copies still landing in its shared memory.
      Abort no_abort{ab.flag + 1};
      for (int i = max(0, issued - C::NSTAGE); i < issued; ++i)
        if (i != skipped) mbar_wait(bar_full + 8 * (i % C::NSTAGE), (i / C::NSTAGE) & 1, ctl, no_abort);
    }
  } else if (warp == 2) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc_s = idesc_bf16(128, C::T, 0, 0);  // Q (TMEM) x K^T (K-major)
    constexpr uint32_t idesc_pv = idesc_bf16(128, D, 0, 1);    // P (TMEM) x V (MN-major)
    bool ok = mbar_wait_warp(bar_q, 0, ctl, ab);
    tc_fence_after();
    for (int it = 0; ok && it < n_st; ++it) {
      const int s = it % C::NSTAGE;
      if (!(ok = mbar_wait_warp(bar_full + 8 * s, (it / C::NSTAGE) & 1, ctl, ab))) break;
      tc_fence_after();
      const uint32_t kslot = sbase + s * C::STAGE_BYTES;
      // S = Q K^T over D in 64-wide boxes (the previous stage's P.V, issued before, has
      // read the P these columns held: the MMAs of a CTA run in issue order)
#pragma unroll
      for (int x = 0; x < C::NBOX; ++x)
        mma_ts_kmaj_k64_el(tmem + C::S_COL, tmem + C::Q_COL + x * 32,
                           sdesc_sw128(kslot + x * C::BOX_BYTES, 16, 1024), idesc_s, x > 0 ? 1u : 0u);
      tc_commit_el(bar_s);
      if (!(ok = mbar_wait_warp(bar_p, it & 1, ctl, ab))) break;
      tc_fence_after();
      // O += P V over the stage's 64 keys
      decode_tc_issue_pv<C>(tmem, kslot + C::TILE_BYTES, idesc_pv, it > 0);
      tc_commit_el(bar_o);
      tc_commit_el(bar_empty + 8 * s);
    }
    // every MMA issued above is done before TMEM is released
    Abort no_abort{ab.flag + 1};
    tc_commit_el(bar_drain);
    mbar_wait_warp(bar_drain, 0, ctl, no_abort);
  } else {
    // ------------------------------------------------------------ query rows (warp 0)
    decode_tc_rows<D>(q, o_part, lse_part, tmem, b, h0, G, Hq, splits, row0, t_begin, t_end, n_st, c, smem, bar_full,
                      bar_q, bar_s, bar_p, bar_o, ctl, ab);
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------- tensor-core persistent split kernel
// decode_tc_persist_kernel: the tensor-core split kernel as persistent CTAs (two per SM,
// the TMEM and shared memory of DecodeTcCfg).  The loader takes (sequence, kv head, split)
// items from the workspace counter (one atomic per item; the sequences sorted by length,
// longest first) and streams each item's q (TMA, 128-byte swizzled, 64 dims per box) and
// K/V stages into the ring without a break between items.  With every stage it records in
// the slot which item and which stage of it the slot holds; the MMA warp and the softmax
// warp walk the ring and learn the item boundaries from those records, so neither needs
// the counter.  A final record with b = -1 ends both.
template <int D>
struct DecodeTcPersistCfg {
  using C = DecodeTcCfg<D>;
  static constexpr int kMaxSortedB = 256;                 // sequences sorted by length
  static constexpr uint32_t Q_BOX_BYTES = C::MAX_G * 128;  // up to 32 heads x 64 dims
  static constexpr uint32_t Q_OFF = C::NSTAGE * C::STAGE_BYTES;
  static constexpr uint32_t META_OFF = Q_OFF + C::NBOX * Q_BOX_BYTES;  // [NSTAGE] x 8 int32
  static constexpr uint32_t ORDER_OFF = META_OFF + C::NSTAGE * 32;     // [kMaxSortedB] int32
  static constexpr uint32_t LENS_OFF = ORDER_OFF + kMaxSortedB * 4;     // [kMaxSortedB] int32
  static constexpr uint32_t BAR_OFF = LENS_OFF + kMaxSortedB * 4;
  // barriers: full[NSTAGE], empty[NSTAGE], q_full, q_empty, q, s, p, o, drain
  static constexpr int NBAR = 2 * C::NSTAGE + 7;
  static constexpr uint32_t TMEM_PTR_OFF = BAR_OFF + NBAR * 8;
  static constexpr uint32_t ABORT_OFF = TMEM_PTR_OFF + 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16 + 1024;  // + 1024-byte alignment slack
  static_assert(Q_OFF % 1024 == 0 && Q_BOX_BYTES % 1024 == 0, "q boxes start on the swizzle period");
  static_assert(2 * (BYTES + 1024) <= 228 * 1024 && 3 * (BYTES + 1024) > 228 * 1024, "exactly two CTAs per SM");
};

// Warp 0 of decode_tc_persist_kernel: the softmax of decode_tc_rows over the ring's
// records.  At an item's first stage it moves the item's q rows from the swizzled boxes
// into TMEM (lane h reads head h, its 16-byte chunks in swizzled order: no bank conflicts)
// and starts a fresh running state; at its last stage it writes the item's partial.
template <int D>
__device__ __forceinline__ void decode_tc_persist_rows(const uint8_t* smem, float* __restrict__ o_part,
                                                       float* __restrict__ lse_part, uint32_t tmem, int G, int Hq,
                                                       int splits, float c, uint32_t bar_full, uint32_t bar_qf,
                                                       uint32_t bar_qe, uint32_t bar_q, uint32_t bar_s, uint32_t bar_p,
                                                       uint32_t bar_o, const KernelCtl& ctl, const Abort& ab) {
  using C = DecodeTcCfg<D>;
  using L = DecodeTcPersistCfg<D>;
  const int lane = threadIdx.x & 31;
  const bool real = lane < G;
  float m_run = -INFINITY, l_run = 0.f;
  int nq = 0;
  for (int st = 0;; ++st) {
    const int slot = st % C::NSTAGE;
    if (!mbar_wait_warp(bar_full + 8 * slot, (st / C::NSTAGE) & 1, ctl, ab)) return;
    const volatile int* rec = reinterpret_cast<const volatile int*>(smem + L::META_OFF + slot * 32);
    const int b = rec[0];
    if (b < 0) return;  // no more items
    const int hk = rec[1], split = rec[2], j = rec[3], n_st = rec[4], ntok = rec[6];
    if (j == 0) {
      if (!mbar_wait_warp(bar_qf, nq & 1, ctl, ab)) return;
#pragma unroll
      for (int x = 0; x < C::NBOX; ++x) {
        uint32_t w[32];
        const uint8_t* row = smem + L::Q_OFF + x * L::Q_BOX_BYTES + (real ? lane : 0) * 128;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const uint4 v = real ? *reinterpret_cast<const uint4*>(row + ((i ^ (lane & 7)) << 4))
                               : make_uint4(0u, 0u, 0u, 0u);
          w[4 * i] = v.x;
          w[4 * i + 1] = v.y;
          w[4 * i + 2] = v.z;
          w[4 * i + 3] = v.w;
        }
        tmem_st32(tmem + C::Q_COL + x * 32, w);
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(bar_qe);  // the q boxes may take the next item's rows
        mbar_arrive(bar_q);   // q is in TMEM
      }
      ++nq;
      m_run = -INFINITY;
      l_run = 0.f;
    }
    if (!mbar_wait_warp(bar_s, st & 1, ctl, ab)) return;
    tc_fence_after();
    float alpha;
    bool need;
    const float psum = decode_tc_softmax<C>(tmem, ntok, c, &m_run, &alpha, &need);
    if (ntok < C::T) {
      // V rows past the split's end may hold anything: zero them (P = 0 meets 0)
      uint4* vt = reinterpret_cast<uint4*>(const_cast<uint8_t*>(smem) + slot * C::STAGE_BYTES + C::TILE_BYTES);
#pragma unroll
      for (int x = 0; x < C::NBOX; ++x)
        for (int i = lane; i < (C::T - ntok) * 8; i += 32)
          vt[x * (C::BOX_BYTES / 16) + ntok * 8 + i] = make_uint4(0u, 0u, 0u, 0u);
      fence_proxy_async_smem();
    }
    // O holds the previous stage's P.V (committed before this stage's S) when rescaled
    if (j > 0 && __any_sync(0xffffffffu, need)) {
      if (!mbar_wait_warp(bar_o, (st - 1) & 1, ctl, ab)) return;
      tc_fence_after();
      const uint64_t a2 = f2(alpha, alpha);
#pragma unroll 1
      for (int ch = 0; ch < D / 32; ++ch) {
        uint32_t rr[32];
        tmem_ld32(tmem + C::O_COL + ch * 32, rr);
        tmem_wait_ld();
        reg_fence32(rr);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const uint64_t x = mul2(f2(__uint_as_float(rr[2 * i]), __uint_as_float(rr[2 * i + 1])), a2);
          rr[2 * i] = __float_as_uint(f2lo(x));
          rr[2 * i + 1] = __float_as_uint(f2hi(x));
        }
        tmem_st32(tmem + C::O_COL + ch * 32, rr);
      }
      tmem_wait_st();
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_p);
    l_run = l_run * alpha + psum;
    if (j == n_st - 1) {
      // the item's last P.V, then O / l and the log-sum-exp of each real row
      if (!mbar_wait_warp(bar_o, st & 1, ctl, ab)) return;
      tc_fence_after();
      const size_t row0 = (static_cast<size_t>(b) * Hq + static_cast<size_t>(hk) * G) * splits + split;
      const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
      float* dst = o_part + (row0 + static_cast<size_t>(real ? lane : 0) * splits) * D;
#pragma unroll 1
      for (int ch = 0; ch < D / 32; ++ch) {
        uint32_t rr[32];
        tmem_ld32(tmem + C::O_COL + ch * 32, rr);
        tmem_wait_ld();
        reg_fence32(rr);
        if (real) {
#pragma unroll
          for (int i = 0; i < 8; ++i)
            reinterpret_cast<float4*>(dst + ch * 32)[i] =
                make_float4(__uint_as_float(rr[4 * i]) * inv_l, __uint_as_float(rr[4 * i + 1]) * inv_l,
                            __uint_as_float(rr[4 * i + 2]) * inv_l, __uint_as_float(rr[4 * i + 3]) * inv_l);
        }
      }
      if (real)
        lse_part[row0 + static_cast<size_t>(lane) * splits] = l_run > 0.f ? (m_run + log2f(l_run)) * kLn2 : -INFINITY;
    }
  }
}

// PAGED: K/V from a paged cache.  A stage of T keys is then copied in pieces of min(page
// size, 64) keys, one per page it touches (each page looked up in the block table, each
// piece looked up and copied by its own loader lane), into the same 128-byte-swizzled
// tile: a piece of r rows starts r x 128 bytes into its box, a multiple of 1024 (page
// sizes 8, 16, 32 or multiples of 64), so the swizzle pattern is the one a single 64-row
// box leaves.  Pieces past the split's end are not copied (their keys are masked and
// their V rows zeroed).
template <int D, bool PAGED>
__global__ void __launch_bounds__(DecodeTcCfg<D>::THREADS, 2)
    decode_tc_persist_kernel(const int32_t* __restrict__ seqlens, float* __restrict__ o_part,
                             float* __restrict__ lse_part, unsigned long long* __restrict__ sched, int B, int Hq,
                             int Hkv, int Skv, int splits, float c, KernelCtl ctl, const __grid_constant__ CUtensorMap tm_q,
                             const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                             PagedView pv) {
  using C = DecodeTcCfg<D>;
  using L = DecodeTcPersistCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  // Let the merge grid launch as soon as every CTA is resident.
  asm volatile("griddepcontrol.launch_dependents;");
  const uint32_t raw_base = smem_u32(smem_raw);
  const uint32_t sbase = (raw_base + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (sbase - raw_base);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = Hq / Hkv;
  const long long per_seq = static_cast<long long>(Hkv) * splits;
  const long long n_items = B * per_seq;

  const uint32_t bar_full = sbase + L::BAR_OFF;
  const uint32_t bar_empty = bar_full + 8 * C::NSTAGE;
  const uint32_t bar_qf = bar_empty + 8 * C::NSTAGE;  // an item's q rows are in the boxes
  const uint32_t bar_qe = bar_qf + 8;                 // the boxes were read
  const uint32_t bar_q = bar_qe + 8;                  // q is in TMEM
  const uint32_t bar_s = bar_q + 8;                   // S of the stage is in TMEM
  const uint32_t bar_p = bar_s + 8;                   // P of the stage is in TMEM (O rescaled)
  const uint32_t bar_o = bar_p + 8;                   // the stage's P.V is done
  const uint32_t bar_drain = bar_o + 8;
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + L::TMEM_PTR_OFF);
  Abort ab{reinterpret_cast<volatile int*>(smem + L::ABORT_OFF)};
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    mbar_init(bar_qf, 1);
    mbar_init(bar_qe, 1);
    mbar_init(bar_q, 1);
    mbar_init(bar_s, 1);
    mbar_init(bar_p, 1);
    mbar_init(bar_o, 1);
    mbar_init(bar_drain, 1);
    *ab.flag = 0;
    *(ab.flag + 1) = 0;
    fence_barrier_init();
  }
  if (warp == 2) tmem_alloc(smem_u32(tmem_ptr), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_ptr;
  // Launched as a dependent of the previous kernel in the stream (the previous call's
  // merge lets it start early): everything above touches no global memory; from here on
  // the previous kernel's writes must be complete and visible.
  asm volatile("griddepcontrol.wait;" ::: "memory");

  // the sequences in order of decreasing length (ties by index): items are taken in it
  int* order = reinterpret_cast<int*>(smem + L::ORDER_OFF);
  const bool sorted = seqlens != nullptr && B <= L::kMaxSortedB;
  if (sorted) {
    int* lens = reinterpret_cast<int*>(smem + L::LENS_OFF);
    for (int bb = threadIdx.x; bb < B; bb += blockDim.x) lens[bb] = seqlens[bb];
    __syncthreads();
    for (int bb = threadIdx.x; bb < B; bb += blockDim.x) {
      const int lb = lens[bb];
      int r = 0;
      for (int x = 0; x < B; ++x) {
        const int lx = lens[x];
        r += (lx > lb) || (lx == lb && x < bb);
      }
      order[r] = bb;
    }
    __syncthreads();
  }

  if (warp == 1) {
    // ------------------------------------------------------------ loader (whole warp)
    // Lane 0 takes the tickets, waits on the ring and writes the records; a paged stage's
    // pieces are looked up and copied by one lane each, so that the copies of a stage go
    // out together.
    if (lane == 0) {
      prefetch_tensormap(&tm_q);
      prefetch_tensormap(&tm_k);
      prefetch_tensormap(&tm_v);
    }
    // Item blockIdx.x first.  An armed counter deals the items past the first gridDim.x
    // on demand, one ticket fetched an item ahead so that its latency is hidden; a
    // workspace never armed (its first call) deals them statically, item blockIdx.x +
    // k * gridDim.x (every CTA reads the same unarmed tag: all take the same branch).
    unsigned long long ticket = lane == 0 ? atomicAdd(sched, 1ull) : 0ull;
    int dynamic = -1;  // read from the first ticket once the first item is under way
    long long item = blockIdx.x;
    int st = 0, nq = 0, skipped = -1;
    bool ok = true;
    for (long long kk = 1; ok && item < n_items; ++kk) {
      const int rb = static_cast<int>(item / per_seq);
      const int rem = static_cast<int>(item - rb * per_seq);
      const int b = sorted ? order[rb] : rb;
      const int split = rem / Hkv, hk = rem - split * Hkv;
      int len = seqlens ? seqlens[b] : Skv;
      len = max(0, min(len, Skv));
      int chunk = (len + splits - 1) / splits;
      chunk = (chunk + kDecodeChunkAlign - 1) / kDecodeChunkAlign * kDecodeChunkAlign;
      const int t_begin = min(split * chunk, len);
      const int t_end = min(t_begin + chunk, len);
      if (t_begin >= t_end) {
        // empty split: contributes nothing to the merge
        const size_t row0 = (static_cast<size_t>(b) * Hq + static_cast<size_t>(hk) * G) * splits + split;
        for (int i = lane; i < G * (D / 4); i += 32) {
          const int r = i / (D / 4);
          reinterpret_cast<float4*>(o_part + (row0 + static_cast<size_t>(r) * splits) * D)[i % (D / 4)] =
              make_float4(0.f, 0.f, 0.f, 0.f);
        }
        for (int r = lane; r < G; r += 32) lse_part[row0 + static_cast<size_t>(r) * splits] = -INFINITY;
      } else {
        // the item's q rows, once the softmax warp has moved the previous ones to TMEM
        if (!(ok = mbar_wait_warp(bar_qe, (nq & 1) ^ 1, ctl, ab))) break;
        if (lane == 0) {
          mbar_expect_tx(bar_qf, static_cast<uint32_t>(C::NBOX * G * 128));
#pragma unroll
          for (int x = 0; x < C::NBOX; ++x)
            tma_load_3d(sbase + L::Q_OFF + x * L::Q_BOX_BYTES, &tm_q, x * 64, b * Hq + hk * G, 0, bar_qf);
        }
        ++nq;
        const int n_st = (t_end - t_begin + C::T - 1) / C::T;
        const int kv_z = b * Hkv + hk;
        for (int j = 0; j < n_st; ++j, ++st) {
          const int s = st % C::NSTAGE;
          if (!(ok = mbar_wait_warp(bar_empty + 8 * s, ((st / C::NSTAGE) & 1) ^ 1, ctl, ab))) break;
          if (ctl.inject == 1 && st == 1) {  // test hook: never fill this stage
            skipped = st;
            continue;
          }
          const int tok0 = t_begin + j * C::T;
          const int ntok = min(C::T, t_end - tok0);
          const uint32_t dst = sbase + s * C::STAGE_BYTES;
          if (lane == 0) {
            volatile int* rec = reinterpret_cast<volatile int*>(smem + L::META_OFF + s * 32);
            rec[0] = b;
            rec[1] = hk;
            rec[2] = split;
            rec[3] = j;
            rec[4] = n_st;
            rec[5] = tok0;
            rec[6] = ntok;
          }
          if constexpr (PAGED) {
            // pieces of min(page, 64) keys: a stage starts on a multiple of 64, so a piece
            // never crosses a page even when a stage (128 keys at D = 64) does
            const int P = pv.page_size;
            const int rows = P < kDecodeChunkAlign ? P : kDecodeChunkAlign;
            const int npiece = (ntok + rows - 1) / rows;  // at most T / 8 <= 16 (pages of 8 keys or more)
            if (lane == 0) mbar_expect_tx(bar_full + 8 * s, 2u * C::NBOX * npiece * rows * 128);
            __syncwarp();
            if (lane < npiece) {
              // An out-of-range page (a caller error) is sent past the end of the cache,
              // where the copy engine reads zeros.  HND view [pages x Hkv, page_size, D]:
              // (dim, row in page, page x Hkv + hk); NHD view [keys of all pages, Hkv, D]:
              // (dim, hk, key).
              const int t = tok0 + lane * rows;
              const int page = pv.block_table[static_cast<size_t>(b) * pv.max_pages + t / P];
              const bool bad = page < 0 || page >= pv.num_pages;
              const int y = pv.hnd ? t % P : hk;
              const int z = pv.hnd ? (bad ? pv.num_pages * Hkv : page * Hkv + hk)
                                   : (bad ? pv.num_pages * P : page * P + t % P);
#pragma unroll
              for (int x = 0; x < C::NBOX; ++x) {
                const uint32_t off = x * C::BOX_BYTES + lane * rows * 128;
                tma_load_3d(dst + off, &tm_k, x * 64, y, z, bar_full + 8 * s);
                tma_load_3d(dst + C::TILE_BYTES + off, &tm_v, x * 64, y, z, bar_full + 8 * s);
              }
            }
          } else {
            if (lane == 0) {
              mbar_expect_tx(bar_full + 8 * s, C::STAGE_BYTES);
#pragma unroll
              for (int x = 0; x < C::NBOX; ++x) {
                tma_load_3d(dst + x * C::BOX_BYTES, &tm_k, x * 64, tok0, kv_z, bar_full + 8 * s);
                tma_load_3d(dst + C::TILE_BYTES + x * C::BOX_BYTES, &tm_v, x * 64, tok0, kv_z, bar_full + 8 * s);
              }
            }
          }
          __syncwarp();
        }
      }
      if (!ok) break;
      if (lane == 0) {
        if (dynamic < 0) dynamic = static_cast<uint32_t>(ticket >> 32) == kDecodeSchedTag ? 1 : 0;
        if (dynamic) {
          item = static_cast<long long>(gridDim.x) + static_cast<uint32_t>(ticket);
          if (item < n_items) ticket = atomicAdd(sched, 1ull);
        } else {
          item = blockIdx.x + kk * static_cast<long long>(gridDim.x);
        }
      }
      item = __shfl_sync(0xffffffffu, item, 0);
    }
    // the end record
    bool ended = false;
    if (ok) {
      const int s = st % C::NSTAGE;
      if (mbar_wait_warp(bar_empty + 8 * s, ((st / C::NSTAGE) & 1) ^ 1, ctl, ab)) {
        if (lane == 0) {
          *reinterpret_cast<volatile int*>(smem + L::META_OFF + s * 32) = -1;
          mbar_arrive(bar_full + 8 * s);
        }
        ended = true;
      }
    }
    // Drain: never leave the CTA with copies still landing in its shared memory (after
    // the end record the stage it replaced has been consumed).
    if (lane == 0) {
      Abort no_abort{ab.flag + 1};
      for (int i = max(0, st - C::NSTAGE + (ended ? 1 : 0)); i < st; ++i)
        if (i != skipped) mbar_wait(bar_full + 8 * (i % C::NSTAGE), (i / C::NSTAGE) & 1, ctl, no_abort);
      if (nq > 0) mbar_wait(bar_qf, (nq - 1) & 1, ctl, no_abort);
    }
  } else if (warp == 2) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc_s = idesc_bf16(128, C::T, 0, 0);  // Q (TMEM) x K^T (K-major)
    constexpr uint32_t idesc_pv = idesc_bf16(128, D, 0, 1);    // P (TMEM) x V (MN-major)
    int nq = 0;
    for (int st = 0;; ++st) {
      const int s = st % C::NSTAGE;
      if (!mbar_wait_warp(bar_full + 8 * s, (st / C::NSTAGE) & 1, ctl, ab)) break;
      tc_fence_after();
      const volatile int* rec = reinterpret_cast<const volatile int*>(smem + L::META_OFF + s * 32);
      if (rec[0] < 0) break;  // no more items
      const int j = rec[3];
      if (j == 0) {  // an item's first stage: its q must be in TMEM
        if (!mbar_wait_warp(bar_q, nq & 1, ctl, ab)) break;
        tc_fence_after();
        ++nq;
      }
      const uint32_t kslot = sbase + s * C::STAGE_BYTES;
      // S = Q K^T (the previous stage's P.V, issued before, has read the P these columns
      // held: the MMAs of a CTA run in issue order)
#pragma unroll
      for (int x = 0; x < C::NBOX; ++x)
        mma_ts_kmaj_k64_el(tmem + C::S_COL, tmem + C::Q_COL + x * 32,
                           sdesc_sw128(kslot + x * C::BOX_BYTES, 16, 1024), idesc_s, x > 0 ? 1u : 0u);
      tc_commit_el(bar_s);
      if (!mbar_wait_warp(bar_p, st & 1, ctl, ab)) break;
      tc_fence_after();
      decode_tc_issue_pv<C>(tmem, kslot + C::TILE_BYTES, idesc_pv, j > 0);
      tc_commit_el(bar_o);
      tc_commit_el(bar_empty + 8 * s);
    }
    // every MMA issued above is done before TMEM is released
    Abort no_abort{ab.flag + 1};
    tc_commit_el(bar_drain);
    mbar_wait_warp(bar_drain, 0, ctl, no_abort);
  } else {
    // ------------------------------------------------------------ softmax (warp 0)
    decode_tc_persist_rows<D>(smem, o_part, lse_part, tmem, G, Hq, splits, c, bar_full, bar_qf, bar_qe, bar_q, bar_s,
                              bar_p, bar_o, ctl, ab);
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------- persistent forms
// Two persistent kernels share one body (decode_persistent_kernel):
//   CLUSTER = true: the single-kernel form.  Clusters of cs CTAs walk units (batch, kv
//     head, head group); CTA r of a cluster takes splits r, r + cs, ... of each unit and the
//     cluster merges its partials over distributed shared memory.
//   CLUSTER = false: the persistent split kernel of the split + merge form.  Each CTA walks
//     items (unit, split) and writes each item's partial (O_i, lse_i) to the workspace for
//     the merge kernel, exactly as decode_split_kernel does, but without a CTA launch, a
//     pipeline fill and a tail per item: the loader streams the next item's q and K/V
//     while the compute warps finish the current one.
// Both deal their work in a snake order over the sequences sorted by length (longest
// first), which evens out the work per cluster or CTA when lengths differ.
template <int D, int GT>
struct PersistSmem {
  using C = DecodeCfg<D>;
  static constexpr int kMaxSortedB = 256;  // sequences sorted by length for the dealing
  // ring first (16-byte aligned bulk-copy destinations), then the small arrays
  static constexpr uint32_t P_OFF = C::RING_BYTES;                        // [NCW][TW][GT] f32
  static constexpr uint32_t ALPHA_OFF = P_OFF + C::NCW * C::TW * GT * 4;  // [NCW][GT] f32
  static constexpr uint32_t WM_OFF = ALPHA_OFF + C::NCW * GT * 4;         // [NCW][GT] f32
  static constexpr uint32_t WL_OFF = WM_OFF + C::NCW * GT * 4;            // [NCW][GT] f32
  static constexpr uint32_t Q_OFF = (WL_OFF + C::NCW * GT * 4 + 15) / 16 * 16;  // [GT][D] bf16, q of an item
  static constexpr uint32_t PO_OFF = Q_OFF + GT * D * 2;                 // [GT][D] f32, the CTA's partial O
  static constexpr uint32_t PL_OFF = PO_OFF + GT * D * 4;                // [GT] f32, its log-sum-exps
  static constexpr uint32_t ORDER_OFF = (PL_OFF + GT * 4 + 15) / 16 * 16;  // [kMaxSortedB] int32
  static constexpr uint32_t BAR_OFF = ORDER_OFF + kMaxSortedB * 4;
  // full[NSTAGE], empty[NSTAGE], q_full, q_empty, ready, consumed
  static constexpr uint32_t ABORT_OFF = BAR_OFF + (2 * C::NSTAGE + 4) * 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16;
  static_assert(C::NCW * GT * D * 4 <= C::STAGE_BYTES, "the warps' merge fits in one ring slot");
  static_assert(C::CTAS_PER_SM * (BYTES + 1024) <= 228 * 1024, "CTAs per SM of the stage plan");
};

// The k-th work index of worker `w` of n_workers: a snake order over the sorted work
// (even rounds left to right, odd rounds right to left); -1 past the last.
__device__ __forceinline__ int snake_index(int kk, int w, int n_workers, int n_work) {
  const long long i = static_cast<long long>(kk) * n_workers + ((kk & 1) ? n_workers - 1 - w : w);
  return i < n_work ? static_cast<int>(i) : -1;
}

template <int D, int GT, bool PAGED, bool CLUSTER>
__global__ void __launch_bounds__(DecodeCfg<D>::THREADS, DecodeCfg<D>::CTAS_PER_SM)
    decode_persistent_kernel(const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ k,
                             const __nv_bfloat16* __restrict__ v, const int32_t* __restrict__ seqlens,
                             __nv_bfloat16* __restrict__ o, float* __restrict__ lse, float* __restrict__ o_part,
                             float* __restrict__ lse_part, int B, int Hq, int Hkv, int Skv, int splits,
                             int n_groups, float c, KernelCtl ctl, const __grid_constant__ CUtensorMap tm_k,
                             const __grid_constant__ CUtensorMap tm_v, PagedView pv) {
  using C = DecodeCfg<D>;
  using L = PersistSmem<D, GT>;
  extern __shared__ __align__(128) uint8_t smem[];
  // split + merge form: let the merge grid launch as soon as every CTA is resident
  if constexpr (!CLUSTER) asm volatile("griddepcontrol.launch_dependents;");
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int cs = CLUSTER ? static_cast<int>(cluster_nctarank()) : 1;
  const int rank = CLUSTER ? static_cast<int>(cluster_ctarank()) : 0;
  const int worker = static_cast<int>(blockIdx.x) / cs;         // cluster (or CTA) index
  const int n_workers = static_cast<int>(gridDim.x) / cs;
  const int G = Hq / Hkv;
  const int upb = Hkv * n_groups;  // units per sequence
  // work: units (cluster form; CTA r takes splits r, r + cs, ...) or (unit, split) items
  // ordered sequence (by length), then split, then unit
  const int per_seq = CLUSTER ? upb : upb * splits;
  const int n_work = B * per_seq;
  const int per_cta = CLUSTER ? splits / cs : 1;  // splits of a work piece this CTA streams

  const uint32_t s_base = smem_u32(smem);
  const uint32_t bar_full = s_base + L::BAR_OFF;
  const uint32_t bar_empty = bar_full + C::NSTAGE * 8;
  const uint32_t bar_qf = bar_empty + C::NSTAGE * 8;
  const uint32_t bar_qe = bar_qf + 8;
  const uint32_t bar_ready = bar_qe + 8;        // cluster form: every CTA's partial of the unit is written
  const uint32_t bar_consumed = bar_ready + 8;  // cluster form: every CTA has read this CTA's partial
  Abort ab{reinterpret_cast<volatile int*>(smem + L::ABORT_OFF)};

  // the sequences in order of decreasing length (ties by index): the dealing order
  int* order = reinterpret_cast<int*>(smem + L::ORDER_OFF);
  const bool sorted = seqlens != nullptr && B <= L::kMaxSortedB;
  if (sorted) {
    for (int bb = threadIdx.x; bb < B; bb += blockDim.x) {
      const int lb = seqlens[bb];
      int r = 0;
      for (int x = 0; x < B; ++x) {
        const int lx = seqlens[x];
        r += (lx > lb) || (lx == lb && x < bb);
      }
      order[r] = bb;
    }
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, C::NCW);
    }
    mbar_init(bar_qf, 1);
    mbar_init(bar_qe, C::NCW);
    mbar_init(bar_ready, cs);
    mbar_init(bar_consumed, cs);
    *ab.flag = 0;
    *(ab.flag + 1) = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if constexpr (CLUSTER) cluster_sync_all();  // every CTA's barriers exist before a peer arrives on them

  // work index i -> sequence, kv head, head group, first split, and the sequence's chunk
  struct Work {
    int b, hk, grp, h0, nh, len, chunk, split0;
  };
  auto work = [&](int i) {
    Work u;
    const int br = i / per_seq, rem = i % per_seq;
    const int j = CLUSTER ? rem : rem % upb;
    u.b = sorted ? order[br] : br;
    u.split0 = CLUSTER ? rank : rem / upb;
    u.hk = j / n_groups;
    u.grp = j % n_groups;
    u.h0 = u.hk * G + u.grp * GT;
    u.nh = min(GT, G - u.grp * GT);
    u.len = max(0, min(seqlens ? seqlens[u.b] : Skv, Skv));
    const int ch = (u.len + splits - 1) / splits;
    u.chunk = (ch + kDecodeChunkAlign - 1) / kDecodeChunkAlign * kDecodeChunkAlign;
    return u;
  };
  // keys [*t0, *t1) of this CTA's jj-th split of work u
  auto split_range = [&](const Work& u, int jj, int* t0, int* t1) {
    const int s = u.split0 + jj * cs;
    *t0 = min(s * u.chunk, u.len);
    *t1 = min(*t0 + u.chunk, u.len);
  };

  if (warp == C::NCW) {
    // ------------------------------------------------------------ loader warp (whole warp)
    PagedLoader pl;
    int pos = 0, skipped = -1, q_loads = 0;
    bool ok = true;
    for (int kk = 0, wi; ok && (wi = snake_index(kk, worker, n_workers, n_work)) >= 0; ++kk) {
      const Work u = work(wi);
      // the work's q rows (one bulk copy), once the compute warps have read the previous ones
      if (kk > 0 && !(ok = mbar_wait_warp(bar_qe, (kk - 1) & 1, ctl, ab))) break;
      if (lane == 0) {
        const uint32_t qbytes = static_cast<uint32_t>(u.nh) * D * 2;
        mbar_expect_tx(bar_qf, qbytes);
        bulk_g2s(s_base + L::Q_OFF, q + (static_cast<size_t>(u.b) * Hq + u.h0) * D, qbytes, bar_qf);
      }
      q_loads = kk + 1;
      if constexpr (PAGED) pl.reset();
      const size_t kv_row0 = (static_cast<size_t>(u.b) * Hkv + u.hk) * Skv;
      const int32_t* tbl = PAGED ? pv.block_table + static_cast<size_t>(u.b) * pv.max_pages : nullptr;
      for (int jj = 0; ok && jj < per_cta; ++jj) {
        int t0, t1;
        split_range(u, jj, &t0, &t1);
        for (int tok0 = t0; tok0 < t1; tok0 += C::T, ++pos) {
          const int slot = pos % C::NSTAGE, round = pos / C::NSTAGE;
          if (!(ok = mbar_wait_warp(bar_empty + 8 * slot, (round & 1) ^ 1, ctl, ab))) break;
          if (ctl.inject == 1 && pos == 1) {  // test hook: never fill this stage
            skipped = pos;
            continue;
          }
          const int ntok = min(C::T, t1 - tok0);
          const uint32_t dst = s_base + slot * C::STAGE_BYTES;
          if constexpr (PAGED) {
            pl.stage<D>(pv, tbl, Hkv, u.hk, tok0, ntok, dst, bar_full + 8 * slot, C::TILE_BYTES, &tm_k, &tm_v,
                        lane);
          } else if (lane == 0) {
            const uint32_t bytes = static_cast<uint32_t>(ntok) * D * 2;
            mbar_expect_tx(bar_full + 8 * slot, 2 * bytes);
            bulk_g2s(dst, k + (kv_row0 + tok0) * D, bytes, bar_full + 8 * slot);
            bulk_g2s(dst + C::TILE_BYTES, v + (kv_row0 + tok0) * D, bytes, bar_full + 8 * slot);
          }
        }
      }
    }
    // Drain: never leave the CTA with copies still landing in its shared memory.
    if (lane == 0) {
      Abort no_abort{ab.flag + 1};
      for (int it = max(0, pos - C::NSTAGE); it < pos; ++it)
        if (it != skipped) mbar_wait(bar_full + 8 * (it % C::NSTAGE), (it / C::NSTAGE) & 1, ctl, no_abort);
      if (q_loads > 0) mbar_wait(bar_qf, (q_loads - 1) & 1, ctl, no_abort);
    }
    __syncwarp();
  } else {
    // -------------------------------------------------------------- compute warps
    const LaneRole<D, GT> lr(lane);
    float* ps = reinterpret_cast<float*>(smem + L::P_OFF) + warp * C::TW * GT;
    float* alpha_s = reinterpret_cast<float*>(smem + L::ALPHA_OFF) + warp * GT;
    float* part_o = reinterpret_cast<float*>(smem + L::PO_OFF);
    float* part_l = reinterpret_cast<float*>(smem + L::PL_OFF);
    int pos = 0;
    // A failed (timed-out) wait is made known to all compute warps at the work piece's next
    // common point (a barrier reduction), so that they leave together and none is left
    // waiting at a barrier of the merge.
    for (int kk = 0, wi; (wi = snake_index(kk, worker, n_workers, n_work)) >= 0; ++kk) {
      const Work u = work(wi);
      bool ok = mbar_wait_warp(bar_qf, kk & 1, ctl, ab);
      float qf[GT][8];
      load_q<D, GT>(reinterpret_cast<const __nv_bfloat16*>(smem + L::Q_OFF), u.nh, lr.kl, c, qf);
      __syncwarp();
      if (ok && lane == 0) mbar_arrive(bar_qe);

      float m_run = -INFINITY, l_run = 0.f;
      float acc_o[GT][C::VD];
#pragma unroll
      for (int h = 0; h < GT; ++h)
#pragma unroll
        for (int d = 0; d < C::VD; ++d) acc_o[h][d] = 0.f;

      int n_st = 0;  // this CTA's stages of the work piece
      for (int jj = 0; jj < per_cta; ++jj) {
        int t0, t1;
        split_range(u, jj, &t0, &t1);
        n_st += (t1 - t0 + C::T - 1) / C::T;
      }
      int st = 0;
      for (int jj = 0; ok && jj < per_cta; ++jj) {
        int t0, t1;
        split_range(u, jj, &t0, &t1);
        for (int tok0 = t0; tok0 < t1; tok0 += C::T, ++pos, ++st) {
          const int slot = pos % C::NSTAGE;
          if (!(ok = mbar_wait_warp(bar_full + 8 * slot, (pos / C::NSTAGE) & 1, ctl, ab))) break;
          const uint8_t* ks = smem + slot * C::STAGE_BYTES;
          decode_stage<C, GT>(ks, ks + C::TILE_BYTES, min(C::T, t1 - tok0), warp, lane, lr, qf, m_run, l_run, acc_o,
                              ps, alpha_s);
          __syncwarp();
          // the last slot of the work piece stays held: it is the scratch of the merge below
          if (st + 1 < n_st && lane == 0) mbar_arrive(bar_empty + 8 * slot);
        }
      }
      // cluster form: this CTA's partial, once every CTA has read its previous one
      if (CLUSTER && ok && kk > 0) ok = mbar_wait_cluster_warp(bar_consumed, (kk - 1) & 1, ctl, ab);
      if (named_bar_any(1, C::NCW * 32, !ok)) break;
      const size_t part_row0 = (static_cast<size_t>(u.b) * Hq + u.h0) * splits + u.split0;  // split form
      if (n_st > 0) {
        const int last = (pos - 1) % C::NSTAGE;
        merge_warps<D, GT>(reinterpret_cast<float*>(smem + last * C::STAGE_BYTES),
                           reinterpret_cast<float*>(smem + L::WM_OFF), reinterpret_cast<float*>(smem + L::WL_OFF),
                           u.nh, warp, lane, lr, m_run, l_run, acc_o, [&](int idx, int h, int d, float ov, float lv) {
                             if constexpr (CLUSTER) {
                               part_o[idx] = ov;
                               if (d == 0) part_l[h] = lv;
                             } else {
                               const size_t row = part_row0 + static_cast<size_t>(h) * splits;
                               o_part[row * D + d] = ov;
                               if (d == 0) lse_part[row] = lv;
                             }
                           });
        asm volatile("bar.sync 1, %0;" ::"n"(C::NCW * 32) : "memory");  // partial written, slot read
        if (lane == 0) mbar_arrive(bar_empty + 8 * last);
      } else {  // no key of the work piece falls to this CTA
        for (int idx = threadIdx.x; idx < u.nh * D; idx += C::NCW * 32) {
          if constexpr (CLUSTER) {
            part_o[idx] = 0.f;
          } else {
            o_part[(part_row0 + static_cast<size_t>(idx / D) * splits) * D + idx % D] = 0.f;
          }
        }
        if (threadIdx.x < u.nh) {
          if constexpr (CLUSTER) {
            part_l[threadIdx.x] = -INFINITY;
          } else {
            lse_part[part_row0 + static_cast<size_t>(threadIdx.x) * splits] = -INFINITY;
          }
        }
        if constexpr (CLUSTER) asm volatile("bar.sync 1, %0;" ::"n"(C::NCW * 32) : "memory");
      }
      if constexpr (!CLUSTER) continue;

      if (static_cast<int>(threadIdx.x) < cs) mbar_arrive_cluster(map_shared_rank(bar_ready, threadIdx.x));
      ok = mbar_wait_cluster_warp(bar_ready, kk & 1, ctl, ab);
      if (named_bar_any(1, C::NCW * 32, !ok)) break;

      // gather, global softmax and final scaling of this CTA's share of the unit's outputs
      const int total = u.nh * D;
      const int per = (total + cs - 1) / cs;
      const int e1 = min(total, (rank + 1) * per);
      const size_t o_row0 = static_cast<size_t>(u.b) * Hq + u.h0;
      for (int e = rank * per + static_cast<int>(threadIdx.x); e < e1; e += C::NCW * 32) {
        const int h = e / D, d = e % D;
        float l[model::kMaxClusterSize];
        float M = -INFINITY;
#pragma unroll
        for (int i = 0; i < model::kMaxClusterSize; ++i) {
          l[i] = i < cs ? ld_dsmem_f32(map_shared_rank(s_base + L::PL_OFF + 4u * h, i)) : -INFINITY;
          M = fmaxf(M, l[i]);
        }
        float W = 0.f, acc = 0.f;
        if (M != -INFINITY) {
#pragma unroll
          for (int i = 0; i < model::kMaxClusterSize; ++i) {
            if (i < cs) {
              const float w = ex2((l[i] - M) * kLog2e);  // 0 for a CTA without keys
              W += w;
              acc = fmaf(w, ld_dsmem_f32(map_shared_rank(s_base + L::PO_OFF + 4u * e, i)), acc);
            }
          }
        }
        const bool any = W > 0.f;
        o[(o_row0 + h) * D + d] = __float2bfloat16_rn(any ? acc / W : 0.f);
        if (lse && d == 0) lse[o_row0 + h] = any ? M + log2f(W) * kLn2 : -INFINITY;
      }
      asm volatile("bar.sync 1, %0;" ::"n"(C::NCW * 32) : "memory");  // this CTA's reads are done
      if (static_cast<int>(threadIdx.x) < cs) mbar_arrive_cluster(map_shared_rank(bar_consumed, threadIdx.x));
    }
  }
  // Cluster form: leave together -- no CTA exits while a peer may still read its partial or
  // arrive on its barriers.
  if constexpr (CLUSTER) cluster_sync_all();
}

// One CTA (D threads) per (batch, query head).  The split log-sum-exps are read in
// parallel (one per thread), reduced, turned into weights in shared memory, and the
// partial rows are streamed with 8 independent loads in flight per thread.
template <int D>
__global__ void __launch_bounds__(D) decode_merge_kernel(const float* __restrict__ o_part,
                                                         const float* __restrict__ lse_part,
                                                         __nv_bfloat16* __restrict__ o,
                                                         float* __restrict__ lse, int splits,
                                                         unsigned long long* __restrict__ sched) {
  constexpr int NW = D / 32;
  __shared__ float w_s[kMaxDecodeSplits];
  __shared__ float red[NW];
  // Let the next kernel in the stream (the next call's split kernel) launch early; it
  // waits for this grid before it touches global memory.
  asm volatile("griddepcontrol.launch_dependents;");
  // Wait until the split kernel's partials are complete and visible.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // The split kernel has taken its last item: arm the workspace's item counter for the next call.
  if (sched != nullptr && blockIdx.x == 0 && threadIdx.x == 0)
    *sched = static_cast<unsigned long long>(kDecodeSchedTag) << 32;
  const int bh = blockIdx.x, d = threadIdx.x, lane = d & 31, wid = d >> 5;
  const float* lp = lse_part + static_cast<size_t>(bh) * splits;
  const float* op = o_part + static_cast<size_t>(bh) * splits * D + d;
  // Up to kMergeRegSplits splits, every partial of this thread's dimension is requested
  // before the weights are known, so the merge waits for one round trip to memory
  // instead of one per reduction step and per batch of partials.
  constexpr int kMergeRegSplits = 64;
  const bool in_regs = splits <= kMergeRegSplits;
  float pre[kMergeRegSplits];
  if (in_regs) {
#pragma unroll
    for (int i = 0; i < kMergeRegSplits; ++i) pre[i] = i < splits ? op[static_cast<size_t>(i) * D] : 0.f;
  }

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

  // the same order of additions either way: eight running sums over whole groups of
  // eight splits, the remainder into the first
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (in_regs) {
    const int full = splits & ~7;
#pragma unroll
    for (int i = 0; i < kMergeRegSplits; ++i) {
      if (i < full)
        acc[i & 7] = fmaf(w_s[i], pre[i], acc[i & 7]);
      else if (i < splits)
        acc[0] = fmaf(w_s[i], pre[i], acc[0]);
    }
  } else {
    int i = 0;
    for (; i + 8 <= splits; i += 8) {
#pragma unroll
      for (int u = 0; u < 8; ++u) acc[u] = fmaf(w_s[i + u], op[static_cast<size_t>(i + u) * D], acc[u]);
    }
    for (; i < splits; ++i) acc[0] = fmaf(w_s[i], op[static_cast<size_t>(i) * D], acc[0]);
  }
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
// kernel, clusters of up to 16 CTAs (beyond the portable 8).
template <class Kernel>
bool prepare_kernel(Kernel kernel, uint32_t smem, bool cluster, PerDeviceOnce& once) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  return once.run(dev, [&] {
    const void* fn = reinterpret_cast<const void*>(kernel);
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess) return false;
    return !cluster || cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess;
  });
}

template <int D, int GT, bool PAGED, class Cfg = DecodeCfg<D>>
bool prepare_split() {
  static PerDeviceOnce once;
  return prepare_kernel(decode_split_kernel<D, GT, PAGED, Cfg>, DecodeSmem<Cfg, GT>::BYTES, false, once);
}

template <int D, int GT, bool PAGED, bool CLUSTER>
bool prepare_persistent() {
  static PerDeviceOnce once;
  return prepare_kernel(decode_persistent_kernel<D, GT, PAGED, CLUSTER>, PersistSmem<D, GT>::BYTES, CLUSTER, once);
}

cudaLaunchConfig_t launch_config(dim3 grid, uint32_t smem, int cluster, cudaStream_t stream, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(DecodeCfg<128>::THREADS);
  static_assert(DecodeCfg<128>::THREADS == DecodeCfg<64>::THREADS, "one block shape");
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 0;
  if (cluster > 0) {
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(cluster);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.numAttrs = 1;
  }
  return cfg;
}

// Clusters of `cs` cluster-kernel CTAs that fit on the current device at once
// (cudaOccupancyMaxActiveClusters); 0 if none or the device cannot be asked.  Cached per
// device and cluster size.
template <int D, int GT, bool PAGED>
int max_clusters(int cs) {
  static std::atomic<int> cache[64][model::kMaxClusterSize + 1];  // value + 1 once known
  int dev = 0;
  if (cs < 1 || cs > model::kMaxClusterSize || cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 0;
  if (dev < 64) {
    const int c = cache[dev][cs].load(std::memory_order_relaxed);
    if (c != 0) return c - 1;
  }
  int clusters = 0;
  if (prepare_persistent<D, GT, PAGED, true>()) {
    cudaLaunchAttribute attr[1];
    const cudaLaunchConfig_t cfg = launch_config(dim3(cs * 64), PersistSmem<D, GT>::BYTES, cs, nullptr, attr);
    if (cudaOccupancyMaxActiveClusters(&clusters, decode_persistent_kernel<D, GT, PAGED, true>, &cfg) !=
        cudaSuccess) {
      cudaGetLastError();
      clusters = 0;
    }
  }
  if (dev < 64) cache[dev][cs].store(clusters + 1, std::memory_order_relaxed);
  return clusters;
}

// CTAs of the persistent split kernel resident on the current device at once (blocks per
// SM x SMs); 0 if the device cannot be asked.  Cached per device.
template <int D, int GT, bool PAGED>
int persistent_slots() {
  static std::atomic<int> cache[64];  // value + 1 once known
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 0;
  if (dev < 64) {
    const int c = cache[dev].load(std::memory_order_relaxed);
    if (c != 0) return c - 1;
  }
  int per_sm = 0, sms = 0;
  if (!prepare_persistent<D, GT, PAGED, false>() ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_persistent_kernel<D, GT, PAGED, false>,
                                                    DecodeCfg<D>::THREADS, PersistSmem<D, GT>::BYTES) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    per_sm = sms = 0;
  }
  if (dev < 64) cache[dev].store(per_sm * sms + 1, std::memory_order_relaxed);
  return per_sm * sms;
}

// Views of the K and V caches for the split kernels' loaders: paged caches as TMA tensors,
// contiguous caches need none (1-D bulk copies).
template <int D, bool PAGED>
bool kv_views(const DecodeArgs& a, const PagedKV* pk, CUtensorMap* tk, CUtensorMap* tv, PagedView* view) {
  *view = PagedView{nullptr, 0, 0, 0, 0};
  if constexpr (PAGED) {
    const int rows = pk->page_size < kDecodeChunkAlign ? pk->page_size : kDecodeChunkAlign;
    if (!paged_map(tk, a.k, *pk, a.Hkv, D, rows) || !paged_map(tv, a.v, *pk, a.Hkv, D, rows)) return false;
    *view = PagedView{pk->block_table, pk->page_size, pk->max_pages, pk->num_pages, pk->layout == kPagedHND ? 1 : 0};
  } else {
    (void)a;
    (void)pk;
    memset(tk, 0, sizeof(*tk));
    memset(tv, 0, sizeof(*tv));
  }
  return true;
}

template <int D, int GT, bool PAGED, class Cfg = DecodeCfg<D>>
cudaError_t launch_split(const DecodeArgs& a, const PagedKV* pk, const KernelCtl& ctl, cudaStream_t stream) {
  if (!prepare_split<D, GT, PAGED, Cfg>()) return cudaErrorInvalidValue;
  CUtensorMap tk, tv;
  PagedView view;
  if (!kv_views<D, PAGED>(a, pk, &tk, &tv, &view)) return cudaErrorInvalidValue;
  const int G = a.Hq / a.Hkv;
  const int n_groups = (G + GT - 1) / GT;
  dim3 grid(a.splits, a.Hkv * n_groups, a.B);
  decode_split_kernel<D, GT, PAGED, Cfg><<<grid, Cfg::THREADS, DecodeSmem<Cfg, GT>::BYTES, stream>>>(
      static_cast<const __nv_bfloat16*>(a.q), static_cast<const __nv_bfloat16*>(a.k),
      static_cast<const __nv_bfloat16*>(a.v), a.seqlens, a.o_part, a.lse_part, a.Hq, a.Hkv, a.Skv,
      a.splits, n_groups, a.scale * kLog2e, ctl, tk, tv, view);
  return cudaGetLastError();
}

// The contiguous cache [B, Hkv, Skv, D] as a 3-D tensor (dim, key, kv head of a sequence)
// in 64-dim x T-key boxes (T: the tensor-core stage's keys at this D), 128-byte swizzled:
// the tensor-core split kernels' K and V tiles.
bool kv_map_sw128(CUtensorMap* map, const void* cache, int B, int Hkv, int Skv, int D) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(Skv),
                        static_cast<cuuint64_t>(B) * Hkv};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(Skv) * D * 2};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(model::decode_tc_stage_keys(D)), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(cache), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Whether the tensor-core split kernel takes this decode: a contiguous cache, at most 32
// query heads per kv head, the model's stage plan.
bool decode_tc_eligible(const DecodeArgs& a) {
  const int G = a.Hq / a.Hkv;
  return a.tc != 0 && a.stage_plan == 0 && G <= DecodeTcCfg<128>::MAX_G && (a.D == 64 || a.D == 128);
}

template <int D>
cudaError_t launch_tc_split(const DecodeArgs& a, const KernelCtl& ctl, cudaStream_t stream) {
  using C = DecodeTcCfg<D>;
  static PerDeviceOnce once;
  if (!prepare_kernel(decode_tc_split_kernel<D>, C::BYTES, false, once)) return cudaErrorInvalidValue;
  CUtensorMap tk, tv;
  if (!kv_map_sw128(&tk, a.k, a.B, a.Hkv, a.Skv, D) || !kv_map_sw128(&tv, a.v, a.B, a.Hkv, a.Skv, D))
    return cudaErrorInvalidValue;
  dim3 grid(a.splits, a.Hkv, a.B);
  decode_tc_split_kernel<D><<<grid, C::THREADS, C::BYTES, stream>>>(
      static_cast<const __nv_bfloat16*>(a.q), a.seqlens, a.o_part, a.lse_part, a.Hq, a.Hkv, a.Skv, a.splits,
      a.scale * kLog2e, ctl, tk, tv);
  return cudaGetLastError();
}

// The queries [B * Hq rows, D] as a 3-D tensor (dim, row, 1) in 64-dim x G-row boxes,
// 128-byte swizzled: an item's q rows for the persistent tensor-core split kernel.
bool q_map_sw128(CUtensorMap* map, const void* q, int rows, int D, int G) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(rows), 1};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(rows) * D * 2};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(G), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// A paged cache as the paged loader's 3-D view (paged_map) in 64-dim boxes of `rows`
// keys, 128-byte swizzled: the persistent tensor-core split kernel's K/V pieces.
bool paged_map_sw128(CUtensorMap* map, const void* cache, const PagedKV& pk, int Hkv, int D, int rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  const bool hnd = pk.layout == kPagedHND;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(hnd ? pk.page_size : Hkv),
                        static_cast<cuuint64_t>(pk.num_pages) * (hnd ? Hkv : pk.page_size)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(hnd ? pk.page_size : Hkv) * D * 2};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(hnd ? rows : 1), static_cast<cuuint32_t>(hnd ? 1 : rows)};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(cache), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The persistent tensor-core split kernel: two CTAs per SM (or one per item when fewer).
template <int D, bool PAGED>
cudaError_t launch_tc_persist(const DecodeArgs& a, const PagedKV* pk, const KernelCtl& ctl, cudaStream_t stream) {
  using L = DecodeTcPersistCfg<D>;
  if (a.sched == nullptr) return cudaErrorInvalidValue;
  static PerDeviceOnce once;
  if (!prepare_kernel(decode_tc_persist_kernel<D, PAGED>, L::BYTES, false, once)) return cudaErrorInvalidValue;
  const int G = a.Hq / a.Hkv;
  CUtensorMap tq, tk, tv;
  PagedView view{nullptr, 0, 0, 0, 0};
  if (!q_map_sw128(&tq, a.q, a.B * a.Hq, D, G)) return cudaErrorInvalidValue;
  if constexpr (PAGED) {
    const int rows = pk->page_size < kDecodeChunkAlign ? pk->page_size : kDecodeChunkAlign;
    if (!paged_map_sw128(&tk, a.k, *pk, a.Hkv, D, rows) || !paged_map_sw128(&tv, a.v, *pk, a.Hkv, D, rows))
      return cudaErrorInvalidValue;
    view = PagedView{pk->block_table, pk->page_size, pk->max_pages, pk->num_pages, pk->layout == kPagedHND ? 1 : 0};
  } else {
    if (!kv_map_sw128(&tk, a.k, a.B, a.Hkv, a.Skv, D) || !kv_map_sw128(&tv, a.v, a.B, a.Hkv, a.Skv, D))
      return cudaErrorInvalidValue;
  }
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                cudaSuccess)
    return cudaErrorInvalidValue;
  const long long items = static_cast<long long>(a.B) * a.Hkv * a.splits;
  const long long ctas = items < 2LL * sms ? items : 2LL * sms;
  // programmatic dependent launch: the CTAs set up their barriers and TMEM while the
  // previous kernel in the stream finishes (the kernel waits for it before any global access)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(ctas));
  cfg.blockDim = dim3(DecodeTcCfg<D>::THREADS);
  cfg.dynamicSmemBytes = L::BYTES;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decode_tc_persist_kernel<D, PAGED>, a.seqlens, a.o_part, a.lse_part, a.sched, a.B,
                            a.Hq, a.Hkv, a.Skv, a.splits, a.scale * kLog2e, ctl, tq, tk, tv, view);
}

template <int D, int GT, bool PAGED, bool CLUSTER>
cudaError_t launch_persistent_kernel(const DecodeArgs& a, dim3 grid, int cs, const PagedKV* pk, const KernelCtl& ctl,
                                     cudaStream_t stream) {
  if (!prepare_persistent<D, GT, PAGED, CLUSTER>()) return cudaErrorInvalidConfiguration;
  CUtensorMap tk, tv;
  PagedView view;
  if (!kv_views<D, PAGED>(a, pk, &tk, &tv, &view)) return cudaErrorInvalidValue;
  const int G = a.Hq / a.Hkv;
  const int n_groups = (G + GT - 1) / GT;
  cudaLaunchAttribute attr[1];
  const cudaLaunchConfig_t cfg = launch_config(grid, PersistSmem<D, GT>::BYTES, CLUSTER ? cs : 0, stream, attr);
  return cudaLaunchKernelEx(&cfg, decode_persistent_kernel<D, GT, PAGED, CLUSTER>,
                            static_cast<const __nv_bfloat16*>(a.q), static_cast<const __nv_bfloat16*>(a.k),
                            static_cast<const __nv_bfloat16*>(a.v), a.seqlens, static_cast<__nv_bfloat16*>(a.o),
                            a.lse, a.o_part, a.lse_part, a.B, a.Hq, a.Hkv, a.Skv, a.splits, n_groups,
                            a.scale * kLog2e, ctl, tk, tv, view);
}

// The cluster kernel with clusters of cs CTAs: as many clusters as fit at once, at most one
// per unit.
template <int D, int GT, bool PAGED>
cudaError_t launch_cluster(const DecodeArgs& a, int cs, const PagedKV* pk, const KernelCtl& ctl,
                           cudaStream_t stream) {
  const int fit = max_clusters<D, GT, PAGED>(cs);
  if (fit < 1) return cudaErrorInvalidConfiguration;
  const int G = a.Hq / a.Hkv;
  const long long units = static_cast<long long>(a.B) * a.Hkv * ((G + GT - 1) / GT);
  const long long n_clusters = units < fit ? units : fit;
  return launch_persistent_kernel<D, GT, PAGED, true>(a, dim3(static_cast<unsigned>(n_clusters * cs)), cs, pk, ctl,
                                                      stream);
}

// The persistent split kernel: as many CTAs as fit at once, evened out so that every CTA
// walks the same number of (unit, split) items (the last round is the only short one).
template <int D, int GT, bool PAGED>
cudaError_t launch_persist(const DecodeArgs& a, const PagedKV* pk, const KernelCtl& ctl, cudaStream_t stream) {
  const int slots = persistent_slots<D, GT, PAGED>();
  if (slots < 1) return cudaErrorInvalidConfiguration;
  const int G = a.Hq / a.Hkv;
  const long long items = static_cast<long long>(a.B) * a.Hkv * ((G + GT - 1) / GT) * a.splits;
  const long long per = (items + slots - 1) / slots;
  const long long ctas = (items + per - 1) / per;
  return launch_persistent_kernel<D, GT, PAGED, false>(a, dim3(static_cast<unsigned>(ctas)), 1, pk, ctl, stream);
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
                            static_cast<__nv_bfloat16*>(a.o), a.lse, a.splits, a.sched);
}

// The Flash Decode form of a launch: kDecodeSplitMerge, kDecodePersistent (both with the
// merge kernel) or kDecodeCluster with *cs CTAs per cluster.  A split count the caller fixed
// runs the split + merge form; a split count the model chose comes with the model's form
// (Eq. 9 over the forms at that count, which is the form of the joint argmin).  a.form
// pins a form (a pinned form that cannot run falls back to the rule above); a.cluster pins
// the cluster size (when it divides the split count and such clusters fit).
template <int D, int GT, bool PAGED>
int decode_form(const DecodeArgs& a, int* cs_out) {
  *cs_out = 0;
  if (a.form == 0 && !a.by_model) return kDecodeSplitMerge;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                cudaSuccess)
    return kDecodeSplitMerge;
  const int slots = persistent_slots<D, GT, PAGED>();
  const model::DecodeClusterChoice ch = model::choose_decode_cluster(
      a.splits, a.B, a.Hq, a.Hkv, a.Skv, D, [](int cs) { return max_clusters<D, GT, PAGED>(cs); }, a.cluster);
  if (a.form == kDecodeSplitMerge) return kDecodeSplitMerge;
  if (a.form == kDecodePersistent && slots > 0) return kDecodePersistent;
  if (a.form == kDecodeCluster && ch.cs > 0) {
    *cs_out = ch.cs;
    return kDecodeCluster;
  }
  // Where the split + merge form's split kernel runs on the tensor cores it is priced as
  // such, and the CUDA-core persistent split kernel (the same schedule with a slower
  // stage, measured slower or equal on every shape) is not a candidate.
  const bool tc = decode_tc_eligible(a) && !(PAGED && a.tc == 2);
  const double t_split = tc ? model::decode_tc_time_us(a.splits, a.B, a.Hq, a.Hkv, a.Skv, D, sms)
                            : model::decode_time_us(a.splits, a.B, a.Hq, a.Hkv, a.Skv, D, sms);
  const double t_persist =
      (slots > 0 && !tc) ? model::decode_persistent_time_us(a.splits, a.B, a.Hq, a.Hkv, a.Skv, D, slots) : 1e300;
  int form = kDecodeSplitMerge;
  double best = t_split;
  if (t_persist < best * (1.0 - 1e-9)) {
    form = kDecodePersistent;
    best = t_persist;
  }
  if (ch.cs > 0 && ch.t_us < best * (1.0 - 1e-9)) {
    form = kDecodeCluster;
    *cs_out = ch.cs;
  }
  return form;
}

// Stage plans compiled beside the model's for the block-size ablation (contiguous cache,
// D = 128, four query heads per CTA, split + merge form): {tokens per stage, stages, CTAs
// per SM}; index + 1 is DecodeArgs::stage_plan.
constexpr int kDecodeAblationPlans[][3] = {{32, 2, 2}, {32, 3, 2}, {32, 4, 2}, {64, 2, 2},
                                           {64, 4, 1}, {128, 2, 1}, {128, 3, 1}};

template <int I>
cudaError_t launch_ablation_split(const DecodeArgs& a, const KernelCtl& ctl, cudaStream_t stream) {
  constexpr const int* P = kDecodeAblationPlans[I];
  return launch_split<128, 4, false, DecodeCfg<128, P[0], P[1], P[2]>>(a, nullptr, ctl, stream);
}

cudaError_t launch_ablation(const DecodeArgs& a, const KernelCtl& ctl, cudaStream_t stream) {
  cudaError_t e;
  switch (a.stage_plan) {
    case 1: e = launch_ablation_split<0>(a, ctl, stream); break;
    case 2: e = launch_ablation_split<1>(a, ctl, stream); break;
    case 3: e = launch_ablation_split<2>(a, ctl, stream); break;
    case 4: e = launch_ablation_split<3>(a, ctl, stream); break;
    case 5: e = launch_ablation_split<4>(a, ctl, stream); break;
    case 6: e = launch_ablation_split<5>(a, ctl, stream); break;
    default: e = launch_ablation_split<6>(a, ctl, stream); break;
  }
  if (e != cudaSuccess) return e;
  return launch_merge<128>(a, stream);
}

template <int D, int GT, bool PAGED>
cudaError_t launch_form(const DecodeArgs& a, const PagedKV* pk, const KernelCtl& ctl, cudaStream_t stream) {
  if (D == 128 && GT == 4 && !PAGED && a.stage_plan > 0) return launch_ablation(a, ctl, stream);
  int cs = 0;
  const int form = decode_form<D, GT, PAGED>(a, &cs);
  if (form == kDecodeCluster) return launch_cluster<D, GT, PAGED>(a, cs, pk, ctl, stream);
  cudaError_t e;
  if (form == kDecodePersistent)
    e = launch_persist<D, GT, PAGED>(a, pk, ctl, stream);
  else if (decode_tc_eligible(a) && !(PAGED && a.tc == 2))
    e = a.tc == 2 ? launch_tc_split<D>(a, ctl, stream) : launch_tc_persist<D, PAGED>(a, pk, ctl, stream);
  else
    e = launch_split<D, GT, PAGED>(a, pk, ctl, stream);
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
int decode_form_d(const DecodeArgs& a, int* cs) {
  const int G = a.Hq / a.Hkv;
  if (G >= 8) return decode_form<D, 8, PAGED>(a, cs);
  if (G >= 4) return decode_form<D, 4, PAGED>(a, cs);
  if (G >= 2) return decode_form<D, 2, PAGED>(a, cs);
  return decode_form<D, 1, PAGED>(a, cs);
}

template <int D>
int persistent_slots_d(int G) {
  if (G >= 8) return persistent_slots<D, 8, false>();
  if (G >= 4) return persistent_slots<D, 4, false>();
  if (G >= 2) return persistent_slots<D, 2, false>();
  return persistent_slots<D, 1, false>();
}

template <int D>
int max_clusters_d(int G, int cs) {
  if (G >= 8) return max_clusters<D, 8, false>(cs);
  if (G >= 4) return max_clusters<D, 4, false>(cs);
  if (G >= 2) return max_clusters<D, 2, false>(cs);
  return max_clusters<D, 1, false>(cs);
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

int decode_form_of(const DecodeArgs& a, bool paged, int* cs) {
  if (a.D == 128) return paged ? decode_form_d<128, true>(a, cs) : decode_form_d<128, false>(a, cs);
  return paged ? decode_form_d<64, true>(a, cs) : decode_form_d<64, false>(a, cs);
}

int decode_persistent_slots(int D, int G) { return D == 128 ? persistent_slots_d<128>(G) : persistent_slots_d<64>(G); }

int decode_max_clusters(int D, int G, int cs) { return D == 128 ? max_clusters_d<128>(G, cs) : max_clusters_d<64>(G, cs); }

int decode_ablation_plan(int tokens, int stages, int ctas_per_sm) {
  for (int i = 0; i < static_cast<int>(sizeof(kDecodeAblationPlans) / sizeof(kDecodeAblationPlans[0])); ++i)
    if (kDecodeAblationPlans[i][0] == tokens && kDecodeAblationPlans[i][1] == stages &&
        kDecodeAblationPlans[i][2] == ctas_per_sm)
      return i + 1;
  return 0;
}

}  // namespace loom
