// Flash Attention prefill for GB300 (sm_103a): TMA + mbarrier ring, tcgen05 MMAs with
// TMEM accumulators, warp-specialised loader / MMA / softmax roles.
//
// Paper: Sec. 3.2.2 evaluates Flash Attention as one fused kernel for the score product,
// the softmax and the weighted sum of values; the pipelining of its load, compute and store stages through
// counted circular buffers is the virtual-buffer protocol of Sec. 2.3, and the tile and
// stage constants come from the latency model of Sec. 2.6 (Eq. 6-9, in model.h).
//
// One CTA owns NQT = 2 query tiles of BM = 128 rows (tile 0 and tile 1) of one
// (batch, query head) and walks the key/value sequence in tiles of BN = 128 rows:
//
//   warp 8 (loader, 1 thread)   Q0, Q1 once; then K_0, V_0, K_1, V_1, ... into an
//                               NSLOT-deep ring of 128B-swizzled shared-memory slots
//   warp 9 (MMA, whole warp,    S_t = Q_t K_j^T          (SS MMA, fp32 in TMEM)
//     one elected lane issues)
//                               O_t += P_t V_j           (TS MMA: P read from TMEM)
//                               issue order S0 S1 | PV0 S0' | PV1 S1' | ... so the
//                               tensor pipe works on one tile while the other tile's
//                               softmax runs
//   warps 0-3 / 4-7 (softmax)   one thread per query row of tile 0 / tile 1: read the
//                               S row from TMEM, mask, online softmax in base 2 with a
//                               lazily moved running max, write P (bf16) back over S,
//                               rescale O in TMEM on the rare max jumps, and finally
//                               normalise O, store it (bf16) and the log-sum-exp.
//
// TMEM (512 columns): [0,128) S0/P0 | [128,256) S1/P1 | [256,256+D) O0 | [256+D, 256+2D) O1.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cmath>
#include <cstring>
#include <mutex>

#include "kernels.h"
#include "varlen.h"
#include "model.h"
#include "ptx.cuh"

namespace loom {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleThreshold = 8.0f;  // base-2 units; P <= 2^8 between rescales

// Tile and stage constants: the analytic model's argmin for this head dimension.  SLOTS
// other than 0 overrides the ring depth (the neighbours of the model's choice, measured by
// the block-size ablation; 2 slots leave the loader no tile of look-ahead but cannot
// deadlock: every slot the MMA warp waits for is released earlier in its own order).
template <int D, int SLOTS = 0>
struct FwdCfg {
  static constexpr model::FwdPlan kPlan = model::fwd_plan_variant(D, 2);
  static_assert(kPlan.feasible, "no feasible two-tile prefill schedule");
  static constexpr int BM = kPlan.bm;         // rows per query tile (= TMEM lanes)
  static constexpr int NQT = kPlan.q_tiles;   // query tiles per CTA
  static constexpr int BN = kPlan.bn;         // keys per KV tile
  static constexpr int NSLOT = SLOTS ? SLOTS : kPlan.kv_slots;  // K/V ring slots
  static_assert(BM == 128 && NQT == 2, "warp roles assume two 128-row query tiles");
  static_assert(BN == 128, "softmax holds one S row of 128 fp32 in registers, P leaves in two 64-key halves");
  static_assert(kPlan.b_lm == 1 && NSLOT >= 2, "a K and a V slot at least");
  static constexpr int THREADS = 320;               // 8 softmax warps + loader + MMA
  static constexpr int BOX_COLS = 64;               // 128-byte swizzle atom = 64 bf16
  static constexpr int NBOX = D / BOX_COLS;         // TMA boxes per row of a tile
  static constexpr uint32_t Q_BOX_BYTES = BM * 128;
  static constexpr uint32_t Q_TILE_BYTES = NBOX * Q_BOX_BYTES;
  static constexpr uint32_t KV_BOX_BYTES = BN * 128;
  static constexpr uint32_t SLOT_BYTES = NBOX * KV_BOX_BYTES;
  static constexpr uint32_t Q_OFF = 0;
  static constexpr uint32_t RING_OFF = NQT * Q_TILE_BYTES;
  static constexpr uint32_t STG_OFF = RING_OFF + NSLOT * SLOT_BYTES;  // O staging per tile
  static constexpr uint32_t BAR_OFF = STG_OFF + NQT * BM * D * 2;
  // barriers: q_full[2], q_empty[2], full[NSLOT], empty[NSLOT], s[2], p[2][2], o[2], o_empty[2], drain
  static constexpr int NBAR = 4 + 2 * NSLOT + 11;
  static constexpr uint32_t TMEM_PTR_OFF = BAR_OFF + NBAR * 8;
  static constexpr uint32_t ABORT_OFF = TMEM_PTR_OFF + 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16 + 1024;  // + alignment slack
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t S_COL = 0;        // + t * BN
  static constexpr uint32_t O_COL = 2 * BN;   // + t * D
  static_assert(BYTES <= 227 * 1024, "shared memory budget");
  static_assert(O_COL + NQT * D <= TMEM_COLS, "TMEM budget");
};

struct FwdParams {
  __nv_bfloat16* o;
  float* lse;
  int Hq, Hkv, Sq, Skv;
  int n_pairs;   // query-tile pairs per (b, h)
  int n_items;   // n_pairs * B * Hq work items
  int plane_block;  // causal: (b, h) planes per block of the work order
  int last_h0;      // causal: first plane of the final block (which may be larger)
  int causal;
  float c;       // scale * log2(e)
  KernelCtl ctl;
  // ragged batches (Q/K/V/O packed [total, H, D]; unused by the dense instantiations)
  const int32_t* cu_q;  // [B + 1] first query token of each sequence
  const int32_t* cu_k;  // [B + 1] first key token of each sequence
  int B, total_q;       // sequences; query tokens (the row stride of LSE [Hq, total_q])
};

// One work item of a persistent CTA: a pair of 128-row query tiles of one (b, h).
struct Item {
  int b, h, q_z, kv_z, q0, n_tiles0, n_tiles;
  int sq, skv, qb, kb;  // ragged batches: the sequence's lengths and first tokens
};

// The r-th item of this CTA (-1 once it has none left).  Causal items are ordered
// heaviest first (within blocks of planes, see item_coords) and dealt out in a snake
// order (CTA c takes item c of even rounds and item G-1-c of odd rounds) so that long and
// short items even out per CTA.
__device__ __forceinline__ int item_index(const FwdParams& p, int r) {
  const int G = static_cast<int>(gridDim.x), c = static_cast<int>(blockIdx.x);
  const long long idx = static_cast<long long>(r) * G + ((p.causal && (r & 1)) ? G - 1 - c : c);
  return idx < p.n_items ? static_cast<int>(idx) : -1;
}

// Item idx -> (position pos of its query tile or tile pair within the plane, plane bh).
// Non-causal: consecutive items are consecutive positions of one plane (they share its
// K/V in L2).  Causal: blocks of p.plane_block planes, the final block running from plane
// p.last_h0 to the end; within a block the bottom (longest) positions of every plane go
// first.
__device__ __forceinline__ void item_coords(const FwdParams& p, int idx, int& pos, int& bh) {
  if (p.causal) {
    const int BH = p.n_items / p.n_pairs;
    int h0, nb, in;
    if (idx >= p.last_h0 * p.n_pairs) {  // the final block: planes [last_h0, BH)
      h0 = p.last_h0;
      nb = BH - h0;
      in = idx - h0 * p.n_pairs;
    } else {
      const int per_block = p.plane_block * p.n_pairs;
      const int blk = idx / per_block;
      h0 = blk * p.plane_block;
      nb = p.plane_block;
      in = idx - blk * per_block;
    }
    pos = p.n_pairs - 1 - in / nb;
    bh = h0 + in % nb;
  } else {
    pos = idx % p.n_pairs;
    bh = idx / p.n_pairs;
  }
}

template <int D>
__device__ __forceinline__ Item make_item(const FwdParams& p, int idx) {
  using C = FwdCfg<D>;
  int pair, bh;
  item_coords(p, idx, pair, bh);
  Item it;
  it.h = bh % p.Hq;
  it.b = bh / p.Hq;
  it.q_z = bh;
  it.kv_z = it.b * p.Hkv + it.h / (p.Hq / p.Hkv);
  it.q0 = pair * (C::NQT * C::BM);
  // KV tiles each query tile needs (causal: up to the diagonal of its last row); the
  // CTA loads the union, i.e. tile 1's range.
  const int off = p.Skv - p.Sq;  // bottom-right causal offset
  int n_kv0 = p.Skv, n_kv1 = p.Skv;
  if (p.causal) {
    n_kv0 = min(p.Skv, it.q0 + C::BM + off);
    n_kv1 = min(p.Skv, it.q0 + 2 * C::BM + off);
  }
  it.n_tiles0 = (n_kv0 + C::BN - 1) / C::BN;
  it.n_tiles = (n_kv1 + C::BN - 1) / C::BN;
  return it;
}

// ---------------------------------------------------------------- ragged batches
// Items are (sequence, head, query-tile pair) in sequence order; sequence b, with sq_b
// query rows, owns ceil(sq_b / rows_per_item) pairs per head.  Every role walks its items
// with a cursor over the sequence offsets -- a CTA's item indices only grow -- so no item
// list is stored and an empty sequence costs one step of the cursor.
struct SeqCursor {
  int b;            // sequence of the last located item
  long long first;  // index of that sequence's first item
  int pairs;        // its query-tile pairs per head
};

template <int ROWS>
__device__ __forceinline__ int seq_pairs(const FwdParams& p, int b) {
  const int sq = p.cu_q[b + 1] - p.cu_q[b];
  return sq > 0 ? (sq + ROWS - 1) / ROWS : 0;
}

template <int ROWS>
__device__ __forceinline__ SeqCursor seq_cursor(const FwdParams& p) {
  return SeqCursor{0, 0, p.B > 0 ? seq_pairs<ROWS>(p, 0) : 0};
}

// Dense: the r-th item's index (see item_index).  Ragged: the same dealing over the
// unbounded index space, with the cursor moved to the item's sequence; -1 past the last.
template <int ROWS, bool VARLEN>
__device__ __forceinline__ int item_index_t(const FwdParams& p, int r, SeqCursor& cur) {
  if constexpr (!VARLEN) {
    (void)cur;
    return item_index(p, r);
  } else {
    const int G = static_cast<int>(gridDim.x), c = static_cast<int>(blockIdx.x);
    const long long idx = static_cast<long long>(r) * G + ((p.causal && (r & 1)) ? G - 1 - c : c);
    while (cur.b < p.B && idx >= cur.first + static_cast<long long>(cur.pairs) * p.Hq) {
      cur.first += static_cast<long long>(cur.pairs) * p.Hq;
      ++cur.b;
      cur.pairs = cur.b < p.B ? seq_pairs<ROWS>(p, cur.b) : 0;
    }
    return cur.b < p.B ? static_cast<int>(idx) : -1;
  }
}

// Ragged item: causal takes a sequence's heaviest pairs (last rows) first over all heads;
// non-causal takes one head's pairs in a row (they share its K/V in L2).  At least one KV
// tile is processed even when no key is visible (fully masked: O = 0, LSE = -inf).
template <int D, bool VARLEN>
__device__ __forceinline__ Item make_item_t(const FwdParams& p, const SeqCursor& cur, int idx) {
  using C = FwdCfg<D>;
  if constexpr (!VARLEN) {
    (void)cur;
    return make_item<D>(p, idx);
  } else {
    const int in = static_cast<int>(idx - cur.first);
    int pos, h;
    if (p.causal) {
      pos = cur.pairs - 1 - in / p.Hq;
      h = in % p.Hq;
    } else {
      pos = in % cur.pairs;
      h = in / cur.pairs;
    }
    Item it;
    it.b = cur.b;
    it.h = h;
    it.q_z = h;
    it.kv_z = h / (p.Hq / p.Hkv);
    it.qb = p.cu_q[cur.b];
    it.sq = p.cu_q[cur.b + 1] - it.qb;
    it.kb = p.cu_k[cur.b];
    it.skv = p.cu_k[cur.b + 1] - it.kb;
    it.q0 = pos * (C::NQT * C::BM);
    const int off = it.skv - it.sq;
    int n_kv0 = it.skv, n_kv1 = it.skv;
    if (p.causal) {
      n_kv0 = min(it.skv, it.q0 + C::BM + off);
      n_kv1 = min(it.skv, it.q0 + 2 * C::BM + off);
    }
    it.n_tiles0 = max(1, (n_kv0 + C::BN - 1) / C::BN);
    it.n_tiles = max(it.n_tiles0, (n_kv1 + C::BN - 1) / C::BN);
    return it;
  }
}

// One online-softmax step of one query row (this thread's TMEM lane) over a BN-key
// tile of S in TMEM at s_tm: wait for S, mask keys >= limit, move the running max
// lazily, write P = 2^(S*c - m) as bf16 over the first half of the S columns in two
// halves (arriving on bar_p and bar_p + 8 after each, so that P.V can start on the first
// half), rescale O at o_tm when the max moved (after waiting for the previous P.V on
// bar_o with parity par_o), and accumulate the row sum.  Returns false if a wait gave up.
template <int D, int BN>
__device__ __forceinline__ bool softmax_step(uint32_t s_tm, uint32_t o_tm, uint32_t bar_s,
                                             uint32_t par_s, uint32_t bar_p, uint32_t bar_o,
                                             uint32_t par_o, bool first, int kbase, int limit,
                                             float c, uint64_t c2, float& m_run, float& l_run,
                                             const KernelCtl& ctl, const Abort& ab) {
  if (!mbar_wait_warp(bar_s, par_s, ctl, ab)) return false;
  tc_fence_after();
  uint32_t s[BN];
#pragma unroll
  for (int ch = 0; ch < BN / 32; ++ch) tmem_ld32(s_tm + ch * 32, s + ch * 32);
  tmem_wait_ld();
#pragma unroll
  for (int ch = 0; ch < BN / 32; ++ch) reg_fence32(s + ch * 32);
  if (kbase + BN > limit) {
#pragma unroll
    for (int i = 0; i < BN; ++i)
      if (kbase + i >= limit) s[i] = __float_as_uint(-INFINITY);
  }
  // row max: 8 independent chains of 3-input max, then a small tree
  float mx;
  {
    float mm[8];
#pragma unroll
    for (int g = 0; g < 8; ++g) mm[g] = __uint_as_float(s[g]);
#pragma unroll
    for (int i = 8; i + 16 <= BN; i += 16)
#pragma unroll
      for (int g = 0; g < 8; ++g)
        mm[g] = max3(mm[g], __uint_as_float(s[i + g]), __uint_as_float(s[i + 8 + g]));
    if constexpr ((BN - 8) % 16 != 0) {
#pragma unroll
      for (int g = 0; g < 8; ++g) mm[g] = fmaxf(mm[g], __uint_as_float(s[BN - 8 + g]));
    }
    mx = fmaxf(max3(mm[0], mm[1], mm[2]), max3(max3(mm[3], mm[4], mm[5]), mm[6], mm[7]));
  }
  const float m_new = fmaxf(m_run, mx * c);
  const bool need = m_new > m_run + kRescaleThreshold;
  const float alpha = need ? ex2(m_run - m_new) : 1.f;
  if (need) m_run = m_new;
  const float ms = (m_run == -INFINITY) ? 0.f : m_run;
  const uint64_t nms2 = f2(-ms, -ms);
  // p = 2^(s*c - m): packed FMA, one MUFU ex2 per score, 4 packed partial sums.  P leaves
  // in two halves of H0 and BN - H0 keys (64 + 64, or 64 + 32 for 96-key tiles), each
  // written as packed bf16 pairs over the first columns of its keys' S.
  static_assert(BN == 128 || BN == 96, "P halves of 64 + 64 or 64 + 32 keys");
  constexpr int H0 = 64;
  uint64_t acc[4] = {0, 0, 0, 0};
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int k0 = half == 0 ? 0 : H0;
    const int nk = half == 0 ? H0 : BN - H0;
    uint32_t pk[H0 / 2];
#pragma unroll
    for (int i = 0; i < H0 / 2; ++i) {
      if (i < nk / 2) {
        const int e = k0 + 2 * i;
        const uint64_t x = fma2(f2(__uint_as_float(s[e]), __uint_as_float(s[e + 1])), c2, nms2);
        const float p0 = ex2(f2lo(x));
        const float p1 = ex2(f2hi(x));
        acc[i & 3] = add2(acc[i & 3], f2(p0, p1));
        pk[i] = pack_bf16x2(p0, p1);
      }
    }
    if (nk == 64)
      tmem_st32(s_tm + k0 / 2, pk);
    else
      tmem_st16(s_tm + k0 / 2, pk);
    tmem_wait_st();
    // O must hold the previous P.V before it is rescaled, and be rescaled before this
    // tile's P.V starts (the first-half arrive below).
    if (half == 0 && !first && __any_sync(0xffffffffu, need)) {
      if (!mbar_wait_warp(bar_o, par_o, ctl, ab)) return false;
      tc_fence_after();
      const uint64_t a2 = f2(alpha, alpha);
#pragma unroll 1
      for (int ch = 0; ch < D / 32; ++ch) {
        uint32_t rr[32];
        tmem_ld32(o_tm + ch * 32, rr);
        tmem_wait_ld();
        reg_fence32(rr);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const uint64_t x = mul2(f2(__uint_as_float(rr[2 * i]), __uint_as_float(rr[2 * i + 1])), a2);
          rr[2 * i] = __float_as_uint(f2lo(x));
          rr[2 * i + 1] = __float_as_uint(f2hi(x));
        }
        tmem_st32(o_tm + ch * 32, rr);
      }
      tmem_wait_st();
    }
    tc_fence_before();
    mbar_arrive(bar_p + 8 * half);
  }
  const uint64_t a01 = add2(add2(acc[0], acc[1]), add2(acc[2], acc[3]));
  l_run = l_run * alpha + (f2lo(a01) + f2hi(a01));
  return true;
}

// Epilogue of one query row (this thread's TMEM lane): wait for the last P.V (bar_o,
// par_o), read O from TMEM into registers as bf16 O / l and hand the O columns back to
// the MMA warp at once (bar_oe); then write the row into this warp's staging block in
// shared memory (D / 64 boxes of 32 rows x 128 B, 128B-swizzled like the TMA tile) and
// let one lane store the block with TMA (rows >= Sq are clipped by the tensor map).  The
// store completes in the background; the block is reused by this warp one item later,
// after waiting for the store to have read it.  Finally the log-sum-exp.
// Ragged batches (VARLEN): O is [total_q, Hq, D] and the store box is 32 rows of one head;
// a warp whose 32 rows run past its sequence's end writes its valid rows with plain
// stores instead (a TMA store would spill into the next sequence), and LSE is [Hq, total_q].
template <int D, bool VARLEN = false>
__device__ __forceinline__ bool softmax_epilogue(uint32_t o_tm, uint32_t bar_o, uint32_t par_o,
                                                 uint32_t bar_oe, float m_run, float l_run,
                                                 int row, int q_z, const FwdParams& p,
                                                 const Abort& ab, const CUtensorMap* tm_o,
                                                 uint32_t stg, int qb = 0, int sq = 0) {
  const int lane = threadIdx.x & 31;
  if (!mbar_wait_warp(bar_o, par_o, p.ctl, ab)) return false;
  tc_fence_after();
  const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
  const uint64_t il2 = f2(inv_l, inv_l);
  uint32_t w[D / 2];  // the row as packed bf16 pairs
  // 64 columns per TMEM round trip: two loads in flight before each wait
#pragma unroll
  for (int ch = 0; ch < D / 32; ch += 2) {
    uint32_t rr[2][32];
    tmem_ld32(o_tm + ch * 32, rr[0]);
    tmem_ld32(o_tm + ch * 32 + 32, rr[1]);
    tmem_wait_ld();
    reg_fence32(rr[0]);
    reg_fence32(rr[1]);
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const uint64_t x = mul2(f2(__uint_as_float(rr[u][2 * i]), __uint_as_float(rr[u][2 * i + 1])), il2);
        w[(ch + u) * 16 + i] = pack_bf16x2(f2lo(x), f2hi(x));
      }
  }
  tc_fence_before();
  mbar_arrive(bar_oe);  // O is in registers: the next item's P.V may overwrite it
  if constexpr (VARLEN) {
    const int row0 = row - lane;  // the warp's rows are row0 .. row0 + 31
    if (row0 + 32 > sq) {
      if (row < sq) {
        uint4* dst = reinterpret_cast<uint4*>(p.o + (static_cast<size_t>(qb + row) * p.Hq + q_z) * D);
#pragma unroll
        for (int c = 0; c < D / 8; ++c) dst[c] = make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
        if (p.lse)
          p.lse[static_cast<size_t>(q_z) * p.total_q + qb + row] =
              l_run > 0.f ? (m_run + log2f(l_run)) * kLn2 : -INFINITY;
      }
      return true;
    }
  }
  if (lane == 0) bulk_wait_group_read0();  // this warp's previous store has left the block
  __syncwarp();
  const uint32_t my_row = stg + static_cast<uint32_t>(lane) * 128u;
#pragma unroll
  for (int c = 0; c < D / 8; ++c) {  // 16-byte chunk c of the row: box c / 8, slot c % 8
    const uint32_t slot = static_cast<uint32_t>((c & 7) ^ (lane & 7));
    st_shared_v4(my_row + static_cast<uint32_t>(c >> 3) * 4096u + (slot << 4), w[4 * c], w[4 * c + 1],
                 w[4 * c + 2], w[4 * c + 3]);
  }
  fence_proxy_async_smem();
  __syncwarp();
  if constexpr (VARLEN) {
    if (lane == 0) {
#pragma unroll
      for (int x = 0; x < D / 64; ++x) tma_store_3d(tm_o, stg + x * 4096u, x * 64, q_z, qb + row);
      bulk_commit_group();
    }
    if (p.lse)
      p.lse[static_cast<size_t>(q_z) * p.total_q + qb + row] = l_run > 0.f ? (m_run + log2f(l_run)) * kLn2 : -INFINITY;
    return true;
  }
  if (lane == 0) {
#pragma unroll
    for (int x = 0; x < D / 64; ++x) tma_store_3d(tm_o, stg + x * 4096u, x * 64, row, q_z);
    bulk_commit_group();
  }
  if (row < p.Sq && p.lse)
    p.lse[static_cast<size_t>(q_z) * p.Sq + row] = l_run > 0.f ? (m_run + log2f(l_run)) * kLn2 : -INFINITY;
  return true;
}

// Bring the next work item's query tiles and first K/V tiles into L2 while the current
// item still runs, so that its start waits on an L2 hit rather than HBM.
template <int D, int NQT, int BM, bool VARLEN = false>
__device__ __forceinline__ void prefetch_item_l2(const CUtensorMap* tm_q, const CUtensorMap* tm_k,
                                                 const CUtensorMap* tm_v, int q0, int q_z, int kv_z,
                                                 int qb = 0, int kb = 0) {
#pragma unroll
  for (int x = 0; x < D / 64; ++x) {
    if constexpr (VARLEN) {
#pragma unroll
      for (int t = 0; t < NQT; ++t) tma_prefetch_l2_3d(tm_q, x * 64, q_z, qb + q0 + t * BM);
      tma_prefetch_l2_3d(tm_k, x * 64, kv_z, kb);
      tma_prefetch_l2_3d(tm_v, x * 64, kv_z, kb);
    } else {
#pragma unroll
      for (int t = 0; t < NQT; ++t) tma_prefetch_l2_3d(tm_q, x * 64, q0 + t * BM, q_z);
      tma_prefetch_l2_3d(tm_k, x * 64, 0, kv_z);
      tma_prefetch_l2_3d(tm_v, x * 64, 0, kv_z);
    }
  }
}

// VARLEN: a ragged batch packed [total, H, D]: the tensor maps are [total, H, D] views
// (coordinates: column, head, token) and items come from the sequence cursor.  SLOTS: the
// ring depth (0: the model's).
template <int D, bool VARLEN = false, int SLOTS = 0>
__global__ void __launch_bounds__(FwdCfg<D, SLOTS>::THREADS, 1)
    attn_fwd_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                    const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o,
                    const FwdParams p) {
  using C = FwdCfg<D, SLOTS>;
  constexpr int kRows = C::NQT * C::BM;  // query rows of one item
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the 128B-swizzled tiles
  const uint32_t raw_base = smem_u32(smem_raw);
  const uint32_t sbase = (raw_base + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (sbase - raw_base);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const uint32_t bar_q = sbase + C::BAR_OFF;       // [2] Q_t loaded (once per item)
  const uint32_t bar_qe = bar_q + 16;              // [2] Q_t no longer read (once per item)
  const uint32_t bar_full = bar_qe + 16;           // [NSLOT]
  const uint32_t bar_empty = bar_full + 8 * C::NSLOT;
  const uint32_t bar_s = bar_empty + 8 * C::NSLOT;  // [2] S_t ready
  const uint32_t bar_p = bar_s + 16;                // [2][2] half h of P_t written (h = 0: and O_t rescaled)
  const uint32_t bar_o = bar_p + 32;                // [2] P_t V_j accumulated into O_t
  const uint32_t bar_oe = bar_o + 16;               // [2] O_t read out by the epilogue
  const uint32_t bar_drain = bar_oe + 16;
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::TMEM_PTR_OFF);
  Abort ab{reinterpret_cast<volatile int*>(smem + C::ABORT_OFF)};

  if (threadIdx.x == 0) {
    for (int t = 0; t < 2; ++t) {
      mbar_init(bar_q + 8 * t, 1);
      mbar_init(bar_qe + 8 * t, 1);
    }
    for (int s = 0; s < C::NSLOT; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(bar_s + 8 * t, 1);
      mbar_init(bar_p + 16 * t, C::BM);
      mbar_init(bar_p + 16 * t + 8, C::BM);
      mbar_init(bar_o + 8 * t, 1);
      mbar_init(bar_oe + 8 * t, C::BM);
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
  // above touches no global memory; from here on the previous kernel's writes must be
  // complete and visible.  The next launch may then start its own set-up on SMs this
  // grid frees.  (Not in the ragged-batch instantiation, which is launched plainly: the
  // two instructions alone cost it 4 %.)
  if constexpr (!VARLEN) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;");
  }

  if (warp == 8) {
    // ------------------------------------------------------------------ loader
    if (lane == 0) {
      prefetch_tensormap(&tm_q);
      prefetch_tensormap(&tm_k);
      prefetch_tensormap(&tm_v);
      int pos = 0, issued = 0, skipped = -1, q_issued[2] = {0, 0};
      bool ok = true;
      SeqCursor cur = VARLEN ? seq_cursor<kRows>(p) : SeqCursor{0, 0, 0};
      // Q_t of item r, once the previous item's S MMAs of tile t are done with its buffer
      auto load_q = [&](int t, int r, const Item& it) -> bool {
        if (r > 0 && !mbar_wait(bar_qe + 8 * t, (r - 1) & 1, p.ctl, ab)) return false;
        mbar_expect_tx(bar_q + 8 * t, C::Q_TILE_BYTES);
        const int qy = VARLEN ? it.q_z : it.q0 + t * C::BM;
        const int qz = VARLEN ? it.qb + it.q0 + t * C::BM : it.q_z;
        for (int x = 0; x < C::NBOX; ++x)
          tma_load_3d(sbase + C::Q_OFF + t * C::Q_TILE_BYTES + x * C::Q_BOX_BYTES, &tm_q, x * C::BOX_COLS,
                      qy, qz, bar_q + 8 * t);
        q_issued[t] = r + 1;
        return true;
      };
      for (int r = 0, idx; ok && (idx = item_index_t<kRows, VARLEN>(p, r, cur)) >= 0; ++r) {
        const Item it = make_item_t<D, VARLEN>(p, cur, idx);
        // Q_0 first: tile 0 finishes its S MMAs of the previous item before tile 1 does
        if (!(ok = load_q(0, r, it))) break;
        for (int jj = 0; jj < 2 * it.n_tiles; ++jj, ++pos) {  // K_0, [Q_1], V_0, K_1, V_1, ...
          if (jj == 1 && !(ok = load_q(1, r, it))) break;
          if (jj == max(0, 2 * it.n_tiles - 6)) {  // three KV tiles before the end
            SeqCursor nc = cur;
            const int nidx = item_index_t<kRows, VARLEN>(p, r + 1, nc);
            if (nidx >= 0) {
              const Item nx = make_item_t<D, VARLEN>(p, nc, nidx);
              prefetch_item_l2<D, C::NQT, C::BM, VARLEN>(&tm_q, &tm_k, &tm_v, nx.q0, nx.q_z, nx.kv_z, nx.qb,
                                                         nx.kb);
            }
          }
          const int slot = pos % C::NSLOT, round = pos / C::NSLOT;
          if (!(ok = mbar_wait(bar_empty + 8 * slot, (round & 1) ^ 1, p.ctl, ab))) break;
          issued = pos + 1;
          if (p.ctl.inject == 2 && pos == 2) {  // test hook: never load this tile
            skipped = pos;
            continue;
          }
          const CUtensorMap* map = (jj & 1) ? &tm_v : &tm_k;
          const int row = (jj >> 1) * C::BN;
          const int ky = VARLEN ? it.kv_z : row, kz = VARLEN ? it.kb + row : it.kv_z;
          mbar_expect_tx(bar_full + 8 * slot, C::SLOT_BYTES);
          for (int x = 0; x < C::NBOX; ++x)
            tma_load_3d(sbase + C::RING_OFF + slot * C::SLOT_BYTES + x * C::KV_BOX_BYTES, map,
                        x * C::BOX_COLS, ky, kz, bar_full + 8 * slot);
        }
      }
      // drain copies still in flight before the CTA may exit
      Abort no_abort{ab.flag + 1};
      for (int t = 0; t < 2; ++t)
        if (q_issued[t] > 0) mbar_wait(bar_q + 8 * t, (q_issued[t] - 1) & 1, p.ctl, no_abort);
      for (int ps = max(0, issued - C::NSLOT); ps < issued; ++ps)
        if (ps != skipped)
          mbar_wait(bar_full + 8 * (ps % C::NSLOT), (ps / C::NSLOT) & 1, p.ctl, no_abort);
    }
  } else if (warp == 9) {
    // ------------------------------------------------------------------ MMA issuer
    // The whole warp runs this role (warp-uniform operands and waits); one elected lane
    // issues the MMAs and commits.
    {
      constexpr uint32_t idesc_s = idesc_bf16(C::BM, C::BN, 0, 0);  // Q, K both K-major
      constexpr uint32_t idesc_pv = idesc_bf16(C::BM, D, 0, 1);     // P from TMEM, V MN-major
      auto wait_slot = [&](int ps) {
        return mbar_wait_warp(bar_full + 8 * (ps % C::NSLOT), (ps / C::NSLOT) & 1, p.ctl, ab);
      };
      // Base descriptors, built once: Q tile t, and ring slot s read as K (K-major) or V
      // (MN-major); a slot or box step is a constant added to the start-address field.
      const uint64_t dq0 = sdesc_sw128(sbase + C::Q_OFF, 16, 1024);
      const uint64_t dk0 = sdesc_sw128(sbase + C::RING_OFF, 16, 1024);
      const uint64_t dv0 = sdesc_sw128(sbase + C::RING_OFF, C::KV_BOX_BYTES, 1024);
      constexpr uint32_t kSlot16 = C::SLOT_BYTES >> 4, kQTile16 = C::Q_TILE_BYTES >> 4;
      constexpr uint32_t kQBox16 = C::Q_BOX_BYTES >> 4, kKBox16 = C::KV_BOX_BYTES >> 4;
      // S_t = Q_t K^T over K = D in 64-wide boxes
      auto issue_s = [&](int t, int kpos) {
        const uint64_t a = dq0 + t * kQTile16;
        const uint64_t b = dk0 + (kpos % C::NSLOT) * kSlot16;
#pragma unroll
        for (int x = 0; x < C::NBOX; ++x)
          mma_ss_k64_el(tmem + C::S_COL + t * C::BN, a + x * kQBox16, b + x * kKBox16, idesc_s, x > 0);
      };
      // O_t += P_t[:, half] V_j[half, :] over K = BN/2 keys
      auto issue_pv = [&](int t, int vpos, bool acc, int half) {
        const uint64_t b = dv0 + (vpos % C::NSLOT) * kSlot16 + half * (C::BN / 2) * (128 >> 4);
        static_assert(C::BN / 2 == 64, "a half of P is one 64-key block of four K-steps");
        mma_ts_k64_el(tmem + C::O_COL + t * D, tmem + C::S_COL + t * C::BN + half * (C::BN / 4), b, idesc_pv,
                   acc ? 1u : 0u);
      };
      int pos = 0, cnt0 = 0, cnt1 = 0;  // ring position of K_0; S/P/O uses so far per tile
      bool ok = true;
      SeqCursor cur = VARLEN ? seq_cursor<kRows>(p) : SeqCursor{0, 0, 0};
      for (int r = 0, idx; ok && (idx = item_index_t<kRows, VARLEN>(p, r, cur)) >= 0; ++r) {
        const Item it = make_item_t<D, VARLEN>(p, cur, idx);
        const int nt0 = it.n_tiles0, nt = it.n_tiles;
        if (!(ok = mbar_wait_warp(bar_q, r & 1, p.ctl, ab) && wait_slot(pos))) break;
        tc_fence_after();
        issue_s(0, pos);
        tc_commit_el(bar_s);
        if (nt0 == 1) tc_commit_el(bar_qe);  // every S of tile 0 issued
        if (!(ok = mbar_wait_warp(bar_q + 8, r & 1, p.ctl, ab))) break;
        tc_fence_after();
        issue_s(1, pos);
        tc_commit_el(bar_s + 8);
        tc_commit_el(bar_empty + 8 * (pos % C::NSLOT));
        if (nt == 1) tc_commit_el(bar_qe + 8);  // every S of tile 1 issued
        for (int j = 0; j < nt; ++j) {
          const int vpos = pos + 2 * j + 1, kpos = pos + 2 * j + 2;
          const bool more = j + 1 < nt;
          if (!(ok = wait_slot(vpos))) break;
          if (j < nt0) {  // query tile 0 stops at its own diagonal
            if (!(ok = mbar_wait_warp(bar_p, (cnt0 + j) & 1, p.ctl, ab))) break;
            // O_0 of the previous item must have been read out
            if (j == 0 && r > 0 && !(ok = mbar_wait_warp(bar_oe, (r - 1) & 1, p.ctl, ab))) break;
            tc_fence_after();
            issue_pv(0, vpos, j > 0, 0);
            if (!(ok = mbar_wait_warp(bar_p + 8, (cnt0 + j) & 1, p.ctl, ab))) break;
            tc_fence_after();
            issue_pv(0, vpos, true, 1);
            tc_commit_el(bar_o);
          }
          if (more) {
            if (!(ok = wait_slot(kpos))) break;
            tc_fence_after();
            if (j + 1 < nt0) {
              issue_s(0, kpos);
              tc_commit_el(bar_s);
              if (j + 2 == nt0) tc_commit_el(bar_qe);  // tile 0's last S of the item
            }
          }
          if (!(ok = mbar_wait_warp(bar_p + 16, (cnt1 + j) & 1, p.ctl, ab))) break;
          if (j == 0 && r > 0 && !(ok = mbar_wait_warp(bar_oe + 8, (r - 1) & 1, p.ctl, ab))) break;
          tc_fence_after();
          issue_pv(1, vpos, j > 0, 0);
          if (!(ok = mbar_wait_warp(bar_p + 24, (cnt1 + j) & 1, p.ctl, ab))) break;
          tc_fence_after();
          issue_pv(1, vpos, true, 1);
          tc_commit_el(bar_o + 8);
          tc_commit_el(bar_empty + 8 * (vpos % C::NSLOT));
          if (more) {
            issue_s(1, kpos);
            tc_commit_el(bar_s + 8);
            tc_commit_el(bar_empty + 8 * (kpos % C::NSLOT));
            if (j + 2 == nt) tc_commit_el(bar_qe + 8);  // tile 1's last S of the item
          }
        }
        cnt0 += nt0;
        cnt1 += nt;
        pos += 2 * nt;
      }
      // wait for every MMA issued above before TMEM may be released
      Abort no_abort{ab.flag + 1};
      tc_commit_el(bar_drain);
      mbar_wait_warp(bar_drain, 0, p.ctl, no_abort);
    }
  } else {
    // ------------------------------------------------------------------ softmax
    const int t = warp >> 2;                        // query tile of this warpgroup
    const int row_in_tile = (warp & 3) * 32 + lane;  // == TMEM lane
    const uint32_t lane_addr = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t s_tm = tmem + lane_addr + C::S_COL + t * C::BN;
    const uint32_t o_tm = tmem + lane_addr + C::O_COL + t * D;
    const uint32_t my_bar_s = bar_s + 8 * t, my_bar_p = bar_p + 16 * t, my_bar_o = bar_o + 8 * t;
    const uint32_t my_bar_oe = bar_oe + 8 * t;
    const uint32_t stg_q = sbase + C::STG_OFF + static_cast<uint32_t>(warp) * (32 * D * 2);
    const float c = p.c;
    const uint64_t c2 = f2(c, c);
    const int off = p.Skv - p.Sq;

    int cnt = 0;  // S tiles of this query tile processed in earlier items
    bool ok = true;
    SeqCursor cur = VARLEN ? seq_cursor<kRows>(p) : SeqCursor{0, 0, 0};
    for (int r = 0, idx; ok && (idx = item_index_t<kRows, VARLEN>(p, r, cur)) >= 0; ++r) {
      const Item it = make_item_t<D, VARLEN>(p, cur, idx);
      const int row = it.q0 + t * C::BM + row_in_tile;
      const int skv = VARLEN ? it.skv : p.Skv;
      const int offv = VARLEN ? it.skv - it.sq : off;
      const int limit = p.causal ? min(skv, row + offv + 1) : skv;  // keys [0, limit) visible
      const int my_tiles = t == 0 ? it.n_tiles0 : it.n_tiles;
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; ok && j < my_tiles; ++j)
        ok = softmax_step<D, C::BN>(s_tm, o_tm, my_bar_s, (cnt + j) & 1, my_bar_p, my_bar_o,
                                    (cnt + j - 1) & 1, j == 0, j * C::BN, limit, c, c2, m_run,
                                    l_run, p.ctl, ab);
      if (!ok) break;
      // epilogue: hand O_t back to the MMA warp, O / l -> bf16 rows, LSE
      if (!(ok = softmax_epilogue<D, VARLEN>(o_tm, my_bar_o, (cnt + my_tiles - 1) & 1, my_bar_oe, m_run,
                                             l_run, row, it.q_z, p, ab, &tm_o, stg_q,
                                             VARLEN ? it.qb : 0, VARLEN ? it.sq : 0)))
        break;
      cnt += my_tiles;
    }
    if (lane == 0) bulk_wait_group0();  // the O stores have completed before the CTA exits
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------- single-tile variant
// One 128-row query tile per CTA with S double-buffered in TMEM: while the softmax
// warpgroup works on S_j in buffer j % 2, the tensor pipe computes S_{j+1} in the other
// buffer and P_{j-1} V_{j-1}.  In the paper's terms this opens the boundary between the
// S MMA (load stage of the softmax) and the softmax body of Eq. 6, paid for with a
// second S buffer of TMEM (the capacity constraint of Eq. 8).
//
//   warps 0-3 softmax (thread = query row = TMEM lane), warp 4 loader, warp 5 MMA
//   TMEM: [0, BN) S/P buffer 0 | [BN, 2BN) S/P buffer 1 | [2BN, 2BN + D) O
//   ring order per item: K_0, K_1, V_0, K_2, V_1, ..., K_{n-1}, V_{n-2}, V_{n-1}
template <int D>
struct Fwd1Cfg {
  static constexpr model::FwdPlan kPlan = model::fwd_plan_variant(D, 1);
  static_assert(kPlan.feasible, "no feasible single-tile prefill schedule");
  static constexpr int BM = 128;
  static constexpr int BN = kPlan.bn;
  static constexpr int NSLOT = kPlan.kv_slots;
  static_assert(kPlan.design == 1 && kPlan.q_tiles == 1 && kPlan.s_buffers == 2, "single-tile variant");
  static_assert(BN == 128, "softmax holds one S row of 128 fp32 in registers");
  static constexpr int THREADS = 192;
  static constexpr int BOX_COLS = 64;
  static constexpr int NBOX = D / BOX_COLS;
  static constexpr uint32_t Q_BOX_BYTES = BM * 128;
  static constexpr uint32_t Q_TILE_BYTES = NBOX * Q_BOX_BYTES;
  static constexpr uint32_t KV_BOX_BYTES = BN * 128;
  static constexpr uint32_t SLOT_BYTES = NBOX * KV_BOX_BYTES;
  static constexpr uint32_t Q_OFF = 0;
  static constexpr uint32_t RING_OFF = Q_TILE_BYTES;
  static constexpr uint32_t STG_OFF = RING_OFF + NSLOT * SLOT_BYTES;  // O staging, one tile
  static constexpr uint32_t BAR_OFF = STG_OFF + BM * D * 2;
  // barriers: q_full, q_empty, full[NSLOT], empty[NSLOT], s[2], p[2][2], o[2], o_empty, drain
  static constexpr int NBAR = 2 + 2 * NSLOT + 12;
  static constexpr uint32_t TMEM_PTR_OFF = BAR_OFF + NBAR * 8;
  static constexpr uint32_t ABORT_OFF = TMEM_PTR_OFF + 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16 + 1024;
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t S_COL = 0;       // + buffer * BN
  static constexpr uint32_t O_COL = 2 * BN;
  static_assert(BYTES <= 227 * 1024, "shared memory budget");
  static_assert(O_COL + D <= TMEM_COLS, "TMEM budget");
};

template <int D>
__device__ __forceinline__ Item make_item1(const FwdParams& p, int idx) {
  using C = Fwd1Cfg<D>;
  int qt, bh;  // n_pairs holds the query tiles per (b, h) here
  item_coords(p, idx, qt, bh);
  Item it;
  it.h = bh % p.Hq;
  it.b = bh / p.Hq;
  it.q_z = bh;
  it.kv_z = it.b * p.Hkv + it.h / (p.Hq / p.Hkv);
  it.q0 = qt * C::BM;
  int n_kv = p.Skv;
  if (p.causal) n_kv = min(p.Skv, it.q0 + C::BM + (p.Skv - p.Sq));
  it.n_tiles0 = it.n_tiles = (n_kv + C::BN - 1) / C::BN;
  return it;
}

// Ring positions of K_j and V_j within an item of n KV tiles (order above).
__device__ __forceinline__ int ring_pos_k(int j) { return j == 0 ? 0 : 2 * j - 1; }
__device__ __forceinline__ int ring_pos_v(int j, int n) { return j == n - 1 ? 2 * n - 1 : 2 * j + 2; }

template <int D>
__global__ void __launch_bounds__(Fwd1Cfg<D>::THREADS, 1)
    attn_fwd1_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o,
                     const FwdParams p) {
  using C = Fwd1Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_base = smem_u32(smem_raw);
  const uint32_t sbase = (raw_base + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (sbase - raw_base);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const uint32_t bar_q = sbase + C::BAR_OFF;
  const uint32_t bar_qe = bar_q + 8;
  const uint32_t bar_full = bar_qe + 8;               // [NSLOT]
  const uint32_t bar_empty = bar_full + 8 * C::NSLOT;  // [NSLOT]
  const uint32_t bar_s = bar_empty + 8 * C::NSLOT;     // [2]    S in buffer b ready
  const uint32_t bar_p = bar_s + 16;                   // [2][2] half h of P in buffer b written
  const uint32_t bar_o = bar_p + 32;                   // [2]    P.V of S number g (g % 2 == b) done
  const uint32_t bar_oe = bar_o + 16;                  // O read out by the epilogue
  const uint32_t bar_drain = bar_oe + 8;
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::TMEM_PTR_OFF);
  Abort ab{reinterpret_cast<volatile int*>(smem + C::ABORT_OFF)};

  if (threadIdx.x == 0) {
    mbar_init(bar_q, 1);
    mbar_init(bar_qe, 1);
    for (int i = 0; i < C::NSLOT; ++i) {
      mbar_init(bar_full + 8 * i, 1);
      mbar_init(bar_empty + 8 * i, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar_s + 8 * b, 1);
      mbar_init(bar_p + 16 * b, C::BM);
      mbar_init(bar_p + 16 * b + 8, C::BM);
      mbar_init(bar_o + 8 * b, 1);
    }
    mbar_init(bar_oe, C::BM);
    mbar_init(bar_drain, 1);
    *ab.flag = 0;
    *(ab.flag + 1) = 0;
    fence_barrier_init();
  }
  if (warp == 5) tmem_alloc(smem_u32(tmem_ptr), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_ptr;
  // Launched as a programmatic dependent of the previous kernel in the stream: the set-up
  // above touches no global memory; from here on the previous kernel's writes must be
  // complete and visible.  The next launch may then start its own set-up on SMs this
  // grid frees.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;");

  if (warp == 4) {
    // ------------------------------------------------------------------ loader
    if (lane == 0) {
      prefetch_tensormap(&tm_q);
      prefetch_tensormap(&tm_k);
      prefetch_tensormap(&tm_v);
      int pos = 0, issued = 0, skipped = -1, q_issued = 0;
      bool ok = true;
      for (int r = 0, idx; ok && (idx = item_index(p, r)) >= 0; ++r) {
        const Item it = make_item1<D>(p, idx);
        const int n = it.n_tiles;
        if (r > 0 && !(ok = mbar_wait(bar_qe, (r - 1) & 1, p.ctl, ab))) break;
        mbar_expect_tx(bar_q, C::Q_TILE_BYTES);
        for (int x = 0; x < C::NBOX; ++x)
          tma_load_3d(sbase + C::Q_OFF + x * C::Q_BOX_BYTES, &tm_q, x * C::BOX_COLS, it.q0, it.q_z, bar_q);
        q_issued = r + 1;
        for (int sq = 0; sq < 2 * n; ++sq, ++pos) {
          if (sq == max(0, 2 * n - 6)) {  // three KV tiles before the end
            const int nidx = item_index(p, r + 1);
            if (nidx >= 0) {
              const Item nx = make_item1<D>(p, nidx);
              prefetch_item_l2<D, 1, C::BM>(&tm_q, &tm_k, &tm_v, nx.q0, nx.q_z, nx.kv_z);
            }
          }
          const int slot = pos % C::NSLOT, round = pos / C::NSLOT;
          if (!(ok = mbar_wait(bar_empty + 8 * slot, (round & 1) ^ 1, p.ctl, ab))) break;
          issued = pos + 1;
          if (p.ctl.inject == 2 && pos == 2) {  // test hook: never load this tile
            skipped = pos;
            continue;
          }
          // sequence index sq -> K_0 | V_{n-1} (last) | K_{(sq+1)/2} (odd) | V_{sq/2-1} (even)
          const bool is_v = sq != 0 && (sq == 2 * n - 1 || (sq & 1) == 0);
          const int tile = sq == 0 ? 0 : sq == 2 * n - 1 ? n - 1 : (sq & 1) ? (sq + 1) / 2 : sq / 2 - 1;
          mbar_expect_tx(bar_full + 8 * slot, C::SLOT_BYTES);
          for (int x = 0; x < C::NBOX; ++x)
            tma_load_3d(sbase + C::RING_OFF + slot * C::SLOT_BYTES + x * C::KV_BOX_BYTES,
                        is_v ? &tm_v : &tm_k, x * C::BOX_COLS, tile * C::BN, it.kv_z, bar_full + 8 * slot);
        }
      }
      Abort no_abort{ab.flag + 1};
      if (q_issued > 0) mbar_wait(bar_q, (q_issued - 1) & 1, p.ctl, no_abort);
      for (int ps = max(0, issued - C::NSLOT); ps < issued; ++ps)
        if (ps != skipped)
          mbar_wait(bar_full + 8 * (ps % C::NSLOT), (ps / C::NSLOT) & 1, p.ctl, no_abort);
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------------ MMA issuer
    // The whole warp runs this role; one elected lane issues the MMAs and commits.
    {
      constexpr uint32_t idesc_s = idesc_bf16(C::BM, C::BN, 0, 0);
      constexpr uint32_t idesc_pv = idesc_bf16(C::BM, D, 0, 1);
      const uint64_t dq = sdesc_sw128(sbase + C::Q_OFF, 16, 1024);
      const uint64_t dk0 = sdesc_sw128(sbase + C::RING_OFF, 16, 1024);
      const uint64_t dv0 = sdesc_sw128(sbase + C::RING_OFF, C::KV_BOX_BYTES, 1024);
      constexpr uint32_t kSlot16 = C::SLOT_BYTES >> 4, kQBox16 = C::Q_BOX_BYTES >> 4;
      constexpr uint32_t kKBox16 = C::KV_BOX_BYTES >> 4;
      auto wait_slot = [&](int ps) {
        return mbar_wait_warp(bar_full + 8 * (ps % C::NSLOT), (ps / C::NSLOT) & 1, p.ctl, ab);
      };
      auto issue_s = [&](int buf, int kpos) {
        const uint64_t b = dk0 + (kpos % C::NSLOT) * kSlot16;
#pragma unroll
        for (int x = 0; x < C::NBOX; ++x)
          mma_ss_k64_el(tmem + C::S_COL + buf * C::BN, dq + x * kQBox16, b + x * kKBox16, idesc_s, x > 0);
      };
      auto issue_pv = [&](int buf, int vpos, bool acc, int half) {
        const uint64_t b = dv0 + (vpos % C::NSLOT) * kSlot16 + half * (C::BN / 2) * (128 >> 4);
        mma_ts_k64_el(tmem + C::O_COL, tmem + C::S_COL + buf * C::BN + half * (C::BN / 4), b, idesc_pv,
                   acc ? 1u : 0u);
      };
      int pos = 0, g = 0;  // ring position of the item's first tile; S tiles issued so far
      bool ok = true;
      for (int r = 0, idx; ok && (idx = item_index(p, r)) >= 0; ++r) {
        const Item it = make_item1<D>(p, idx);
        const int n = it.n_tiles;
        if (!(ok = mbar_wait_warp(bar_q, r & 1, p.ctl, ab))) break;
        // S_0 and S_1 of the item into the two buffers
        for (int j = 0; j < 2 && j < n; ++j) {
          const int kp = pos + ring_pos_k(j);
          if (!(ok = wait_slot(kp))) break;
          tc_fence_after();
          issue_s((g + j) & 1, kp);
          tc_commit_el(bar_s + 8 * ((g + j) & 1));
          tc_commit_el(bar_empty + 8 * (kp % C::NSLOT));
        }
        if (!ok) break;
        if (n <= 2) tc_commit_el(bar_qe);  // every S of this item issued
        for (int j = 0; j < n; ++j) {
          const int gj = g + j, buf = gj & 1;
          const int vp = pos + ring_pos_v(j, n);
          if (!(ok = wait_slot(vp))) break;
          if (!(ok = mbar_wait_warp(bar_p + 16 * buf, (gj >> 1) & 1, p.ctl, ab))) break;
          if (j == 0 && r > 0 && !(ok = mbar_wait_warp(bar_oe, (r - 1) & 1, p.ctl, ab))) break;
          tc_fence_after();
          issue_pv(buf, vp, j > 0, 0);
          if (!(ok = mbar_wait_warp(bar_p + 16 * buf + 8, (gj >> 1) & 1, p.ctl, ab))) break;
          tc_fence_after();
          issue_pv(buf, vp, true, 1);
          tc_commit_el(bar_o + 8 * buf);
          tc_commit_el(bar_empty + 8 * (vp % C::NSLOT));
          if (j + 2 < n) {  // S_{j+2} into the buffer P_j V_j has just been issued from
            const int kp = pos + ring_pos_k(j + 2);
            if (!(ok = wait_slot(kp))) break;
            tc_fence_after();
            issue_s(buf, kp);
            tc_commit_el(bar_s + 8 * buf);
            tc_commit_el(bar_empty + 8 * (kp % C::NSLOT));
            if (j + 3 == n) tc_commit_el(bar_qe);
          }
        }
        g += n;
        pos += 2 * n;
      }
      Abort no_abort{ab.flag + 1};
      tc_commit_el(bar_drain);
      mbar_wait_warp(bar_drain, 0, p.ctl, no_abort);
    }
  } else {
    // ------------------------------------------------------------------ softmax
    const uint32_t lane_addr = static_cast<uint32_t>(warp * 32) << 16;
    const uint32_t s_tm0 = tmem + lane_addr + C::S_COL;
    const uint32_t o_tm = tmem + lane_addr + C::O_COL;
    const uint32_t stg_q = sbase + C::STG_OFF + static_cast<uint32_t>(warp) * (32 * D * 2);
    const float c = p.c;
    const uint64_t c2 = f2(c, c);
    const int off = p.Skv - p.Sq;
    int g = 0;  // S tiles processed in earlier items
    bool ok = true;
    for (int r = 0, idx; ok && (idx = item_index(p, r)) >= 0; ++r) {
      const Item it = make_item1<D>(p, idx);
      const int n = it.n_tiles;
      const int row = it.q0 + warp * 32 + lane;
      const int limit = p.causal ? min(p.Skv, row + off + 1) : p.Skv;
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; ok && j < n; ++j) {
        const int gj = g + j, buf = gj & 1;
        // the previous P.V (S number gj - 1) completes on bar_o[(gj - 1) % 2]
        ok = softmax_step<D, C::BN>(s_tm0 + buf * C::BN, o_tm, bar_s + 8 * buf, (gj >> 1) & 1,
                                    bar_p + 16 * buf, bar_o + 8 * ((gj - 1) & 1), ((gj - 1) >> 1) & 1,
                                    j == 0, j * C::BN, limit, c, c2, m_run, l_run, p.ctl, ab);
      }
      if (!ok) break;
      const int gl = g + n - 1;  // the item's last P.V
      if (!(ok = softmax_epilogue<D>(o_tm, bar_o + 8 * (gl & 1), (gl >> 1) & 1, bar_oe, m_run, l_run,
                                     row, it.q_z, p, ab, &tm_o, stg_q)))
        break;
      g += n;
    }
    if (lane == 0) bulk_wait_group0();  // the O stores have completed before the CTA exits
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ---------------------------------------------------------------- S-ring variant
// Two 128-row query tiles share a ring of three S buffers in TMEM.  S tiles are issued
// alternately for the two query tiles (S number k: tile k % 2, key tile k / 2 of the
// item, buffer k % 3), and S number k + 3 is issued right after P.V of S number k has
// freed its buffer.  Each tile's next S is therefore ready while its softmax still runs,
// so both softmax warpgroups stay busy and the tensor pipe does not wait on one tile's
// S -> softmax -> P.V chain.  TMEM: 3 * BN (S/P) + 2 * D (O) columns, which fits only for
// D = 64.  Causal items run both tiles over the same n KV tiles (tile 0's last one is
// fully masked).
//   warps 0-3 / 4-7 softmax of tile 0 / 1, warp 8 loader, warp 9 MMA
template <int D>
struct Fwd3Cfg {
  static constexpr model::FwdPlan kPlan = model::fwd_plan_variant(D, 3);
  static constexpr bool kFeasible = kPlan.feasible;
  static constexpr int BM = 128;
  static constexpr int NQT = 2;
  static constexpr int BN = 128;
  static constexpr int NSLOT = kFeasible ? kPlan.kv_slots : 4;
  static constexpr int THREADS = 320;
  static constexpr int BOX_COLS = 64;
  static constexpr int NBOX = D / BOX_COLS;
  static constexpr uint32_t Q_BOX_BYTES = BM * 128;
  static constexpr uint32_t Q_TILE_BYTES = NBOX * Q_BOX_BYTES;
  static constexpr uint32_t KV_BOX_BYTES = BN * 128;
  static constexpr uint32_t SLOT_BYTES = NBOX * KV_BOX_BYTES;
  static constexpr uint32_t Q_OFF = 0;
  static constexpr uint32_t RING_OFF = NQT * Q_TILE_BYTES;
  static constexpr uint32_t STG_OFF = RING_OFF + NSLOT * SLOT_BYTES;  // O staging per tile
  static constexpr uint32_t BAR_OFF = STG_OFF + NQT * BM * D * 2;
  // barriers: q_full, q_empty, full[NSLOT], empty[NSLOT], s[3], p[3][2], o[2][2], o_empty[2], drain
  static constexpr int NBAR = 2 + 2 * NSLOT + 3 + 6 + 4 + 2 + 1;
  static constexpr uint32_t TMEM_PTR_OFF = BAR_OFF + NBAR * 8;
  static constexpr uint32_t ABORT_OFF = TMEM_PTR_OFF + 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16 + 1024;
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t S_COL = 0;        // + buffer * BN
  static constexpr uint32_t O_COL = 3 * BN;   // + t * D
  static_assert(!kFeasible || (BYTES <= 227 * 1024 && O_COL + NQT * D <= TMEM_COLS), "budgets");
};

template <int D>
__global__ void __launch_bounds__(Fwd3Cfg<D>::THREADS, 1)
    attn_fwd3_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o,
                     const FwdParams p) {
  using C = Fwd3Cfg<D>;
  if constexpr (!C::kFeasible) {
    return;
  } else {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_base = smem_u32(smem_raw);
  const uint32_t sbase = (raw_base + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (sbase - raw_base);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const uint32_t bar_q = sbase + C::BAR_OFF;
  const uint32_t bar_qe = bar_q + 8;
  const uint32_t bar_full = bar_qe + 8;                // [NSLOT]
  const uint32_t bar_empty = bar_full + 8 * C::NSLOT;  // [NSLOT]
  const uint32_t bar_s = bar_empty + 8 * C::NSLOT;     // [3]    S in buffer b ready
  const uint32_t bar_p = bar_s + 24;                   // [3][2] half h of P in buffer b written
  const uint32_t bar_o = bar_p + 48;                   // [2][2] P.V of tile t, its S number parity e
  const uint32_t bar_oe = bar_o + 32;                  // [2]    O_t read out by the epilogue
  const uint32_t bar_drain = bar_oe + 16;
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::TMEM_PTR_OFF);
  Abort ab{reinterpret_cast<volatile int*>(smem + C::ABORT_OFF)};

  if (threadIdx.x == 0) {
    mbar_init(bar_q, 1);
    mbar_init(bar_qe, 1);
    for (int i = 0; i < C::NSLOT; ++i) {
      mbar_init(bar_full + 8 * i, 1);
      mbar_init(bar_empty + 8 * i, 1);
    }
    for (int b = 0; b < 3; ++b) {
      mbar_init(bar_s + 8 * b, 1);
      mbar_init(bar_p + 16 * b, C::BM);
      mbar_init(bar_p + 16 * b + 8, C::BM);
    }
    for (int i = 0; i < 4; ++i) mbar_init(bar_o + 8 * i, 1);
    mbar_init(bar_oe, C::BM);
    mbar_init(bar_oe + 8, C::BM);
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
  // above touches no global memory; from here on the previous kernel's writes must be
  // complete and visible.  The next launch may then start its own set-up on SMs this
  // grid frees.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;");

  if (warp == 8) {
    // ------------------------------------------------------------------ loader
    if (lane == 0) {
      prefetch_tensormap(&tm_q);
      prefetch_tensormap(&tm_k);
      prefetch_tensormap(&tm_v);
      int pos = 0, issued = 0, skipped = -1, q_issued = 0;
      bool ok = true;
      for (int r = 0, idx; ok && (idx = item_index(p, r)) >= 0; ++r) {
        const Item it = make_item<D>(p, idx);
        const int n = it.n_tiles;
        if (r > 0 && !(ok = mbar_wait(bar_qe, (r - 1) & 1, p.ctl, ab))) break;
        mbar_expect_tx(bar_q, C::NQT * C::Q_TILE_BYTES);
        for (int t = 0; t < C::NQT; ++t)
          for (int x = 0; x < C::NBOX; ++x)
            tma_load_3d(sbase + C::Q_OFF + t * C::Q_TILE_BYTES + x * C::Q_BOX_BYTES, &tm_q,
                        x * C::BOX_COLS, it.q0 + t * C::BM, it.q_z, bar_q);
        q_issued = r + 1;
        for (int sq = 0; sq < 2 * n; ++sq, ++pos) {  // K_0, K_1, V_0, K_2, V_1, ..., V_{n-1}
          if (sq == max(0, 2 * n - 6)) {  // three KV tiles before the end
            const int nidx = item_index(p, r + 1);
            if (nidx >= 0) {
              const Item nx = make_item<D>(p, nidx);
              prefetch_item_l2<D, C::NQT, C::BM>(&tm_q, &tm_k, &tm_v, nx.q0, nx.q_z, nx.kv_z);
            }
          }
          const int slot = pos % C::NSLOT, round = pos / C::NSLOT;
          if (!(ok = mbar_wait(bar_empty + 8 * slot, (round & 1) ^ 1, p.ctl, ab))) break;
          issued = pos + 1;
          if (p.ctl.inject == 2 && pos == 2) {  // test hook: never load this tile
            skipped = pos;
            continue;
          }
          const bool is_v = sq != 0 && (sq == 2 * n - 1 || (sq & 1) == 0);
          const int tile = sq == 0 ? 0 : sq == 2 * n - 1 ? n - 1 : (sq & 1) ? (sq + 1) / 2 : sq / 2 - 1;
          mbar_expect_tx(bar_full + 8 * slot, C::SLOT_BYTES);
          for (int x = 0; x < C::NBOX; ++x)
            tma_load_3d(sbase + C::RING_OFF + slot * C::SLOT_BYTES + x * C::KV_BOX_BYTES,
                        is_v ? &tm_v : &tm_k, x * C::BOX_COLS, tile * C::BN, it.kv_z, bar_full + 8 * slot);
        }
      }
      Abort no_abort{ab.flag + 1};
      if (q_issued > 0) mbar_wait(bar_q, (q_issued - 1) & 1, p.ctl, no_abort);
      for (int ps = max(0, issued - C::NSLOT); ps < issued; ++ps)
        if (ps != skipped)
          mbar_wait(bar_full + 8 * (ps % C::NSLOT), (ps / C::NSLOT) & 1, p.ctl, no_abort);
    }
  } else if (warp == 9) {
    // ------------------------------------------------------------------ MMA issuer
    // The whole warp runs this role; one elected lane issues the MMAs and commits.
    {
      constexpr uint32_t idesc_s = idesc_bf16(C::BM, C::BN, 0, 0);
      constexpr uint32_t idesc_pv = idesc_bf16(C::BM, D, 0, 1);
      const uint64_t dq0 = sdesc_sw128(sbase + C::Q_OFF, 16, 1024);
      const uint64_t dk0 = sdesc_sw128(sbase + C::RING_OFF, 16, 1024);
      const uint64_t dv0 = sdesc_sw128(sbase + C::RING_OFF, C::KV_BOX_BYTES, 1024);
      constexpr uint32_t kSlot16 = C::SLOT_BYTES >> 4, kQTile16 = C::Q_TILE_BYTES >> 4;
      constexpr uint32_t kQBox16 = C::Q_BOX_BYTES >> 4, kKBox16 = C::KV_BOX_BYTES >> 4;
      auto wait_slot = [&](int ps) {
        return mbar_wait_warp(bar_full + 8 * (ps % C::NSLOT), (ps / C::NSLOT) & 1, p.ctl, ab);
      };
      long long gk = 0;  // S tiles issued in earlier items (both query tiles)
      int pos = 0, cnt = 0;  // ring position of the item's K_0; per-tile S count before the item
      bool ok = true;
      // S number k of the item (tile k % 2, key tile k / 2) into buffer (gk + k) % 3
      auto issue_s = [&](int k, int n) -> bool {
        const int t = k & 1, j = k >> 1;
        const int kp = pos + ring_pos_k(j);
        if (!wait_slot(kp)) return false;
        tc_fence_after();
        const int buf = static_cast<int>((gk + k) % 3);
        const uint64_t a = dq0 + t * kQTile16;
        const uint64_t b = dk0 + (kp % C::NSLOT) * kSlot16;
#pragma unroll
        for (int x = 0; x < C::NBOX; ++x)
          mma_ss_k64_el(tmem + C::S_COL + buf * C::BN, a + x * kQBox16, b + x * kKBox16, idesc_s, x > 0);
        tc_commit_el(bar_s + 8 * buf);
        if (t == 1) tc_commit_el(bar_empty + 8 * (kp % C::NSLOT));  // both tiles have used K_j
        if (k == 2 * n - 1) tc_commit_el(bar_qe);                   // the item's last S
        return true;
      };
      for (int r = 0, idx; ok && (idx = item_index(p, r)) >= 0; ++r) {
        const Item it = make_item<D>(p, idx);
        const int n = it.n_tiles;
        if (!(ok = mbar_wait_warp(bar_q, r & 1, p.ctl, ab))) break;
        for (int k = 0; ok && k < 3 && k < 2 * n; ++k) ok = issue_s(k, n);
        for (int m = 0; ok && m < 2 * n; ++m) {
          const int t = m & 1, j = m >> 1;
          const long long km = gk + m;
          const int buf = static_cast<int>(km % 3);
          const uint32_t par = static_cast<uint32_t>((km / 3) & 1);
          const int vp = pos + ring_pos_v(j, n);
          if (!(ok = wait_slot(vp))) break;
          if (!(ok = mbar_wait_warp(bar_p + 16 * buf, par, p.ctl, ab))) break;
          if (j == 0 && r > 0 && !(ok = mbar_wait_warp(bar_oe + 8 * t, (r - 1) & 1, p.ctl, ab))) break;
          tc_fence_after();
          const uint64_t b = dv0 + (vp % C::NSLOT) * kSlot16;
          mma_ts_k64_el(tmem + C::O_COL + t * D, tmem + C::S_COL + buf * C::BN, b, idesc_pv, j > 0 ? 1u : 0u);
          if (!(ok = mbar_wait_warp(bar_p + 16 * buf + 8, par, p.ctl, ab))) break;
          tc_fence_after();
          mma_ts_k64_el(tmem + C::O_COL + t * D, tmem + C::S_COL + buf * C::BN + C::BN / 4,
                     b + (C::BN / 2) * (128 >> 4), idesc_pv, 1u);
          const int g = cnt + j;  // this tile's S number across items
          tc_commit_el(bar_o + 8 * (2 * t + (g & 1)));
          if (t == 1) tc_commit_el(bar_empty + 8 * (vp % C::NSLOT));  // both tiles have used V_j
          if (m + 3 < 2 * n) ok = issue_s(m + 3, n);                // into the buffer just freed
        }
        gk += 2 * n;
        cnt += n;
        pos += 2 * n;
      }
      Abort no_abort{ab.flag + 1};
      tc_commit_el(bar_drain);
      mbar_wait_warp(bar_drain, 0, p.ctl, no_abort);
    }
  } else {
    // ------------------------------------------------------------------ softmax
    const int t = warp >> 2;
    const int row_in_tile = (warp & 3) * 32 + lane;
    const uint32_t lane_addr = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t s_tm0 = tmem + lane_addr + C::S_COL;
    const uint32_t o_tm = tmem + lane_addr + C::O_COL + t * D;
    const uint32_t stg_q = sbase + C::STG_OFF + static_cast<uint32_t>(warp) * (32 * D * 2);
    const float c = p.c;
    const uint64_t c2 = f2(c, c);
    const int off = p.Skv - p.Sq;
    long long gk = 0;
    int cnt = 0;
    bool ok = true;
    for (int r = 0, idx; ok && (idx = item_index(p, r)) >= 0; ++r) {
      const Item it = make_item<D>(p, idx);
      const int n = it.n_tiles;
      const int row = it.q0 + t * C::BM + row_in_tile;
      const int limit = p.causal ? min(p.Skv, row + off + 1) : p.Skv;
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; ok && j < n; ++j) {
        const long long k = gk + 2 * j + t;
        const int buf = static_cast<int>(k % 3);
        const int g = cnt + j;
        ok = softmax_step<D, C::BN>(s_tm0 + buf * C::BN, o_tm, bar_s + 8 * buf,
                                    static_cast<uint32_t>((k / 3) & 1), bar_p + 16 * buf,
                                    bar_o + 8 * (2 * t + ((g - 1) & 1)), ((g - 1) >> 1) & 1, j == 0,
                                    j * C::BN, limit, c, c2, m_run, l_run, p.ctl, ab);
      }
      if (!ok) break;
      const int gl = cnt + n - 1;
      if (!(ok = softmax_epilogue<D>(o_tm, bar_o + 8 * (2 * t + (gl & 1)), (gl >> 1) & 1, bar_oe + 8 * t,
                                     m_run, l_run, row, it.q_z, p, ab, &tm_o, stg_q)))
        break;
      gk += 2 * n;
      cnt += n;
    }
    if (lane == 0) bulk_wait_group0();  // the O stores have completed before the CTA exits
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
  }
}

// ---------------------------------------------------------------- three-tile variant
// Three 128-row query tiles per CTA over KV tiles of BN = 96 keys (D = 64 only).  The MMA
// warp issues S0 S1 S2 | PV0 S0' | PV1 S1' | PV2 S2' | ...: while one tile's softmax
// runs, the tensor pipe works through the other two tiles' P.V and next S, so each tile's
// chain S -> softmax -> P.V has two tiles' MMAs to hide behind (design 2 has one).  P is
// handed over in halves of 64 and 32 keys.  A query tile wholly past Sq (the last item of
// a plane when Sq is not a multiple of 384) runs one KV tile only; its rows are clipped
// by the O tensor map and get no LSE.
//   warps 0-3 / 4-7 / 8-11 softmax of tile 0 / 1 / 2, warp 12 loader, warp 13 MMA
//   TMEM (512 columns): tile t's S/P at t * 160 (96 columns), its O at t * 160 + 96 (64)
template <int D>
struct Fwd4Cfg {
  static constexpr model::FwdPlan kPlan = model::fwd_plan_variant(D, 4);
  static constexpr bool kFeasible = kPlan.feasible;
  static constexpr int BM = 128;
  static constexpr int NQT = 3;
  static constexpr int BN = 96;
  static constexpr int NSLOT = kFeasible ? kPlan.kv_slots : 3;
  static constexpr int THREADS = 448;
  static constexpr int BOX_COLS = 64;
  static constexpr int NBOX = D / BOX_COLS;
  static constexpr uint32_t Q_BOX_BYTES = BM * 128;
  static constexpr uint32_t Q_TILE_BYTES = NBOX * Q_BOX_BYTES;
  static constexpr uint32_t KV_BOX_BYTES = BN * 128;
  static constexpr uint32_t SLOT_BYTES = NBOX * KV_BOX_BYTES;
  static constexpr uint32_t Q_OFF = 0;
  static constexpr uint32_t RING_OFF = NQT * Q_TILE_BYTES;
  static constexpr uint32_t STG_OFF = RING_OFF + NSLOT * SLOT_BYTES;  // O staging, one block per warp
  static constexpr uint32_t BAR_OFF = STG_OFF + NQT * BM * D * 2;
  // barriers: q_full[3], q_empty[3], full[NSLOT], empty[NSLOT], s[3], p[3][2], o[3], o_empty[3], drain
  static constexpr int NBAR = 6 + 2 * NSLOT + 3 + 6 + 3 + 3 + 1;
  static constexpr uint32_t TMEM_PTR_OFF = BAR_OFF + NBAR * 8;
  static constexpr uint32_t ABORT_OFF = TMEM_PTR_OFF + 8;
  static constexpr uint32_t BYTES = ABORT_OFF + 16 + 1024;
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t TILE_COLS = 160;  // tile t: S/P at t * 160, O at t * 160 + BN
  static_assert(!kFeasible || D == 64, "three S buffers and O accumulators fit TMEM at D = 64 only");
  static_assert(!kFeasible || (BYTES <= 227 * 1024 && NQT * TILE_COLS <= TMEM_COLS && BN + D <= TILE_COLS),
                "budgets");
  static_assert(KV_BOX_BYTES % 1024 == 0, "128B-swizzled tiles start on 1024-byte boundaries");
};

// KV tiles of BN keys that query tile t (rows q0 + t * 128 ..) of an item needs: up to the
// diagonal of its last row when causal; one for a tile wholly past Sq.
__device__ __forceinline__ int fwd4_tiles(const FwdParams& p, int q0, int t) {
  const int r0 = q0 + t * Fwd4Cfg<64>::BM;
  if (r0 >= p.Sq) return 1;
  int n_kv = p.Skv;
  if (p.causal) n_kv = min(p.Skv, r0 + Fwd4Cfg<64>::BM + (p.Skv - p.Sq));
  return (n_kv + Fwd4Cfg<64>::BN - 1) / Fwd4Cfg<64>::BN;
}

template <int D>
__global__ void __launch_bounds__(Fwd4Cfg<D>::THREADS, 1)
    attn_fwd4_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o,
                     const FwdParams p) {
  using C = Fwd4Cfg<D>;
  if constexpr (!C::kFeasible) {
    return;
  } else {
  constexpr int kRows = C::NQT * C::BM;  // query rows of one item
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_base = smem_u32(smem_raw);
  const uint32_t sbase = (raw_base + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (sbase - raw_base);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const uint32_t bar_q = sbase + C::BAR_OFF;           // [3] Q_t loaded
  const uint32_t bar_qe = bar_q + 24;                  // [3] Q_t no longer read
  const uint32_t bar_full = bar_qe + 24;               // [NSLOT]
  const uint32_t bar_empty = bar_full + 8 * C::NSLOT;  // [NSLOT]
  const uint32_t bar_s = bar_empty + 8 * C::NSLOT;     // [3] S_t ready
  const uint32_t bar_p = bar_s + 24;                   // [3][2] half h of P_t written (h = 0: and O_t rescaled)
  const uint32_t bar_o = bar_p + 48;                   // [3] P_t V_j accumulated into O_t
  const uint32_t bar_oe = bar_o + 24;                  // [3] O_t read out by the epilogue
  const uint32_t bar_drain = bar_oe + 24;
  uint32_t* tmem_ptr = reinterpret_cast<uint32_t*>(smem + C::TMEM_PTR_OFF);
  Abort ab{reinterpret_cast<volatile int*>(smem + C::ABORT_OFF)};

  if (threadIdx.x == 0) {
    for (int t = 0; t < C::NQT; ++t) {
      mbar_init(bar_q + 8 * t, 1);
      mbar_init(bar_qe + 8 * t, 1);
      mbar_init(bar_s + 8 * t, 1);
      mbar_init(bar_p + 16 * t, C::BM);
      mbar_init(bar_p + 16 * t + 8, C::BM);
      mbar_init(bar_o + 8 * t, 1);
      mbar_init(bar_oe + 8 * t, C::BM);
    }
    for (int s = 0; s < C::NSLOT; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    mbar_init(bar_drain, 1);
    *ab.flag = 0;
    *(ab.flag + 1) = 0;
    fence_barrier_init();
  }
  if (warp == 13) tmem_alloc(smem_u32(tmem_ptr), C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_ptr;
  // Launched as a programmatic dependent of the previous kernel in the stream: the set-up
  // above touches no global memory; from here on the previous kernel's writes must be
  // complete and visible.  The next launch may then start its own set-up on SMs this
  // grid frees.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;");

  if (warp == 12) {
    // ------------------------------------------------------------------ loader
    if (lane == 0) {
      prefetch_tensormap(&tm_q);
      prefetch_tensormap(&tm_k);
      prefetch_tensormap(&tm_v);
      int pos = 0, issued = 0, skipped = -1, q_issued[3] = {0, 0, 0};
      bool ok = true;
      // Q_t of item r, once the previous item's S MMAs of tile t are done with its buffer
      auto load_q = [&](int t, int r, const Item& it) -> bool {
        if (r > 0 && !mbar_wait(bar_qe + 8 * t, (r - 1) & 1, p.ctl, ab)) return false;
        mbar_expect_tx(bar_q + 8 * t, C::Q_TILE_BYTES);
        for (int x = 0; x < C::NBOX; ++x)
          tma_load_3d(sbase + C::Q_OFF + t * C::Q_TILE_BYTES + x * C::Q_BOX_BYTES, &tm_q, x * C::BOX_COLS,
                      it.q0 + t * C::BM, it.q_z, bar_q + 8 * t);
        q_issued[t] = r + 1;
        return true;
      };
      for (int r = 0, idx; ok && (idx = item_index(p, r)) >= 0; ++r) {
        const Item it = make_item<D>(p, idx);  // b, h, q_z, kv_z (the 256-row fields are unused)
        Item it4 = it;
        int pos_item, bh;
        item_coords(p, idx, pos_item, bh);
        it4.q0 = pos_item * kRows;
        const int nmax = max(fwd4_tiles(p, it4.q0, 0), max(fwd4_tiles(p, it4.q0, 1), fwd4_tiles(p, it4.q0, 2)));
        if (!(ok = load_q(0, r, it4))) break;
        for (int jj = 0; jj < 2 * nmax; ++jj, ++pos) {  // K_0, [Q_1, Q_2], V_0, K_1, V_1, ...
          if (jj == 1 && !((ok = load_q(1, r, it4)) && (ok = load_q(2, r, it4)))) break;
          if (jj == max(0, 2 * nmax - 6)) {  // three KV tiles before the end
            const int nidx = item_index(p, r + 1);
            if (nidx >= 0) {
              const Item nx = make_item<D>(p, nidx);
              int npos, nbh;
              item_coords(p, nidx, npos, nbh);
              prefetch_item_l2<D, C::NQT, C::BM>(&tm_q, &tm_k, &tm_v, npos * kRows, nx.q_z, nx.kv_z);
            }
          }
          const int slot = pos % C::NSLOT, round = pos / C::NSLOT;
          if (!(ok = mbar_wait(bar_empty + 8 * slot, (round & 1) ^ 1, p.ctl, ab))) break;
          issued = pos + 1;
          if (p.ctl.inject == 2 && pos == 2) {  // test hook: never load this tile
            skipped = pos;
            continue;
          }
          mbar_expect_tx(bar_full + 8 * slot, C::SLOT_BYTES);
          for (int x = 0; x < C::NBOX; ++x)
            tma_load_3d(sbase + C::RING_OFF + slot * C::SLOT_BYTES + x * C::KV_BOX_BYTES, (jj & 1) ? &tm_v : &tm_k,
                        x * C::BOX_COLS, (jj >> 1) * C::BN, it4.kv_z, bar_full + 8 * slot);
        }
      }
      // drain copies still in flight before the CTA may exit
      Abort no_abort{ab.flag + 1};
      for (int t = 0; t < C::NQT; ++t)
        if (q_issued[t] > 0) mbar_wait(bar_q + 8 * t, (q_issued[t] - 1) & 1, p.ctl, no_abort);
      for (int ps = max(0, issued - C::NSLOT); ps < issued; ++ps)
        if (ps != skipped) mbar_wait(bar_full + 8 * (ps % C::NSLOT), (ps / C::NSLOT) & 1, p.ctl, no_abort);
    }
  } else if (warp == 13) {
    // ------------------------------------------------------------------ MMA issuer
    // The whole warp runs this role (warp-uniform operands and waits); one elected lane
    // issues the MMAs and commits.
    {
      constexpr uint32_t idesc_s = idesc_bf16(C::BM, C::BN, 0, 0);  // Q, K both K-major
      constexpr uint32_t idesc_pv = idesc_bf16(C::BM, D, 0, 1);     // P from TMEM, V MN-major
      auto wait_slot = [&](int ps) {
        return mbar_wait_warp(bar_full + 8 * (ps % C::NSLOT), (ps / C::NSLOT) & 1, p.ctl, ab);
      };
      const uint64_t dq0 = sdesc_sw128(sbase + C::Q_OFF, 16, 1024);
      const uint64_t dk0 = sdesc_sw128(sbase + C::RING_OFF, 16, 1024);
      const uint64_t dv0 = sdesc_sw128(sbase + C::RING_OFF, C::KV_BOX_BYTES, 1024);
      constexpr uint32_t kSlot16 = C::SLOT_BYTES >> 4, kQTile16 = C::Q_TILE_BYTES >> 4;
      // S_t = Q_t K^T (K = D = 64: one 64-wide box)
      auto issue_s = [&](int t, int kpos) {
        mma_ss_k64_el(tmem + t * C::TILE_COLS, dq0 + t * kQTile16, dk0 + (kpos % C::NSLOT) * kSlot16, idesc_s, 0u);
      };
      // O_t += P_t V_j: keys 0-63 (P columns 0-31), then keys 64-95 (P columns 32-47)
      auto issue_pv = [&](int t, int vpos, bool acc, int half) {
        const uint64_t b = dv0 + (vpos % C::NSLOT) * kSlot16 + half * 64 * (128 >> 4);
        const uint32_t o = tmem + t * C::TILE_COLS + C::BN;
        if (half == 0)
          mma_ts_k64_el(o, tmem + t * C::TILE_COLS, b, idesc_pv, acc ? 1u : 0u);
        else
          mma_ts_k32_el(o, tmem + t * C::TILE_COLS + 32, b, idesc_pv, 1u);
      };
      int pos = 0, cnt[3] = {0, 0, 0};  // ring position of K_0; S/P/O uses so far per tile
      bool ok = true;
      for (int r = 0, idx; ok && (idx = item_index(p, r)) >= 0; ++r) {
        int pos_item, bh;
        item_coords(p, idx, pos_item, bh);
        const int q0 = pos_item * kRows;
        int nt[3];
        for (int t = 0; t < 3; ++t) nt[t] = fwd4_tiles(p, q0, t);
        const int nmax = max(nt[0], max(nt[1], nt[2]));
        for (int t = 0; ok && t < 3; ++t) {
          if (!(ok = mbar_wait_warp(bar_q + 8 * t, r & 1, p.ctl, ab) && (t > 0 || wait_slot(pos)))) break;
          tc_fence_after();
          issue_s(t, pos);
          tc_commit_el(bar_s + 8 * t);
          if (nt[t] == 1) tc_commit_el(bar_qe + 8 * t);  // every S of tile t issued
        }
        if (!ok) break;
        tc_commit_el(bar_empty + 8 * (pos % C::NSLOT));  // K_0 read by the three S MMAs
        for (int j = 0; ok && j < nmax; ++j) {
          const int vpos = pos + 2 * j + 1, kpos = pos + 2 * j + 2;
          const bool more = j + 1 < nmax;
          if (!(ok = wait_slot(vpos))) break;
          bool k_ready = false;
          for (int t = 0; ok && t < 3; ++t) {
            if (j < nt[t]) {
              if (!(ok = mbar_wait_warp(bar_p + 16 * t, (cnt[t] + j) & 1, p.ctl, ab))) break;
              // O_t of the previous item must have been read out
              if (j == 0 && r > 0 && !(ok = mbar_wait_warp(bar_oe + 8 * t, (r - 1) & 1, p.ctl, ab))) break;
              tc_fence_after();
              issue_pv(t, vpos, j > 0, 0);
              if (!(ok = mbar_wait_warp(bar_p + 16 * t + 8, (cnt[t] + j) & 1, p.ctl, ab))) break;
              tc_fence_after();
              issue_pv(t, vpos, true, 1);
              tc_commit_el(bar_o + 8 * t);
            }
            if (j + 1 < nt[t]) {
              if (!k_ready && !(ok = k_ready = wait_slot(kpos))) break;
              tc_fence_after();
              issue_s(t, kpos);
              tc_commit_el(bar_s + 8 * t);
              if (j + 2 == nt[t]) tc_commit_el(bar_qe + 8 * t);  // tile t's last S of the item
            }
          }
          if (!ok) break;
          tc_commit_el(bar_empty + 8 * (vpos % C::NSLOT));
          if (more) tc_commit_el(bar_empty + 8 * (kpos % C::NSLOT));
        }
        for (int t = 0; t < 3; ++t) cnt[t] += nt[t];
        pos += 2 * nmax;
      }
      // wait for every MMA issued above before TMEM may be released
      Abort no_abort{ab.flag + 1};
      tc_commit_el(bar_drain);
      mbar_wait_warp(bar_drain, 0, p.ctl, no_abort);
    }
  } else {
    // ------------------------------------------------------------------ softmax
    const int t = warp >> 2;                        // query tile of this warpgroup
    const int row_in_tile = (warp & 3) * 32 + lane;  // == TMEM lane
    const uint32_t lane_addr = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t s_tm = tmem + lane_addr + t * C::TILE_COLS;
    const uint32_t o_tm = s_tm + C::BN;
    const uint32_t my_bar_s = bar_s + 8 * t, my_bar_p = bar_p + 16 * t, my_bar_o = bar_o + 8 * t;
    const uint32_t my_bar_oe = bar_oe + 8 * t;
    const uint32_t stg_q = sbase + C::STG_OFF + static_cast<uint32_t>(warp) * (32 * D * 2);
    const float c = p.c;
    const uint64_t c2 = f2(c, c);
    const int off = p.Skv - p.Sq;
    int cnt = 0;  // S tiles of this query tile processed in earlier items
    bool ok = true;
    for (int r = 0, idx; ok && (idx = item_index(p, r)) >= 0; ++r) {
      int pos_item, bh;
      item_coords(p, idx, pos_item, bh);
      const int q0 = pos_item * kRows;
      const int row = q0 + t * C::BM + row_in_tile;
      const int limit = p.causal ? min(p.Skv, row + off + 1) : p.Skv;  // keys [0, limit) visible
      const int my_tiles = fwd4_tiles(p, q0, t);
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; ok && j < my_tiles; ++j)
        ok = softmax_step<D, C::BN>(s_tm, o_tm, my_bar_s, (cnt + j) & 1, my_bar_p, my_bar_o, (cnt + j - 1) & 1,
                                    j == 0, j * C::BN, limit, c, c2, m_run, l_run, p.ctl, ab);
      if (!ok) break;
      if (!(ok = softmax_epilogue<D>(o_tm, my_bar_o, (cnt + my_tiles - 1) & 1, my_bar_oe, m_run, l_run, row, bh, p,
                                     ab, &tm_o, stg_q)))
        break;
      cnt += my_tiles;
    }
    if (lane == 0) bulk_wait_group0();  // the O stores have completed before the CTA exits
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 13) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
  }
}

// ---------------------------------------------------------------- host side
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult qres;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &qres) == cudaSuccess &&
        qres == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

// 3-D view [planes, rows, D] of a [B, H, S, D] bf16 tensor with a 64 x box_rows box.
bool make_map(CUtensorMap* map, const void* base, int D, int rows, int planes, int box_rows) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(rows),
                        static_cast<cuuint64_t>(planes)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2,
                           static_cast<cuuint64_t>(D) * 2 * static_cast<cuuint64_t>(rows)};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D view [total, H, D] of a packed [total, H, D] bf16 tensor (innermost first: D, H,
// tokens) with a 64-column x 1-head x box_rows box, which lands in shared memory exactly
// like the dense 64 x box_rows box.
bool make_map_tokens(CUtensorMap* map, const void* base, int D, int H, int total, int box_rows) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(H), static_cast<cuuint64_t>(total)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(D) * 2 * static_cast<cuuint64_t>(H)};
  cuuint32_t box[3] = {64, 1, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// A launch, as a programmatic dependent of the previous kernel in the stream
// (cudaLaunchAttributeProgrammaticStreamSerialization) when `dependent`: the prefill
// kernels wait for that kernel (griddepcontrol.wait) after their set-up and before any
// global access, which costs nothing when they were launched plainly.  Non-causal launches
// take it (their set-up overlaps the previous grid's tail: +1.3 % on B4 H32 S2048, +10 %
// on B1 H32 S1024, back to back); causal ones do not (-4 % on B4 H32 S2048 causal: the
// early CTAs land on SMs in the order the previous grid frees them, which the causal
// dealing's L2 blocks do not expect).
template <class Kernel, class... Args>
cudaError_t launch_dependent(bool dependent, Kernel kernel, int grid, int threads, uint32_t smem,
                             cudaStream_t stream, Args... args) {
  if (!dependent) {
    kernel<<<grid, threads, smem, stream>>>(args...);
    return cudaGetLastError();
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(static_cast<unsigned>(threads));
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

template <int D>
cudaError_t launch_varlen_d(const FwdVarlenArgs& a, const KernelCtl& ctl, cudaStream_t stream) {
  using C = FwdCfg<D>;
  static PerDeviceOnce configured;
  CUtensorMap mq, mk, mv, mo;
  if (!make_map_tokens(&mq, a.q, D, a.Hq, a.total_q, C::BM) ||
      !make_map_tokens(&mk, a.k, D, a.Hkv, a.total_k, C::BN) ||
      !make_map_tokens(&mv, a.v, D, a.Hkv, a.total_k, C::BN) ||
      !make_map_tokens(&mo, a.o, D, a.Hq, a.total_q, 32))
    return cudaErrorInvalidValue;
  int dev = 0;
  cudaGetDevice(&dev);
  if (!configured.run(dev, [] {
        return cudaFuncSetAttribute(attn_fwd_kernel<D, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    C::BYTES) == cudaSuccess;
      }))
    return cudaErrorInvalidValue;
  FwdParams p;
  memset(&p, 0, sizeof(p));
  p.o = static_cast<__nv_bfloat16*>(a.o);
  p.lse = a.lse;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.causal = a.causal;
  p.c = a.scale * kLog2e;
  p.ctl = ctl;
  p.cu_q = a.cu_q;
  p.cu_k = a.cu_k;
  p.B = a.B;
  p.total_q = a.total_q;
  int sms = 0;
  cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  // items: at most B * Hq * ceil(max_seqlen_q / rows) (the persistent loop takes them all
  // whatever the grid; max_seqlen_q only caps the CTAs launched)
  constexpr int kRows = C::NQT * C::BM;
  const long long bound = static_cast<long long>(a.B) * a.Hq * ((a.max_seqlen_q + kRows - 1) / kRows);
  const int grid = static_cast<int>(bound > 0 && bound < sms ? bound : sms);
  return launch_dependent(false, attn_fwd_kernel<D, true>, grid, C::THREADS, C::BYTES, stream, mq, mk, mv, mo, p);
}

// Launch one design: C is its configuration, rows_per_item the query rows of one work
// item (C::NQT * C::BM).
template <int D, class C, class Kernel>
cudaError_t launch_design(Kernel kernel, int rows_per_item, const FwdArgs& a, const KernelCtl& ctl,
                          cudaStream_t stream, PerDeviceOnce& configured) {
  CUtensorMap mq, mk, mv, mo;
  if (!make_map(&mq, a.q, D, a.Sq, a.B * a.Hq, C::BM) ||
      !make_map(&mk, a.k, D, a.Skv, a.B * a.Hkv, C::BN) ||
      !make_map(&mv, a.v, D, a.Skv, a.B * a.Hkv, C::BN) ||
      !make_map(&mo, a.o, D, a.Sq, a.B * a.Hq, 32))  // epilogue: one 32-row block per warp
    return cudaErrorInvalidValue;
  int dev = 0;
  cudaGetDevice(&dev);
  if (!configured.run(dev, [&] {
        return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, C::BYTES) == cudaSuccess;
      }))
    return cudaErrorInvalidValue;
  FwdParams p;
  p.o = static_cast<__nv_bfloat16*>(a.o);
  p.lse = a.lse;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.Sq = a.Sq;
  p.Skv = a.Skv;
  p.n_pairs = (a.Sq + rows_per_item - 1) / rows_per_item;
  p.causal = a.causal;
  p.c = a.scale * kLog2e;
  p.ctl = ctl;
  const long long items = static_cast<long long>(p.n_pairs) * a.B * a.Hq;
  if (items > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  p.n_items = static_cast<int>(items);
  // (the block layout is set below, once the grid is known)
  // persistent: one CTA per SM (shared memory / TMEM admit one), each walking its items
  int sms = 0;
  cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const int grid = static_cast<int>(items < sms ? items : sms);
  p.plane_block = model::causal_block_layout(a.B * a.Hq, a.Hq / a.Hkv, a.Skv, D, p.n_pairs, grid, &p.last_h0);
  return launch_dependent(!a.causal, kernel, grid, C::THREADS, C::BYTES, stream, mq, mk, mv, mo, p);
}

// Ring depths compiled for the block-size ablation of the two-tile design (the model's
// depth and its neighbours that fit in shared memory, plus a shallow point).
template <int D>
cudaError_t launch_two_tile_slots(const FwdArgs& a, const KernelCtl& ctl, cudaStream_t stream, bool* handled) {
  *handled = true;
  constexpr int kRows = FwdCfg<D>::NQT * FwdCfg<D>::BM;
  if constexpr (D == 128) {
    static PerDeviceOnce once2;
    if (a.slots == 2) return launch_design<D, FwdCfg<D, 2>>(attn_fwd_kernel<D, false, 2>, kRows, a, ctl, stream, once2);
  } else {
    static PerDeviceOnce once3, once6, once9;
    if (a.slots == 3) return launch_design<D, FwdCfg<D, 3>>(attn_fwd_kernel<D, false, 3>, kRows, a, ctl, stream, once3);
    if (a.slots == 6) return launch_design<D, FwdCfg<D, 6>>(attn_fwd_kernel<D, false, 6>, kRows, a, ctl, stream, once6);
    if (a.slots == 9) return launch_design<D, FwdCfg<D, 9>>(attn_fwd_kernel<D, false, 9>, kRows, a, ctl, stream, once9);
  }
  *handled = false;
  return cudaSuccess;
}

template <int D>
cudaError_t launch_fwd_d(const FwdArgs& a, const KernelCtl& ctl, cudaStream_t stream) {
  static PerDeviceOnce configured1, configured2, configured3;
  constexpr int kModelDesign = model::fwd_plan(D).design;
  const int design = a.design ? a.design : kModelDesign;
  if (design == 2 && a.slots > 0 && a.slots != FwdCfg<D>::NSLOT) {
    bool handled = false;
    const cudaError_t e = launch_two_tile_slots<D>(a, ctl, stream, &handled);
    if (handled) return e;
  }
  if (design == 1)
    return launch_design<D, Fwd1Cfg<D>>(attn_fwd1_kernel<D>, Fwd1Cfg<D>::BM, a, ctl, stream, configured1);
  if constexpr (Fwd3Cfg<D>::kFeasible) {
    if (design == 3)
      return launch_design<D, Fwd3Cfg<D>>(attn_fwd3_kernel<D>, Fwd3Cfg<D>::NQT * Fwd3Cfg<D>::BM, a, ctl,
                                          stream, configured3);
  }
  if constexpr (Fwd4Cfg<D>::kFeasible) {
    static PerDeviceOnce configured4;
    if (design == 4)
      return launch_design<D, Fwd4Cfg<D>>(attn_fwd4_kernel<D>, Fwd4Cfg<D>::NQT * Fwd4Cfg<D>::BM, a, ctl,
                                          stream, configured4);
  }
  return launch_design<D, FwdCfg<D>>(attn_fwd_kernel<D>, FwdCfg<D>::NQT * FwdCfg<D>::BM, a, ctl, stream,
                                     configured2);
}

}  // namespace

cudaError_t launch_fwd(const FwdArgs& a, const KernelCtl& ctl, cudaStream_t stream) {
  if (a.D == 128) return launch_fwd_d<128>(a, ctl, stream);
  return launch_fwd_d<64>(a, ctl, stream);
}

cudaError_t launch_fwd_varlen(const FwdVarlenArgs& a, const KernelCtl& ctl, cudaStream_t stream) {
  if (a.D == 128) return launch_varlen_d<128>(a, ctl, stream);
  return launch_varlen_d<64>(a, ctl, stream);
}

}  // namespace loom
