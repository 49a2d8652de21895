// Analytic schedule model: the paper's Hierarchical Execution Graph latency model
// (Sec. 2.6, Eq. 5-7) and its constrained selection (Eq. 8-9), restated for one GB300
// SM and evaluated by exhaustive enumeration over a small finite domain instead of a
// CP-SAT solve.  Everything is constexpr: the kernels take their tile and stage
// constants from `fwd_plan(D)` / `decode_stage_plan(D)` at compile time, and the host
// picks the decode split count with `choose_decode_splits` at run time.
//
// Architecture description (Sec. 2.7): structural numbers are GB300 specifications;
// throughput numbers are measurements on this GPU type (HBM copy bandwidth and dense
// bf16 GEMM throughput measured with a STREAM-style copy and a cuBLAS GEMM).  Numbers
// marked "assumed" are placeholders for per-architecture microbenchmarks.
#pragma once

#include <cstddef>
#include <cstdint>
#include <initializer_list>

namespace loom {
namespace model {

struct ArchDesc {
  // structural (specifications)
  int num_sms;              // streaming multiprocessors
  int smem_per_sm;          // bytes of shared memory per SM usable by CTAs
  int smem_per_cta;         // bytes of dynamic shared memory one CTA may opt into
  int tmem_cols;            // 32-bit TMEM columns per SM (x 128 lanes)
  int regs_per_sm;          // 32-bit registers per SM
  // performance (measured / assumed)
  double sm_ghz;            // SM clock under sustained load (measured median)
  double hbm_gbs;           // HBM copy bandwidth, GB/s (measured)
  double mma_tflops;        // dense bf16 tensor throughput of the GPU (measured burst)
  double l2_smem_gbs_sm;    // L2 -> shared memory bandwidth of one SM, GB/s (assumed)
  double ex2_per_clk_sm;    // MUFU.EX2 results per clock per SM (assumed)
  double fp32_per_clk_sm;   // fp32 FMA-pipe lane-ops per clock per SM (specification)
  double mem_latency_ns;    // loaded HBM latency of a bulk copy (assumed)
  double sync_ns;           // fixed per-iteration cost of an mbarrier/TMEM round trip (assumed)
  double launch_ns;         // fixed cost of one dependent kernel launch (assumed)
  double decode_cta_gbs;    // KV stream rate of a lone decode split CTA on an SM (measured)
  double cta_start_ns;      // start-up of a decode split CTA: launch, first copies (measured)
  double mma_clk_per_n;     // clocks of one 128xNx16 bf16 MMA per unit of N (measured: 0.5)
  double mma_min_clk;       // floor on one MMA's clocks (measured: 48 at N = 64)
  double softmax_clk_per_key;       // softmax of one 128-row tile alone, clocks per key (measured)
  double softmax_pair_clk_per_key;  // two tiles' softmax running together, clocks per key (measured)
  double l2_bytes;                  // L2 cache capacity (specification)
  double mma_issue_busy_factor;     // MMA stream slowdown while high-ILP warps share the SM with
                                    // the MMA warp issuing warp-wide (measured: 546 vs 512 clk
                                    // per 128^3 GEMM; 1338 when a lone lane issues)
  double item_boundary_ns;  // prefill: per work item of a CTA, the part that does not overlap
                            // the previous item: its first S -> softmax -> P.V chain, the causal
                            // diagonal steps and the last P.V with the O read-out (in-kernel
                            // clock trace of causal B4 H32 S2048: ~6300 clk per item at ~1.9 GHz;
                            // with fwd_launch_ns fitted to B1 S1024 and B16 S512 non-causal)
  double decode_item_ns;    // persistent decode: per (unit, split) item, the warps' merge with
                            // the item's last ring slot held, the partial write and the next
                            // item's q (fitted: B4 H32/8 S16384 measured 56 / 60 us with one / two
                            // items per CTA)
  double softmax_triple_clk_per_key;  // three tiles' softmax running together (design 4, 96-key
                                      // tiles, 14 warps at 128 registers), clocks per key of a
                                      // round (measured: 876 TFLOP/s on B1 H64 S8192 D64 causal)
  double cluster_merge_ns;          // per unit and CTA of a cluster-decode cluster: the
                                    // handshakes waiting on the slowest CTA and the DSMEM gather
                                    // (fitted: 147 us measured with clusters of 16 on the batched
                                    // decode, 123 us with clusters of 4 on B64 S2048)
  double fwd_launch_ns;             // prefill: once per launch, the launch itself, the first Q
                                    // and K/V loads from HBM and the last item's epilogue
                                    // (fitted: B1 H32 S1024 measured 18.9 us, B16 H16 S512 41.3 us,
                                    // one and four items per CTA, launches timed back to back)
  double decode_tc_item_ns;         // persistent tensor-core decode: per (sequence, kv head, split)
                                    // item, the stall of the S -> softmax -> P.V chain at the item's
                                    // boundary (O read-out, next q into TMEM) that the full ring does
                                    // not hide (fitted: batched B16 H32/8 lengths U[4096, 8192], 16 vs
                                    // 32 splits, 70.9 vs 74.2 us, less the merge's extra partials)
  double decode_tc_cta_gbs;         // persistent tensor-core decode: KV stream rate one CTA sustains
                                    // when HBM is not the bound (fitted: B1 H32/8 Skv 131072 with
                                    // 8 and 16 splits, 64 and 128 CTAs, 218.6 and 117.2 us)
  double decode_tc_stage_ns;        // persistent tensor-core decode: the S -> softmax -> P.V chain
                                    // per 64 keys of a stage, the floor of a stage when its bytes
                                    // arrive faster (fitted: D = 64, B1 H64/16 Skv 65536, 19 splits
                                    // in 128-key stages: 54.4 us for 3456 keys per CTA)
  double decode_merge_ns;           // the merge launch's fixed cost in a decode step: the dependent
                                    // launch, its wait for the split grid, one round trip to the
                                    // partials (fitted: a timing probe without the merge launch,
                                    // 3.2-4.8 us per step less the partials' traffic)
};

inline constexpr ArchDesc kGb300 = {
    152, 228 * 1024, 227 * 1024, 512, 65536,
    1.447, 6783.5, 1910.3, 110.0, 32.0, 128.0, 1500.0, 150.0, 2500.0, 32.0, 6000.0, 0.5, 48.0, 9.8, 10.75,
    129.0e6, 1.07, 3400.0, 3000.0, 28.4, 150.0, 2000.0, 300.0, 39.0, 835.0, 3000.0,
};

// ------------------------------------------------------------------ HEG composition
// Eq. 6: latency of pipe(l, body, s) under the two-bit pipeline knob (b_lm, b_ms).
constexpr double heg_pipe(double l, double m, double s, int b_lm, int b_ms) {
  if (!b_lm && !b_ms) return l + m + s;
  if (!b_lm && b_ms) return (l + m) > s ? (l + m) : s;
  if (b_lm && !b_ms) return l > (m + s) ? l : (m + s);
  double x = l > m ? l : m;
  return x > s ? x : s;
}
// Eq. 7: for(i, g)
constexpr double heg_for(double trips, double body) { return trips * body; }
// Eq. 5: g1 ; g2
constexpr double heg_seq(double a, double b) { return a + b; }

constexpr double dmax(double a, double b) { return a > b ? a : b; }
constexpr long long cdiv(long long a, long long b) { return (a + b - 1) / b; }

// ------------------------------------------------------------------ prefill
// Candidates: design x BN keys per tile x KV ring slots x knob b = (b_lm, b_ms).
// BM = 128 query rows per tile (one per TMEM lane).  Three designs are implemented:
//   design 2: two query tiles, one S buffer each; the tiles alternate on the tensor
//     pipe, and each tile's chain S -> softmax -> P.V -> next S is serial;
//   design 1: one query tile, S double-buffered: the boundary between the S MMA and
//     the softmax body is opened (Eq. 6 knob) at the price of a second S buffer;
//   design 3: two query tiles sharing a ring of three S buffers: both tiles' next S is
//     computed while their softmax runs, so the two softmaxes overlap each other and the
//     MMAs (TMEM: 3 BN + 2 D columns).
//   design 4: three query tiles, one S buffer each, over KV tiles of BN = 96 keys (TMEM:
//     3 (BN + D) columns, D = 64 only): the tiles take turns on the tensor pipe like
//     design 2's two, so each tile's chain has two other tiles' MMAs to hide behind.
struct FwdPlan {
  int design, bm, bn, q_tiles, s_buffers, kv_slots, b_lm, b_ms;
  int smem_bytes, tmem_cols;
  double t_load_ns, t_mma_ns, t_softmax_ns, t_iter_ns;  // per KV tile, per query tile
  bool feasible;
};

// Primitive latencies of one KV-tile iteration (per query tile, ns).
constexpr FwdPlan fwd_eval(const ArchDesc& a, int D, int design, int bn, int slots, int b_lm,
                           int b_ms) {
  FwdPlan p{};
  p.design = design;
  p.bm = 128;
  p.q_tiles = design == 1 ? 1 : design == 4 ? 3 : 2;
  p.s_buffers = design == 1 ? 2 : design == 3 ? 3 : 1;
  p.bn = bn;
  p.kv_slots = slots;
  p.b_lm = b_lm;
  p.b_ms = b_ms;
  const double clk = a.sm_ghz;  // clocks per ns
  // load stage: K_j and V_j tiles (mostly L2 hits), shared by the CTA's query tiles
  p.t_load_ns = 2.0 * bn * D * 2 / a.l2_smem_gbs_sm / p.q_tiles;
  // compute leaf: S = Q K^T (N = BN) and O += P V (N = D), K/16 MMAs each
  auto mma_clk = [&](int n) { return dmax(a.mma_clk_per_n * n, a.mma_min_clk); };
  p.t_mma_ns = ((D / 16.0) * mma_clk(bn) + (bn / 16.0) * mma_clk(D)) / clk;
  // softmax leaf of one query tile (measured clocks per key of a 128-row tile)
  p.t_softmax_ns = a.softmax_clk_per_key * bn / clk;
  const double sync = a.sync_ns;
  double body = 0.0;
  if (design == 2 || design == 4) {
    // per round of tile-iterations (one per query tile) the tensor pipe needs q_tiles *
    // mma; each tile's chain (its softmax, then its P.V and next S on the tensor pipe, one
    // barrier round trip: the warp-wide MMA issuer picks P up at once) must fit in the
    // round, while the other tiles' softmaxes overlap it.  With three tiles the three
    // softmaxes share the SM sub-partitions' MUFU and issue slots (and 14 warps cap a thread
    // at 128 registers): a round takes at least their measured joint time.
    body = dmax(p.q_tiles * p.t_mma_ns, p.t_softmax_ns + p.t_mma_ns + sync);
    if (design == 4) body = dmax(body, a.softmax_triple_clk_per_key * bn / clk);
    body /= p.q_tiles;
  } else if (design == 1) {
    body = dmax(p.t_mma_ns, p.t_softmax_ns) + sync;  // softmax and MMA overlap fully
  } else {
    // both softmaxes run together (sharing MUFU and issue slots) and overlap the MMAs,
    // whose stream is stretched by the busy warps; yet every S is issued behind a P.V of
    // the other tile on the single MMA stream, so a tile's chain still holds its softmax,
    // a P.V + S and two barrier round trips (in-kernel clock counters: the softmax waits
    // ~1060 clk per step for S, against ~760 in design 2)
    const double pair = a.softmax_pair_clk_per_key * bn / clk;
    body = dmax(dmax(2 * p.t_mma_ns * a.mma_issue_busy_factor, pair),
                p.t_softmax_ns + p.t_mma_ns + 2 * sync) / 2;
  }
  p.t_iter_ns = heg_pipe(p.t_load_ns, body, 0.0, b_lm, b_ms);
  // resources (Eq. 8 constraints)
  // Q tiles + K/V ring + an O staging tile per query tile (TMA-store epilogue) +
  // barriers and alignment
  p.smem_bytes = 2 * p.q_tiles * p.bm * D * 2 + slots * bn * D * 2 + 1024 + 256;
  // design 4 keeps each tile's S and O adjacent at 32-column aligned bases (t * 160)
  p.tmem_cols = design == 1 ? 2 * bn + D : design == 2 ? 2 * (bn + D) : design == 3 ? 3 * bn + 2 * D
                                                                      : 3 * (bn + D);
  p.feasible = true;
  if (design < 1 || design > 4) p.feasible = false;
  if (bn % 16 != 0 || bn < 16 || bn > 256) p.feasible = false;   // MMA N for M = 128
  // softmax: one S row per thread, P handed over in two halves: 128 keys (64 + 64) for
  // designs 1-3, 96 keys (64 + 32) for design 4
  if (bn != (design == 4 ? 96 : 128)) p.feasible = false;
  if (design == 4 && D != 64) p.feasible = false;  // 3 S buffers + 3 O accumulators in 512 columns
  if (D % 64 != 0) p.feasible = false;                            // 128 B swizzle atoms
  if (p.smem_bytes > a.smem_per_cta) p.feasible = false;          // L1 footprint
  if (p.tmem_cols > a.tmem_cols) p.feasible = false;
  // an open load boundary needs loads in flight while the MMAs read the current tiles:
  // the MMA warp holds two slots (V_j and K_{j+1}); the other slots - 2 are the
  // look-ahead, each consumed in half a KV-tile period, which must cover the latency of
  // an L2-resident tile (half the HBM latency)
  if (slots < 3) p.feasible = false;
  if (b_lm && (slots - 2) * body * p.q_tiles / 2 < a.mem_latency_ns * 0.5) p.feasible = false;
  if (!b_lm) p.feasible = false;  // every kernel prefetches through the ring
  return p;
}

// Eq. 8 for one design by enumeration over BN, slots and knobs; ties go to the deeper
// ring (more latency slack for the same modeled time).
constexpr FwdPlan fwd_plan_variant(int D, int design, const ArchDesc& a = kGb300) {
  FwdPlan best{};
  best.feasible = false;
  for (int bn = 32; bn <= 256; bn += 16)
    for (int slots = 2; slots <= 16; ++slots)
      for (int b_lm = 0; b_lm <= 1; ++b_lm)
        for (int b_ms = 0; b_ms <= 1; ++b_ms) {
          FwdPlan p = fwd_eval(a, D, design, bn, slots, b_lm, b_ms);
          if (!p.feasible) continue;
          const double cost = p.t_iter_ns / bn;  // per key and query tile
          const double best_cost = best.feasible ? best.t_iter_ns / best.bn : 1e300;
          if (cost < best_cost * (1.0 - 1e-9) ||
              (cost <= best_cost * (1.0 + 1e-9) && slots > best.kv_slots))
            best = p;
        }
  return best;
}

// Eq. 9: the design with the lowest modeled latency (ties keep the earlier design).
constexpr FwdPlan fwd_plan(int D, const ArchDesc& a = kGb300) {
  FwdPlan best = fwd_plan_variant(D, 2, a);
  for (int design : {1, 3, 4}) {
    const FwdPlan p = fwd_plan_variant(D, design, a);
    if (!p.feasible) continue;
    if (!best.feasible || p.t_iter_ns / p.bn < best.t_iter_ns / best.bn * (1.0 - 1e-9)) best = p;
  }
  return best;
}

// Causal work order: (b, h) planes per block such that the distinct K/V bytes the block
// streams (a K/V plane is shared by `group` query heads) stay within 40% of L2, leaving
// room for Q, O and the next block's first tiles.  Items are dealt block by block, so
// the CTAs working at the same time re-read K/V from L2 rather than HBM.
constexpr int causal_plane_block(int planes, int group, int Skv, int D, const ArchDesc& a = kGb300) {
  const double per_plane = 2.0 * Skv * D * 2 / (group > 0 ? group : 1);
  double blk = 0.4 * a.l2_bytes / per_plane;
  if (blk < 1.0) blk = 1.0;
  return blk >= planes ? planes : static_cast<int>(blk);
}

// Block layout of the causal order for `grid` persistent CTAs dealing `items_per_plane`
// items of every plane heaviest first, in a snake order (CTA c takes the c-th item of even
// rounds and the (grid-1-c)-th of odd ones): a block whose items fill whole pairs of
// rounds gives every CTA one item from the heavy end and one from the light end of each
// pair, so blocks are sized to whole round pairs where the plane count allows, and the
// remainder joins the last block (its items are then dealt heaviest first together with a
// whole round pair, instead of forming a final round of heavy items on a few CTAs).
// Returns the regular block size; *last_h0 is the first plane of the final block.
constexpr int causal_block_layout(int planes, int group, int Skv, int D, int items_per_plane, int grid,
                                  int* last_h0, const ArchDesc& a = kGb300) {
  const int budget = causal_plane_block(planes, group, Skv, D, a);
  *last_h0 = 0;
  if (budget >= planes) return planes;  // everything fits: one heaviest-first order
  const long long pair_items = 2LL * grid;
  if (items_per_plane <= 0 || pair_items % items_per_plane != 0) {
    *last_h0 = (planes - 1) / budget * budget;  // blocks of the budget, the last one partial
    return budget;
  }
  const int unit = static_cast<int>(pair_items / items_per_plane);  // planes per round pair
  if (unit > budget) {
    *last_h0 = (planes - 1) / budget * budget;
    return budget;
  }
  const int blk = budget / unit * unit;
  const int full = planes / blk;              // whole blocks
  *last_h0 = full >= 1 ? (full - 1) * blk : 0;  // the last whole block absorbs the remainder
  if (planes % blk == 0) *last_h0 = (full - 1) * blk;
  return blk;
}

// Modeled time (us) of a whole prefill launch under a plan (Eq. 5-7 over the CTA's
// items: launch ; for(items, item boundary ; for(KV tiles, pipe))).  The query tiles of
// an item take turns on the tensor pipe, so a KV-tile step costs a full round of
// q_tiles iterations even when some tile (causal: the item's upper tiles) has no work left
// in it: an item costs its slowest tile's KV tiles x q_tiles x t_iter, plus the part of
// the item that overlaps nothing (item_boundary_ns: its first S -> softmax -> P.V chain,
// the diagonal steps, the last P.V and the O read-out), and a launch adds fwd_launch_ns.
constexpr double fwd_time_us(const FwdPlan& p, int B, int Hq, int Sq, int Skv, int D, int causal,
                             const ArchDesc& a = kGb300) {
  (void)D;
  const long long rows_per_item = 1LL * p.q_tiles * p.bm;
  const long long groups = cdiv(Sq, rows_per_item);
  const long long items = groups * B * Hq;
  double item_tiles = 0;  // average over an item's of its slowest query tile's KV tiles
  for (long long g = 0; g < groups; ++g) {
    long long n_max = 0;
    for (long long t = 0; t < p.q_tiles; ++t) {
      const long long i = g * p.q_tiles + t;  // query tile
      if (i * p.bm >= Sq) break;
      long long n_kv = Skv;
      if (causal) {
        const long long lim = (i + 1) * p.bm + (Skv - Sq);
        n_kv = lim < Skv ? lim : Skv;
      }
      const long long n = cdiv(n_kv, p.bn);
      n_max = n > n_max ? n : n_max;
    }
    item_tiles += static_cast<double>(n_max);
  }
  item_tiles /= static_cast<double>(groups);
  const double t_item = heg_seq(a.item_boundary_ns, heg_for(item_tiles * p.q_tiles, p.t_iter_ns));
  // Persistent CTAs take whole items.  Equal items (non-causal): the busiest CTA runs
  // ceil(items / SMs) of them.  Causal items differ in length and the snake dealing evens
  // the work per CTA out, so the average share is priced (at least one item).
  const double share = static_cast<double>(items) / a.num_sms;
  const double w = causal ? (share < 1.0 ? 1.0 : share) : static_cast<double>(cdiv(items, a.num_sms));
  return heg_seq(a.fwd_launch_ns, w * t_item) * 1e-3;
}

// ------------------------------------------------------------------ decode
// Stage plan of the split kernel: T keys per stage, NSTAGE ring depth, CTAs per SM.
struct DecodeStagePlan {
  int tokens, stages, ctas_per_sm;
  int smem_bytes;
  double t_stage_ns;      // one stage of one CTA at its share of HBM bandwidth
  double bytes_in_flight_sm;
  bool feasible;
};

constexpr DecodeStagePlan decode_stage_eval(const ArchDesc& a, int D, int tokens, int stages,
                                            int ctas_per_sm) {
  DecodeStagePlan p{};
  p.tokens = tokens;
  p.stages = stages;
  p.ctas_per_sm = ctas_per_sm;
  const double stage_bytes = 2.0 * tokens * D * 2;
  p.smem_bytes = static_cast<int>(stages * stage_bytes) + 4096;
  p.bytes_in_flight_sm = stage_bytes * (stages - 1) * ctas_per_sm;
  const double bw_cta = a.hbm_gbs / (a.num_sms * ctas_per_sm);  // bytes/ns per CTA
  const double l = stage_bytes / bw_cta;
  p.t_stage_ns = heg_pipe(l, 0.0, 0.0, 1, 1);
  // Little's law: enough bytes in flight per SM to cover the memory latency
  const double need = a.hbm_gbs / a.num_sms * a.mem_latency_ns;
  // while the compute warps read one stage, the other stages-1 are in flight
  p.feasible = p.smem_bytes * ctas_per_sm <= a.smem_per_sm && p.smem_bytes <= a.smem_per_cta &&
               stage_bytes * (stages - 1) * ctas_per_sm >= need && stages >= 2 &&
               tokens % 64 == 0 && (tokens / 8) % (256 / D) == 0;
  return p;
}

// Smallest footprint that keeps HBM saturated: among feasible (tokens, stages,
// CTAs/SM), prefer 2 CTAs per SM (latency tolerance of the compute warps), then the
// smallest ring.
constexpr DecodeStagePlan decode_stage_plan(int D, const ArchDesc& a = kGb300) {
  DecodeStagePlan best{};
  best.feasible = false;
  for (int ctas = 2; ctas >= 1; --ctas)
    for (int tokens = 64; tokens <= 256; tokens += 64)
      for (int stages = 2; stages <= 8; ++stages) {
        DecodeStagePlan p = decode_stage_eval(a, D, tokens, stages, ctas);
        if (!p.feasible) continue;
        if (!best.feasible || p.ctas_per_sm > best.ctas_per_sm ||
            (p.ctas_per_sm == best.ctas_per_sm && p.smem_bytes < best.smem_bytes))
          best = p;
      }
  return best;
}

// The stage plans of the two supported head dimensions, evaluated at compile time.
inline constexpr DecodeStagePlan kDecodeStage64 = decode_stage_plan(64);
inline constexpr DecodeStagePlan kDecodeStage128 = decode_stage_plan(128);
constexpr const DecodeStagePlan& decode_stage(int D) { return D == 64 ? kDecodeStage64 : kDecodeStage128; }

struct DecodeSplitPlan {
  int splits;
  double t_us;  // modeled time of the chosen form
  int cluster;  // 0: split kernel + merge kernel; cs > 0: the cluster kernel, clusters of cs CTAs
};

// Largest cluster of the single-kernel (cluster) Flash Decode: 16 CTAs, the largest
// (non-portable) thread-block cluster.
constexpr int kMaxClusterSize = 16;

// Number of q heads one split CTA serves (must match the kernel dispatch).
constexpr int decode_group_tile(int G) { return G >= 8 ? 8 : G >= 4 ? 4 : G >= 2 ? 2 : 1; }

// The split loop of Flash Decode (Eq. 6-7 with an open load boundary), evaluated on the
// busiest SM: it runs ceil(CTAs / SMs) split CTAs in rounds of at most CTAs-per-SM at a
// time; a round of k CTAs streams at min(the SM's share of HBM / k, the rate one CTA
// sustains), and each round pays the CTA start-up (launch and first copies).
constexpr double decode_split_loop_ns(int splits, int B, int Hq, int Hkv, int Skv, int D, int num_sms,
                                      const ArchDesc& a) {
  const DecodeStagePlan& sp = decode_stage(D);
  const int G = Hq / Hkv;
  const int gt = decode_group_tile(G);
  const long long units = 1LL * B * Hkv * cdiv(G, gt);
  const long long ctas = units * splits;
  const long long chunk = cdiv(cdiv(Skv, splits), 64) * 64;
  const double chunk_bytes = 2.0 * chunk * D * 2;
  const long long per_sm = cdiv(ctas, num_sms);
  const double active_sms = static_cast<double>(ctas < num_sms ? ctas : num_sms);
  const double share = a.hbm_gbs / active_sms;  // bytes/ns for one SM
  double t_split = 0.0;
  for (long long left = per_sm; left > 0;) {
    const long long k = left < sp.ctas_per_sm ? left : sp.ctas_per_sm;
    left -= k;
    double bw = share / static_cast<double>(k);
    if (bw > a.decode_cta_gbs) bw = a.decode_cta_gbs;
    t_split += heg_seq(a.cta_start_ns, chunk_bytes / bw);
  }
  return t_split;
}

// Stream rate (bytes/ns) of one of `ctas` CTAs resident at once: the busiest SM holds
// ceil(ctas / SMs) of them and they share its part of HBM, up to the rate one CTA sustains.
constexpr double decode_cta_rate(double ctas, int num_sms, const ArchDesc& a) {
  const double active = ctas < num_sms ? ctas : static_cast<double>(num_sms);
  long long k = static_cast<long long>(ctas / num_sms);
  if (static_cast<double>(k) * num_sms < ctas) ++k;
  if (k < 1) k = 1;
  const double rate = a.hbm_gbs / active / static_cast<double>(k);
  return rate < a.decode_cta_gbs ? rate : a.decode_cta_gbs;
}

// Eq. 5 for Flash Decode in the split + merge form: T = T_split-loop ; T_merge (gather +
// global softmax + final scaling), the merge a second, dependent launch that reads the
// partials back.
constexpr double decode_time_us(int splits, int B, int Hq, int Hkv, int Skv, int D, int num_sms,
                                const ArchDesc& a = kGb300) {
  const double t_split = decode_split_loop_ns(splits, B, Hq, Hkv, Skv, D, num_sms, a);
  const double part_bytes = 1.0 * B * Hq * splits * (D + 1) * 4;
  const double t_merge = a.decode_merge_ns + 2.0 * part_bytes / a.hbm_gbs;
  return heg_seq(t_split, t_merge) * 1e-3;
}

// Eq. 5 for the single-kernel form: persistent clusters of cs CTAs (cs divides the split
// count); the min(fit_clusters, units) clusters each walk ceil(units / clusters) units, and
// a CTA streams splits / cs chunks of every unit at min(its share of HBM, the rate one CTA
// sustains), without a break between units.  Per unit it pays what the persistent split
// kernel pays per item (decode_item_ns) and the gather + global softmax + scaling over DSMEM
// with its handshakes, which wait for the slowest of the cluster's CTAs (cluster_merge_ns
// per CTA of the cluster); the start-up once.  No merge launch, no workspace.
constexpr double decode_cluster_time_us(int splits, int cs, int B, int Hq, int Hkv, int Skv, int D,
                                        int fit_clusters, const ArchDesc& a = kGb300) {
  if (cs < 1 || cs > kMaxClusterSize || splits < cs || splits % cs != 0 || fit_clusters < 1) return 1e300;
  const int G = Hq / Hkv;
  const long long units = 1LL * B * Hkv * cdiv(G, decode_group_tile(G));
  const long long clusters = units < fit_clusters ? units : fit_clusters;
  const double ctas = static_cast<double>(clusters * cs);
  const long long chunk = cdiv(cdiv(Skv, splits), 64) * 64;
  const double cta_unit_bytes = static_cast<double>(splits / cs) * 2.0 * chunk * D * 2;
  const double rate = decode_cta_rate(ctas, a.num_sms, a);
  const double per_unit = heg_seq(cta_unit_bytes / rate, heg_seq(a.decode_item_ns, a.cluster_merge_ns * cs));
  return heg_seq(a.cta_start_ns, heg_for(static_cast<double>(cdiv(units, clusters)), per_unit)) * 1e-3;
}

// Eq. 5 for the persistent split kernel + merge: ctas persistent CTAs walk the units x
// splits items (ceil(items / ctas) each, as evened out by the launch), each CTA streaming
// its items back to back at min(its share of HBM, the rate one CTA sustains); the start-up
// once, a per-item cost for the warps' merge and the partial write (item_ns), then the
// merge launch of the split + merge form.
constexpr double decode_persistent_time_us(int splits, int B, int Hq, int Hkv, int Skv, int D, int slots,
                                           const ArchDesc& a = kGb300) {
  if (splits < 1 || slots < 1) return 1e300;
  const int G = Hq / Hkv;
  const long long items = 1LL * B * Hkv * cdiv(G, decode_group_tile(G)) * splits;
  const long long per = cdiv(items, slots);
  const double ctas = static_cast<double>(cdiv(items, per));
  const long long chunk = cdiv(cdiv(Skv, splits), 64) * 64;
  const double chunk_bytes = 2.0 * chunk * D * 2;
  const double rate = decode_cta_rate(ctas, a.num_sms, a);
  const double t_split = heg_seq(a.cta_start_ns, heg_for(static_cast<double>(per),
                                                         heg_seq(chunk_bytes / rate, a.decode_item_ns)));
  const double part_bytes = 1.0 * B * Hq * splits * (D + 1) * 4;
  const double t_merge = a.decode_merge_ns + 2.0 * part_bytes / a.hbm_gbs;
  return heg_seq(t_split, t_merge) * 1e-3;
}

// Keys per stage of the tensor-core decode split kernels: 64 at D = 128 (TMEM: q 64, S 64
// and O 128 columns of a CTA's 256); 128 at D = 64 (q 32, S 128, O 64), where a 64-key
// stage carries too few bytes to cover its S -> softmax -> P.V chain.
constexpr int decode_tc_stage_keys(int D) { return D == 64 ? 128 : 64; }

// Eq. 5 for the split + merge form whose split kernel runs on the tensor cores as
// persistent CTAs (two per SM) taking the items on demand: the start-up once; the items,
// all of one length, go in rounds of at most 2 x SMs (the last round may be partial).
// Within a round the active CTAs share HBM (the stage runs on the tensor pipe, so two CTAs
// on an SM do not slow each other), each up to the rate one CTA sustains; an item streams
// its chunk at that rate, or at one S -> softmax -> P.V chain per 64-key stage when that is
// slower (Eq. 6 with an open load boundary), and pays decode_tc_item_ns at its boundary;
// then the merge launch.
constexpr double decode_tc_time_us(int splits, int B, int Hq, int Hkv, int Skv, int D, int num_sms,
                                   const ArchDesc& a = kGb300) {
  if (splits < 1 || num_sms < 1) return 1e300;
  const long long items = 1LL * B * Hkv * splits;
  const long long slots = 2LL * num_sms;
  const long long chunk = cdiv(cdiv(Skv, splits), 64) * 64;
  const double chunk_bytes = 2.0 * chunk * D * 2;
  const double chain = static_cast<double>(chunk / 64) * a.decode_tc_stage_ns;  // per 64 keys of the chunk
  double t_split = a.cta_start_ns;
  for (long long left = items; left > 0;) {
    const long long active = left < slots ? left : slots;
    left -= active;
    double rate = a.hbm_gbs / static_cast<double>(active);
    if (rate > a.decode_tc_cta_gbs) rate = a.decode_tc_cta_gbs;
    t_split += heg_pipe(chunk_bytes / rate, chain, 0.0, 1, 1) + a.decode_tc_item_ns;
  }
  const double part_bytes = 1.0 * B * Hq * splits * (D + 1) * 4;
  const double t_merge = a.decode_merge_ns + 2.0 * part_bytes / a.hbm_gbs;
  return heg_seq(t_split, t_merge) * 1e-3;
}

// Clusters of cs decode CTAs in one GPC-sized group when no device can be asked: whole
// clusters in 8 equal groups of SMs at the stage plan's CTAs per SM.
constexpr int decode_default_clusters(int num_sms, int cs, int D) {
  if (cs < 1) return 0;
  const int per_gpc = num_sms / 8 * decode_stage(D).ctas_per_sm;
  return per_gpc / cs * 8;
}

struct DecodeClusterChoice {
  int cs;       // 0: no cluster size can run
  double t_us;
};

// The cluster size of the single-kernel form for a split count: Eq. 9 over the sizes that
// divide it and fit (fit(cs): clusters of cs CTAs resident at once, 0 if none); forced_cs
// > 0 admits that size only.  Ties keep the smaller cluster.
template <class Fit>
constexpr DecodeClusterChoice choose_decode_cluster(int splits, int B, int Hq, int Hkv, int Skv, int D, Fit fit,
                                                    int forced_cs = 0, const ArchDesc& a = kGb300) {
  DecodeClusterChoice best{0, 1e300};
  for (int cs = 1; cs <= kMaxClusterSize && cs <= splits; ++cs) {
    if (splits % cs != 0 || (forced_cs > 0 && cs != forced_cs)) continue;
    const int f = fit(cs);
    if (f < 1) continue;
    const double t = decode_cluster_time_us(splits, cs, B, Hq, Hkv, Skv, D, f, a);
    if (t < best.t_us * (1.0 - 1e-9)) best = {cs, t};
  }
  return best;
}

// Eq. 9 over the Flash Decode forms and every split count: the split + merge form (its
// split kernel on the tensor cores when `tc`), the persistent split + merge form on
// `slots` CTAs (0: not considered) and the cluster form with fit(cs) clusters of cs CTAs
// (always 0: not considered).  Ties keep the earlier form and fewer splits.
// DecodeSplitPlan::cluster: 0 split + merge, -1 persistent, cs cluster.
template <class Fit>
constexpr DecodeSplitPlan choose_decode_plan(int B, int Hq, int Hkv, int Skv, int D, int num_sms, Fit fit,
                                             int slots = 0, const ArchDesc& a = kGb300, bool tc = false) {
  DecodeSplitPlan best{1, 1e300, 0};
  const long long max_splits = cdiv(Skv, 64) < 1024 ? cdiv(Skv, 64) : 1024;
  for (int s = 1; s <= max_splits; ++s) {
    const double t = tc ? decode_tc_time_us(s, B, Hq, Hkv, Skv, D, num_sms, a)
                        : decode_time_us(s, B, Hq, Hkv, Skv, D, num_sms, a);
    if (t < best.t_us * (1.0 - 1e-9)) best = {s, t, 0};
  }
  for (int s = 1; slots > 0 && s <= max_splits; ++s) {
    const double t = decode_persistent_time_us(s, B, Hq, Hkv, Skv, D, slots, a);
    if (t < best.t_us * (1.0 - 1e-9)) best = {s, t, -1};
  }
  for (int s = 1; s <= max_splits; ++s) {
    const DecodeClusterChoice c = choose_decode_cluster(s, B, Hq, Hkv, Skv, D, fit, 0, a);
    if (c.cs > 0 && c.t_us < best.t_us * (1.0 - 1e-9)) best = {s, c.t_us, c.cs};
  }
  return best;
}

// The split + merge form alone (Eq. 9 over its split counts).
constexpr DecodeSplitPlan choose_decode_splits(int B, int Hq, int Hkv, int Skv, int D, int num_sms,
                                               const ArchDesc& a = kGb300) {
  return choose_decode_plan(B, Hq, Hkv, Skv, D, num_sms, [](int) { return 0; }, 0, a);
}

}  // namespace model
}  // namespace loom
