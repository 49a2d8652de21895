// Analytic model of the BF16 GEMM (C = A B), the paper's third kernel (Sec. 4): the HEG
// latency composition of Eq. 5-7 and the enumerated choice of Eq. 8-9, restated for one
// GB300 SM.  It shares the architecture description and the HEG operators of model.h.
#pragma once

#include "model.h"

namespace loom {
namespace model {

// ------------------------------------------------------------------ persistent tiles
// The paper's third kernel.  A CTA computes BM = 128 rows x BN columns of C at a time,
// with K in BK = 64 stages through an NSTAGE ring (Eq. 6 with the load boundary open)
// and the accumulator double-buffered in TMEM, so that one tile's epilogue overlaps the
// next tile's MMAs.  Candidates: BN in {64, 128, 192, 256} x ring depth.
struct GemmPlan {
  int bm, bn, bk, stages, smem_bytes, tmem_cols;
  double t_load_ns, t_mma_ns, t_iter_ns, t_epi_ns;
  double t_epi_tile_ns;  // the epilogue's time for one tile: it bounds the tile rate when K is short
  bool feasible;
};

constexpr int kGemmStagingBytes = 8 * 32 * 128;  // 8 epilogue warps x 32 rows x 128 B
// Epilogue of one tile by the eight epilogue warps: a fixed part plus 64-column chunks
// (TMEM -> registers -> bf16 -> staging -> TMA store), and the factor of a CTA pair's
// cross-SM accumulator release (fitted to K = 256 tiles in steady state, 54 tiles per SM:
// 128 x 256 take 2.89 us single and 2.9-3.2 us per SM as a pair across boxes, 128 x 128
// 1.66 us).
constexpr double kGemmEpiTileNs = 430.0;
constexpr double kGemmEpiChunkNs = 615.0;
constexpr double kGemmPairEpiFactor = 1.1;

constexpr GemmPlan gemm_eval(const ArchDesc& a, int bn, int stages) {
  GemmPlan p{};
  p.bm = 128;
  p.bn = bn;
  p.bk = 64;
  p.stages = stages;
  const double stage_bytes = (p.bm + bn) * p.bk * 2.0;
  p.t_load_ns = stage_bytes / a.l2_smem_gbs_sm;  // A and B tiles from L2
  p.t_mma_ns = (p.bk / 16.0) * dmax(a.mma_clk_per_n * bn, a.mma_min_clk) / a.sm_ghz;
  p.t_iter_ns = heg_pipe(p.t_load_ns, p.t_mma_ns, 0.0, 1, 0);
  p.t_epi_ns = p.bm * bn * 2.0 / a.l2_smem_gbs_sm;  // the C tile leaves through L2
  p.t_epi_tile_ns = kGemmEpiTileNs + (bn / 64) * kGemmEpiChunkNs;
  p.smem_bytes = static_cast<int>(stages * stage_bytes) + kGemmStagingBytes + 1024 + 256;
  p.tmem_cols = 2 * bn;
  p.feasible = p.smem_bytes <= a.smem_per_cta && p.tmem_cols <= a.tmem_cols && stages >= 2 && bn % 64 == 0 &&
               bn >= 64 && bn <= 256 && (stages - 1) * p.t_iter_ns >= a.mem_latency_ns * 0.5;
  return p;
}

// Eq. 8 for one tile width: the ring depth with the lowest modeled iteration, ties to the
// deeper ring.
constexpr GemmPlan gemm_plan_variant(int bn, const ArchDesc& a = kGb300) {
  GemmPlan best{};
  best.feasible = false;
  for (int stages = 2; stages <= 12; ++stages) {
    const GemmPlan p = gemm_eval(a, bn, stages);
    if (!p.feasible) continue;
    if (!best.feasible || p.t_iter_ns < best.t_iter_ns * (1.0 - 1e-9) ||
        (p.t_iter_ns <= best.t_iter_ns * (1.0 + 1e-9) && p.stages > best.stages))
      best = p;
  }
  return best;
}

// Eq. 5-7 for a whole launch: the busiest SM runs ceil(tiles / SMs) tiles of ceil(K / BK)
// iterations back to back; the first load and the last epilogue are exposed.
constexpr double gemm_time_us(const GemmPlan& p, long long M, long long N, long long K, int num_sms,
                              const ArchDesc& a = kGb300) {
  const long long tiles = cdiv(M, p.bm) * cdiv(N, p.bn);
  const long long per_sm = cdiv(tiles, num_sms);
  // the next tile's K loop overlaps this tile's epilogue (two accumulators): a tile takes
  // the longer of the two
  const double t_tile = dmax(heg_for(cdiv(K, p.bk), p.t_iter_ns), p.t_epi_tile_ns);
  const double t = heg_seq(heg_seq(p.t_load_ns, heg_for(per_sm, t_tile)), p.t_epi_ns);
  return (t + a.launch_ns * 0.2) * 1e-3;
}

// Eq. 9: the tile width with the lowest modeled launch time (ties to the wider tile).
constexpr int gemm_choose_bn(long long M, long long N, long long K, int num_sms, const ArchDesc& a = kGb300) {
  int best_bn = 0;
  double best_t = 1e300;
  for (int bn = 256; bn >= 64; bn -= 64) {
    const GemmPlan p = gemm_plan_variant(bn, a);
    if (!p.feasible) continue;
    const double t = gemm_time_us(p, M, N, K, num_sms, a);
    if (t < best_t * (1.0 - 1e-9)) {
      best_t = t;
      best_bn = bn;
    }
  }
  return best_bn;
}

// ------------------------------------------------------------------ split-K clusters
// When there are few C tiles for the SMs (small M x N, long K), a cluster of S CTAs shares
// one tile, each CTA taking a contiguous 1/S of the K stages into its own TMEM
// accumulator.  The S fp32 partial tiles are then summed through distributed shared
// memory: every CTA parks its partial in its own shared memory and, after a cluster
// barrier, reduces BM / S rows of the tile over all S CTAs and stores them.  So each CTA
// reads one tile's worth of fp32 over DSMEM, and the reduction adds two cluster barriers.
struct GemmClusterArch {
  double dsmem_gbs_sm;    // distributed-shared-memory read rate of one SM, GB/s (assumed)
  double cluster_sync_ns; // one cluster-wide barrier.cluster round trip (assumed)
};
inline constexpr GemmClusterArch kGb300Cluster = {120.0, 300.0};

constexpr int kGemmMaxSplits = 16;

// Time of one launch with split S (S >= 2) when `cta_slots` CTAs of clusters of S fit on the
// GPU at once: every CTA of the busiest wave loads and multiplies ceil(k_iters / S) stages,
// then reduces and stores its BM / S rows.
constexpr double gemm_splitk_time_us(const GemmPlan& p, long long M, long long N, long long K, int S, int cta_slots,
                                     const ArchDesc& a = kGb300, const GemmClusterArch& c = kGb300Cluster) {
  const long long tiles = cdiv(M, p.bm) * cdiv(N, p.bn);
  const long long units = tiles * S;
  const long long waves = cdiv(units, cta_slots < S ? S : cta_slots);
  const long long iters = cdiv(cdiv(K, p.bk), S);
  const double t_red = p.bm * p.bn * 4.0 / c.dsmem_gbs_sm + 2.0 * c.cluster_sync_ns;
  const double t_unit = heg_seq(heg_seq(p.t_load_ns, heg_for(iters, p.t_iter_ns)), t_red + p.t_epi_ns / S);
  return (static_cast<double>(waves) * t_unit + a.launch_ns * 0.2) * 1e-3;
}

// Split counts the kernel supports, and the plan of the split-K kernel for one tile width
// (the same ring as the persistent kernel: the partial tile reuses the ring's memory).
constexpr bool gemm_split_supported(int S) { return S == 1 || S == 2 || S == 4 || S == 8 || S == 16; }

// Eq. 9 over (tile width, split count).  `slots(bn, S)` is the number of CTAs of clusters
// of S that fit on the GPU at once with tile width bn; zero rules the split out.  A
// non-zero `only_bn` / `only_splits` restricts the search to that value (and a forced
// split may leave a CTA fewer than two stages).  Ties go to the wider tile and then to
// fewer splits; bn = 0 when nothing is feasible.
struct GemmChoiceModel {
  int bn, splits;
  double t_us;
  bool pair;  // CTA-pair 256 x 256 tiles (bn = 256, splits = 1)
};

// ------------------------------------------------------------------ CTA pairs
// Two CTAs of a cluster compute a 256 x 256 tile with one M = 256 MMA stream: each SM
// loads its 128 rows of A and half of B, (128 + 128) x 64 x 2 = 32 KB per K stage, against
// the same four 128 x 256 x 16 MMAs per SM as a 128 x 256 single-CTA tile (48 KB).
constexpr GemmPlan gemm_pair_plan(const ArchDesc& a = kGb300) {
  GemmPlan p{};
  p.bm = 256;
  p.bn = 256;
  p.bk = 64;
  p.stages = 6;
  const double stage_bytes = (128 + 128) * p.bk * 2.0;
  p.t_load_ns = stage_bytes / a.l2_smem_gbs_sm;
  p.t_mma_ns = (p.bk / 16.0) * dmax(a.mma_clk_per_n * 256, a.mma_min_clk) / a.sm_ghz;
  p.t_iter_ns = heg_pipe(p.t_load_ns, p.t_mma_ns, 0.0, 1, 0);
  p.t_epi_ns = 128 * 256 * 2.0 / a.l2_smem_gbs_sm;
  p.t_epi_tile_ns = (kGemmEpiTileNs + (256 / 64) * kGemmEpiChunkNs) * kGemmPairEpiFactor;
  p.smem_bytes = static_cast<int>(p.stages * stage_bytes) + kGemmStagingBytes + 1024 + 256;
  p.tmem_cols = 512;
  p.feasible = p.smem_bytes <= a.smem_per_cta && p.tmem_cols <= a.tmem_cols;
  return p;
}

// `pair_ctas` CTAs (whole pairs) fit on the GPU at once.  A last round that would keep at
// most a quarter of the pairs busy runs its tiles as two 256 x 128 halves each (N = 128
// pair MMAs, each SM loading 64 columns of B: 24 KB per stage), about half a round.
constexpr double gemm_pair_time_us(long long M, long long N, long long K, int pair_ctas, const ArchDesc& a = kGb300) {
  const GemmPlan p = gemm_pair_plan(a);
  const long long tiles = cdiv(M, 256) * cdiv(N, 256);
  const long long pairs = pair_ctas / 2 > 0 ? pair_ctas / 2 : 1;
  const long long full = tiles / pairs, rest = tiles % pairs;
  const long long k_iters = cdiv(K, p.bk);
  const double t_tile = dmax(heg_for(k_iters, p.t_iter_ns), p.t_epi_tile_ns);
  const double t_load_n = (128 + 64) * p.bk * 2.0 / a.l2_smem_gbs_sm;
  const double t_mma_n = (p.bk / 16.0) * dmax(a.mma_clk_per_n * 128, a.mma_min_clk) / a.sm_ghz;
  const double t_tile_n = dmax(heg_for(k_iters, heg_pipe(t_load_n, t_mma_n, 0.0, 1, 0)),
                               (kGemmEpiTileNs + 2 * kGemmEpiChunkNs) * kGemmPairEpiFactor);
  const double last = rest == 0 ? 0.0 : (4 * rest <= pairs ? t_tile_n : t_tile);
  const double t = heg_seq(heg_seq(p.t_load_ns, heg_seq(heg_for(full, t_tile), last)), p.t_epi_ns);
  return (t + a.launch_ns * 0.2) * 1e-3;
}

// Eq. 9 over the kernel variants.  only_pair: 0 = the model decides, 1 = the pair kernel
// only, -1 = never the pair kernel.
template <typename SlotsFn>
constexpr GemmChoiceModel gemm_choose(long long M, long long N, long long K, int num_sms, SlotsFn slots,
                                      const ArchDesc& a = kGb300, int only_bn = 0, int only_splits = 0,
                                      int pair_ctas = 0, int only_pair = 0) {
  GemmChoiceModel best{0, 0, 1e300, false};
  if (only_pair >= 0 && pair_ctas >= 2 && (only_bn == 0 || only_bn == 256) && only_splits <= 1 &&
      gemm_pair_plan(a).feasible) {
    best = {256, 1, gemm_pair_time_us(M, N, K, pair_ctas, a), true};
    if (only_pair == 1) return best;
  }
  if (only_pair == 1) return GemmChoiceModel{0, 0, 1e300, false};
  for (int bn = 256; bn >= 64; bn -= 64) {
    if (only_bn != 0 && bn != only_bn) continue;
    const GemmPlan p = gemm_plan_variant(bn, a);
    if (!p.feasible) continue;
    for (int S = 1; S <= kGemmMaxSplits; S *= 2) {
      if (only_splits != 0 && S != only_splits) continue;
      double t;
      if (S == 1) {
        t = gemm_time_us(p, M, N, K, num_sms, a);
      } else {
        if (only_splits == 0 && cdiv(K, p.bk) < 2LL * S) break;  // every CTA takes two stages or more
        const int s = slots(bn, S);
        if (s <= 0) continue;
        t = gemm_splitk_time_us(p, M, N, K, S, s, a);
      }
      if (t < best.t_us * (1.0 - 1e-9)) best = {bn, S, t, false};
    }
  }
  return best;
}

// Cluster slots when nothing better is known: whole clusters of S on `num_sms` SMs with the
// GPU's SMs in 8 groups (GPCs) of equal size; a cluster never spans two groups.
constexpr int gemm_default_slots(int num_sms, int S) {
  const int per_gpc = num_sms / 8;
  return (per_gpc / S) * S * 8;
}

}  // namespace model
}  // namespace loom
