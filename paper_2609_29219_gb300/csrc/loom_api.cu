// C ABI of the library (declared in include/loom_attn.h): argument validation, the
// device error word, the analytic model hook for the decode split count, and dispatch
// to the kernels.  No device memory is allocated here: the error word is a
// file-scope __device__ variable whose address is looked up once per device.
#include <cmath>
#include <cstdint>
#include <mutex>
#include <utility>
#include <vector>

#include "../../include/loom_attn.h"
#include "gemm.h"
#include "gemm_model.h"
#include "kernels.h"
#include "model.h"
#include "paged.h"
#include "varlen.h"

namespace loom {
namespace {

__device__ uint32_t g_error_word = 0;

constexpr uint64_t kDefaultTimeoutNs = 2000000000ull;  // 2 s
uint64_t g_timeout_ns = kDefaultTimeoutNs;
int g_inject = 0;
int g_prefill_design = 0;
int g_prefill_slots = 0;  // test hook: the two-tile prefill's K/V ring depth (0: the model's)
int g_gemm_tile_n = 0;  // test hook: forced GEMM tile width (0: the model's choice)
int g_gemm_splits = 0;  // test hook: forced GEMM split count (0: the model's choice)
int g_gemm_pair = 0;    // test hook: 1 forces CTA-pair tiles, -1 forbids them, 0: the model's choice
int g_gemm_stages = 0;  // test hook: GEMM ring depth (0: the model's; a compiled neighbour otherwise)
int g_gemm_group = 0;   // test hook: tile rows per group of the GEMM tile order (0: the default)
int g_gemm_k_alt = 0;   // test hook: -1 stops the CTA-pair GEMM walking K backwards every other round
int g_decode_form = 0;     // test hook: the Flash Decode form (0: the model's; kDecode* otherwise)
int g_decode_cluster = 0;  // test hook: the cluster decode form's cluster size (0: the model's)
int g_decode_stage_plan = 0;  // test hook: a compiled ablation stage plan of the decode split kernel
// test hook: the split + merge form's split kernel on a contiguous cache (DecodeArgs::tc)
int g_decode_tc = 1;

constexpr int kMaxDevices = 64;
uint32_t* g_err_ptr[kMaxDevices] = {};
std::mutex g_err_mutex;

// Device address of the error word on the current device (looked up once per device).
uint32_t* error_word_ptr() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_err_mutex);
  if (!g_err_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_error_word) != cudaSuccess) return nullptr;
    g_err_ptr[dev] = static_cast<uint32_t*>(p);
  }
  return g_err_ptr[dev];
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int current_sm_count() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return sms;
}

struct SplitKey {
  int B, Hq, Hkv, Skv, D, sms, tc;
  bool operator==(const SplitKey& o) const {
    return B == o.B && Hq == o.Hq && Hkv == o.Hkv && Skv == o.Skv && D == o.D && sms == o.sms && tc == o.tc;
  }
};
std::vector<std::pair<SplitKey, int>> g_split_cache;
std::mutex g_split_mutex;

bool make_ctl(KernelCtl* ctl) {
  ctl->err = error_word_ptr();
  ctl->timeout_ns = g_timeout_ns;
  ctl->inject = g_inject;
  return ctl->err != nullptr;
}

}  // namespace
}  // namespace loom

using namespace loom;

extern "C" {

const char* loom_status_string(loom_status s) {
  switch (s) {
    case LOOM_OK: return "LOOM_OK";
    case LOOM_ERR_INVALID_ARG: return "LOOM_ERR_INVALID_ARG";
    case LOOM_ERR_UNSUPPORTED: return "LOOM_ERR_UNSUPPORTED";
    case LOOM_ERR_MISALIGNED: return "LOOM_ERR_MISALIGNED";
    case LOOM_ERR_WORKSPACE: return "LOOM_ERR_WORKSPACE";
    case LOOM_ERR_CUDA: return "LOOM_ERR_CUDA";
    case LOOM_ERR_TIMEOUT: return "LOOM_ERR_TIMEOUT";
  }
  return "LOOM_ERR_UNKNOWN";
}

loom_status loom_attn_fwd(const void* q, const void* k, const void* v, void* o, float* lse, int B,
                          int Hq, int Hkv, int Sq, int Skv, int D, int causal, float scale,
                          void* stream) {
  if (!q || !k || !v || !o) return LOOM_ERR_INVALID_ARG;
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || Sq <= 0 || Skv <= 0 || D <= 0) return LOOM_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return LOOM_ERR_INVALID_ARG;
  if (causal != 0 && causal != 1) return LOOM_ERR_INVALID_ARG;
  if (causal && Sq > Skv) return LOOM_ERR_INVALID_ARG;
  if (!std::isfinite(scale) || scale <= 0.f) return LOOM_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return LOOM_ERR_UNSUPPORTED;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o)) return LOOM_ERR_MISALIGNED;
  if (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)) return LOOM_ERR_MISALIGNED;
  // TMA views use 32-bit coordinates: rows and planes must fit
  if (static_cast<long long>(B) * Hq > 0x7fffffff || static_cast<long long>(B) * Hkv > 0x7fffffff)
    return LOOM_ERR_UNSUPPORTED;
  KernelCtl ctl;
  if (!make_ctl(&ctl)) return LOOM_ERR_CUDA;
  FwdArgs a{q, k, v, o, lse, B, Hq, Hkv, Sq, Skv, D, causal, scale, g_prefill_design, g_prefill_slots};
  return launch_fwd(a, ctl, static_cast<cudaStream_t>(stream)) == cudaSuccess ? LOOM_OK
                                                                               : LOOM_ERR_CUDA;
}

int loom_attn_decode_num_splits(int B, int Hq, int Hkv, int Skv, int D) {
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || Skv <= 0 || Hq % Hkv != 0) return 0;
  if (D != 64 && D != 128) return 0;
  int sms = current_sm_count();
  if (sms <= 0) sms = model::kGb300.num_sms;
  // The enumeration costs ~0.1 ms of host time: remember the answer per problem shape.
  // the split + merge form's split kernel runs on the tensor cores for a contiguous cache
  // (a paged cache takes the same split count, with the CUDA-core kernel)
  const int tc = (g_decode_tc != 0 && Hq / Hkv <= kDecodeTcMaxGroup) ? 1 : 0;
  const SplitKey key{B, Hq, Hkv, Skv, D, sms, tc};
  {
    std::lock_guard<std::mutex> lock(g_split_mutex);
    for (const auto& e : g_split_cache)
      if (e.first == key) return e.second;
  }
  // Both Flash Decode forms compete (Eq. 9); the cluster form's CTA slots come from the
  // device, or from the GB300 estimate when no device answers.
  const bool device = current_sm_count() > 0;
  const int G = Hq / Hkv;
  // (the CUDA-core persistent split kernel is a candidate only where the tensor-core one
  // does not run)
  const int slots = tc ? 0 : device ? decode_persistent_slots(D, G) : sms * model::decode_stage(D).ctas_per_sm;
  const int splits = model::choose_decode_plan(
                         B, Hq, Hkv, Skv, D, sms,
                         [&](int cs) {
                           return device ? decode_max_clusters(D, G, cs) : model::decode_default_clusters(sms, cs, D);
                         },
                         slots, model::kGb300, tc != 0)
                         .splits;
  std::lock_guard<std::mutex> lock(g_split_mutex);
  if (g_split_cache.size() >= 256) g_split_cache.erase(g_split_cache.begin());
  g_split_cache.emplace_back(key, splits);
  return splits;
}

size_t loom_attn_decode_workspace_bytes(int B, int Hq, int Hkv, int Skv, int D, int num_splits) {
  if (num_splits == 0) num_splits = loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D);
  if (num_splits <= 0 || num_splits > kMaxDecodeSplits) return 0;
  if (B <= 0 || Hq <= 0 || (D != 64 && D != 128)) return 0;
  return decode_workspace_bytes(B, Hq, D, num_splits);
}

}  // extern "C"

namespace loom {
// Every check of the contiguous decode entry points that comes before the workspace: on
// LOOM_OK, *splits is the split count the call will use (the model's when num_splits = 0).
int decode_check_args(const void* q, const void* k_cache, const void* v_cache, const int32_t* seqlens_k,
                      const void* o, const float* lse, int B, int Hq, int Hkv, int Skv, int D, float scale,
                      int num_splits, int* splits) {
  if (!q || !k_cache || !v_cache || !o) return LOOM_ERR_INVALID_ARG;
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || Skv <= 0 || D <= 0) return LOOM_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return LOOM_ERR_INVALID_ARG;
  if (!std::isfinite(scale) || scale <= 0.f) return LOOM_ERR_INVALID_ARG;
  if (num_splits < 0) return LOOM_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return LOOM_ERR_UNSUPPORTED;
  if (num_splits > kMaxDecodeSplits) return LOOM_ERR_UNSUPPORTED;
  if (static_cast<long long>(B) * Hq * (num_splits ? num_splits : 1) > 0x7fffffffLL ||
      static_cast<long long>(B) > 65535)
    return LOOM_ERR_UNSUPPORTED;
  if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(o))
    return LOOM_ERR_MISALIGNED;
  if ((lse && (reinterpret_cast<uintptr_t>(lse) & 3u)) ||
      (seqlens_k && (reinterpret_cast<uintptr_t>(seqlens_k) & 3u)))
    return LOOM_ERR_MISALIGNED;
  if (num_splits == 0) num_splits = loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D);
  if (num_splits <= 0) return LOOM_ERR_INVALID_ARG;
  *splits = num_splits;
  return LOOM_OK;
}
}  // namespace loom

extern "C" {

loom_status loom_attn_decode(const void* q, const void* k_cache, const void* v_cache,
                             const int32_t* seqlens_k, void* o, float* lse, void* workspace,
                             size_t workspace_bytes, int B, int Hq, int Hkv, int Skv, int D,
                             float scale, int num_splits, void* stream) {
  const int by_model = num_splits == 0 ? 1 : 0;
  const int st = decode_check_args(q, k_cache, v_cache, seqlens_k, o, lse, B, Hq, Hkv, Skv, D, scale, num_splits,
                                   &num_splits);
  if (st != LOOM_OK) return static_cast<loom_status>(st);
  const size_t need = decode_workspace_bytes(B, Hq, D, num_splits);
  if (!workspace || workspace_bytes < need) return LOOM_ERR_WORKSPACE;
  if (!aligned16(workspace)) return LOOM_ERR_MISALIGNED;
  KernelCtl ctl;
  if (!make_ctl(&ctl)) return LOOM_ERR_CUDA;
  const size_t rows = static_cast<size_t>(B) * Hq * num_splits;
  float* o_part = static_cast<float*>(workspace);
  float* lse_part = reinterpret_cast<float*>(static_cast<char*>(workspace) +
                                             (rows * D * sizeof(float) + 255) / 256 * 256);
  DecodeArgs a{q, k_cache, v_cache, seqlens_k, o, lse, o_part, lse_part, B, Hq, Hkv, Skv, D,
               num_splits, scale, g_decode_form, g_decode_cluster, g_decode_stage_plan, by_model, g_decode_tc,
               decode_sched_word(workspace, B, Hq, D, num_splits)};
  return launch_decode(a, ctl, static_cast<cudaStream_t>(stream)) == cudaSuccess ? LOOM_OK
                                                                                 : LOOM_ERR_CUDA;
}

loom_status loom_attn_fwd_varlen(const void* q, const void* k, const void* v, void* o, float* lse,
                                 const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k, int B,
                                 int Hq, int Hkv, int total_q, int total_k, int max_seqlen_q, int D,
                                 int causal, float scale, void* stream) {
  if (!q || !k || !v || !o || !cu_seqlens_q || !cu_seqlens_k) return LOOM_ERR_INVALID_ARG;
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || D <= 0 || total_q < 0 || total_k < 0 || max_seqlen_q < 0)
    return LOOM_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return LOOM_ERR_INVALID_ARG;
  if (!std::isfinite(scale) || scale <= 0.f) return LOOM_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return LOOM_ERR_UNSUPPORTED;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o)) return LOOM_ERR_MISALIGNED;
  if ((reinterpret_cast<uintptr_t>(cu_seqlens_q) & 3u) || (reinterpret_cast<uintptr_t>(cu_seqlens_k) & 3u) ||
      (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)))
    return LOOM_ERR_MISALIGNED;
  if (total_q == 0) return LOOM_OK;
  if (total_k == 0) return LOOM_ERR_UNSUPPORTED;
  // work items (query-tile pairs x heads) are at most (total_q / 256 + B) * Hq
  if ((static_cast<long long>(total_q) / 256 + B) * Hq > 0x7fffffffLL) return LOOM_ERR_UNSUPPORTED;
  KernelCtl ctl;
  if (!make_ctl(&ctl)) return LOOM_ERR_CUDA;
  FwdVarlenArgs a{q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, B, Hq, Hkv, total_q, total_k, max_seqlen_q, D,
                  causal ? 1 : 0, scale};
  return launch_fwd_varlen(a, ctl, static_cast<cudaStream_t>(stream)) == cudaSuccess ? LOOM_OK : LOOM_ERR_CUDA;
}

loom_status loom_attn_decode_paged(const void* q, const void* k_cache, const void* v_cache,
                                   const int32_t* block_table, const int32_t* seqlens_k, void* o,
                                   float* lse, void* workspace, size_t workspace_bytes, int B, int Hq,
                                   int Hkv, int num_pages, int page_size, int max_pages, int kv_layout,
                                   int D, float scale, int num_splits, void* stream) {
  if (!q || !k_cache || !v_cache || !o || !block_table || !seqlens_k) return LOOM_ERR_INVALID_ARG;
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || num_pages <= 0 || page_size <= 0 || max_pages <= 0 || D <= 0)
    return LOOM_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return LOOM_ERR_INVALID_ARG;
  if (!std::isfinite(scale) || scale <= 0.f) return LOOM_ERR_INVALID_ARG;
  if (num_splits < 0) return LOOM_ERR_INVALID_ARG;
  if (kv_layout != kPagedNHD && kv_layout != kPagedHND) return LOOM_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return LOOM_ERR_UNSUPPORTED;
  if (!paged_page_size_ok(page_size)) return LOOM_ERR_UNSUPPORTED;
  if (static_cast<long long>(num_pages) * page_size > 0x7fffffffLL ||
      static_cast<long long>(num_pages) * Hkv > 0x7fffffffLL ||
      static_cast<long long>(max_pages) * page_size > 0x7fffffffLL ||
      static_cast<long long>(B) * max_pages > 0x7fffffffLL)
    return LOOM_ERR_UNSUPPORTED;
  if (num_splits > kMaxDecodeSplits) return LOOM_ERR_UNSUPPORTED;
  if (static_cast<long long>(B) * Hq * (num_splits ? num_splits : 1) > 0x7fffffffLL ||
      static_cast<long long>(B) > 65535)
    return LOOM_ERR_UNSUPPORTED;
  if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(o)) return LOOM_ERR_MISALIGNED;
  if ((reinterpret_cast<uintptr_t>(block_table) & 3u) || (reinterpret_cast<uintptr_t>(seqlens_k) & 3u) ||
      (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)))
    return LOOM_ERR_MISALIGNED;
  const int Skv = max_pages * page_size;
  const int by_model = num_splits == 0 ? 1 : 0;
  if (num_splits == 0) num_splits = loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D);
  if (num_splits <= 0) return LOOM_ERR_INVALID_ARG;
  const size_t need = decode_workspace_bytes(B, Hq, D, num_splits);
  if (!workspace || workspace_bytes < need) return LOOM_ERR_WORKSPACE;
  if (!aligned16(workspace)) return LOOM_ERR_MISALIGNED;
  KernelCtl ctl;
  if (!make_ctl(&ctl)) return LOOM_ERR_CUDA;
  const size_t rows = static_cast<size_t>(B) * Hq * num_splits;
  float* o_part = static_cast<float*>(workspace);
  float* lse_part = reinterpret_cast<float*>(static_cast<char*>(workspace) +
                                             (rows * D * sizeof(float) + 255) / 256 * 256);
  DecodeArgs a{q, k_cache, v_cache, seqlens_k, o, lse, o_part, lse_part, B, Hq, Hkv, Skv, D, num_splits, scale,
               g_decode_form, g_decode_cluster, 0, by_model, g_decode_tc,
               decode_sched_word(workspace, B, Hq, D, num_splits)};
  PagedKV pk{block_table, num_pages, page_size, max_pages, kv_layout};
  return launch_decode_paged(a, pk, ctl, static_cast<cudaStream_t>(stream)) == cudaSuccess ? LOOM_OK
                                                                                          : LOOM_ERR_CUDA;
}

namespace {
loom_status gemm_call(const void* a, const void* b, void* c, int M, int N, int K, int b_kmajor, void* stream) {
  if (!a || !b || !c) return LOOM_ERR_INVALID_ARG;
  if (M <= 0 || N <= 0 || K <= 0) return LOOM_ERR_INVALID_ARG;
  if (!aligned16(a) || !aligned16(b) || !aligned16(c)) return LOOM_ERR_MISALIGNED;
  if (K % 8 != 0 || N % 8 != 0) return LOOM_ERR_UNSUPPORTED;  // 16-byte row strides for TMA
  KernelCtl ctl;
  if (!make_ctl(&ctl)) return LOOM_ERR_CUDA;
  GemmArgs g{a, b, c, M, N, K, g_gemm_tile_n, g_gemm_splits, g_gemm_pair, b_kmajor, g_gemm_stages, g_gemm_group, g_gemm_k_alt};
  return launch_gemm(g, ctl, static_cast<cudaStream_t>(stream)) == cudaSuccess ? LOOM_OK : LOOM_ERR_CUDA;
}
}  // namespace

loom_status loom_gemm_bf16(const void* a, const void* b, void* c, int M, int N, int K, void* stream) {
  return gemm_call(a, b, c, M, N, K, 0, stream);
}

loom_status loom_gemm_bf16_bt(const void* a, const void* b, void* c, int M, int N, int K, void* stream) {
  return gemm_call(a, b, c, M, N, K, 1, stream);
}

namespace {
// The model's GEMM choice: with the device's cluster occupancy when a device answers, else
// with the estimate of whole clusters in 8 equal SM groups of a GB300.
GemmChoice gemm_choice_any(int M, int N, int K, GemmChoice forced) {
  const GemmChoice c = gemm_choice(M, N, K, forced);
  if (c.tile_n != 0) return c;
  cudaGetLastError();
  const int sms = model::kGb300.num_sms;
  const model::GemmChoiceModel m = model::gemm_choose(
      M, N, K, sms, [sms](int, int S) { return model::gemm_default_slots(sms, S); }, model::kGb300,
      forced.tile_n, forced.splits, forced.pair >= 0 ? model::gemm_default_slots(sms, 2) : 0, forced.pair);
  return {m.bn, m.splits, m.pair ? 1 : 0};
}
}  // namespace

int loom_gemm_tile_n(int M, int N, int K) {
  if (M <= 0 || N <= 0 || K <= 0) return 0;
  return gemm_choice_any(M, N, K, {g_gemm_tile_n, g_gemm_splits, g_gemm_pair}).tile_n;
}

int loom_gemm_splits(int M, int N, int K) {
  if (M <= 0 || N <= 0 || K <= 0) return 0;
  return gemm_choice_any(M, N, K, {g_gemm_tile_n, g_gemm_splits, g_gemm_pair}).splits;
}

int loom_gemm_cta_pair(int M, int N, int K) {
  if (M <= 0 || N <= 0 || K <= 0) return 0;
  return gemm_choice_any(M, N, K, {g_gemm_tile_n, g_gemm_splits, g_gemm_pair}).pair;
}

double loom_model_gemm_time_us(int M, int N, int K, int tile_n, int splits, int num_sms) {
  if (M <= 0 || N <= 0 || K <= 0 || num_sms <= 0) return -1.0;
  if (tile_n == 512 && splits == 1)  // CTA-pair 256 x 256 tiles
    return model::gemm_pair_time_us(M, N, K, model::gemm_default_slots(num_sms, 2));
  if (tile_n != 64 && tile_n != 128 && tile_n != 192 && tile_n != 256) return -1.0;
  if (!model::gemm_split_supported(splits)) return -1.0;
  const model::GemmPlan p = model::gemm_plan_variant(tile_n);
  if (!p.feasible) return -1.0;
  if (splits == 1) return model::gemm_time_us(p, M, N, K, num_sms);
  return model::gemm_splitk_time_us(p, M, N, K, splits, model::gemm_default_slots(num_sms, splits));
}

void loom_debug_gemm_tile_n(int tile_n) {
  g_gemm_tile_n = (tile_n == 64 || tile_n == 128 || tile_n == 192 || tile_n == 256) ? tile_n : 0;
}

void loom_debug_gemm_splits(int splits) { g_gemm_splits = model::gemm_split_supported(splits) ? splits : 0; }

void loom_debug_gemm_cta_pair(int mode) { g_gemm_pair = (mode == 1 || mode == -1) ? mode : 0; }

void loom_debug_gemm_stages(int stages) { g_gemm_stages = stages > 0 ? stages : 0; }

void loom_debug_decode_tensor_cores(int mode) { g_decode_tc = (mode >= 0 && mode <= 2) ? mode : 1; }

void loom_debug_gemm_order(int group_rows, int k_alternate) {
  g_gemm_group = (group_rows >= 1 && group_rows <= 1024) ? group_rows : 0;
  g_gemm_k_alt = k_alternate < 0 ? -1 : 0;
}

loom_status loom_attn_check_error(void* stream) {
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return LOOM_ERR_CUDA;
  uint32_t* p = error_word_ptr();
  if (!p) return LOOM_ERR_CUDA;
  uint32_t word = 0;
  if (cudaMemcpy(&word, p, sizeof word, cudaMemcpyDeviceToHost) != cudaSuccess) return LOOM_ERR_CUDA;
  if (word) {
    const uint32_t zero = 0;
    if (cudaMemcpy(p, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess) return LOOM_ERR_CUDA;
  }
  return (word & kErrTimeout) ? LOOM_ERR_TIMEOUT : LOOM_OK;
}

namespace {
void fill_plan(const model::FwdPlan& p, loom_fwd_plan* out) {
  out->design = p.design;
  out->s_buffers = p.s_buffers;
  out->bm = p.bm;
  out->bn = p.bn;
  out->q_tiles = p.q_tiles;
  out->kv_slots = p.kv_slots;
  out->b_lm = p.b_lm;
  out->b_ms = p.b_ms;
  out->smem_bytes = p.smem_bytes;
  out->tmem_cols = p.tmem_cols;
  out->t_load_ns = p.t_load_ns;
  out->t_mma_ns = p.t_mma_ns;
  out->t_softmax_ns = p.t_softmax_ns;
  out->t_iter_ns = p.t_iter_ns;
}
}  // namespace

loom_status loom_model_fwd_plan(int D, loom_fwd_plan* out) {
  if (!out) return LOOM_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return LOOM_ERR_UNSUPPORTED;
  fill_plan(model::fwd_plan(D), out);
  return LOOM_OK;
}

loom_status loom_model_fwd_plan_variant(int D, int design, loom_fwd_plan* out) {
  if (!out) return LOOM_ERR_INVALID_ARG;
  if ((D != 64 && D != 128) || design < 1 || design > 4) return LOOM_ERR_UNSUPPORTED;
  const model::FwdPlan p = model::fwd_plan_variant(D, design);
  if (!p.feasible) return LOOM_ERR_UNSUPPORTED;
  fill_plan(p, out);
  return LOOM_OK;
}

double loom_model_heg_pipe(double l, double m, double s, int b_lm, int b_ms) {
  return model::heg_pipe(l, m, s, b_lm != 0, b_ms != 0);
}

double loom_model_fwd_time_us(int B, int Hq, int Sq, int Skv, int D, int causal) {
  if (B <= 0 || Hq <= 0 || Sq <= 0 || Skv <= 0 || (D != 64 && D != 128)) return -1.0;
  return model::fwd_time_us(model::fwd_plan(D), B, Hq, Sq, Skv, D, causal != 0);
}

double loom_model_fwd_time_us_design(int design, int B, int Hq, int Sq, int Skv, int D, int causal) {
  if (B <= 0 || Hq <= 0 || Sq <= 0 || Skv <= 0 || (D != 64 && D != 128) || design < 1 || design > 4) return -1.0;
  const model::FwdPlan p = model::fwd_plan_variant(D, design);
  if (!p.feasible) return -1.0;
  return model::fwd_time_us(p, B, Hq, Sq, Skv, D, causal != 0);
}

double loom_model_decode_time_us(int splits, int B, int Hq, int Hkv, int Skv, int D, int num_sms) {
  if (splits <= 0 || B <= 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv || Skv <= 0 || num_sms <= 0 ||
      (D != 64 && D != 128))
    return -1.0;
  return model::decode_time_us(splits, B, Hq, Hkv, Skv, D, num_sms);
}

double loom_model_decode_tc_time_us(int splits, int B, int Hq, int Hkv, int Skv, int D, int num_sms) {
  if (splits <= 0 || B <= 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv || Skv <= 0 || num_sms <= 0 ||
      (D != 64 && D != 128) || Hq / Hkv > kDecodeTcMaxGroup)
    return -1.0;
  return model::decode_tc_time_us(splits, B, Hq, Hkv, Skv, D, num_sms);
}

int loom_attn_decode_form(int B, int Hq, int Hkv, int Skv, int D, int num_splits, int paged, int* cluster) {
  if (cluster) *cluster = 0;
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || Skv <= 0 || Hq % Hkv != 0 || (D != 64 && D != 128) || num_splits < 0 ||
      num_splits > kMaxDecodeSplits)
    return -1;
  const int by_model = num_splits == 0 ? 1 : 0;
  if (num_splits == 0) num_splits = loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D);
  if (num_splits <= 0) return -1;
  DecodeArgs a{};
  a.by_model = by_model;
  a.B = B;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.Skv = Skv;
  a.D = D;
  a.splits = num_splits;
  a.form = g_decode_form;
  a.cluster = g_decode_cluster;
  a.tc = g_decode_tc;
  int cs = 0;
  const int form = decode_form_of(a, paged != 0, &cs);
  cudaGetLastError();
  if (cluster) *cluster = cs;
  return form;
}

double loom_model_decode_cluster_time_us(int splits, int cluster, int B, int Hq, int Hkv, int Skv, int D,
                                         int clusters) {
  if (splits <= 0 || B <= 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv || Skv <= 0 || clusters <= 0 ||
      (D != 64 && D != 128))
    return -1.0;
  const double t = model::decode_cluster_time_us(splits, cluster, B, Hq, Hkv, Skv, D, clusters);
  return t > 1e299 ? -1.0 : t;
}

double loom_model_decode_persistent_time_us(int splits, int B, int Hq, int Hkv, int Skv, int D, int ctas) {
  if (splits <= 0 || B <= 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv || Skv <= 0 || ctas <= 0 || (D != 64 && D != 128))
    return -1.0;
  return model::decode_persistent_time_us(splits, B, Hq, Hkv, Skv, D, ctas);
}

int loom_decode_max_clusters(int D, int G, int cluster) {
  if ((D != 64 && D != 128) || G <= 0 || cluster <= 0 || cluster > model::kMaxClusterSize) return 0;
  const int sms = current_sm_count();
  if (sms <= 0) return model::decode_default_clusters(model::kGb300.num_sms, cluster, D);
  const int n = decode_max_clusters(D, G, cluster);
  cudaGetLastError();
  return n;
}

int loom_decode_persistent_slots(int D, int G) {
  if ((D != 64 && D != 128) || G <= 0) return 0;
  const int sms = current_sm_count();
  if (sms <= 0) return model::kGb300.num_sms * model::decode_stage(D).ctas_per_sm;
  const int n = decode_persistent_slots(D, G);
  cudaGetLastError();
  return n;
}

void loom_debug_decode_form(int form, int cluster) {
  g_decode_form = (form == kDecodeSplitMerge || form == kDecodePersistent || form == kDecodeCluster) ? form : 0;
  g_decode_cluster = (cluster >= 1 && cluster <= model::kMaxClusterSize) ? cluster : 0;
}

int loom_debug_decode_stage_plan(int tokens, int stages, int ctas_per_sm) {
  const model::DecodeStagePlan& m = model::decode_stage(128);
  if (tokens == 0 || (tokens == m.tokens && stages == m.stages && ctas_per_sm == m.ctas_per_sm)) {
    g_decode_stage_plan = 0;
    return 1;
  }
  g_decode_stage_plan = decode_ablation_plan(tokens, stages, ctas_per_sm);
  return g_decode_stage_plan > 0 ? 1 : 0;
}

void loom_debug_set_timeout_ns(uint64_t ns) { g_timeout_ns = ns ? ns : kDefaultTimeoutNs; }

void loom_debug_inject(int mode) { g_inject = mode; }

void loom_debug_prefill_design(int design) {
  g_prefill_design = (design >= 1 && design <= 4) ? design : 0;
}

int loom_debug_prefill_slots(int D, int slots) {
  if (slots == 0 || (D == 128 && slots == model::fwd_plan_variant(128, 2).kv_slots) ||
      (D == 64 && slots == model::fwd_plan_variant(64, 2).kv_slots) || fwd_slots_compiled(D, slots)) {
    g_prefill_slots = slots;
    return 1;
  }
  g_prefill_slots = 0;
  return 0;
}

}  // extern "C"
