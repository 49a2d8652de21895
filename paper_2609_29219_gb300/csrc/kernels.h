// Internal launch interface between the C ABI (loom_api.cu) and the kernel files.
#pragma once

#include <atomic>
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "ptx.cuh"

namespace loom {

// One-time set-up per device (a kernel's shared-memory opt-in, a cluster-size opt-in),
// safe when several host threads launch at once: the first call on a device runs `fn`,
// later calls skip it once it has succeeded.  Devices beyond the 64 tracked bits run `fn`
// on every call (the set-up calls it guards are idempotent).
class PerDeviceOnce {
 public:
  template <class F>
  bool run(int dev, F&& fn) {
    if (dev < 0 || dev >= 64) return fn();
    const unsigned long long bit = 1ull << dev;
    if (bits_.load(std::memory_order_acquire) & bit) return true;
    if (!fn()) return false;
    bits_.fetch_or(bit, std::memory_order_acq_rel);
    return true;
  }

 private:
  std::atomic<unsigned long long> bits_{0};
};

// Split rule of the decode path: chunk length of a sequence of `len` keys cut into
// `splits` pieces, ceil(len / splits) rounded up to a multiple of kDecodeChunkAlign.
constexpr int kDecodeChunkAlign = 64;
constexpr int kMaxDecodeSplits = 1024;

struct DecodeArgs {
  const void* q;            // [B, Hq, 1, D] bf16
  const void* k;            // [B, Hkv, Skv, D] bf16
  const void* v;            // [B, Hkv, Skv, D] bf16
  const int32_t* seqlens;   // [B] or null
  void* o;                  // [B, Hq, 1, D] bf16
  float* lse;               // [B, Hq] or null
  float* o_part;            // [B, Hq, splits, D] fp32 (workspace)
  float* lse_part;          // [B, Hq, splits] fp32 (workspace)
  int B, Hq, Hkv, Skv, D, splits;
  float scale;
  int form;     // 0: the model's form; else a kDecode* form (when it can run)
  int cluster;  // cluster form: 0 = the model's cluster size, else this size (if it divides splits and fits)
  int stage_plan;  // 0: the model's stage plan; i > 0: the i-th compiled ablation plan (split + merge form)
  int by_model;    // 1: the split count is the model's (num_splits = 0), which then also picks the form
  int tc;          // split + merge form's split kernel on a contiguous cache: 0 CUDA cores; tensor
                   // cores, 1 persistent CTAs taking items from the workspace counter, 2 one CTA per split
  unsigned long long* sched;  // the workspace's item counter (tag kDecodeSchedTag in the high word)
};

// High word of an armed item counter: a signalling-NaN pattern that no float the decode
// path writes to the workspace carries, so that a workspace never used before is told
// apart (its first call deals items statically; the merge kernel then arms the counter).
constexpr uint32_t kDecodeSchedTag = 0x7FBADC0Du;
// Query heads per kv head that the tensor-core split kernels take (the lanes of one warp).
constexpr int kDecodeTcMaxGroup = 32;

struct FwdArgs {
  const void* q;  // [B, Hq, Sq, D] bf16
  const void* k;  // [B, Hkv, Skv, D] bf16
  const void* v;  // [B, Hkv, Skv, D] bf16
  void* o;        // [B, Hq, Sq, D] bf16
  float* lse;     // [B, Hq, Sq] or null
  int B, Hq, Hkv, Sq, Skv, D, causal;
  float scale;
  int design;  // prefill design: 0 = the analytic model's choice, 1..3 forced
  int slots;   // two-tile design's K/V ring depth: 0 = the model's; a compiled neighbour otherwise
};

// K/V ring depths of the two-tile prefill compiled beside the model's, for the block-size
// ablation (D = 128: 2; D = 64: 3, 6, 9).
inline bool fwd_slots_compiled(int D, int slots) {
  return D == 128 ? slots == 2 : (slots == 3 || slots == 6 || slots == 9);
}

// Bytes of workspace the decode path needs for `splits` splits.
inline size_t decode_workspace_bytes(int B, int Hq, int D, int splits) {
  const size_t rows = static_cast<size_t>(B) * Hq * splits;
  const size_t opart = rows * D * sizeof(float);
  const size_t lpart = rows * sizeof(float);
  return ((opart + 255) / 256) * 256 + ((lpart + 255) / 256) * 256 + 256;  // + the item counter
}

// The item counter's place in a decode workspace (after the partial O and LSE).
inline unsigned long long* decode_sched_word(void* workspace, int B, int Hq, int D, int splits) {
  return reinterpret_cast<unsigned long long*>(static_cast<char*>(workspace) + decode_workspace_bytes(B, Hq, D, splits) -
                                               256);
}

// Argument checks of the contiguous decode entry points, in their order, up to (not
// including) the workspace; returns a loom_status value and, on success, the split count.
int decode_check_args(const void* q, const void* k_cache, const void* v_cache, const int32_t* seqlens_k,
                      const void* o, const float* lse, int B, int Hq, int Hkv, int Skv, int D, float scale,
                      int num_splits, int* splits);

cudaError_t launch_decode(const DecodeArgs& a, const KernelCtl& ctl, cudaStream_t stream);
// Flash Decode forms: a split kernel of one CTA per (split, unit) + the merge kernel; a
// persistent split kernel walking (unit, split) items + the merge kernel; one persistent
// kernel whose clusters merge over distributed shared memory.
constexpr int kDecodeSplitMerge = 1, kDecodePersistent = 2, kDecodeCluster = 3;
// The form a decode launch with these arguments runs (and, for the cluster form, its
// cluster size in *cs).
int decode_form_of(const DecodeArgs& a, bool paged, int* cs);
// CTAs of the persistent split kernel resident at once on the current device (0: unknown).
int decode_persistent_slots(int D, int G);
// Clusters of cs cluster-decode CTAs (G query heads per kv head) resident at once on the
// current device; 0 if none fit or the device cannot be asked.
int decode_max_clusters(int D, int G, int cs);
// Index (> 0) of a compiled ablation stage plan of the decode split kernel (contiguous
// cache, D = 128, 4 query heads per kv head), 0 if that plan is not compiled.
int decode_ablation_plan(int tokens, int stages, int ctas_per_sm);
cudaError_t launch_fwd(const FwdArgs& a, const KernelCtl& ctl, cudaStream_t stream);

}  // namespace loom
