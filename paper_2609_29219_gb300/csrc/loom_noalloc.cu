// Flash Decode entry point that allocates nothing and takes no workspace argument.
//
// Some callers have no way to obtain device scratch memory for a call: serving engines
// that reserve all device memory when they start and forbid allocation on the request
// path (cudaMalloc synchronises the whole device and can fail in the middle of a
// request), and plug-in hosts that hand a kernel library only the tensors of the call
// and no allocator.  For them, loom_attn_decode_noalloc runs the same split + merge
// kernels as loom_attn_decode, with the per-split partials kept in a fixed scratch array
// that lives in this file as a `static __device__` variable.  Every GPU that loads the
// library holds that array (kNoallocScratchBytes) until the process exits.
//
// In host code `g_decode_scratch` is only a host-side stand-in for the device array; its
// device address is obtained with cudaGetSymbolAddress, once per device, with that
// device current, the first time the entry point runs there.  Do that first call before
// any stream capture.  All calls share the array and it keeps the last call's contents;
// nothing in it needs to start at zero (the split kernel writes every partial, empty
// splits included, before the merge kernel reads them).  Calls whose kernels overlap on
// the GPU (concurrent streams, or two host threads) race on the array.  The cached
// address belongs to the device's context: after cudaDeviceReset on a device this entry
// point must not be called there again in the same process.
//
// Arguments are checked exactly as loom_attn_decode checks them, in the same order; only
// then is the problem's need compared with the array's size (LOOM_ERR_WORKSPACE).
#include <mutex>

#include "../../include/loom_attn.h"
#include "kernels.h"

namespace loom {
namespace {

constexpr size_t kNoallocScratchBytes = LOOM_DECODE_NOALLOC_SCRATCH_BYTES;

static __device__ __align__(256) unsigned char g_decode_scratch[kNoallocScratchBytes];

constexpr int kMaxScratchDevices = 64;
void* g_scratch_dev_ptr[kMaxScratchDevices] = {};
std::mutex g_scratch_mutex;

// Device address of the scratch array on the current device (looked up once per device).
void* scratch_ptr() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxScratchDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (!g_scratch_dev_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || p == nullptr) return nullptr;
    g_scratch_dev_ptr[dev] = p;
  }
  return g_scratch_dev_ptr[dev];
}

}  // namespace
}  // namespace loom

extern "C" loom_status loom_attn_decode_noalloc(const void* q, const void* k_cache,
                                                const void* v_cache, const int32_t* seqlens_k,
                                                void* o, float* lse, int B, int Hq, int Hkv,
                                                int Skv, int D, float scale, int num_splits,
                                                void* stream) {
  int splits = 0;
  const int st = loom::decode_check_args(q, k_cache, v_cache, seqlens_k, o, lse, B, Hq, Hkv, Skv, D, scale,
                                         num_splits, &splits);
  if (st != LOOM_OK) return static_cast<loom_status>(st);
  if (loom::decode_workspace_bytes(B, Hq, D, splits) > loom::kNoallocScratchBytes) return LOOM_ERR_WORKSPACE;
  void* scratch = loom::scratch_ptr();
  if (!scratch) return LOOM_ERR_CUDA;
  return loom_attn_decode(q, k_cache, v_cache, seqlens_k, o, lse, scratch, loom::kNoallocScratchBytes,
                          B, Hq, Hkv, Skv, D, scale, num_splits, stream);
}
