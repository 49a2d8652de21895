// Internal launch interface between the C ABI (loom_api.cu) and the kernel files.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "ptx.cuh"

namespace loom {

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
};

struct FwdArgs {
  const void* q;  // [B, Hq, Sq, D] bf16
  const void* k;  // [B, Hkv, Skv, D] bf16
  const void* v;  // [B, Hkv, Skv, D] bf16
  void* o;        // [B, Hq, Sq, D] bf16
  float* lse;     // [B, Hq, Sq] or null
  int B, Hq, Hkv, Sq, Skv, D, causal;
  float scale;
  int design;  // prefill design: 0 = the analytic model's choice, 1..3 forced
};

// Bytes of workspace the decode path needs for `splits` splits.
inline size_t decode_workspace_bytes(int B, int Hq, int D, int splits) {
  const size_t rows = static_cast<size_t>(B) * Hq * splits;
  const size_t opart = rows * D * sizeof(float);
  const size_t lpart = rows * sizeof(float);
  return ((opart + 255) / 256) * 256 + ((lpart + 255) / 256) * 256;
}

cudaError_t launch_decode(const DecodeArgs& a, const KernelCtl& ctl, cudaStream_t stream);
cudaError_t launch_fwd(const FwdArgs& a, const KernelCtl& ctl, cudaStream_t stream);

}  // namespace loom
