// Ragged-batch (varlen) prefill: the launch interface between the C ABI (loom_api.cu)
// and the prefill kernel (attn_fwd.cu).
#pragma once

#include <cstdint>

#include "kernels.h"

namespace loom {

struct FwdVarlenArgs {
  const void* q;           // [total_q, Hq, D] bf16
  const void* k;           // [total_k, Hkv, D] bf16
  const void* v;           // [total_k, Hkv, D] bf16
  void* o;                 // [total_q, Hq, D] bf16
  float* lse;              // [Hq, total_q] or null
  const int32_t* cu_q;     // [B + 1] on the device
  const int32_t* cu_k;     // [B + 1] on the device
  int B, Hq, Hkv, total_q, total_k, max_seqlen_q, D, causal;
  float scale;
};

cudaError_t launch_fwd_varlen(const FwdVarlenArgs& a, const KernelCtl& ctl, cudaStream_t stream);

}  // namespace loom
