// Launch interface of the BF16 GEMM (gemm.cu) for the C ABI (loom_api.cu).
#pragma once

#include <cuda_runtime.h>

#include "ptx.cuh"

namespace loom {

struct GemmArgs {
  const void* a;  // [M, K] bf16 row-major
  const void* b;  // [K, N] bf16 row-major
  void* c;        // [M, N] bf16 row-major
  int M, N, K;
  int tile_n;     // 0: the analytic model's choice, else 64, 128, 192 or 256
  int splits;     // 0: the model's choice, else 1 (persistent tiles) or 2, 4, 8, 16 (split-K clusters)
};

struct GemmChoice {
  int tile_n, splits;
};

cudaError_t launch_gemm(const GemmArgs& a, const KernelCtl& ctl, cudaStream_t stream);
// The model's (tile width, split count) for this shape on the current device; fields of
// `forced` that are non-zero are kept.  {0, 0} if the device cannot be queried.
GemmChoice gemm_choice(int M, int N, int K, GemmChoice forced);

}  // namespace loom
