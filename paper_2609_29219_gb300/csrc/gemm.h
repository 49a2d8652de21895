// Launch interface of the BF16 GEMM (gemm.cu) for the C ABI (loom_api.cu).
#pragma once

#include <cuda_runtime.h>

#include "ptx.cuh"

namespace loom {

struct GemmArgs {
  const void* a;  // [M, K] bf16 row-major
  const void* b;  // [K, N] bf16 row-major ([N, K] when b_kmajor)
  void* c;        // [M, N] bf16 row-major
  int M, N, K;
  int tile_n;     // 0: the analytic model's choice, else 64, 128, 192 or 256
  int splits;     // 0: the model's choice, else 1 (persistent tiles) or 2, 4, 8, 16 (split-K clusters)
  int pair;       // 0: the model's choice, 1: CTA-pair 256 x 256 tiles, -1: never CTA pairs
  int b_kmajor;   // 1: b is [N, K] row-major and C = A B^T
  int stages;     // 0: the model's ring depth; a compiled neighbour of it otherwise (block-size ablation)
  int group;      // tile rows per group of the tile order (0: 12 for CTA-pair tiles, 8 otherwise)
  int k_alt;      // CTA-pair kernel: K walked backwards in every other round of tiles (0, 1: yes; -1: no)
};

struct GemmChoice {
  int tile_n, splits;
  int pair;  // as a choice: 1 = CTA-pair tiles; as a restriction: see GemmArgs::pair
};

cudaError_t launch_gemm(const GemmArgs& a, const KernelCtl& ctl, cudaStream_t stream);
// The model's (tile width, split count, CTA pair) for this shape on the current device;
// fields of `forced` that are non-zero restrict the choice.  tile_n = 0 if the device
// cannot be queried or nothing fits the restriction.
GemmChoice gemm_choice(int M, int N, int K, GemmChoice forced);

}  // namespace loom
