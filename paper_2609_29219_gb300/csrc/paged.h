// Paged KV cache for Flash Decode: the launch interface between the C ABI (loom_api.cu)
// and the decode kernels (attn_decode.cu).
#pragma once

#include <cstdint>

#include "kernels.h"

namespace loom {

// A page holds page_size consecutive keys of one sequence.  Key t of sequence b lives in
// row t % page_size of page block_table[b * max_pages + t / page_size].  Layouts (bf16):
//   kPagedNHD  [num_pages, page_size, Hkv, D]  (a key's rows of all kv heads adjacent)
//   kPagedHND  [num_pages, Hkv, page_size, D]  (a page's rows of one kv head contiguous)
constexpr int kPagedNHD = 0, kPagedHND = 1;

struct PagedKV {
  const int32_t* block_table;  // [B, max_pages]
  int num_pages;               // pages in each of the K and V caches
  int page_size;               // keys per page
  int max_pages;               // logical pages per sequence (row stride of block_table)
  int layout;                  // kPagedNHD or kPagedHND
};

// Page sizes the loader supports: each 64-key copy (the split-chunk alignment) lies in one
// page, or a stage's keys span whole pages of at least 8 keys.
constexpr bool paged_page_size_ok(int p) { return p == 8 || p == 16 || p == 32 || (p >= 64 && p % 64 == 0); }

// a.k / a.v are the caches, a.Skv = max_pages * page_size, a.seqlens is required.
cudaError_t launch_decode_paged(const DecodeArgs& a, const PagedKV& pk, const KernelCtl& ctl, cudaStream_t stream);

}  // namespace loom
