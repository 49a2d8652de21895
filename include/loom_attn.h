/*
 * loom_attn.h -- C ABI of the GB300 (sm_103a) fused-attention library.
 *
 * The library computes scaled-dot-product attention
 *
 *     O = softmax(scale * Q K^T [+ causal mask]) V,   LSE = ln sum_j exp(scale * q . k_j)
 *
 * in the two forms the Loom paper evaluates: Flash Attention prefill (Sec. 3.2.2: the
 * score product, the softmax and the weighted sum of values fused in one kernel) and
 * Flash Decode (Sec. 2.6 Flash Decode example and Sec. 3.2.3: the sequence axis is
 * split across cores, each split runs a local softmax loop, and the partial results
 * are gathered, globally softmaxed and finally scaled).
 *
 * Conventions shared by every entry point:
 *   - Tensors are dense, contiguous, row-major device buffers:
 *       Q, O   [B, Hq,  Sq,  D]  bfloat16
 *       K, V   [B, Hkv, Skv, D]  bfloat16
 *       LSE    [B, Hq,  Sq]      float32 (natural log)
 *   - Grouped-query attention: query head h reads kv head h / (Hq / Hkv).
 *   - Causal masking is bottom-right aligned: query i sees key j iff j <= i + (Skv - Sq).
 *   - D must be 64 or 128; scale must be finite and > 0.
 *   - Every device pointer must be 16-byte aligned.
 *   - All calls are asynchronous on `stream` (a cudaStream_t passed as void*; NULL is
 *     the legacy default stream).  The caller owns every buffer, including the decode
 *     workspace; the library allocates no device memory.
 *   - Argument errors are reported synchronously by the return value and nothing is
 *     launched.  Launch failures return LOOM_ERR_CUDA.  A kernel that gives up on a
 *     bounded internal wait sets a device error word, which loom_attn_check_error
 *     reports as LOOM_ERR_TIMEOUT.
 */
#ifndef LOOM_ATTN_H_
#define LOOM_ATTN_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  LOOM_OK = 0,
  LOOM_ERR_INVALID_ARG = 1, /* null pointer, non-positive size, Hq % Hkv != 0, bad scale, ... */
  LOOM_ERR_UNSUPPORTED = 2, /* D not in {64, 128}, too many splits, ... */
  LOOM_ERR_MISALIGNED = 3,  /* a pointer is not 16-byte aligned */
  LOOM_ERR_WORKSPACE = 4,   /* decode workspace missing or too small */
  LOOM_ERR_CUDA = 5,        /* a CUDA runtime/driver call or kernel launch failed */
  LOOM_ERR_TIMEOUT = 6      /* a kernel abandoned a bounded wait (reported by check_error) */
} loom_status;

/*
 * Flash Attention forward (prefill), paper Sec. 3.2.2.
 *   q      [B, Hq, Sq, D]  bf16, read
 *   k, v   [B, Hkv, Skv, D] bf16, read
 *   o      [B, Hq, Sq, D]  bf16, written
 *   lse    [B, Hq, Sq]     fp32, written; may be NULL
 *   causal 0 or 1 (bottom-right aligned; causal requires Sq <= Skv)
 * Errors: INVALID_ARG (null q/k/v/o, any size <= 0, Hq % Hkv, causal with Sq > Skv,
 * scale not finite or <= 0), UNSUPPORTED (D), MISALIGNED, CUDA.
 */
loom_status loom_attn_fwd(const void* q, const void* k, const void* v, void* o, float* lse, int B,
                          int Hq, int Hkv, int Sq, int Skv, int D, int causal, float scale,
                          void* stream);

/*
 * Prefill over a ragged batch packed token-major (the packed-varlen layout; the paper has
 * no counterpart -- irregular grids are outside its Sec. 2.6 scope note).
 *   q             [total_q, Hq, D]   bf16, read
 *   k, v          [total_k, Hkv, D]  bf16, read
 *   o             [total_q, Hq, D]   bf16, written
 *   lse           [Hq, total_q]      fp32, written (natural log); may be NULL
 *   cu_seqlens_q,
 *   cu_seqlens_k  [B + 1] int32 on the device: sequence b owns query tokens
 *                 cu_seqlens_q[b] .. cu_seqlens_q[b+1] - 1 and key tokens likewise; both
 *                 start at 0, never decrease and end at total_q / total_k.
 *   max_seqlen_q  an upper bound of the query lengths (it only sizes the launch; every
 *                 sequence is computed whatever its value).
 * Each sequence is attention on its own tokens (GQA as loom_attn_fwd); causal masking is
 * bottom-right aligned per sequence, and a query with no visible key (causal with more
 * queries than keys, or no keys) gets O = 0 and LSE = -inf.  Runs the two-tile prefill
 * kernel (design 2) with a sequence cursor over the offsets.
 * Errors: INVALID_ARG (NULL pointer, B, Hq, Hkv or D <= 0, total_q, total_k or
 * max_seqlen_q < 0, Hq % Hkv, scale), UNSUPPORTED (D not 64 or 128; total_k = 0 while
 * total_q > 0; more than 2^31 work items), MISALIGNED (q, k, v, o not 16-byte aligned;
 * cu_seqlens, lse not 4-byte aligned), CUDA.  total_q = 0 returns LOOM_OK at once.
 */
loom_status loom_attn_fwd_varlen(const void* q, const void* k, const void* v, void* o, float* lse,
                                 const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k, int B,
                                 int Hq, int Hkv, int total_q, int total_k, int max_seqlen_q, int D,
                                 int causal, float scale, void* stream);

/*
 * Number of KV splits the decode path uses for this problem when the caller passes
 * num_splits = 0: the analytic model's choice (one wave of split CTAs over the GPU's
 * SMs, Sec. 2.6 Eq. 8-9 restated for GB300).  Returns 0 on invalid sizes.
 * Skv is the KV-cache capacity (the longest possible sequence).
 */
int loom_attn_decode_num_splits(int B, int Hq, int Hkv, int Skv, int D);

/*
 * Device workspace (bytes) that loom_attn_decode needs: the per-split partial outputs
 * O_i [B, Hq, splits, D] fp32 and log-sum-exps lse_i [B, Hq, splits] fp32 (each from a
 * 256-byte boundary), then 256 bytes holding the persistent split kernel's item counter.
 * num_splits = 0 means the model's choice.  Returns 0 on invalid sizes.
 */
size_t loom_attn_decode_workspace_bytes(int B, int Hq, int Hkv, int Skv, int D, int num_splits);

/*
 * Flash Decode (Sq = 1), paper Sec. 2.6 (Flash Decode HEG) and Sec. 3.2.3.
 *   q          [B, Hq, 1, D]      bf16, read
 *   k_cache,
 *   v_cache    [B, Hkv, Skv, D]   bf16, read (Skv = cache capacity)
 *   seqlens_k  [B] int32 on the device: valid length of each sequence, 0..Skv; NULL means
 *              every sequence has Skv keys.  Lengths outside [0, Skv] are clamped.
 *   o          [B, Hq, 1, D]      bf16, written
 *   lse        [B, Hq]            fp32, written; may be NULL
 *   workspace  device scratch of at least loom_attn_decode_workspace_bytes(...) bytes;
 *              its contents on entry do not matter and are overwritten (the item
 *              counter in its last 256 bytes is left armed for the next call; a
 *              workspace serves one call at a time).
 *   num_splits 0 = analytic model, otherwise 1..1024 splits of each sequence.
 * Split i of sequence b covers keys [i*C, min((i+1)*C, len_b)), C = ceil(len_b/splits)
 * rounded up to a multiple of 64; empty splits contribute nothing.  A sequence of
 * length 0 yields O = 0 and LSE = -inf.
 * Three forms compute it, chosen by the analytic model (see loom_attn_decode_form):
 *   1  a split kernel writing the partials (O_i, lse_i) into the workspace, then a merge
 *      kernel (the gather, global softmax and final scaling of the Flash Decode HEG).
 *      The split kernel runs on the tensor cores (D 64 or 128, at most 32 query heads
 *      per kv head): persistent CTAs take the (sequence, kv head, split) items from a
 *      counter in the workspace (loom_debug_decode_tensor_cores); otherwise it is a
 *      CUDA-core kernel of one CTA per (split, batch, kv head);
 *   2  the same partials and merge kernel, with a persistent CUDA-core split kernel whose
 *      CTAs walk the (split, batch, kv head) items in a fixed order, streaming K/V across
 *      item boundaries (the model considers it only where the tensor-core kernel does not
 *      run);
 *   3  one persistent kernel in which clusters of cs CTAs (cs divides num_splits, cs <= 16)
 *      walk the (batch, kv head) pairs, CTA r taking splits r, r + cs, ... of each, and
 *      merge their partials over distributed shared memory; it leaves the workspace
 *      untouched, but the call checks and requires it all the same.
 * All three follow the split rule above and give the same result up to rounding order.
 * With num_splits = 0 the model picks the split count and the form together (Eq. 9 over
 * both); a split count the caller fixes runs form 1 (loom_debug_decode_form pins another).
 * Errors: INVALID_ARG, UNSUPPORTED, MISALIGNED, WORKSPACE, CUDA.
 */
loom_status loom_attn_decode(const void* q, const void* k_cache, const void* v_cache,
                             const int32_t* seqlens_k, void* o, float* lse, void* workspace,
                             size_t workspace_bytes, int B, int Hq, int Hkv, int Skv, int D,
                             float scale, int num_splits, void* stream);

/*
 * Flash Decode over a paged KV cache (the layout of paged serving engines; the paper has
 * no counterpart -- it belongs to the irregular grids its Sec. 2.6 scope note sets aside).
 *   q            [B, Hq, 1, D]                     bf16, read
 *   k_cache,
 *   v_cache      bf16, read; a page holds page_size consecutive keys of one sequence:
 *                kv_layout 0 (NHD): [num_pages, page_size, Hkv, D], a key's rows of all kv
 *                heads adjacent; kv_layout 1 (HND): [num_pages, Hkv, page_size, D], a page's
 *                rows of one kv head contiguous
 *   block_table  [B, max_pages] int32 on the device: key t of sequence b is row
 *                t % page_size of page block_table[b * max_pages + t / page_size].  Only
 *                the first ceil(len_b / page_size) entries of a row are read; an entry
 *                outside [0, num_pages) reads zeros (no fault).
 *   seqlens_k    [B] int32 on the device (required): 0 .. max_pages * page_size, clamped
 *   o, lse, workspace, num_splits, scale: as loom_attn_decode, with Skv = max_pages *
 *                page_size in loom_attn_decode_workspace_bytes / loom_attn_decode_num_splits.
 * page_size: 8, 16, 32 or a multiple of 64.  The split rule and results are those of
 * loom_attn_decode on the gathered (logical) cache.
 * Errors: INVALID_ARG (NULL q/k/v/o/block_table/seqlens_k, a size <= 0, Hq % Hkv, scale,
 * kv_layout not 0 or 1), UNSUPPORTED (D, page_size, more than 2^31 - 1 keys in the cache or
 * per sequence, too many splits), MISALIGNED (q, caches, o, workspace not 16-byte aligned; block_table, seqlens_k,
 * lse not 4-byte aligned), WORKSPACE, CUDA.
 */
loom_status loom_attn_decode_paged(const void* q, const void* k_cache, const void* v_cache,
                                   const int32_t* block_table, const int32_t* seqlens_k, void* o,
                                   float* lse, void* workspace, size_t workspace_bytes, int B, int Hq,
                                   int Hkv, int num_pages, int page_size, int max_pages, int kv_layout,
                                   int D, float scale, int num_splits, void* stream);

/*
 * Flash Decode without any allocation and without a workspace argument.  The paper has
 * no counterpart; this entry point exists for callers that cannot obtain device scratch
 * memory for a call -- serving engines that reserve all device memory at start-up and
 * forbid allocation on the request path (cudaMalloc synchronises the whole device and
 * can fail mid-request), and plug-in hosts that pass a library only the call's tensors.
 *
 * Arguments, layouts and results are those of loom_attn_decode.  The per-split partials
 * live in a scratch array built into the library (LOOM_DECODE_NOALLOC_SCRATCH_BYTES,
 * 8 MiB), held by every GPU that loads the library until the process exits.  A problem
 * whose partials need more (loom_attn_decode_workspace_bytes(...) larger than that)
 * returns LOOM_ERR_WORKSPACE without launching anything.  The first call on a device
 * looks up the array's device address (cudaGetSymbolAddress, current device); make that
 * first call before any stream capture.  All calls share the array, which keeps the last
 * call's contents (nothing in it needs to start at zero); calls whose kernels overlap on
 * the GPU race on it.  This entry point itself calls no cudaMalloc or cudaFree.  The
 * looked-up address belongs to the device's context: after cudaDeviceReset the entry
 * point must not be called on that device again in the same process.
 * Errors: those of loom_attn_decode, checked in the same order (INVALID_ARG,
 * UNSUPPORTED, MISALIGNED); then WORKSPACE when the partials exceed the array; CUDA.
 */
#define LOOM_DECODE_NOALLOC_SCRATCH_BYTES ((size_t)8 << 20)
loom_status loom_attn_decode_noalloc(const void* q, const void* k_cache, const void* v_cache,
                                     const int32_t* seqlens_k, void* o, float* lse, int B, int Hq,
                                     int Hkv, int Skv, int D, float scale, int num_splits,
                                     void* stream);

/*
 * Analytic schedule model (paper Sec. 2.6: HEG latency, Eq. 5-7, and the constrained
 * selection of Eq. 8-9, solved by enumeration) with the GB300 architecture description
 * of Sec. 2.7.  The kernels are compiled with the plan these functions report.
 *
 * loom_model_fwd_plan: the prefill plan for head dimension D (64 or 128): the design, rows
 *   per query tile, keys per KV tile, query tiles per CTA, S buffers, K/V ring slots, the pipeline knob
 *   (b_lm, b_ms) of Eq. 6, shared-memory bytes, TMEM columns, and the modeled latencies
 *   (ns) of one KV-tile iteration: load stage, MMA leaf, softmax leaf, and the pipe node.
 *   Returns LOOM_ERR_UNSUPPORTED for other D, LOOM_ERR_INVALID_ARG for a NULL out.
 * loom_model_fwd_plan_variant: the best plan of one design (1, 2 or 3) for head dimension
 *   D, the candidates Eq. 9 ranks; LOOM_ERR_UNSUPPORTED if that design has no feasible plan
 *   at this D (the TMEM or shared-memory capacity of Eq. 8 rules it out).
 * loom_model_heg_pipe: Eq. 6, the latency of a three-stage pipe node with load stage l,
 *   body m and store stage s under the pipeline knob (b_lm, b_ms), each 0 or 1.
 * loom_model_fwd_time_us: modeled time of a whole prefill launch (us); < 0 on bad sizes.
 * loom_model_decode_time_us: modeled split + merge time (us) of Flash Decode with
 *   `splits` splits on `num_sms` SMs (every sequence Skv keys); < 0 on bad sizes.
 */
typedef struct {
  int design; /* 2: two alternating query tiles; 1: one tile, S double-buffered; 3: two tiles, S ring of 3 */
  int bm, bn, q_tiles, s_buffers, kv_slots, b_lm, b_ms, smem_bytes, tmem_cols;
  double t_load_ns, t_mma_ns, t_softmax_ns, t_iter_ns;
} loom_fwd_plan;
loom_status loom_model_fwd_plan(int D, loom_fwd_plan* out);
loom_status loom_model_fwd_plan_variant(int D, int design, loom_fwd_plan* out);
double loom_model_heg_pipe(double l, double m, double s, int b_lm, int b_ms);
double loom_model_fwd_time_us(int B, int Hq, int Sq, int Skv, int D, int causal);
/* Modeled prefill launch time (us) with design 1, 2 or 3 forced; < 0 if infeasible. */
double loom_model_fwd_time_us_design(int design, int B, int Hq, int Sq, int Skv, int D, int causal);
double loom_model_decode_time_us(int splits, int B, int Hq, int Hkv, int Skv, int D, int num_sms);
/* Modeled time (us) of the single-kernel (cluster) Flash Decode with `splits` splits and
 * clusters of `cluster` CTAs (dividing splits, at most 16) when `clusters` such clusters
 * fit on the GPU at once; < 0 on bad sizes. */
double loom_model_decode_cluster_time_us(int splits, int cluster, int B, int Hq, int Hkv, int Skv, int D,
                                         int clusters);

/* Modeled time (us) of the persistent split kernel + merge with `splits` splits on `ctas`
 * resident CTAs; < 0 on bad sizes. */
double loom_model_decode_persistent_time_us(int splits, int B, int Hq, int Hkv, int Skv, int D, int ctas);

/* Modeled time (us) of the split + merge form with its split kernel on the tensor cores
 * (persistent CTAs, two per SM of `num_sms`, taking the items on demand): the start-up
 * once, the items in rounds of at most 2 * num_sms, each streaming its chunk and paying a
 * fixed boundary cost, then the merge.  The split count with num_splits = 0 and the form
 * of a contiguous-cache call use it where that kernel takes the shape (at most 32 query
 * heads per kv head); < 0 on bad sizes or more heads per kv head. */
double loom_model_decode_tc_time_us(int splits, int B, int Hq, int Hkv, int Skv, int D, int num_sms);

/*
 * Which Flash Decode form a call with these sizes runs on the current device: 1 = split
 * kernel + merge kernel, 2 = persistent split kernel + merge kernel, 3 = the single-kernel
 * cluster form (Sec. 2.6's gather, global softmax and final scaling done inside one kernel,
 * over distributed shared memory) with *cluster CTAs per cluster; -1 = invalid sizes.
 * num_splits = 0 means the model's split count; paged = 1 asks about
 * loom_attn_decode_paged (Skv = max_pages * page_size).  cluster may be NULL.  Follows
 * loom_debug_decode_form.
 * loom_decode_max_clusters: clusters of `cluster` decode CTAs (G query heads per kv head,
 * head dimension D) resident on the current device at once, 0 if none; with no device, the
 * model's GB300 estimate (whole clusters in 8 equal groups of SMs).
 * loom_decode_persistent_slots: CTAs of the persistent split kernel resident at once (with
 * no device: the model's 2 per SM x 152 SMs).  These are what the split-count choice
 * (num_splits = 0) prices the persistent forms with.
 */
int loom_attn_decode_form(int B, int Hq, int Hkv, int Skv, int D, int num_splits, int paged, int* cluster);
int loom_decode_max_clusters(int D, int G, int cluster);
int loom_decode_persistent_slots(int D, int G);

/*
 * BF16 GEMM, the third kernel the paper evaluates (GEMM shapes, Sec. 4): C = A B with
 *   a  [M, K] bf16 row-major, read
 *   b  [K, N] bf16 row-major, read
 *   c  [M, N] bf16 row-major, written (fp32 accumulation, rounded to nearest even)
 * The caller owns the buffers; the call is asynchronous on `stream` and needs no
 * workspace.  The analytic model picks the kernel: persistent CTAs over 128-row tiles of
 * 64, 128, 192 or 256 columns; persistent CTA pairs over 256 x 256 tiles; or, for few
 * tiles and a long K, split-K over clusters of S = 2, 4, 8 or 16 CTAs that sum their fp32
 * partials through distributed shared memory in a fixed order (so the result depends on
 * S but not on timing).  loom_gemm_tile_n / loom_gemm_splits report the
 * choice for a shape on the current device.
 * Errors: INVALID_ARG (NULL pointer, M, N or K < 1), MISALIGNED (pointer not 16-byte
 * aligned), UNSUPPORTED (K or N not a multiple of 8: rows must be 16-byte multiples for
 * the tensor-memory-access copies), CUDA (launch failure).
 */
loom_status loom_gemm_bf16(const void* a, const void* b, void* c, int M, int N, int K, void* stream);
/* C = A B^T with b [N, K] bf16 row-major (a linear layer's weight layout: c_ij = sum_k a_ik
 * b_jk); B's tiles are then K-major like A's.  Everything else as loom_gemm_bf16, including
 * the model's choice of kernel (it depends on the shape only). */
loom_status loom_gemm_bf16_bt(const void* a, const void* b, void* c, int M, int N, int K, void* stream);
/* The model's tile width / split count for this shape (0 for a non-positive size).  Without a
 * device the cluster occupancy is estimated as whole clusters in 8 equal SM groups. */
int loom_gemm_tile_n(int M, int N, int K);
int loom_gemm_splits(int M, int N, int K);
/* 1 if the model computes this shape with CTA-pair tiles: a cluster of two CTAs per 256 x 256
 * tile of C with M = 256 pair MMAs (each SM holds its 128 rows of A and half of B), else 0. */
int loom_gemm_cta_pair(int M, int N, int K);
/* Modeled GEMM launch time (us) with tile width tile_n and split count splits on num_sms SMs
 * (cluster occupancy estimated as above; tile_n = 512 with splits = 1 prices the CTA-pair
 * tiles); < 0 if infeasible. */
double loom_model_gemm_time_us(int M, int N, int K, int tile_n, int splits, int num_sms);
/* Test hooks: force the GEMM tile width (64, 128, 192, 256) / split count (1, 2, 4, 8, 16);
 * any other value restores the model's choice.  A forced split may leave CTAs no K stage:
 * their partial is zero. */
void loom_debug_gemm_tile_n(int tile_n);
void loom_debug_gemm_splits(int splits);
/* Test hook: 1 forces CTA-pair tiles, -1 forbids them, anything else restores the model's choice. */
void loom_debug_gemm_cta_pair(int mode);

/*
 * Synchronises `stream`, then reads and clears the current device's error word.
 * Returns LOOM_OK, LOOM_ERR_TIMEOUT if a kernel abandoned a bounded wait since the last
 * check, or LOOM_ERR_CUDA if the synchronisation itself failed.
 */
loom_status loom_attn_check_error(void* stream);

/* Static, human-readable name of a status code. */
const char* loom_status_string(loom_status status);

/*
 * Test hooks (not needed for normal use).
 * loom_debug_set_timeout_ns: upper bound, in nanoseconds of %globaltimer, on every
 *   internal wait of the kernels (default 2e9).  0 restores the default.
 * loom_debug_inject: 0 = off; 1 = the decode split kernel's loader skips the copy of
 *   its second stage; 2 = the prefill kernel's loader skips its second K tile; 3 = the
 *   GEMM loader skips its third stage (of each CTA's K range).  The
 *   waits on the skipped data then expire, the kernel unwinds and the next
 *   loom_attn_check_error returns LOOM_ERR_TIMEOUT.  Host-side switch; no fault.
 */
void loom_debug_set_timeout_ns(uint64_t ns);
void loom_debug_inject(int mode);

/*
 * Test hook: force the prefill design instead of the analytic model's choice (used to
 * measure the alternatives the model ranks).  2: two query tiles per CTA that alternate
 * on the tensor pipe; 1: one query tile with S double-buffered in TMEM; 3: two query
 * tiles sharing a ring of three S buffers (D = 64 only; D = 128 falls back to 2);
 * anything else: the model's choice (default).
 */
void loom_debug_prefill_design(int design);

/*
 * Block-size ablation hooks (the paper's block-size ablation, Sec. 3 "Ablation Studies":
 * the neighbourhood of the solver's choice, measured).  Each pins a compiled neighbour of
 * the analytic model's constant and returns 1, or returns 0 (and restores the model's
 * constant) when that value is not compiled:
 * loom_debug_prefill_slots: the two-tile prefill's K/V ring depth for head dimension D
 *   (compiled beside the model's 3 at D = 128: 2; beside 10 at D = 64: 3, 6, 9; deeper
 *   rings do not fit in shared memory).  0 restores the model's.
 * loom_debug_decode_stage_plan: the decode split kernel's keys per stage, ring stages and
 *   CTAs per SM (contiguous cache, D = 128, 4 query heads per kv head, split + merge form;
 *   compiled: 32x2x2, 32x3x2, 32x4x2, 64x2x2, 64x4x1, 128x2x1, 128x3x1 beside the model's
 *   64x3x2).  tokens = 0 restores the model's.
 * loom_debug_gemm_stages: the GEMM's K-stage ring depth ([K, N] B): the CTA pair with 5
 *   (model: 6), 256-wide persistent tiles with 3 (model: 4), 128-wide with 5 (model: 6);
 *   other values or kernels run the model's depth.  0 restores the model's.
 * loom_debug_gemm_order: the GEMM's tile order.  group_rows (1..1024; 0: the default, 12
 *   for CTA-pair tiles and 8 otherwise) tile rows form one group, walked column by column,
 *   so tiles in flight together share rows of A and columns of B in L2.  The CTA-pair
 *   kernel walks K from its end in every other round of tiles, so a round starts on the K
 *   slices the previous round touched last (still in L2); k_alternate = -1 turns that off
 *   (0 or 1: on).  Either changes only which CTA computes which tile when, and the order of
 *   the fp32 sum over K blocks.
 */
int loom_debug_prefill_slots(int D, int slots);
int loom_debug_decode_stage_plan(int tokens, int stages, int ctas_per_sm);
void loom_debug_gemm_stages(int stages);
void loom_debug_gemm_order(int group_rows, int k_alternate);

/*
 * loom_debug_decode_tensor_cores: which split kernel the split + merge form runs (D 64
 * or 128, at most 32 query heads per kv head; the other forms always use the CUDA-core
 * stage).
 *   1 (the default): tensor cores, persistent, contiguous or paged cache.  Two CTAs per
 *     SM take (sequence, kv head, split) items, longest sequence first, from a counter in
 *     the workspace's last 256 bytes until none is left, and stream the next item's q and
 *     K/V without a break (a paged cache: each stage copied page by page); per stage of
 *     64 keys (128 at D = 64) S = Q K^T and O += P V are tcgen05 MMAs with the query heads as rows
 *     of a TMEM tile and the softmax on one warp.  The merge kernel re-arms the counter;
 *     a workspace whose counter was never armed (its first call) is dealt statically.
 *   2: the same stage on the tensor cores, one CTA per (split, kv head, sequence), for a
 *     contiguous cache (a paged cache takes the CUDA-core kernel).
 *   0: the CUDA-core split kernel.
 * Other values select 1.  On the tensor cores P is rounded to bf16 before P V, as in
 * the prefill; the CUDA-core stage keeps it in fp32.
 */
void loom_debug_decode_tensor_cores(int mode);

/*
 * Test hook: the Flash Decode form.  form 1 = split + merge kernels, 2 = persistent split
 * kernel + merge kernel, 3 = the single-kernel cluster form (each when it can run); anything
 * else: the analytic model's choice (default).  cluster in 1..16 pins the cluster form's
 * cluster size (honoured when it divides the split count and such clusters fit); 0: the
 * model's size.
 */
void loom_debug_decode_form(int form, int cluster);

#ifdef __cplusplus
}
#endif

#endif /* LOOM_ATTN_H_ */
