// Architecture microbenchmarks for the analytic schedule model (the paper's Sec. 2.7:
// performance properties of an architecture are characterised once, by isolated
// microbenchmarks, and reused across operators and shapes).
//
// Built as a standalone program (paper_2609_29219_gb300/arch_probe.py builds and runs it)
// and printing one JSON object:
//   pipes : ex2.approx / fma.rn.f32 / fma.rn.f32x2 / cvt.rn.bf16x2.f32 / ex2.approx.bf16x2
//           instruction-lanes per clock per SM, and ex2 beside the bf16x2 packs of the softmax
//           (one per pair)
//   mma   : clocks per tcgen05.mma kind::f16 128xNx16 (SS with N = 64, 128, 256; TS N = 128)
//   mix   : clocks per 128x128x128 GEMM of the prefill kernel's MMA stream (P.V as TS,
//           S = Q.K^T as SS, two query tiles) alone and under added load: bulk copies,
//           TMEM loads/stores, commits, fences, random operands, and neighbour warps that
//           keep the issue ports busy.
// Every kernel runs one CTA per SM, touches only its own shared memory / TMEM and the
// buffers allocated below, and bounds every wait.
#include <cstdint>
#include <cstdio>
#include <initializer_list>

#include "ptx.cuh"

namespace {
using namespace loom;
__device__ __forceinline__ float ex2f_(float x){float y; asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x)); return y;}
// One tcgen05.mma issued by the warp's elected lane while every lane runs the surrounding
// code, so that operands and control flow are warp-uniform.
__device__ __forceinline__ void mma_ss_el(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p, e;\n\tsetp.ne.b32 p, %4, 0;\n\telect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
__device__ __forceinline__ void mma_ts_el(uint32_t d, uint32_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p, e;\n\tsetp.ne.b32 p, %4, 0;\n\telect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
      "r"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
__device__ __forceinline__ void tc_commit_el(uint32_t bar) {
  asm volatile(
      "{\n\t.reg .pred e;\n\telect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(bar)
      : "memory");
}

template <int MODE>
__global__ void pipe_kernel(float* out, long long* cyc, int iters) {
  float v[8];
  for (int i=0;i<8;i++) v[i] = -1e-3f * (threadIdx.x + i);
  unsigned long long w[8];
  for (int i=0;i<8;i++) { float a=v[i], b=v[i]*0.5f; asm("mov.b64 %0, {%1,%2};" : "=l"(w[i]) : "f"(a), "f"(b)); }
  const unsigned long long m2 = 0x3f0000003f000000ull;  // (0.5, 0.5)
  __syncthreads();
  long long t0 = clock64();
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if (MODE == 0) v[i] = ex2f_(v[i]) - 1.5f;              // 1 MUFU + 1 FADD
      if (MODE == 1) v[i] = fmaf(v[i], 0.999f, 1e-7f);       // 1 FFMA
      if (MODE == 2) asm volatile("fma.rn.f32x2 %0, %0, %1, %1;" : "+l"(w[i]) : "l"(m2));  // 1 FFMA2
      if (MODE == 3) {  // 1 bf16x2 pack, its result fed back as the next input
        uint32_t r;
        asm volatile("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(v[i]), "f"(v[i]));
        v[i] = __uint_as_float(r);
      }
      if (MODE == 5) {  // packed exponential: one MUFU instruction for two bf16 results
        uint32_t r = __float_as_uint(v[i]);
        asm volatile("ex2.approx.ftz.bf16x2 %0, %0;" : "+r"(r));
        v[i] = __uint_as_float(r ^ 0x80008000u);  // both halves negative again: results stay in (0, 1]
      }
      if (MODE == 4) {  // the softmax mix: 1 MUFU + 1 FADD per element, a bf16x2 pack per pair
        v[i] = ex2f_(v[i]) - 1.5f;
        if (i & 1) {
          uint32_t r;
          asm volatile("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(v[i - 1]), "f"(v[i]));
          w[i] ^= r;
        }
      }
    }
  }
  __syncthreads();
  long long t1 = clock64();
  float s = 0; for (int i=0;i<8;i++) s += v[i] + __uint_as_float((unsigned)w[i]);
  out[blockIdx.x * blockDim.x + threadIdx.x] = s;
  if (threadIdx.x == 0) cyc[blockIdx.x] = t1 - t0;
}
template <int MODE>  // 0: SS N=128, 1: TS N=128, 2: SS N=256, 3: SS N=64
__global__ void __launch_bounds__(128, 1) mma_kernel(long long* out, int iters) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* sm = smem_raw + (base - raw);
  __shared__ uint64_t bar;
  __shared__ uint32_t tptr;
  for (int i = threadIdx.x; i < 65536 / 4; i += blockDim.x) reinterpret_cast<uint32_t*>(sm)[i] = 0;  // A 16K | B 32K | pad
  const uint32_t bar_a = smem_u32(&bar);
  if (threadIdx.x == 0) { mbar_init(bar_a, 1); fence_barrier_init(); }
  if (threadIdx.x < 32) tmem_alloc(smem_u32(&tptr), 512);
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  tc_fence_before(); __syncthreads(); tc_fence_after();
  const uint32_t tmem = tptr;
  if (threadIdx.x == 0) {
    constexpr int N = MODE == 2 ? 256 : MODE == 3 ? 64 : 128;
    const uint32_t idesc = idesc_bf16(128, N, 0, 0);
    const uint32_t a = base, b = base + 16384;
    // warm-up + timed
    long long t0 = 0;
    for (int rep = 0; rep < 2; ++rep) {
      if (rep == 1) t0 = clock64();
      for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t bd = sdesc_sw128(b + (kk % 4) * 32, 16, 1024);
          if (MODE == 1) mma_ts(tmem, tmem + 256 + kk * 8, bd, idesc, 1);
          else mma_ss(tmem, sdesc_sw128(a + (kk % 4) * 32, 16, 1024), bd, idesc, 1);
        }
      }
      tc_commit(bar_a);
      for (long long spin = 0; spin < (1LL << 26) && !mbar_try_wait(bar_a, rep & 1); ++spin) {}
    }
    long long t1 = clock64();
    out[blockIdx.x] = t1 - t0;
  }
  tc_fence_before(); __syncthreads(); tc_fence_after();
  if (threadIdx.x < 32) tmem_dealloc(tmem, 512);
}
// and concurrent tcgen05.ld/st traffic by 8 other warps.  Reports clocks per 128^3 GEMM.
// smem: Q 2x32K at 0, ring 4x32K at 64K  (total 192K + 1K align)
// bit0: bulk copies; bit1: tcgen05.ld/st traffic; bit2: busy ALU warps; bit3: commit per GEMM;
// bit4: random operands; bit5: fence per GEMM; bit6: high-ILP FMA warps; bit7: prebuilt
// descriptors; bit8: polling warps; bit9: the whole MMA warp runs the issue loop (elected lane issues)
template <int MODE>
__global__ void __launch_bounds__(320, 1) mix_kernel(long long* out, const uint8_t* __restrict__ g, int iters) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  __shared__ uint64_t bars[4];
  __shared__ uint32_t tptr;
  __shared__ volatile int done;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) { for (int i = 0; i < 4; ++i) mbar_init(smem_u32(&bars[i]), 1); done = 0; fence_barrier_init(); }
  {
    uint32_t* w = reinterpret_cast<uint32_t*>(smem_raw + (base - raw));
    for (int i = threadIdx.x; i < 6 * 32768 / 4; i += blockDim.x) {
      uint32_t x = (MODE & 16) ? (uint32_t)i * 2654435761u + 12345u : 0u;
      x ^= x >> 13; x *= 0x5bd1e995u; x ^= x >> 15;
      // two bf16 values with exponent in [2^-2, 2^1] and random sign/mantissa
      const uint32_t lo = (x & 0x807Fu) | 0x3E80u | ((x >> 7) & 0x0180u);
      const uint32_t hi = ((x >> 16) & 0x807Fu) | 0x3E80u | ((x >> 23) & 0x0180u);
      w[i] = (MODE & 16) ? (lo | (hi << 16)) : 0u;
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 9) tmem_alloc(smem_u32(&tptr), 512);
  tc_fence_before(); __syncthreads(); tc_fence_after();
  const uint32_t tmem = tptr;
  if (warp == 9 && (lane == 0 || (MODE & 512))) {
    const uint32_t ids = idesc_bf16(128, 128, 0, 0), idpv = idesc_bf16(128, 128, 0, 1);
    long long t0 = 0;
    for (int rep = 0; rep < 2; ++rep) {
      if (rep == 1) t0 = clock64();
      if (MODE & 128) {
        // lean issue: descriptors built once, then a 32-bit add per MMA on the address field
        const uint64_t dq0 = sdesc_sw128(base, 16, 1024), dq1 = sdesc_sw128(base + 32768, 16, 1024);
        const uint64_t dk = sdesc_sw128(base + 65536, 16, 1024), dv = sdesc_sw128(base + 65536, 16384, 1024);
        for (int it = 0; it < iters; ++it) {
          const uint32_t vs = ((2 * it + 1) % 4) * (32768 >> 4), ks = ((2 * it + 2) % 4) * (32768 >> 4);
#pragma unroll
          for (int t = 0; t < 2; ++t) {
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              if (MODE & 512)
                mma_ts_el(tmem + 256 + t * 128, tmem + t * 128 + kk * 8, dv + vs + kk * (2048 >> 4), idpv, 1);
              else
                mma_ts(tmem + 256 + t * 128, tmem + t * 128 + kk * 8, dv + vs + kk * (2048 >> 4), idpv, 1);
            }
            const uint64_t dq = t ? dq1 : dq0;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              if (MODE & 512)
                mma_ss_el(tmem + t * 128, dq + ((kk / 4) * 16384 + (kk % 4) * 32) / 16,
                          dk + ks + ((kk / 4) * 16384 + (kk % 4) * 32) / 16, ids, 1);
              else
                mma_ss(tmem + t * 128, dq + ((kk / 4) * 16384 + (kk % 4) * 32) / 16,
                       dk + ks + ((kk / 4) * 16384 + (kk % 4) * 32) / 16, ids, 1);
            }
          }
        }
      } else
      for (int it = 0; it < iters; ++it) {
        for (int t = 0; t < 2; ++t) {
          const uint32_t va = base + 65536 + ((2 * it + 1) % 4) * 32768;
          if (MODE & 32) tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
            mma_ts(tmem + 256 + t * 128, tmem + t * 128 + kk * 8, sdesc_sw128(va + kk * 2048, 16384, 1024), idpv, 1);
          if (MODE & 8) tc_commit(smem_u32(&bars[3]));
          const uint32_t qa = base + t * 32768, ka = base + 65536 + ((2 * it + 2) % 4) * 32768;
          if (MODE & 32) tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
            mma_ss(tmem + t * 128, sdesc_sw128(qa + (kk / 4) * 16384 + (kk % 4) * 32, 16, 1024),
                   sdesc_sw128(ka + (kk / 4) * 16384 + (kk % 4) * 32, 16, 1024), ids, 1);
          if (MODE & 8) { tc_commit(smem_u32(&bars[3])); tc_commit(smem_u32(&bars[3])); }
        }
      }
      if (MODE & 512)
        tc_commit_el(smem_u32(&bars[0]));
      else
        tc_commit(smem_u32(&bars[0]));
      for (long long spin = 0; spin < (1LL << 26) && !mbar_try_wait(smem_u32(&bars[0]), rep & 1); ++spin) {}
    }
    if (lane == 0) out[blockIdx.x] = clock64() - t0;
    done = 1;
  } else if (warp == 8 && lane == 0 && (MODE & 1)) {
    // bulk copies of 32 KB into the ring slots, back to back, until the MMA stream is done
    int n = 0;
    for (long long spin = 0; spin < (1LL << 22) && !done; ++spin) {
      const uint32_t b = smem_u32(&bars[1 + (n & 1)]);
      if (n >= 2) for (long long s2 = 0; s2 < (1LL << 24) && !mbar_try_wait(b, ((n >> 1) - 1) & 1); ++s2) {}
      mbar_expect_tx(b, 32768);
      bulk_g2s(base + 65536 + (n % 4) * 32768, g + (size_t)(n % 64) * 32768, 32768, b);
      ++n;
    }
    for (int m = (n >= 2 ? n - 2 : 0); m < n; ++m)
      for (long long s2 = 0; s2 < (1LL << 24) && !mbar_try_wait(smem_u32(&bars[1 + (m & 1)]), (m >> 1) & 1); ++s2) {}
  } else if (warp < 8 && (MODE & 256)) {
    // neighbours polling an mbarrier phase that never completes, the way waiting
    // softmax warps do (all lanes in try_wait, warp-wide vote)
    const uint32_t never = smem_u32(&bars[3]);
    for (long long spin = 0; spin < (1LL << 24) && !done; ++spin)
      if (__all_sync(0xffffffffu, mbar_try_wait(never, 0))) break;
  } else if (warp < 8 && (MODE & 64)) {
    // high-ILP issue pressure: 32 independent FMA chains per thread
    float v[32];
    for (int i = 0; i < 32; ++i) v[i] = 1e-3f * (lane + i);
    for (long long spin = 0; spin < (1LL << 22) && !done; ++spin) {
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = fmaf(v[i], 0.999f, 1e-6f);
    }
    float acc = 0.f;
    for (int i = 0; i < 32; ++i) acc += v[i];
    if (acc == 12345.f) out[0] = 1;
  } else if (warp < 8 && (MODE & 4)) {
    // softmax-like issue pressure: FMA + MUFU work, no sleeping
    float v[8];
    for (int i = 0; i < 8; ++i) v[i] = -1e-3f * (lane + i);
    for (long long spin = 0; spin < (1LL << 22) && !done; ++spin) {
#pragma unroll
      for (int u = 0; u < 16; ++u)
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = ex2(fmaf(v[i], 0.5f, -0.75f)) - 1.5f;
    }
    if (v[0] == 12345.f) out[0] = 1;
  } else if (warp < 8 && (MODE & 2)) {
    // softmax-like TMEM traffic: read 128 columns of S, write 64 columns of P (other tile's columns)
    const uint32_t lane_addr = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t s_tm = tmem + lane_addr + (warp >> 2) * 128;
    for (long long spin = 0; spin < (1LL << 20) && !done; ++spin) {
      uint32_t r[32];
      float acc = 0.f;
      for (int ch = 0; ch < 4; ++ch) { tmem_ld32(s_tm + ch * 32, r); tmem_wait_ld(); reg_fence32(r); acc += __uint_as_float(r[0]); }
      for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(acc);
      for (int ch = 0; ch < 2; ++ch) tmem_st32(s_tm + ch * 32, r);
      tmem_wait_st();
      __nanosleep(600);
    }
  }
  __syncwarp();
  tc_fence_before(); __syncthreads(); tc_fence_after();
  if (warp == 9) tmem_dealloc(tmem, 512);
}

// The prefill softmax step on register data: per 128-key row, a 3-input max tree, then
// p = 2^(s*c - m) with a bf16x2 pack and the row sum.  Each iteration perturbs the row
// so nothing is hoisted.  Reports clocks per row per warp.  Variants of the per-pair work:
//   0: packed FMA (f32x2), two ex2, packed add into 4 accumulators, pack
//   1: scalar FMA, two ex2, scalar adds into 4 accumulators, pack
//   2: like 1 without the row sum (sum delegated elsewhere)
//   3: scalar FMA and ex2 only (no pack, no sum): MUFU-bound reference
//   4: variant 0 with every other pair's exponentials on the FMA pipe (exp2_poly)
//   5: variant 0 with one pair in four on the FMA pipe
//   6, 7, 8: variant 0 with one pair in 8, 4 or 16 on the FMA pipe in packed form (exp2_poly2)
template <int V, int CAP_THREADS = 256>
__global__ void __launch_bounds__(CAP_THREADS, 1) softmax_row_kernel(long long* cyc, float* sink, int iters) {
  if (threadIdx.x >= 256) return;  // extra threads only lower the register cap
  float s[128];
  for (int i = 0; i < 128; ++i) s[i] = 0.01f * ((threadIdx.x * 7 + i * 13) % 97) - 0.5f;
  const float c = 0.18f;
  const uint64_t c2 = f2(c, c);
  uint32_t keep = 0;
  float lsum = 0.f;
  __syncthreads();
  const long long t0 = clock64();
  for (int it = 0; it < iters; ++it) {
    float mm[8];
#pragma unroll
    for (int g = 0; g < 8; ++g) mm[g] = s[g];
#pragma unroll
    for (int i = 8; i + 16 <= 128; i += 16)
#pragma unroll
      for (int g = 0; g < 8; ++g) mm[g] = max3(mm[g], s[i + g], s[i + 8 + g]);
#pragma unroll
    for (int g = 0; g < 8; ++g) mm[g] = fmaxf(mm[g], s[120 + g]);
    const float mx = fmaxf(max3(mm[0], mm[1], mm[2]), max3(max3(mm[3], mm[4], mm[5]), mm[6], mm[7]));
    const float nm = -mx * c;
    if constexpr (V == 0 || V == 4 || V == 5 || V >= 6) {
      const uint64_t nms2 = f2(nm, nm);
      uint64_t acc[4] = {0, 0, 0, 0};
#pragma unroll
      for (int i = 0; i < 64; ++i) {
        const uint64_t x = fma2(f2(s[2 * i], s[2 * i + 1]), c2, nms2);
        const bool poly = (V == 4 && (i & 1)) || (V == 5 && (i & 3) == 3);
        const bool poly2 = (V == 6 && (i & 7) == 7) || (V == 7 && (i & 3) == 3) || (V == 8 && (i & 15) == 15);
        float p0, p1;
        if (poly2) {
          const uint64_t pp = exp2_poly2(x);
          p0 = f2lo(pp);
          p1 = f2hi(pp);
        } else {
          p0 = poly ? exp2_poly(f2lo(x)) : ex2(f2lo(x));
          p1 = poly ? exp2_poly(f2hi(x)) : ex2(f2hi(x));
        }
        acc[i & 3] = add2(acc[i & 3], f2(p0, p1));
        keep ^= pack_bf16x2(p0, p1);
      }
      const uint64_t a01 = add2(add2(acc[0], acc[1]), add2(acc[2], acc[3]));
      lsum += f2lo(a01) + f2hi(a01);
    } else {
      float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < 64; ++i) {
        const float p0 = ex2(fmaf(s[2 * i], c, nm)), p1 = ex2(fmaf(s[2 * i + 1], c, nm));
        if constexpr (V == 1) {
          acc[i & 3] += p0;
          acc[(i + 2) & 3] += p1;
        }
        if constexpr (V != 3) keep ^= pack_bf16x2(p0, p1);
        else keep ^= __float_as_uint(p0) ^ __float_as_uint(p1);
      }
      lsum += (acc[0] + acc[1]) + (acc[2] + acc[3]);
    }
    s[0] += 1e-3f * static_cast<float>(it & 1);  // perturb (static index: stays in registers)
  }
  const long long t1 = clock64();
  if (threadIdx.x == 0) cyc[blockIdx.x] = t1 - t0;
  sink[blockIdx.x * blockDim.x + threadIdx.x] = lsum + __uint_as_float(keep & 0x3f800000u);
}
}  // namespace

#define CHECK(x)                                                           \
  do {                                                                     \
    cudaError_t e_ = (x);                                                  \
    if (e_ != cudaSuccess) {                                               \
      printf("{\"error\": \"%s at line %d\"}\n", cudaGetErrorString(e_), __LINE__); \
      return 1;                                                            \
    }                                                                      \
  } while (0)

template <typename F>
static double avg_cycles(F launch, long long* d, long long* h, int sms) {
  launch();
  if (cudaDeviceSynchronize() != cudaSuccess) return -1.0;
  cudaMemcpy(h, d, sizeof(long long) * sms, cudaMemcpyDeviceToHost);
  double avg = 0;
  for (int i = 0; i < sms; ++i) avg += static_cast<double>(h[i]);
  return avg / sms;
}

int main() {
  int sms = 0;
  CHECK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0));
  long long* d = nullptr;
  CHECK(cudaMalloc(&d, sizeof(long long) * sms));
  float* out = nullptr;
  CHECK(cudaMalloc(&out, sizeof(float) * sms * 1024));
  uint8_t* g = nullptr;
  CHECK(cudaMalloc(&g, 64 * 32768));
  CHECK(cudaMemset(g, 0, 64 * 32768));
  long long* h = new long long[sms];
  printf("{\"sms\": %d", sms);

  // pipes: 1024 threads x 4096 iterations x 8 ops per CTA
  {
    const double ops = 1024.0 * 4096 * 8;
    // mode 4 counts its ex2 (8 per iteration, with 4 bf16x2 packs beside them)
    // mode 5 counts instructions (each gives two bf16 exponentials)
    const char* names[6] = {"ex2_per_clk_sm", "ffma_lanes_per_clk_sm", "ffma2_instr_lanes_per_clk_sm",
                            "cvt_bf16x2_per_clk_sm", "ex2_beside_cvt_per_clk_sm", "ex2_bf16x2_instr_per_clk_sm"};
    for (int mode = 0; mode < 6; ++mode) {
      auto launch = [&] {
        for (int rep = 0; rep < 2; ++rep) {
          if (mode == 0) pipe_kernel<0><<<sms, 1024>>>(out, d, 4096);
          if (mode == 1) pipe_kernel<1><<<sms, 1024>>>(out, d, 4096);
          if (mode == 2) pipe_kernel<2><<<sms, 1024>>>(out, d, 4096);
          if (mode == 3) pipe_kernel<3><<<sms, 1024>>>(out, d, 4096);
          if (mode == 4) pipe_kernel<4><<<sms, 1024>>>(out, d, 4096);
          if (mode == 5) pipe_kernel<5><<<sms, 1024>>>(out, d, 4096);
        }
      };
      const double cyc = avg_cycles(launch, d, h, sms);
      if (cyc <= 0) { printf(", \"error\": \"pipe probe failed\"}\n"); return 1; }
      printf(", \"%s\": %.2f", names[mode], ops / cyc);
    }
  }
  // softmax row step variants: 4 warps (one per SM sub-partition) and 8 warps (two each)
  {
    const int iters = 2000;
    for (int v = 0; v < 9; ++v)
      for (int warps : {4, 8}) {
        auto launch = [&] {
          if (v == 0) softmax_row_kernel<0><<<sms, warps * 32>>>(d, out, iters);
          if (v == 1) softmax_row_kernel<1><<<sms, warps * 32>>>(d, out, iters);
          if (v == 2) softmax_row_kernel<2><<<sms, warps * 32>>>(d, out, iters);
          if (v == 3) softmax_row_kernel<3><<<sms, warps * 32>>>(d, out, iters);
          if (v == 4) softmax_row_kernel<4><<<sms, warps * 32>>>(d, out, iters);
          if (v == 5) softmax_row_kernel<5><<<sms, warps * 32>>>(d, out, iters);
          if (v == 6) softmax_row_kernel<6><<<sms, warps * 32>>>(d, out, iters);
          if (v == 7) softmax_row_kernel<7><<<sms, warps * 32>>>(d, out, iters);
          if (v == 8) softmax_row_kernel<8><<<sms, warps * 32>>>(d, out, iters);
        };
        const double cyc = avg_cycles(launch, d, h, sms);
        if (cyc <= 0) { printf(", \"error\": \"softmax probe failed\"}\n"); return 1; }
        printf(", \"softmax_row128_v%d_clk_%dwarps\": %.1f", v, warps, cyc / iters);
      }
  }
  // variant 0 compiled under the prefill kernel's register cap (10 warps -> 168 registers)
  {
    const int iters = 2000;
    for (int warps : {4, 8}) {
      auto launch = [&] { softmax_row_kernel<0, 320><<<sms, 320>>>(d, out, iters); };
      (void)warps;
      const double cyc = avg_cycles(launch, d, h, sms);
      if (cyc <= 0) { printf(", \"error\": \"softmax probe failed\"}\n"); return 1; }
      printf(", \"softmax_row128_v0_clk_8warps_168regs\": %.1f", cyc / iters);
      auto launch6 = [&] { softmax_row_kernel<6, 320><<<sms, 320>>>(d, out, iters); };
      const double cyc6 = avg_cycles(launch6, d, h, sms);
      if (cyc6 <= 0) { printf(", \"error\": \"softmax probe failed\"}\n"); return 1; }
      printf(", \"softmax_row128_v6_clk_8warps_168regs\": %.1f", cyc6 / iters);
      break;
    }
  }
  // single-MMA rates
  {
    const int smem = 65536 + 2048, iters = 2000;
    CHECK(cudaFuncSetAttribute(mma_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    CHECK(cudaFuncSetAttribute(mma_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    CHECK(cudaFuncSetAttribute(mma_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    CHECK(cudaFuncSetAttribute(mma_kernel<3>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    const char* names[4] = {"mma_ss_128x128x16_clk", "mma_ts_128x128x16_clk", "mma_ss_128x256x16_clk",
                            "mma_ss_128x64x16_clk"};
    for (int mode = 0; mode < 4; ++mode) {
      auto launch = [&] {
        if (mode == 0) mma_kernel<0><<<sms, 128, smem>>>(d, iters);
        if (mode == 1) mma_kernel<1><<<sms, 128, smem>>>(d, iters);
        if (mode == 2) mma_kernel<2><<<sms, 128, smem>>>(d, iters);
        if (mode == 3) mma_kernel<3><<<sms, 128, smem>>>(d, iters);
      };
      const double cyc = avg_cycles(launch, d, h, sms);
      if (cyc <= 0) { printf(", \"error\": \"mma probe failed\"}\n"); return 1; }
      printf(", \"%s\": %.1f", names[mode], cyc / (iters * 8.0));
    }
  }
  // prefill-like MMA stream under load
  {
    const int iters = 500, smem = 6 * 32768 + 1024;
    const int modes[14] = {0, 1, 2, 3, 4, 8, 16, 26, 32, 64, 192, 256, 640, 704};
    const char* names[14] = {"alone", "bulk_copies", "tmem_ld_st", "copies_and_tmem", "mufu_warps",
                             "commit_per_gemm", "random_operands", "random_commits_tmem",
                             "fence_per_gemm", "ilp_fma_warps", "ilp_fma_warps_lean_issue",
                             "polling_warps", "lean_issue_warp_wide", "ilp_fma_warps_lean_issue_warp_wide"};
    printf(", \"mix_clk_per_gemm\": {");
    for (int i = 0; i < 14; ++i) {
      auto launch = [&] {
#define LOOM_MIX(M)                                                                        \
  if (modes[i] == M) {                                                                     \
    cudaFuncSetAttribute(mix_kernel<M>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem); \
    mix_kernel<M><<<sms, 320, smem>>>(d, g, iters);                                        \
  }
        LOOM_MIX(0) LOOM_MIX(1) LOOM_MIX(2) LOOM_MIX(3) LOOM_MIX(4) LOOM_MIX(8) LOOM_MIX(16)
        LOOM_MIX(26) LOOM_MIX(32) LOOM_MIX(64) LOOM_MIX(192) LOOM_MIX(256) LOOM_MIX(640) LOOM_MIX(704)
#undef LOOM_MIX
      };
      const double cyc = avg_cycles(launch, d, h, sms);
      if (cyc <= 0) { printf("}, \"error\": \"mix probe failed\"}\n"); return 1; }
      printf("%s\"%s\": %.1f", i ? ", " : "", names[i], cyc / (iters * 4.0));
    }
    printf("}");
  }
  printf("}\n");
  return 0;
}
