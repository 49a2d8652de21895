// Plain fp64 CPU oracle for scaled-dot-product attention and its Flash Decode form.
//
// TEST INFRASTRUCTURE ONLY.  Nothing on the product path links, loads or calls this
// file; only the tests, the smoke check and the CPU-baseline leg of the benchmark do.
// It shares no code, header or constant with the CUDA library.
//
// What it computes (the paper never prints the formula; the evaluation describes Flash
// Attention as the fusion of the two matrix products with the softmax between them (Sec. 3.2.2) and
// Flash Decode as a local softmax loop followed by gathering partial results, a global
// softmax and a final scaling (Sec. 2.6, Flash Decode example; Sec. 3.2.3)):
//
//   s_ij  = scale * sum_d q_id k_jd             for every key j visible to query i
//   m_i   = max_j s_ij
//   l_i   = sum_j exp(s_ij - m_i)
//   O_i   = sum_j exp(s_ij - m_i) v_j / l_i
//   LSE_i = m_i + ln l_i                         (natural log of sum_j exp(s_ij))
//
// Conventions (readings where the paper is silent):
//   * layouts are contiguous row-major Q/O [B, Hq, Sq, D], K/V [B, Hkv, Skv, D],
//     inputs are bfloat16 bit patterns widened exactly to double;
//   * grouped-query attention: query head h reads kv head h / (Hq / Hkv);
//   * the valid key length of batch b is seqlens_k[b] (all Skv when null);
//   * causal masking is bottom-right aligned: query i sees key j iff
//     j <= i + (len_b - Sq);
//   * a query that sees no key gets O = 0 and LSE = -inf.
//
// Entry points (extern "C", used through ctypes):
//   oracle_attention           the definition above, on all rows or a list of rows
//   oracle_decode_split_merge  Flash Decode: per-chunk partial (O_i, lse_i), then the
//                              log-sum-exp merge (global softmax + final scaling)
//   oracle_attention_naive     a second, deliberately naive formula in long double
//                              (no max subtraction), for brute-force pins on tiny inputs
#include <cmath>
#include <cstdint>
#include <cstring>
#include <limits>
#include <thread>
#include <vector>

namespace {

inline double bf16_to_double(uint16_t bits) {
  uint32_t u = static_cast<uint32_t>(bits) << 16;
  float f;
  std::memcpy(&f, &u, sizeof f);
  return static_cast<double>(f);
}

struct Problem {
  const uint16_t* q;
  const uint16_t* k;
  const uint16_t* v;
  int B, Hq, Hkv, Sq, Skv, D;
  int causal;
  double scale;
  const int32_t* seqlens_k;
};

// Number of visible keys of query row i in batch b: the visible set is always the
// prefix [0, n) of the key sequence.
int64_t visible_keys(const Problem& p, int b, int i) {
  int64_t len = p.seqlens_k ? p.seqlens_k[b] : p.Skv;
  if (len < 0) len = 0;
  if (len > p.Skv) len = p.Skv;
  if (!p.causal) return len;
  int64_t last = static_cast<int64_t>(i) + (len - p.Sq);  // largest visible key index
  int64_t n = last + 1;
  if (n < 0) n = 0;
  if (n > len) n = len;
  return n;
}

const uint16_t* q_row(const Problem& p, int b, int h, int i) {
  return p.q + ((static_cast<int64_t>(b) * p.Hq + h) * p.Sq + i) * p.D;
}
const uint16_t* kv_row(const Problem& p, const uint16_t* base, int b, int hk, int64_t j) {
  return base + ((static_cast<int64_t>(b) * p.Hkv + hk) * p.Skv + j) * p.D;
}

// Attention of one query row over keys [j0, j1): writes O (D doubles) and returns LSE.
// Empty range -> O = 0, LSE = -inf.
double attend_range(const Problem& p, int b, int h, int i, int64_t j0, int64_t j1,
                    double* o, std::vector<double>& s, std::vector<double>& qd) {
  const int D = p.D;
  const int hk = h / (p.Hq / p.Hkv);
  for (int d = 0; d < D; ++d) o[d] = 0.0;
  if (j1 <= j0) return -std::numeric_limits<double>::infinity();
  const uint16_t* qr = q_row(p, b, h, i);
  for (int d = 0; d < D; ++d) qd[d] = bf16_to_double(qr[d]);
  const int64_t n = j1 - j0;
  s.resize(static_cast<size_t>(n));
  double m = -std::numeric_limits<double>::infinity();
  for (int64_t j = j0; j < j1; ++j) {
    const uint16_t* kr = kv_row(p, p.k, b, hk, j);
    double dot = 0.0;
    for (int d = 0; d < D; ++d) dot += qd[d] * bf16_to_double(kr[d]);
    const double sj = p.scale * dot;
    s[static_cast<size_t>(j - j0)] = sj;
    if (sj > m) m = sj;
  }
  double l = 0.0;
  for (int64_t j = j0; j < j1; ++j) {
    const double w = std::exp(s[static_cast<size_t>(j - j0)] - m);
    l += w;
    const uint16_t* vr = kv_row(p, p.v, b, hk, j);
    for (int d = 0; d < D; ++d) o[d] += w * bf16_to_double(vr[d]);
  }
  for (int d = 0; d < D; ++d) o[d] /= l;
  return m + std::log(l);
}

bool valid(const Problem& p) {
  return p.q && p.k && p.v && p.B >= 0 && p.Hq > 0 && p.Hkv > 0 && p.Hq % p.Hkv == 0 &&
         p.Sq >= 0 && p.Skv >= 0 && p.D > 0;
}

template <class F>
void parallel_for(int64_t n, int nthreads, F&& f) {
  if (nthreads <= 0) nthreads = static_cast<int>(std::thread::hardware_concurrency());
  if (nthreads <= 0) nthreads = 1;
  if (nthreads > n) nthreads = static_cast<int>(n > 0 ? n : 1);
  if (nthreads == 1) {
    for (int64_t r = 0; r < n; ++r) f(r);
    return;
  }
  std::vector<std::thread> pool;
  pool.reserve(static_cast<size_t>(nthreads));
  for (int t = 0; t < nthreads; ++t) {
    pool.emplace_back([&, t] {
      // static round-robin over rows: neighbouring rows have similar cost
      for (int64_t r = t; r < n; r += nthreads) f(r);
    });
  }
  for (auto& th : pool) th.join();
}

}  // namespace

extern "C" {

// Attention by definition.  rows == nullptr computes every row (b, h, i) in that
// order; otherwise rows[r] is the flat row index (b * Hq + h) * Sq + i.  o receives
// nrows x D doubles, lse nrows doubles.  Returns 0 on success, -1 on bad arguments.
int oracle_attention(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int Hq,
                     int Hkv, int Sq, int Skv, int D, int causal, double scale,
                     const int32_t* seqlens_k, const int64_t* rows, int64_t nrows, double* o,
                     double* lse, int nthreads) {
  Problem p{q, k, v, B, Hq, Hkv, Sq, Skv, D, causal, scale, seqlens_k};
  if (!valid(p) || !o || !lse) return -1;
  const int64_t total = static_cast<int64_t>(B) * Hq * Sq;
  if (!rows) nrows = total;
  for (int64_t r = 0; rows && r < nrows; ++r)
    if (rows[r] < 0 || rows[r] >= total) return -1;
  parallel_for(nrows, nthreads, [&](int64_t r) {
    thread_local std::vector<double> s, qd;
    qd.resize(static_cast<size_t>(D));
    const int64_t flat = rows ? rows[r] : r;
    const int i = static_cast<int>(flat % Sq);
    const int h = static_cast<int>((flat / Sq) % Hq);
    const int b = static_cast<int>(flat / (static_cast<int64_t>(Sq) * Hq));
    const int64_t n = visible_keys(p, b, i);
    lse[r] = attend_range(p, b, h, i, 0, n, o + r * D, s, qd);
  });
  return 0;
}

// Split boundaries used by the Flash Decode form: the chunk length of a sequence of
// len keys cut into num_splits pieces is ceil(len / num_splits) rounded up to a
// multiple of chunk_align; split i covers [i*C, min((i+1)*C, len)) and may be empty.
int64_t oracle_decode_chunk(int64_t len, int num_splits, int chunk_align) {
  if (len <= 0 || num_splits <= 0) return 0;
  int64_t c = (len + num_splits - 1) / num_splits;
  if (chunk_align > 1) c = (c + chunk_align - 1) / chunk_align * chunk_align;
  return c;
}

// Flash Decode (Sq = 1): for every (b, h) and split i, the local softmax over the
// split's keys gives a normalised partial O_i and lse_i; the gather step then takes
// L = max_i lse_i, w_i = exp(lse_i - L), O = sum_i w_i O_i / sum_i w_i and
// lse = L + ln sum_i w_i.  All splits empty -> O = 0, lse = -inf.
// o_part [B, Hq, num_splits, D] and lse_part [B, Hq, num_splits] may be null.
int oracle_decode_split_merge(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B,
                              int Hq, int Hkv, int Skv, int D, double scale,
                              const int32_t* seqlens_k, int num_splits, int chunk_align,
                              double* o_part, double* lse_part, double* o, double* lse,
                              int nthreads) {
  Problem p{q, k, v, B, Hq, Hkv, 1, Skv, D, 0, scale, seqlens_k};
  if (!valid(p) || num_splits <= 0 || !o || !lse) return -1;
  const int64_t nbh = static_cast<int64_t>(B) * Hq;
  parallel_for(nbh, nthreads, [&](int64_t bh) {
    thread_local std::vector<double> s, qd, part, plse;
    qd.resize(static_cast<size_t>(D));
    part.assign(static_cast<size_t>(num_splits) * D, 0.0);
    plse.assign(static_cast<size_t>(num_splits), 0.0);
    const int b = static_cast<int>(bh / Hq), h = static_cast<int>(bh % Hq);
    const int64_t len = visible_keys(p, b, 0);
    const int64_t c = oracle_decode_chunk(len, num_splits, chunk_align);
    // local softmax loop, one partial per split
    for (int i = 0; i < num_splits; ++i) {
      int64_t j0 = i * c, j1 = (i + 1) * c;
      if (j0 > len) j0 = len;
      if (j1 > len) j1 = len;
      plse[i] = attend_range(p, b, h, 0, j0, j1, &part[static_cast<size_t>(i) * D], s, qd);
    }
    // gather partial results, global softmax, final scaling
    double L = -std::numeric_limits<double>::infinity();
    for (int i = 0; i < num_splits; ++i)
      if (plse[i] > L) L = plse[i];
    double* out = o + bh * D;
    for (int d = 0; d < D; ++d) out[d] = 0.0;
    if (std::isinf(L) && L < 0) {
      lse[bh] = L;
    } else {
      double wsum = 0.0;
      for (int i = 0; i < num_splits; ++i) {
        const double w = std::exp(plse[i] - L);  // exp(-inf) = 0 for empty splits
        wsum += w;
        for (int d = 0; d < D; ++d) out[d] += w * part[static_cast<size_t>(i) * D + d];
      }
      for (int d = 0; d < D; ++d) out[d] /= wsum;
      lse[bh] = L + std::log(wsum);
    }
    if (o_part)
      std::memcpy(o_part + bh * num_splits * D, part.data(), sizeof(double) * num_splits * D);
    if (lse_part) std::memcpy(lse_part + bh * num_splits, plse.data(), sizeof(double) * num_splits);
  });
  return 0;
}

// Naive second formula for brute force on tiny inputs: long double, weights exp(s_ij)
// without subtracting the row maximum, keys visited from last to first.  Only valid
// when every |s_ij| is small enough that exp does not overflow.
int oracle_attention_naive(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B,
                           int Hq, int Hkv, int Sq, int Skv, int D, int causal, double scale,
                           double* o, double* lse) {
  Problem p{q, k, v, B, Hq, Hkv, Sq, Skv, D, causal, scale, nullptr};
  if (!valid(p) || !o || !lse) return -1;
  const int G = Hq / Hkv;
  for (int b = 0; b < B; ++b)
    for (int h = 0; h < Hq; ++h)
      for (int i = 0; i < Sq; ++i) {
        const int64_t r = (static_cast<int64_t>(b) * Hq + h) * Sq + i;
        std::vector<long double> acc(static_cast<size_t>(D), 0.0L);
        long double den = 0.0L;
        for (int j = Skv - 1; j >= 0; --j) {
          if (causal && j > i + (Skv - Sq)) continue;
          long double dot = 0.0L;
          for (int d = D - 1; d >= 0; --d)
            dot += static_cast<long double>(bf16_to_double(q[r * D + d])) *
                   bf16_to_double(k[((static_cast<int64_t>(b) * Hkv + h / G) * Skv + j) * D + d]);
          const long double w = std::exp(static_cast<long double>(scale) * dot);
          den += w;
          for (int d = 0; d < D; ++d)
            acc[d] += w * bf16_to_double(v[((static_cast<int64_t>(b) * Hkv + h / G) * Skv + j) * D + d]);
        }
        for (int d = 0; d < D; ++d)
          o[r * D + d] = den > 0 ? static_cast<double>(acc[d] / den) : 0.0;
        lse[r] = den > 0 ? static_cast<double>(std::log(den))
                         : -std::numeric_limits<double>::infinity();
      }
  return 0;
}

}  // extern "C"
