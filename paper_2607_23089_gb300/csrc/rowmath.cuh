// rowmath.cuh -- per-chunk arithmetic shared by every kernel: the pieces of
// the row statistics and the normalisation, on one 16-byte chunk at a time,
// in packed fp32 pairs.  Elements of a chunk outside [lo, hi) are not part of
// the row (only the first and last chunk of a row can have such elements);
// they are replaced by the identity of the reduction before they are added,
// so a chunk contributes only its row's elements.
//
// Definitions (textbook / PyTorch convention; the paper names the operator
// family through its running-example kernels, §2.1, without formulas):
//   softmax      y = exp(x - M) / S,            M = max x, S = sum exp(x - M)
//   log-softmax  y = (x - M) - log S
//   LayerNorm    y = (x - mu) * rsqrt(var + eps) * gamma + beta  (biased var)
//   RMSNorm      y = x * rsqrt(mean(x^2) + eps) * gamma
#pragma once

#include "common.cuh"

namespace rowop {

// Valid element range [lo, hi) of window chunk c of a row with head offset h
// and end h + n = hn (both in elements from the window start).
__device__ __forceinline__ void chunk_valid_range(int64_t c, int64_t nc, int h, int64_t hn,
                                                  int E, int &lo, int &hi) {
  lo = (c == 0) ? h : 0;
  hi = (c == nc - 1) ? static_cast<int>(hn - c * E) : E;
}

__device__ __forceinline__ bool in_range(int e, int lo, int hi) { return e >= lo && e < hi; }

template <int NP>
__device__ __forceinline__ float chunk_max(const f2 (&p)[NP], float m, int lo, int hi) {
  if (lo == 0 && hi == 2 * NP) {
#pragma unroll
    for (int i = 0; i < NP; ++i) m = fmaxf(m, fmaxf(f2_lo(p[i]), f2_hi(p[i])));
  } else {
#pragma unroll
    for (int e = 0; e < 2 * NP; ++e)
      if (in_range(e, lo, hi)) m = fmaxf(m, pair_elem(p, e));
  }
  return m;
}

// acc += exp(x - m), element-wise in pairs
template <int NP>
__device__ __forceinline__ f2 chunk_sum_exp(const f2 (&p)[NP], f2 m2, f2 acc, int lo, int hi) {
  const bool full = (lo == 0 && hi == 2 * NP);
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    f2 e = f2_exp_shifted(p[i], f2_neg(m2));
    if (!full) e = f2_select(e, in_range(2 * i, lo, hi), in_range(2 * i + 1, lo, hi), 0.f);
    acc = f2_add(acc, e);
  }
  return acc;
}

// acc += x
template <int NP>
__device__ __forceinline__ f2 chunk_sum(const f2 (&p)[NP], f2 acc, int lo, int hi) {
  const bool full = (lo == 0 && hi == 2 * NP);
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    f2 v = p[i];
    if (!full) v = f2_select(v, in_range(2 * i, lo, hi), in_range(2 * i + 1, lo, hi), 0.f);
    acc = f2_add(acc, v);
  }
  return acc;
}

// acc += (x - mean)^2
template <int NP>
__device__ __forceinline__ f2 chunk_sum_sqdev(const f2 (&p)[NP], f2 mean2, f2 acc, int lo,
                                              int hi) {
  const bool full = (lo == 0 && hi == 2 * NP);
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    f2 d = f2_add(p[i], f2_neg(mean2));
    if (!full) d = f2_select(d, in_range(2 * i, lo, hi), in_range(2 * i + 1, lo, hi), 0.f);
    acc = f2_fma(d, d, acc);
  }
  return acc;
}

// acc += x^2
template <int NP>
__device__ __forceinline__ f2 chunk_sum_sq(const f2 (&p)[NP], f2 acc, int lo, int hi) {
  const bool full = (lo == 0 && hi == 2 * NP);
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    f2 v = p[i];
    if (!full) v = f2_select(v, in_range(2 * i, lo, hi), in_range(2 * i + 1, lo, hi), 0.f);
    acc = f2_fma(v, v, acc);
  }
  return acc;
}

// gamma/beta for window chunk c of a row with head offset h, as pairs:
// element e is column j = c*E + e - h; columns outside [0, glen) read `fill`.
template <typename T>
__device__ __forceinline__ void load_param_pairs(const T *__restrict__ g, int64_t glen, int64_t c,
                                                 int h, bool vec, float fill,
                                                 f2 (&out)[Elem<T>::kPerChunk / 2]) {
  constexpr int E = Elem<T>::kPerChunk;
  const int64_t j0 = c * E - h;
  if (vec && h == 0 && j0 + E <= glen) {
    chunk_to_pairs<T>(__ldg(reinterpret_cast<const uint4 *>(g + j0)), out);
    return;
  }
  if (vec && h > 0 && (c + 1) * E <= glen) {
    // columns before 0 (chunk 0 of the row) read as zero: they lie outside
    // the row and are never used
    const uint4 A = c >= 1 ? __ldg(reinterpret_cast<const uint4 *>(g + (c - 1) * E))
                           : make_uint4(0u, 0u, 0u, 0u);
    const uint4 B = __ldg(reinterpret_cast<const uint4 *>(g + c * E));
    chunk_to_pairs<T>(shift_chunk<T>(A, B, h), out);
    return;
  }
  float v[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int64_t j = j0 + e;
    v[e] = (j >= 0 && j < glen) ? load_elem(g + j) : fill;
  }
#pragma unroll
  for (int i = 0; i < E / 2; ++i) out[i] = f2_make(v[2 * i], v[2 * i + 1]);
}

// In place: x pairs -> y pairs.  (s0, s1) are (M, 1/S) for softmax,
// (M, log S) for log-softmax, (mu, rstd) for LayerNorm, (-, rstd) for RMSNorm;
// g / b are the gamma / beta pairs (read only by the norms).
template <int OP, int NP>
__device__ __forceinline__ void normalize_pairs(f2 (&p)[NP], float s0, float s1,
                                                const f2 (&g)[NP], const f2 (&b)[NP]) {
  const f2 na = f2_bcast(-s0);
  const f2 b2 = f2_bcast(s1);
  if constexpr (OP == kSoftmax) {
#pragma unroll
    for (int i = 0; i < NP; ++i) p[i] = f2_mul(f2_exp_shifted(p[i], na), b2);
  } else if constexpr (OP == kLogSoftmax) {
    const f2 nb = f2_bcast(-s1);
#pragma unroll
    for (int i = 0; i < NP; ++i) p[i] = f2_add(f2_add(p[i], na), nb);
  } else if constexpr (OP == kLayerNorm) {
#pragma unroll
    for (int i = 0; i < NP; ++i) p[i] = f2_fma(f2_mul(f2_add(p[i], na), b2), g[i], b[i]);
  } else {
#pragma unroll
    for (int i = 0; i < NP; ++i) p[i] = f2_mul(f2_mul(p[i], b2), g[i]);
  }
}

// chunk_normalize: normalize_pairs with gamma/beta of window chunk c read
// through the general (bounds-checked, any alignment) loader.
template <int OP, typename T>
__device__ __forceinline__ void chunk_normalize(f2 (&p)[Elem<T>::kPerChunk / 2], float s0,
                                                float s1, const T *gamma, int64_t glen_g,
                                                const T *beta, int64_t glen_b, int64_t c, int h,
                                                bool gvec) {
  constexpr int NP = Elem<T>::kPerChunk / 2;
  f2 g[NP], b[NP];
  if constexpr (OP == kLayerNorm || OP == kRmsNorm)
    load_param_pairs<T>(gamma, glen_g, c, h, gvec, 1.f, g);
  if constexpr (OP == kLayerNorm) load_param_pairs<T>(beta, glen_b, c, h, gvec, 0.f, b);
  normalize_pairs<OP, NP>(p, s0, s1, g, b);
}

// Writes the row's elements of chunk c: one 128-bit store when the chunk is
// entirely the row's and the output is 16-byte congruent to the input, else
// one store per element of the row.
template <typename T>
__device__ __forceinline__ void store_chunk(const f2 (&p)[Elem<T>::kPerChunk / 2], char *owin,
                                            T *out_row, int64_t c, int h, int lo, int hi,
                                            bool out_vec) {
  constexpr int E = Elem<T>::kPerChunk;
  if (lo == 0 && hi == E && out_vec) {
    stg_stream(owin + c * kChunkBytes, pairs_to_chunk<T>(p));
  } else {
#pragma unroll
    for (int e = 0; e < E; ++e)
      if (in_range(e, lo, hi)) out_row[c * E + e - h] = from_f32<T>(pair_elem(p, e));
  }
}

// Chunk image of window chunk c holding only the row's own elements (the
// others are zero), read element by element.
template <typename T>
__device__ __forceinline__ uint4 load_chunk_elems(const T *in_row, int64_t c, int h, int64_t n) {
  constexpr int E = Elem<T>::kPerChunk;
  uint32_t w[4] = {0u, 0u, 0u, 0u};
  const unsigned short *p16 = reinterpret_cast<const unsigned short *>(in_row);
  const uint32_t *p32 = reinterpret_cast<const uint32_t *>(in_row);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int64_t j = c * E + e - h;
    if (j >= 0 && j < n) {
      if (sizeof(T) == 2) {
        w[e >> 1] |= static_cast<uint32_t>(p16[j]) << ((e & 1) * 16);
      } else {
        w[e] = p32[j];
      }
    }
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

}  // namespace rowop
