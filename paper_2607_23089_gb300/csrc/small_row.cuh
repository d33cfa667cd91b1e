// small_row.cuh -- the SMALL bucket (small_row_kernel of §2.1): rows of at
// most 4 KiB handled by a group of G lanes (G = 1..32, a power of two;
// BLOCK_ROWS = 32/G rows per warp), read with 128-bit loads and reduced with
// __shfl_xor_sync butterflies.  Statistics are exact two-pass reductions over
// the row (max then sum of exponentials, or mean then squared deviations).
//
// The per-chunk arithmetic lives in rowmath.cuh; small_row_core() runs it on
// chunks handed out by a source functor, so the dense kernel (chunks in
// registers) and the fused ragged kernel (chunks staged in shared memory)
// execute the same operations in the same order.
#pragma once

#include "rowmath.cuh"

namespace rowop {

// Lanes per row for the SMALL bucket: enough lanes that each holds at most
// four chunks even when the row straddles one extra 16-byte chunk.  Depends
// on the row length only, so dense and ragged calls on the same row agree.
__host__ __device__ __forceinline__ int small_group_lanes(int64_t n, int esize) {
  const int64_t e = 16 / esize;
  const int64_t ncd = (n + e - 1) / e;
  const int64_t need = (ncd + 1 + 3) / 4;
  int g = 1;
  while (g < need && g < 32) g <<= 1;
  return g;
}

// Chunk-per-lane capacity the register kernel is compiled for (4, 8 or 9).
__host__ __device__ __forceinline__ int small_cpl_class(int64_t max_chunks, int g) {
  const int64_t need = (max_chunks + g - 1) / g;
  return need <= 4 ? 4 : (need <= 8 ? 8 : 9);
}

struct SmallRowArgs {
  const void *gamma;
  const void *beta;
  int64_t glen;  // length of gamma / beta
  float eps;
  int gvec;      // gamma/beta 16-byte aligned
  int out_vec;   // out is congruent to in modulo 16 bytes
};

// One SMALL row processed by the G-lane group containing this lane (`sub` is
// the lane's index in its group).  `get(k)` returns the 16 bytes of window
// chunk sub + k*G.  All 32 lanes of the warp must call this together (the
// butterflies use the full mask); groups never mix since every xor offset is
// below G.  Inactive groups pass nc = 0.  UNROLL = false keeps the chunk
// loops rolled (for chunk sources that can be indexed at run time); the
// operations and their order do not change.
// Online (one-pass) softmax statistics of a lane's chunks: a running maximum
// m and sum s of exp(x - m), rescaled when a chunk raises the maximum.
// Groups then merge their (m, s) pairs: M = max, S = s e^(m-M) + s' e^(m'-M).
__device__ __forceinline__ void online_merge(float &m, float &s, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    return;
  }
  const float M = fmaxf(m, m2);
  s = __fadd_rn(__fmul_rn(s, exp_shifted(m, M)), __fmul_rn(s2, exp_shifted(m2, M)));
  m = M;
}

template <int OP, typename T, int CPL, bool EXACT, bool UNROLL, bool ONLINE = false, class Get>
__device__ __forceinline__ void small_row_core(Get get, T *out_row, int64_t n, int h, int64_t nc,
                                               int G, int sub, const SmallRowArgs &a) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr int kUnroll = UNROLL ? CPL : 1;
  const int64_t hn = h + n;
  float s0 = 0.f, s1 = 0.f;

  // ---- statistics ----
  if constexpr ((OP == kSoftmax || OP == kLogSoftmax) && ONLINE) {
    float m = -INFINITY, sl = 0.f;
#pragma unroll(kUnroll)
    for (int k = 0; k < CPL; ++k) {
      const int64_t c = sub + static_cast<int64_t>(k) * G;
      if (c < nc) {
        f2 p[NP];
        chunk_to_pairs<T>(get(k), p);
        int lo = 0, hi = E;
        if (!EXACT) chunk_valid_range(c, nc, h, hn, E, lo, hi);
        const float cm = chunk_max<NP>(p, -INFINITY, lo, hi);
        if (cm > m) {  // the chunk raises the maximum: rescale what was summed
          sl = m == -INFINITY ? 0.f : __fmul_rn(sl, exp_shifted(m, cm));
          m = cm;
        }
        if (m != -INFINITY)
          sl = __fadd_rn(sl, f2_total(chunk_sum_exp<NP>(p, f2_bcast(m), f2_bcast(0.f), lo, hi)));
      }
    }
    for (int o = 1; o < G; o <<= 1) {
      const float m2 = __shfl_xor_sync(kFullMask, m, o);
      const float s2 = __shfl_xor_sync(kFullMask, sl, o);
      online_merge(m, sl, m2, s2);
    }
    s0 = m;
    s1 = (OP == kSoftmax) ? __frcp_rn(sl) : logf(sl);
  } else if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
    float m = -INFINITY;
#pragma unroll(kUnroll)
    for (int k = 0; k < CPL; ++k) {
      const int64_t c = sub + static_cast<int64_t>(k) * G;
      if (c < nc) {
        f2 p[NP];
        chunk_to_pairs<T>(get(k), p);
        int lo = 0, hi = E;
        if (!EXACT) chunk_valid_range(c, nc, h, hn, E, lo, hi);
        m = chunk_max<NP>(p, m, lo, hi);
      }
    }
    m = group_max(m, G);
    const f2 m2 = f2_bcast(m);
    f2 acc = f2_bcast(0.f);
#pragma unroll(kUnroll)
    for (int k = 0; k < CPL; ++k) {
      const int64_t c = sub + static_cast<int64_t>(k) * G;
      if (c < nc) {
        f2 p[NP];
        chunk_to_pairs<T>(get(k), p);
        int lo = 0, hi = E;
        if (!EXACT) chunk_valid_range(c, nc, h, hn, E, lo, hi);
        acc = chunk_sum_exp<NP>(p, m2, acc, lo, hi);
      }
    }
    const float s = group_sum(f2_total(acc), G);
    s0 = m;
    s1 = (OP == kSoftmax) ? __frcp_rn(s) : logf(s);
  } else if constexpr (OP == kLayerNorm) {
    f2 acc = f2_bcast(0.f);
#pragma unroll(kUnroll)
    for (int k = 0; k < CPL; ++k) {
      const int64_t c = sub + static_cast<int64_t>(k) * G;
      if (c < nc) {
        f2 p[NP];
        chunk_to_pairs<T>(get(k), p);
        int lo = 0, hi = E;
        if (!EXACT) chunk_valid_range(c, nc, h, hn, E, lo, hi);
        acc = chunk_sum<NP>(p, acc, lo, hi);
      }
    }
    const float mean = __fdiv_rn(group_sum(f2_total(acc), G), static_cast<float>(n));
    const f2 mean2 = f2_bcast(mean);
    acc = f2_bcast(0.f);
#pragma unroll(kUnroll)
    for (int k = 0; k < CPL; ++k) {
      const int64_t c = sub + static_cast<int64_t>(k) * G;
      if (c < nc) {
        f2 p[NP];
        chunk_to_pairs<T>(get(k), p);
        int lo = 0, hi = E;
        if (!EXACT) chunk_valid_range(c, nc, h, hn, E, lo, hi);
        acc = chunk_sum_sqdev<NP>(p, mean2, acc, lo, hi);
      }
    }
    const float q = group_sum(f2_total(acc), G);
    s0 = mean;
    s1 = __frsqrt_rn(__fadd_rn(__fdiv_rn(q, static_cast<float>(n)), a.eps));
  } else {
    f2 acc = f2_bcast(0.f);
#pragma unroll(kUnroll)
    for (int k = 0; k < CPL; ++k) {
      const int64_t c = sub + static_cast<int64_t>(k) * G;
      if (c < nc) {
        f2 p[NP];
        chunk_to_pairs<T>(get(k), p);
        int lo = 0, hi = E;
        if (!EXACT) chunk_valid_range(c, nc, h, hn, E, lo, hi);
        acc = chunk_sum_sq<NP>(p, acc, lo, hi);
      }
    }
    const float q = group_sum(f2_total(acc), G);
    s1 = __frsqrt_rn(__fadd_rn(__fdiv_rn(q, static_cast<float>(n)), a.eps));
  }

  // ---- normalise and store ----
  char *owin = reinterpret_cast<char *>(out_row) - static_cast<int64_t>(h) * Elem<T>::kSize;
#pragma unroll(kUnroll)
  for (int k = 0; k < CPL; ++k) {
    const int64_t c = sub + static_cast<int64_t>(k) * G;
    if (c < nc) {
      f2 p[NP];
      chunk_to_pairs<T>(get(k), p);
      int lo = 0, hi = E;
      if (!EXACT) chunk_valid_range(c, nc, h, hn, E, lo, hi);
      chunk_normalize<OP, T>(p, s0, s1, static_cast<const T *>(a.gamma),
                             a.gamma ? a.glen : 0, static_cast<const T *>(a.beta),
                             a.beta ? a.glen : 0, c, h, a.gvec != 0);
      store_chunk<T>(p, owin, out_row, c, h, lo, hi, a.out_vec != 0);
    }
  }
}

struct SmallParams {
  const void *in;
  void *out;
  int64_t rows;
  int64_t cols;
  int64_t ld;
  int G;
  SmallRowArgs a;
  // fused residual add: sum_out = in + resid (same layout), normalised after
  const void *resid;
  void *sum_out;
  int rvec;  // resid and sum_out 16-byte congruent to in
};

// Residual add for one window chunk c of a row: chunk x (the row's elements,
// zeros elsewhere) plus the same chunk of the residual, rounded to T, stored
// to sum_out and returned -- the norm reads the sum as stored.
template <typename T>
__device__ __forceinline__ uint4 residual_chunk(const uint4 &x, const T *r_row, T *s_row,
                                                const char *rwin, char *swin, int64_t c, int h,
                                                int lo, int hi, int64_t n, bool rvec) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  const bool full = lo == 0 && hi == E;
  const uint4 rr = (full && rvec) ? ldg_stream(rwin + c * kChunkBytes)
                                  : load_chunk_elems<T>(r_row, c, h, n);
  f2 a[NP], b[NP];
  chunk_to_pairs<T>(x, a);
  chunk_to_pairs<T>(rr, b);
#pragma unroll
  for (int i = 0; i < NP; ++i) a[i] = f2_add(a[i], b[i]);
  const uint4 sv = pairs_to_chunk<T>(a);
  if (full && rvec) {
    stg_stream(swin + c * kChunkBytes, sv);
  } else {
    chunk_to_pairs<T>(sv, a);  // the stored (rounded) values, element by element
    store_chunk<T>(a, swin, s_row, c, h, lo, hi, false);
  }
  return sv;
}

// Dense SMALL kernel: persistent grid; each warp takes BLOCK_ROWS = 32/G
// consecutive rows per step, every lane loads its chunks into registers first.
template <int OP, typename T, int CPL, bool EXACT, bool RESID = false, bool ONLINE = false>
__global__ void __launch_bounds__(kCtaThreads) small_row_kernel(const SmallParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  const int lane = threadIdx.x & 31;
  const int G = p.G;
  const int sub = lane & (G - 1);
  const int rows_per_warp = 32 / G;
  const int64_t warp_id = static_cast<int64_t>(blockIdx.x) * kCtaWarps + (threadIdx.x >> 5);
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kCtaWarps;
  const T *in = static_cast<const T *>(p.in);
  T *out = static_cast<T *>(p.out);
  for (int64_t base = warp_id * rows_per_warp; base < p.rows; base += nwarps * rows_per_warp) {
    const int64_t r = base + lane / G;
    const bool active = r < p.rows;
    const T *in_row = in + (active ? r : 0) * p.ld;
    T *out_row = out + (active ? r : 0) * p.ld;
    const uintptr_t ia = reinterpret_cast<uintptr_t>(in_row);
    const int h = EXACT ? 0 : static_cast<int>((ia & 15) / SZ);
    const int64_t nc = active ? (h + p.cols + E - 1) / E : 0;
    const char *win = reinterpret_cast<const char *>(ia - (ia & 15));
    uint4 raw[CPL];
#pragma unroll
    for (int k = 0; k < CPL; ++k) {
      const int64_t c = sub + static_cast<int64_t>(k) * G;
      raw[k] = make_uint4(0u, 0u, 0u, 0u);
      if (c < nc) {
        int lo = 0, hi = E;
        if (!EXACT) chunk_valid_range(c, nc, h, h + p.cols, E, lo, hi);
        raw[k] = (lo == 0 && hi == E) ? ldg_stream(win + c * kChunkBytes)
                                       : load_chunk_elems<T>(in_row, c, h, p.cols);
      }
    }
    if constexpr (RESID) {
      const T *r_row = static_cast<const T *>(p.resid) + (active ? r : 0) * p.ld;
      T *s_row = static_cast<T *>(p.sum_out) + (active ? r : 0) * p.ld;
      const char *rwin = reinterpret_cast<const char *>(r_row) - h * SZ;
      char *swin = reinterpret_cast<char *>(s_row) - h * SZ;
#pragma unroll
      for (int k = 0; k < CPL; ++k) {
        const int64_t c = sub + static_cast<int64_t>(k) * G;
        if (c < nc) {
          int lo = 0, hi = E;
          if (!EXACT) chunk_valid_range(c, nc, h, h + p.cols, E, lo, hi);
          raw[k] = residual_chunk<T>(raw[k], r_row, s_row, rwin, swin, c, h, lo, hi, p.cols,
                                     p.rvec != 0);
        }
      }
    }
    small_row_core<OP, T, CPL, EXACT, true, ONLINE>([&](int k) { return raw[k]; }, out_row, p.cols,
                                                    h, nc, G, sub, p.a);
  }
}

}  // namespace rowop
