// small_row.cuh -- the SMALL bucket (small_row_kernel of §2.1): rows of at
// most 4 KiB held in registers of a group of G lanes (G = 1..32, a power of
// two, BLOCK_ROWS = 32/G rows per warp), read with 128-bit loads and reduced
// with __shfl_xor_sync butterflies; every statistic is an exact two-pass
// reduction over the register-resident row.
#pragma once

#include "common.cuh"

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

// Chunk-per-lane capacity the kernel is compiled for (4, 8 or 9).
__host__ __device__ __forceinline__ int small_cpl_class(int64_t max_chunks, int g) {
  const int64_t need = (max_chunks + g - 1) / g;
  return need <= 4 ? 4 : (need <= 8 ? 8 : 9);
}

struct SmallRowArgs {
  const void *gamma;
  const void *beta;
  int64_t glen;   // length of gamma / beta
  float eps;
  int gvec;       // gamma/beta 16-byte aligned
  int out_vec;    // out is congruent to in modulo 16 bytes
};

// One row (or nothing when !active) processed by the G-lane group that
// contains this lane; `sub` is the lane's index inside its group.  All 32
// lanes of the warp must call this together (the butterflies use the full
// mask); the groups never mix because every xor offset is below G.
template <int OP, typename T, int CPL, bool EXACT>
__device__ __forceinline__ void small_row(const T *__restrict__ in_row, T *out_row, int64_t n,
                                          int G, int sub, bool active,
                                          const SmallRowArgs &a) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  const uintptr_t ia = reinterpret_cast<uintptr_t>(in_row);
  const int h = EXACT ? 0 : static_cast<int>((ia & 15) / SZ);
  const char *win = reinterpret_cast<const char *>(ia - (ia & 15));
  const int64_t nc = active ? (h + n + E - 1) / E : 0;
  const int64_t hn = h + n;

  float v[CPL][E];
  int lo[CPL], hi[CPL];
#pragma unroll
  for (int k = 0; k < CPL; ++k) {
    const int64_t c = sub + static_cast<int64_t>(k) * G;
    if (c < nc) {
      if (EXACT) {
        lo[k] = 0;
        hi[k] = E;
      } else {
        lo[k] = (c == 0) ? h : 0;
        hi[k] = (c == nc - 1) ? static_cast<int>(hn - c * E) : E;
      }
      if (lo[k] == 0 && hi[k] == E) {
        unpack(ldg_stream(win + c * kChunkBytes), v[k]);
      } else {
#pragma unroll
        for (int e = 0; e < E; ++e)
          v[k][e] = (e >= lo[k] && e < hi[k]) ? load_elem(in_row + (c * E + e - h)) : 0.f;
      }
    } else {
      lo[k] = 0;
      hi[k] = 0;
#pragma unroll
      for (int e = 0; e < E; ++e) v[k][e] = 0.f;
    }
  }
#define ROWOP_VALID(k, e) (EXACT ? (hi[k] != 0) : ((e) >= lo[k] && (e) < hi[k]))

  // ---- statistics -----------------------------------------------------------
  float s0 = 0.f, s1 = 0.f;  // op-specific row statistics
  if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
    float m = -INFINITY;
#pragma unroll
    for (int k = 0; k < CPL; ++k)
#pragma unroll
      for (int e = 0; e < E; ++e)
        if (ROWOP_VALID(k, e)) m = fmaxf(m, v[k][e]);
    m = group_max(m, G);
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < CPL; ++k)
#pragma unroll
      for (int e = 0; e < E; ++e)
        if (ROWOP_VALID(k, e)) {
          const float t = expf(__fsub_rn(v[k][e], m));
          s = __fadd_rn(s, t);
          if constexpr (OP == kSoftmax) v[k][e] = t;
        }
    s = group_sum(s, G);
    s0 = m;
    s1 = (OP == kSoftmax) ? __frcp_rn(s) : logf(s);
  } else if constexpr (OP == kLayerNorm) {
    float sum = 0.f;
#pragma unroll
    for (int k = 0; k < CPL; ++k)
#pragma unroll
      for (int e = 0; e < E; ++e)
        if (ROWOP_VALID(k, e)) sum = __fadd_rn(sum, v[k][e]);
    sum = group_sum(sum, G);
    const float mean = __fdiv_rn(sum, static_cast<float>(n));
    float q = 0.f;
#pragma unroll
    for (int k = 0; k < CPL; ++k)
#pragma unroll
      for (int e = 0; e < E; ++e)
        if (ROWOP_VALID(k, e)) {
          const float d = __fsub_rn(v[k][e], mean);
          q = __fmaf_rn(d, d, q);
        }
    q = group_sum(q, G);
    s0 = mean;
    s1 = __frsqrt_rn(__fadd_rn(__fdiv_rn(q, static_cast<float>(n)), a.eps));
  } else {  // RMSNorm
    float q = 0.f;
#pragma unroll
    for (int k = 0; k < CPL; ++k)
#pragma unroll
      for (int e = 0; e < E; ++e)
        if (ROWOP_VALID(k, e)) q = __fmaf_rn(v[k][e], v[k][e], q);
    q = group_sum(q, G);
    s1 = __frsqrt_rn(__fadd_rn(__fdiv_rn(q, static_cast<float>(n)), a.eps));
  }

  // ---- normalise and store -------------------------------------------------
  const uintptr_t oa = reinterpret_cast<uintptr_t>(out_row);
  char *owin = reinterpret_cast<char *>(oa - static_cast<uintptr_t>(h) * SZ);
#pragma unroll
  for (int k = 0; k < CPL; ++k) {
    const int64_t c = sub + static_cast<int64_t>(k) * G;
    if (hi[k] == 0) continue;
    float y[E];
    if constexpr (OP == kSoftmax) {
#pragma unroll
      for (int e = 0; e < E; ++e) y[e] = __fmul_rn(v[k][e], s1);
    } else if constexpr (OP == kLogSoftmax) {
#pragma unroll
      for (int e = 0; e < E; ++e) y[e] = __fsub_rn(__fsub_rn(v[k][e], s0), s1);
    } else if constexpr (OP == kLayerNorm) {
      float g[E], b[E];
      load_param_chunk<T>(static_cast<const T *>(a.gamma), a.gamma ? a.glen : 0, c, h,
                          a.gvec != 0, 1.f, g);
      load_param_chunk<T>(static_cast<const T *>(a.beta), a.beta ? a.glen : 0, c, h,
                          a.gvec != 0, 0.f, b);
#pragma unroll
      for (int e = 0; e < E; ++e)
        y[e] = __fmaf_rn(__fmul_rn(__fsub_rn(v[k][e], s0), s1), g[e], b[e]);
    } else {
      float g[E];
      load_param_chunk<T>(static_cast<const T *>(a.gamma), a.gamma ? a.glen : 0, c, h,
                          a.gvec != 0, 1.f, g);
#pragma unroll
      for (int e = 0; e < E; ++e) y[e] = __fmul_rn(__fmul_rn(v[k][e], s1), g[e]);
    }
    if (lo[k] == 0 && hi[k] == E && a.out_vec) {
      stg_stream(owin + c * kChunkBytes, pack(y));
    } else {
#pragma unroll
      for (int e = 0; e < E; ++e)
        if (e >= lo[k] && e < hi[k]) out_row[c * E + e - h] = from_f32<T>(y[e]);
    }
  }
#undef ROWOP_VALID
}

struct SmallParams {
  const void *in;
  void *out;
  int64_t rows;
  int64_t cols;
  int64_t ld;
  int G;
  SmallRowArgs a;
};

// Dense SMALL kernel: persistent grid, each warp takes BLOCK_ROWS = 32/G
// consecutive rows per step.
template <int OP, typename T, int CPL, bool EXACT>
__global__ void __launch_bounds__(kCtaThreads) small_row_kernel(const SmallParams p) {
  const int lane = threadIdx.x & 31;
  const int G = p.G;
  const int rows_per_warp = 32 / G;
  const int64_t warp_id = static_cast<int64_t>(blockIdx.x) * kCtaWarps + (threadIdx.x >> 5);
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kCtaWarps;
  const T *in = static_cast<const T *>(p.in);
  T *out = static_cast<T *>(p.out);
  for (int64_t base = warp_id * rows_per_warp; base < p.rows; base += nwarps * rows_per_warp) {
    const int64_t r = base + lane / G;
    const bool active = r < p.rows;
    const int64_t rr = active ? r : 0;
    small_row<OP, T, CPL, EXACT>(in + rr * p.ld, out + rr * p.ld, p.cols, G, lane & (G - 1),
                                 active, p.a);
  }
}

}  // namespace rowop
