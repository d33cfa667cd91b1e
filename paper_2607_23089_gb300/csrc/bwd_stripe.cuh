// bwd_stripe.cuh -- the LayerNorm / RMSNorm backward passes over ragged rows
// (the derivatives of §2.1's row-wise norms, as in bwd_row.cuh, on the ragged
// layout), by column stripes, for x, dy and dx congruent modulo 16 bytes.
//
// Two kernels, then bwd_param_finalize_kernel:
//   * bwd_stripe_stats_kernel: CTA (s, g) takes rows [64 g, 64 g + 64) and
//     their columns [s W1, (s+1) W1).  For each row it writes the sums over
//     those columns (LayerNorm: sum (x - k), sum (x - k)^2, sum t and
//     sum t (x - k), with t = dy gamma and k the row's first element;
//     RMSNorm: sum x^2 and sum t x): one float4 per row and stripe;
//   * bwd_stripe_dx_kernel: CTA (s, g) takes the rows of group g and their
//     columns [s W2, (s+1) W2).  It adds each row's stripe sums in stripe
//     order into the row statistics, writes dx over its columns, and sums
//     dy xhat (and dy) over its rows into group g's partial row;
//   * the finalize adds the groups' partial rows in index order.
// x and dy are read twice (10 bytes an element of a 16-bit type against the
// 6 of one pass).  In exchange no CTA holds a whole row, so rows of any
// length keep many loads in flight on every SM, and a lane's dgamma / dbeta
// sums sit in registers at fixed columns.
//
// Alignment.  Lane t of a CTA owns window chunks t, t + NT, ... of the
// stripe.  Window chunks are the 16-byte chunks counted from the boundary
// at or before the row's first element, so every whole-chunk load and store
// is aligned.  A row that starts h elements past a boundary (head class h)
// puts its column j at window position j + h.  Each CTA sorts its rows by
// head class (stably, by row index).  Per class it loads gamma at its
// lanes' columns once; the dx kernel also adds its lanes' sums into the
// CTA's partial row in shared memory when the class ends.  A chunk that
// crosses a row's end is read and written element by element.  A chunk
// that crosses a stripe edge is read whole when it lies inside the row and
// written element by element.
//
// LayerNorm's mean and variance come from the sums about k, the shifted-data
// formula: var = mean((x - k)^2) - mean(x - k)^2, whose cancellation grows
// only with (mean - k)^2 / var.  Nothing is atomic, and every sum has a
// fixed order given the offsets, so the result is bitwise reproducible.
#pragma once

#include "bwd_call.h"
#include "common.cuh"

namespace rowop {

struct StripeParams {
  const void *x;
  const void *dy;
  void *dx;
  const void *gamma;  // NULL = ones
  const int64_t *offsets;
  int64_t rows, max_len;
  float eps;
  int hb;        // element offset of x (dy, dx) past a 16-byte boundary
  float *shift;  // [rows] LayerNorm: each row's first element
  float4 *psum;  // [rows][ns1] the stats kernel's row sums per stripe
  float *part;   // [ng2][nacc][max_len] dgamma (dbeta) partial rows; NULL = not wanted
  int64_t ns1, ng1, ng2, g2;
  unsigned int *status;
};

// Rows of one batch, sorted by head class: seg[c] is where class c starts,
// seg[E] the number listed.
template <int N>
struct StripeRows {
  int64_t off[N];
  int len[N];
  int row[N];
  int seg[10];
  int wcnt[9][kDxThreads / 32];
};

// Rows [r0, r0 + n), one a thread (n <= NT): those that reach column `from`
// (valid, 0 <= length <= max_len, and longer than `from`) are listed in L by
// head class, then by row.  With `first` given, the thread of a listed row
// also stores the row's first element in first_out[position].  Returns
// whether the thread's row is invalid.
template <typename T, int NT, int N>
__device__ __forceinline__ bool stripe_sort(StripeRows<N> &L, const int64_t *offsets, int64_t r0,
                                            int n, int64_t from, int64_t max_len, int hb,
                                            const T *first, float *first_out) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NW = NT / 32;
  static_assert(N <= NT && NW <= kDxThreads / 32, "one row a thread");
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int w = tid >> 5;
  int key = E;
  int len = 0;
  int64_t o = 0;
  bool bad = false;
  float k = 0.f;
  if (tid < n) {
    o = offsets[r0 + tid];
    const int64_t l = offsets[r0 + tid + 1] - o;
    bad = l < 0 || l > max_len;
    if (!bad) {
      len = static_cast<int>(l);
      if (l > from) {
        key = static_cast<int>((o + hb) & (E - 1));
        if (first) k = load_elem(first + o);
      }
    }
  }
  unsigned mine = 0;
#pragma unroll
  for (int c = 0; c <= E; ++c) {
    const unsigned b = __ballot_sync(kFullMask, key == c);
    if (key == c) mine = b;
    if (lane == 0) L.wcnt[c][w] = __popc(b);
  }
  __syncthreads();
  if (tid == 0) {
    int acc = 0;
    for (int c = 0; c <= E; ++c) {
      L.seg[c] = acc;
      for (int q = 0; q < NW; ++q) acc += L.wcnt[c][q];
    }
  }
  __syncthreads();
  if (key < E) {
    int pos = L.seg[key] + __popc(mine & ((1u << lane) - 1u));
    for (int q = 0; q < w; ++q) pos += L.wcnt[key][q];
    L.off[pos] = o;
    L.len[pos] = len;
    L.row[pos] = static_cast<int>(r0 + tid);
    if (first) first_out[pos] = k;
  }
  __syncthreads();
  return bad;
}

// The 16-byte chunk of T at element `src`, raw: read whole when `whole`
// (the chunk lies inside the row), else only its elements [lo, hi), one by
// one (the others zero).
template <typename T>
__device__ __forceinline__ uint4 stripe_load(const T *src, bool whole, int lo, int hi) {
  constexpr int E = Elem<T>::kPerChunk;
  if (whole) return ldg_stream(src);
  uint32_t wd[4] = {0u, 0u, 0u, 0u};
#pragma unroll
  for (int e = 0; e < E; ++e) {
    if (e >= lo && e < hi) {
      if constexpr (sizeof(T) == 4) {
        wd[e] = *reinterpret_cast<const uint32_t *>(src + e);
      } else {
        const uint32_t b = *reinterpret_cast<const unsigned short *>(src + e);
        wd[e >> 1] |= (e & 1) ? (b << 16) : b;
      }
    }
  }
  return make_uint4(wd[0], wd[1], wd[2], wd[3]);
}

// A raw chunk as pairs, elements outside [lo, hi) replaced by `fill`.
template <typename T>
__device__ __forceinline__ void stripe_pairs(const uint4 &raw, int lo, int hi, float fill,
                                             f2 (&v)[Elem<T>::kPerChunk / 2]) {
  constexpr int E = Elem<T>::kPerChunk;
  chunk_to_pairs<T>(raw, v);
  if (lo > 0 || hi < E) {
#pragma unroll
    for (int i = 0; i < E / 2; ++i)
      v[i] = f2_select(v[i], 2 * i >= lo && 2 * i < hi, 2 * i + 1 >= lo && 2 * i + 1 < hi, fill);
  }
}

// gamma at the columns of a lane's M window chunks for head class h: chunk
// m is window chunk tid + NT m of the stripe at column `from`; columns
// outside [from, lim) read as 1 (their data is masked out).
template <typename T, int M, int NT>
__device__ __forceinline__ void stripe_gamma(f2 (&gam)[M][Elem<T>::kPerChunk / 2], const T *gamma,
                                             int64_t from, int64_t lim, int h, int tid) {
  constexpr int E = Elem<T>::kPerChunk;
#pragma unroll
  for (int m = 0; m < M; ++m) {
    float g[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const int64_t col = from + static_cast<int64_t>(E) * (tid + NT * m) + e - h;
      g[e] = (gamma && col >= from && col < lim) ? load_elem(gamma + col) : 1.f;
    }
#pragma unroll
    for (int i = 0; i < E / 2; ++i) gam[m][i] = f2_make(g[2 * i], g[2 * i + 1]);
  }
}

// Sum over a warp of NV values (a power of two up to 32) by recursive
// halving: each stage sends half of a lane's values to the partner lane and
// adds the other half; once one value is left, a butterfly.  Lane l returns
// the total of value (l >> (5 - log2 NV)), so lane i * 32 / NV holds value
// i.  The order of every sum is fixed.
template <int NV>
__device__ __forceinline__ float warp_reduce_scatter(float (&v)[NV], int lane) {
#pragma unroll
  for (int half = NV / 2, o = 16; half >= 1; half >>= 1, o >>= 1) {
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < half; ++i) {
      const float send = up ? v[i] : v[i + half];
      const float keep = up ? v[i + half] : v[i];
      v[i] = __fadd_rn(keep, __shfl_xor_sync(kFullMask, send, o));
    }
  }
  float t = v[0];
#pragma unroll
  for (int o = 16 / NV; o >= 1; o >>= 1) t = __fadd_rn(t, __shfl_xor_sync(kFullMask, t, o));
  return t;
}

// Position of the chunk a lane owns within one row: element index of the
// chunk, the column of its element 0, and its valid elements [lo, hi).
struct StripeChunk {
  int64_t elem;
  bool whole;
  int lo, hi;
};

template <int E>
__device__ __forceinline__ StripeChunk stripe_chunk(int64_t o, int len, int h, int64_t from,
                                                    int64_t width, int q) {
  StripeChunk c;
  const int64_t d0 = from + static_cast<int64_t>(E) * q - h;  // column of element 0
  c.elem = o + d0;
  c.lo = (q == 0) ? h : 0;
  const int64_t lim = min(from + width, static_cast<int64_t>(len));
  c.hi = static_cast<int>(max(static_cast<int64_t>(0), min(static_cast<int64_t>(E), lim - d0)));
  c.whole = d0 >= 0 && d0 + E <= len;
  return c;
}

// ---------------------------------------------------------------------------
// Row sums per stripe.  Every warp walks the CTA's sorted rows two at a time;
// a lane reads its two window chunks of x and dy of both rows before using
// them, then the warp's eight (LayerNorm) or four (RMSNorm) sums are reduced
// by recursive halving into shared memory; the warps are added in warp order
// at the end.
// ---------------------------------------------------------------------------
template <int OP, typename T>
__global__ void __launch_bounds__(kStatThreads, 3) bwd_stripe_stats_kernel(const StripeParams p) {
  static_assert(OP == kLayerNorm || OP == kRmsNorm, "norm backward passes");
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr int M = kStatChunks;
  constexpr int NT = kStatThreads;
  constexpr int NW = NT / 32;
  constexpr int64_t W = static_cast<int64_t>(E) * (NT * M - 1);
  constexpr bool kLN = OP == kLayerNorm;
  constexpr int NV = kLN ? 8 : 4;  // sums of two rows
  __shared__ StripeRows<kStatRows> L;
  __shared__ float kfirst[kStatRows];
  __shared__ float4 wsum[kStatRows][NW];
  // the dx kernel may be scheduled once every CTA of this one has started;
  // it waits for this grid's completion before it reads what this one writes
  asm volatile("griddepcontrol.launch_dependents;");
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int w = tid >> 5;
  const int64_t s = static_cast<int64_t>(blockIdx.x) / p.ng1;  // heavy stripes first
  const int64_t g = static_cast<int64_t>(blockIdx.x) % p.ng1;
  const int64_t r0 = g * kStatRows;
  const int n = static_cast<int>(min(static_cast<int64_t>(kStatRows), p.rows - r0));
  const int64_t from = s * W;
  const int64_t lim = min(from + W, p.max_len);
  const T *x = static_cast<const T *>(p.x);
  const T *dy = static_cast<const T *>(p.dy);
  const T *gamma = static_cast<const T *>(p.gamma);

  const bool bad = stripe_sort<T, NT>(L, p.offsets, r0, n, from, p.max_len, p.hb,
                                      kLN ? x : nullptr, kfirst);
  if (s == 0) {  // uniform over the CTA
    if (__syncthreads_or(bad) && tid == 0) atomicOr(p.status, kStatusBadOffsets);
    if (kLN && tid < L.seg[E]) p.shift[L.row[tid]] = kfirst[tid];
  }
  const int cnt = L.seg[E];
  for (int c = 0; c < E; ++c) {
    const int j0 = L.seg[c], j1 = L.seg[c + 1];
    if (j0 == j1) continue;
    f2 gam[M][NP];
    stripe_gamma<T, M, NT>(gam, gamma, from, lim, c, tid);
    for (int j = j0; j < j1; j += 2) {
      const bool two = j + 1 < j1;
      uint4 xr[2][M], dr[2][M];
      int lo[2][M], hi[2][M];
      float kk[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int jj = (u == 1 && !two) ? j : j + u;
        kk[u] = kLN ? kfirst[jj] : 0.f;
        const int64_t o = L.off[jj];
        const int len = (u == 1 && !two) ? 0 : L.len[jj];
#pragma unroll
        for (int m = 0; m < M; ++m) {
          const StripeChunk ch = stripe_chunk<E>(o, len, c, from, W, tid + NT * m);
          lo[u][m] = ch.lo;
          hi[u][m] = ch.hi;
          xr[u][m] = dr[u][m] = make_uint4(0u, 0u, 0u, 0u);
          if (ch.lo < ch.hi) {
            xr[u][m] = stripe_load<T>(x + ch.elem, ch.whole, ch.lo, ch.hi);
            dr[u][m] = stripe_load<T>(dy + ch.elem, ch.whole, ch.lo, ch.hi);
          }
        }
      }
      float v[NV];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const f2 nk = f2_bcast(-kk[u]);
        f2 s1 = f2_bcast(0.f), s2 = f2_bcast(0.f), s3 = f2_bcast(0.f), s4 = f2_bcast(0.f);
#pragma unroll
        for (int m = 0; m < M; ++m) {
          // elements outside the chunk's valid range read as k (x) and 0 (dy)
          f2 xv[NP], dv[NP];
          stripe_pairs<T>(xr[u][m], lo[u][m], hi[u][m], kk[u], xv);
          stripe_pairs<T>(dr[u][m], lo[u][m], hi[u][m], 0.f, dv);
#pragma unroll
          for (int i = 0; i < NP; ++i) {
            const f2 xs = kLN ? f2_add(xv[i], nk) : xv[i];
            const f2 t = f2_mul(dv[i], gam[m][i]);
            if constexpr (kLN) {
              s1 = f2_add(s1, xs);
              s3 = f2_add(s3, t);
            }
            s2 = f2_fma(xs, xs, s2);
            s4 = f2_fma(t, xs, s4);
          }
        }
        if constexpr (kLN) {
          v[4 * u + 0] = f2_total(s1);
          v[4 * u + 1] = f2_total(s2);
          v[4 * u + 2] = f2_total(s3);
          v[4 * u + 3] = f2_total(s4);
        } else {
          v[2 * u + 0] = f2_total(s2);
          v[2 * u + 1] = f2_total(s4);
        }
      }
      const float t = warp_reduce_scatter<NV>(v, lane);
      constexpr int kStride = 32 / NV;
      if ((lane & (kStride - 1)) == 0) {
        const int i = lane / kStride;  // value index
        const int u = kLN ? (i >> 2) : (i >> 1);
        const int comp = kLN ? (i & 3) : 1 + 2 * (i & 1);  // RMSNorm: .y, .w
        if (u == 0 || two) reinterpret_cast<float *>(&wsum[j + u][w])[comp] = t;
      }
    }
  }
  __syncthreads();
  for (int j = tid; j < cnt; j += NT) {
    float4 t = wsum[j][0];
#pragma unroll
    for (int q = 1; q < NW; ++q) {
      const float4 u = wsum[j][q];
      t.y = __fadd_rn(t.y, u.y);
      t.w = __fadd_rn(t.w, u.w);
      if constexpr (kLN) {
        t.x = __fadd_rn(t.x, u.x);
        t.z = __fadd_rn(t.z, u.z);
      }
    }
    if constexpr (!kLN) t.x = t.z = 0.f;
    p.psum[static_cast<int64_t>(L.row[j]) * p.ns1 + s] = t;
  }
}

// Index of column `local` of a stripe in the padded shared partial row: one
// word of padding every 32, so that lanes E columns apart hit distinct banks.
__device__ __forceinline__ int stripe_pad(int local) { return local + (local >> 5); }

// ---------------------------------------------------------------------------
// dx and the column sums.  Per batch of up to 256 rows of the group: sort,
// then each listed row's statistics from the stats kernel's stripe sums (in
// stripe order), then per head class the rows four at a time: a lane reads
// its window chunk of x and dy of the four rows, then writes its dx chunks
// and adds dy xhat (and dy) to its register sums; at the class's end the
// lane adds those sums into the CTA's partial row in shared memory.  The
// CTA writes its partial row (its stripe of group g's row) at the end.
// ---------------------------------------------------------------------------
template <int OP, typename T>
__global__ void __launch_bounds__(kDxThreads, 3) bwd_stripe_dx_kernel(const StripeParams p) {
  static_assert(OP == kLayerNorm || OP == kRmsNorm, "norm backward passes");
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr int NT = kDxThreads;
  constexpr int64_t W = static_cast<int64_t>(E) * (NT - 1);
  constexpr int64_t W1 = static_cast<int64_t>(E) * (kStatThreads * kStatChunks - 1);
  constexpr bool kLN = OP == kLayerNorm;
  constexpr int NA = kLN ? 2 : 1;
  constexpr int kPadW = static_cast<int>(W + W / 32 + 1);
  constexpr int U = 3;
  __shared__ StripeRows<kDxBatch> L;
  __shared__ float4 coef[kDxBatch];
  __shared__ float spart[NA][kPadW];
  const int tid = threadIdx.x;
  const int64_t s = static_cast<int64_t>(blockIdx.x) / p.ng2;  // heavy stripes first
  const int64_t g = static_cast<int64_t>(blockIdx.x) % p.ng2;
  const int64_t from = s * W;
  const int64_t lim = min(from + W, p.max_len);
  const T *x = static_cast<const T *>(p.x);
  const T *dy = static_cast<const T *>(p.dy);
  T *dx = static_cast<T *>(p.dx);
  const T *gamma = static_cast<const T *>(p.gamma);
  const bool want = p.part != nullptr;
  for (int i = tid; i < NA * kPadW; i += NT) (&spart[0][0])[i] = 0.f;

  f2 accg[NP], accb[NP];
#pragma unroll
  for (int i = 0; i < NP; ++i) accg[i] = accb[i] = f2_bcast(0.f);
  const int64_t gr0 = g * p.g2;
  const int64_t gr1 = min(gr0 + p.g2, p.rows);
  bool waited = false;
  for (int64_t r0 = gr0; r0 < gr1; r0 += kDxBatch) {
    const int n = static_cast<int>(min(static_cast<int64_t>(kDxBatch), gr1 - r0));
    (void)stripe_sort<T, NT>(L, p.offsets, r0, n, from, p.max_len, p.hb,
                             static_cast<const T *>(nullptr), nullptr);
    if (!waited) {
      // launched as a programmatic dependent of the stats kernel: its sums
      // are read, and dx (which may be x or dy) written, only past this
      asm volatile("griddepcontrol.wait;" ::: "memory");
      waited = true;
    }
    const int cnt = L.seg[E];
    if (tid < cnt) {
      const int64_t r = L.row[tid];
      const int len = L.len[tid];
      const int nst = static_cast<int>((len + W1 - 1) / W1);
      const float4 *ps = p.psum + r * p.ns1;
      float4 t = ps[0];
#pragma unroll 4
      for (int q = 1; q < nst; ++q) {
        const float4 u = ps[q];
        t.x = __fadd_rn(t.x, u.x);
        t.y = __fadd_rn(t.y, u.y);
        t.z = __fadd_rn(t.z, u.z);
        t.w = __fadd_rn(t.w, u.w);
      }
      const float inv_n = __frcp_rn(static_cast<float>(len));
      float4 cf;
      if constexpr (kLN) {
        const float m1 = __fmul_rn(t.x, inv_n);  // mean - k
        const float var = fmaxf(__fsub_rn(__fmul_rn(t.y, inv_n), __fmul_rn(m1, m1)), 0.f);
        const float c0 = rsqrtf(__fadd_rn(var, p.eps));        // rstd
        const float mu = __fadd_rn(p.shift[r], m1);            // mean
        const float a = __fmul_rn(t.z, inv_n);                 // mean(t)
        const float b = __fmul_rn(c0, __fsub_rn(__fmul_rn(t.w, inv_n), __fmul_rn(m1, a)));
        cf = make_float4(c0, -__fmul_rn(mu, c0), -__fmul_rn(a, c0), -__fmul_rn(b, c0));
      } else {
        const float c0 = rsqrtf(__fmaf_rn(t.y, inv_n, p.eps));  // rstd
        const float b = __fmul_rn(__fmul_rn(t.w, c0), inv_n);   // mean(t xhat)
        cf = make_float4(c0, 0.f, 0.f, -__fmul_rn(b, c0));
      }
      coef[tid] = cf;
    }
    __syncthreads();
    for (int c = 0; c < E; ++c) {
      const int j0 = L.seg[c], j1 = L.seg[c + 1];
      if (j0 == j1) continue;
      f2 gam[1][NP];
      stripe_gamma<T, 1, NT>(gam, gamma, from, lim, c, tid);
      for (int j = j0; j < j1; j += U) {
        uint4 xr[U], dr[U];
        StripeChunk ch[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const bool on = j + u < j1;
          const int jj = on ? j + u : j;
          ch[u] = stripe_chunk<E>(L.off[jj], on ? L.len[jj] : 0, c, from, W, tid);
          xr[u] = dr[u] = make_uint4(0u, 0u, 0u, 0u);
          if (ch[u].lo < ch[u].hi) {
            xr[u] = stripe_load<T>(x + ch[u].elem, ch[u].whole, ch[u].lo, ch[u].hi);
            dr[u] = stripe_load<T>(dy + ch[u].elem, ch[u].whole, ch[u].lo, ch[u].hi);
          }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
          if (ch[u].lo >= ch[u].hi) continue;
          const float4 cf = coef[j + u];
          const f2 C0 = f2_bcast(cf.x), C1 = f2_bcast(cf.y), NA_ = f2_bcast(cf.z),
                   NB = f2_bcast(cf.w);
          // elements outside the chunk's valid range read as 0: no dy, so
          // they add nothing to the column sums
          f2 xv[NP], dv[NP], o[NP];
          stripe_pairs<T>(xr[u], ch[u].lo, ch[u].hi, 0.f, xv);
          stripe_pairs<T>(dr[u], ch[u].lo, ch[u].hi, 0.f, dv);
#pragma unroll
          for (int i = 0; i < NP; ++i) {
            const f2 xh = f2_fma(xv[i], C0, C1);
            const f2 t = f2_mul(dv[i], gam[0][i]);
            o[i] = f2_fma(t, C0, f2_fma(xh, NB, NA_));
            if (want) {
              accg[i] = f2_fma(dv[i], xh, accg[i]);
              if constexpr (kLN) accb[i] = f2_add(accb[i], dv[i]);
            }
          }
          if (ch[u].lo == 0 && ch[u].hi == E) {
            stg_stream(dx + ch[u].elem, pairs_to_chunk<T>(o));
          } else {
#pragma unroll
            for (int e = 0; e < E; ++e)
              if (e >= ch[u].lo && e < ch[u].hi) dx[ch[u].elem + e] = from_f32<T>(pair_elem(o, e));
          }
        }
      }
      if (want) {  // the class's sums into the partial row, at their columns
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const int local = E * tid + e - c;
          if (local >= 0 && local < W) {
            const int q = stripe_pad(local);
            spart[0][q] = __fadd_rn(spart[0][q], pair_elem(accg, e));
            if constexpr (kLN) spart[NA - 1][q] = __fadd_rn(spart[NA - 1][q], pair_elem(accb, e));
          }
        }
#pragma unroll
        for (int i = 0; i < NP; ++i) accg[i] = accb[i] = f2_bcast(0.f);
      }
      __syncthreads();
    }
  }
  if (!waited) asm volatile("griddepcontrol.wait;" ::: "memory");
  if (!want) return;
  __syncthreads();
  const int64_t ncols = lim - from;
  for (int a = 0; a < NA; ++a) {
    float *prow = p.part + (g * NA + a) * p.max_len + from;
    for (int i = tid; i < ncols; i += NT) prow[i] = spart[a][stripe_pad(i)];
  }
}

}  // namespace rowop
