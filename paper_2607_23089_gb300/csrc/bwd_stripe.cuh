// bwd_stripe.cuh -- the LayerNorm / RMSNorm backward passes over ragged rows
// (the derivatives of §2.1's row-wise norms, as in bwd_row.cuh, on the ragged
// layout), by column stripes, for x, dy and dx congruent modulo 16 bytes.
//
// Two kernels, then bwd_stripe_finalize_kernel:
//   * bwd_stripe_stats_kernel: CTA (s, g) takes rows [64 g, 64 g + 64) and
//     their window chunks [512 s, 512 s + 512).  For each row it writes the
//     statistics
//     of those columns (LayerNorm: mean, sum of squares about it, sum t and
//     sum t (x - mean), with t = dy gamma; RMSNorm: sum x^2 and sum t x): one
//     float4 per row and stripe;
//   * bwd_stripe_dx_kernel: CTA (s, g) takes the rows of group g and their
//     window chunks [256 s, 256 s + 256).  It merges each row's stripe
//     statistics in
//     stripe order into the row's, writes dx over its columns, and sums
//     dy xhat (and dy) over its rows into group g's partial row;
//   * the finalize adds the groups' partial rows in index order.
// x and dy are read twice (10 bytes an element of a 16-bit type against the
// 6 of one pass).  In exchange no CTA holds a whole row, so rows of any
// length keep many loads in flight on every SM, and a lane's dgamma / dbeta
// sums sit in registers at fixed columns.
//
// Alignment.  Window chunks are the 16-byte chunks counted from the
// boundary at or before the row's first element, so every whole-chunk load
// and store is aligned; a row that starts h elements past a boundary (head
// class h) puts its column j at window position j + h.  Stripes are ranges
// of window chunks, so no chunk crosses a stripe edge and a stripe's columns
// move with the head class.  Lane t of a CTA owns window chunks t, t + NT,
// ... of its stripe.  Each CTA sorts its rows by head class (stably, by row
// index).  Per class it loads gamma at its lanes' columns once; the dx
// kernel also adds its lanes' sums into the CTA's partial row (its stripe's
// columns under every head class: E columns of halo before the stripe) in
// shared memory when the class ends.  Only a row's first and last chunks can
// be partial: those are read and written element by element.
//
// LayerNorm's statistics are formed about local means: each warp takes the
// mean of its elements of a row, then the sums about that mean from the same
// registers, and the warps' and then the stripes' statistics are merged
// pairwise (count, mean, M2, sum t, sum t (x - mean)), so no cancellation
// grows with the distance of the values from zero or from one another.
// Nothing is atomic, and every sum and merge has a fixed order given the
// offsets, so the result is bitwise reproducible.
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
  float4 *psum;  // [rows][ns1] the stats kernel's row statistics per stripe
  float *part;   // [ng2][ns2][nacc][W2 + E] dgamma (dbeta) partial rows; NULL = not wanted
  int64_t ns1, ng1;      // stats kernel: stripes, groups of kStatRows rows
  int64_t ns2, ng2, g2;  // dx kernel: stripes, groups, rows a group
  unsigned int *status;
};

// Rows of one batch, sorted by head class: seg[c] is where class c starts,
// seg[E] the number listed.
template <int N>
struct StripeRows {
  int64_t off[N];
  int len[N];
  int row[N];
  int cls[N];
  int seg[10];
  int wcnt[9][kDxThreads / 32];
};

// Rows [r0, r0 + n), one a thread (n <= NT): those that reach window
// position `from` (valid, 0 < length <= max_len, and head class + length >
// from) are listed in L by head class, then by row.  Returns whether the
// thread's row is invalid.
template <typename T, int NT, int N>
__device__ __forceinline__ bool stripe_sort(StripeRows<N> &L, const int64_t *offsets, int64_t r0,
                                            int n, int64_t from, int64_t max_len, int hb) {
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
  if (tid < n) {
    o = offsets[r0 + tid];
    const int64_t l = offsets[r0 + tid + 1] - o;
    bad = l < 0 || l > max_len;
    if (!bad) {
      len = static_cast<int>(l);
      const int c = static_cast<int>((o + hb) & (E - 1));
      if (l > 0 && l + c > from) key = c;
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
    L.cls[pos] = key;
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

// Asynchronous 16-byte copy global -> shared through L2 (cp.async, a lane's
// own copy): only the first `bytes` (0..16) bytes are read, the rest of the
// 16 bytes written as zero.  Groups commit in order; wait_group N returns
// once at most N of the lane's latest groups are pending.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, uint32_t bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr));
  return v;
}

// gamma at the columns of a lane's M window chunks for head class h: the
// lane's chunk m starts at column dc[m] (window position p: p - h);
// columns outside [from, lim) read as 1 (their data is masked out).
template <typename T, int M>
__device__ __forceinline__ void stripe_gamma(f2 (&gam)[M][Elem<T>::kPerChunk / 2], const T *gamma,
                                             int from, int lim, const int (&dc)[M]) {
  constexpr int E = Elem<T>::kPerChunk;
#pragma unroll
  for (int m = 0; m < M; ++m) {
    float g[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const int col = dc[m] + e;
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

// Row statistics of a set of a row's elements, about their own mean:
// count n, mean m, M2 = sum (x - m)^2, St = sum t and Stx = sum t (x - m)
// (t = dy gamma).  stat_merge folds b into a (Chan, Golub and LeVeque's
// pairwise update, with sum t (x - m) carried to the merged mean); the
// order of merges is fixed by the caller.
struct RowStat {
  float n, m, M2, St, Stx;
};
__device__ __forceinline__ void stat_merge(RowStat &a, const RowStat &b) {
  if (b.n == 0.f) return;
  if (a.n == 0.f) {
    a = b;
    return;
  }
  const float nn = __fadd_rn(a.n, b.n);
  const float d = __fsub_rn(b.m, a.m);
  const float fb = __fdividef(b.n, nn);  // the share of b
  const float fa = __fdividef(a.n, nn);
  a.M2 = __fadd_rn(__fadd_rn(a.M2, b.M2), __fmul_rn(__fmul_rn(d, d), __fmul_rn(a.n, fb)));
  a.Stx = __fadd_rn(__fadd_rn(a.Stx, b.Stx),
                    __fmul_rn(d, __fsub_rn(__fmul_rn(b.St, fa), __fmul_rn(a.St, fb))));
  a.St = __fadd_rn(a.St, b.St);
  a.m = __fadd_rn(a.m, __fmul_rn(d, fb));
  a.n = nn;
}

// A warp's statistics of one row over its lanes' M chunks (pairs, elements
// outside [lo, hi) zero when MASK).  LayerNorm: the warp's sum (a
// butterfly) over its n_w elements (n_w > 0, from the row's geometry) gives
// its mean m_w, then the sums about m_w from the same registers are reduced
// by recursive halving: lanes 0, 8 and 16 return M2, St and Stx.  m_w is
// the quotient rounded once more; it stands as the shift of those sums, and
// a shift off the mean by a rounding error changes M2 by n_w times its
// square.  RMSNorm: sum x^2 and sum t x, in lanes 0 and 16.
template <typename T, bool kLN, int M, bool MASK>
__device__ __forceinline__ float warp_row_stats(const f2 (&xv)[M][Elem<T>::kPerChunk / 2],
                                                const f2 (&dv)[M][Elem<T>::kPerChunk / 2],
                                                const int (&lo)[M], const int (&hi)[M],
                                                const f2 (&gam)[M][Elem<T>::kPerChunk / 2],
                                                int lane, float n_w, float &m_w) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  if constexpr (kLN) {
    f2 sx = f2_bcast(0.f);
#pragma unroll
    for (int m = 0; m < M; ++m)
#pragma unroll
      for (int i = 0; i < NP; ++i) sx = f2_add(sx, xv[m][i]);
    float t = f2_total(sx);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t = __fadd_rn(t, __shfl_xor_sync(kFullMask, t, o));
    m_w = __fdividef(t, n_w);
    const f2 nm = f2_bcast(-m_w);
    f2 s2 = f2_bcast(0.f), s3 = f2_bcast(0.f), s4 = f2_bcast(0.f);
#pragma unroll
    for (int m = 0; m < M; ++m)
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        f2 xc = f2_add(xv[m][i], nm);
        if (MASK)
          xc = f2_select(xc, 2 * i >= lo[m] && 2 * i < hi[m], 2 * i + 1 >= lo[m] && 2 * i + 1 < hi[m],
                         0.f);
        const f2 tt = f2_mul(dv[m][i], gam[m][i]);
        s2 = f2_fma(xc, xc, s2);
        s3 = f2_add(s3, tt);
        s4 = f2_fma(tt, xc, s4);
      }
    float v[4] = {f2_total(s2), f2_total(s3), f2_total(s4), 0.f};
    return warp_reduce_scatter<4>(v, lane);
  } else {
    f2 s2 = f2_bcast(0.f), s4 = f2_bcast(0.f);
#pragma unroll
    for (int m = 0; m < M; ++m)
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        const f2 tt = f2_mul(dv[m][i], gam[m][i]);
        s2 = f2_fma(xv[m][i], xv[m][i], s2);
        s4 = f2_fma(tt, xv[m][i], s4);
      }
    float v[2] = {f2_total(s2), f2_total(s4)};
    m_w = 0.f;
    return warp_reduce_scatter<2>(v, lane);
  }
}

// The number of a row's elements in warp w's chunks [64 w, 64 w + 64) of
// the stats kernel's stripe at window position `from`: columns
// [from + 64 E w - c, + 64 E) within [0, len).
template <int E>
__host__ __device__ __forceinline__ int stat_warp_count(int from, int len, int c, int w) {
  const int cs = from + 64 * E * w - c;
  return max(0, min(len, cs + 64 * E) - max(0, cs));
}

// Bytes of a lane's chunk that starting at column dc lie before the end of a
// row of len elements of SZ bytes (0..16): a copy reads no byte past the row.
template <int SZ>
__device__ __forceinline__ uint32_t stripe_bytes(int dc, int len) {
  return static_cast<uint32_t>(max(0, min(16, SZ * (len - dc))));
}

// ---------------------------------------------------------------------------
// Row statistics per stripe.  Warp w owns the stripe's window chunks
// [64 w, 64 w + 64), lane l chunks 64 w + l and 64 w + l + 32.  The lanes
// walk the CTA's sorted rows with their chunks of x and dy of the next
// kStatDepth - 1 rows in flight (cp.async into the lane's own slots of a
// shared-memory ring).  Per row each warp forms its statistics about its
// own mean (LayerNorm: count, mean, M2, sum t, sum t (x - mean); RMSNorm:
// sum x^2, sum t x) into shared memory; at the end they are merged (added)
// in warp order, one RowStat (two sums) per row and stripe.  A row whose
// chunks in the warp are all whole and inside the stripe takes a path
// without masks; a warp with no element of the row skips it (count zero).
// ---------------------------------------------------------------------------
constexpr int kStatDepth = 4;
constexpr size_t kStatRingBytes = static_cast<size_t>(kStatDepth) * kStatChunks * 2 * kStatThreads * 16;

template <int OP, typename T>
__global__ void __launch_bounds__(kStatThreads, 3) bwd_stripe_stats_kernel(const StripeParams p) {
  static_assert(OP == kLayerNorm || OP == kRmsNorm, "norm backward passes");
  static_assert(kStatChunks == 2, "two chunks a lane: 64 a warp");
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  constexpr int NP = E / 2;
  constexpr int M = kStatChunks;
  constexpr int NT = kStatThreads;
  constexpr int NW = NT / 32;
  constexpr int D = kStatDepth;
  constexpr int W = E * NT * M;  // window positions of a stripe
  constexpr bool kLN = OP == kLayerNorm;
  __shared__ StripeRows<kStatRows> L;
  // per row and warp: {mean, M2, St, Stx} (LayerNorm; the warp's count
  // follows from the row's length and head class), {-, sum x^2, -, sum t x}
  // (RMSNorm)
  __shared__ float4 wsa[kStatRows][NW];
  extern __shared__ __align__(16) unsigned char ring[];
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
  const int from = static_cast<int>(s) * W;  // the stripe's first window position
  const int cols = static_cast<int>(p.max_len);
  const T *x = static_cast<const T *>(p.x);
  const T *dy = static_cast<const T *>(p.dy);
  const T *gamma = static_cast<const T *>(p.gamma);
  const uint32_t rbase = smem_addr(ring) + 16u * tid;
  // the lane's bytes of chunk m of tensor t (0 x, 1 dy) in ring slot sl
  // (list entry j takes slot j mod D, counted as the list is walked)
  const auto slot = [&](int sl, int m, int t) -> uint32_t {
    return rbase + static_cast<uint32_t>(sl) * (M * 2 * NT * 16) +
           static_cast<uint32_t>((m * 2 + t) * NT * 16);
  };
  int q[M];
#pragma unroll
  for (int m = 0; m < M; ++m) q[m] = 64 * w + lane + 32 * m;
  for (int i = tid; i < kStatRows * NW; i += NT) (&wsa[0][0])[i] = make_float4(0.f, 0.f, 0.f, 0.f);

  const bool bad = stripe_sort<T, NT>(L, p.offsets, r0, n, from, p.max_len, p.hb);
  if (s == 0) {  // uniform over the CTA
    if (__syncthreads_or(bad) && tid == 0) atomicOr(p.status, kStatusBadOffsets);
  }
  const int cnt = L.seg[E];
  // list entry j's chunks into the ring (a group per entry, empty or not)
  const auto issue = [&](int j, int sl) {
    if (j < cnt) {
      const int c = L.cls[j];
      const int len = L.len[j];
      const int64_t o = L.off[j];
#pragma unroll
      for (int m = 0; m < M; ++m) {
        const int dc = from + E * q[m] - c;
        const int lo = max(0, -dc);
        if (lo < min(E, len - dc)) {
          const uint32_t nb = stripe_bytes<SZ>(dc, len);
          cp_async16(slot(sl, m, 0), x + o + dc, nb);
          cp_async16(slot(sl, m, 1), dy + o + dc, nb);
        }
      }
    }
    cp_async_commit();
  };
#pragma unroll
  for (int j = 0; j < D - 1; ++j) issue(j, j);
  int cur = -1;
  int dc[M], lo[M];
  f2 gam[M][NP];
  // sc: entry j's slot; si: the slot entry j + D - 1 is issued into
  for (int j = 0, sc = 0, si = D - 1; j < cnt;
       ++j, sc = sc + 1 == D ? 0 : sc + 1, si = si + 1 == D ? 0 : si + 1) {
    issue(j + D - 1, si);
    const int c = L.cls[j];
    if (c != cur) {  // a new head class: the lane's columns and gamma there
      cur = c;
#pragma unroll
      for (int m = 0; m < M; ++m) {
        dc[m] = from + E * q[m] - c;
        lo[m] = max(0, -dc[m]);
      }
      stripe_gamma<T, M>(gam, gamma, 0, cols, dc);
    }
    const int rl = L.len[j];
    int hi[M];
    bool full = true, any = false;
#pragma unroll
    for (int m = 0; m < M; ++m) {
      hi[m] = min(E, rl - dc[m]);
      full = full && hi[m] == E && lo[m] == 0;
      any = any || hi[m] > lo[m];
    }
    cp_async_wait<D - 1>();  // entry j's copies have landed
    f2 xv[M][NP], dv[M][NP];
    const float n_w = static_cast<float>(stat_warp_count<E>(from, rl, c, w));
    float t, m_w;
    if (__all_sync(kFullMask, full)) {
#pragma unroll
      for (int m = 0; m < M; ++m) {
        chunk_to_pairs<T>(lds128(slot(sc, m, 0)), xv[m]);
        chunk_to_pairs<T>(lds128(slot(sc, m, 1)), dv[m]);
      }
      t = warp_row_stats<T, kLN, M, false>(xv, dv, lo, hi, gam, lane, n_w, m_w);
    } else if (__any_sync(kFullMask, any)) {
      // elements outside a chunk's valid range read as 0
#pragma unroll
      for (int m = 0; m < M; ++m) {
        const uint4 z = make_uint4(0u, 0u, 0u, 0u);
        stripe_pairs<T>(lo[m] < hi[m] ? lds128(slot(sc, m, 0)) : z, lo[m], hi[m], 0.f, xv[m]);
        stripe_pairs<T>(lo[m] < hi[m] ? lds128(slot(sc, m, 1)) : z, lo[m], hi[m], 0.f, dv[m]);
      }
      t = warp_row_stats<T, kLN, M, true>(xv, dv, lo, hi, gam, lane, n_w, m_w);
    } else {
      continue;  // no element of the row in this warp's chunks
    }
    if constexpr (kLN) {
      if (lane == 0) {
        wsa[j][w].x = m_w;
        wsa[j][w].y = t;
      }
      if (lane == 8) wsa[j][w].z = t;
      if (lane == 16) wsa[j][w].w = t;
    } else {
      if (lane == 0) wsa[j][w].y = t;
      if (lane == 16) wsa[j][w].w = t;
    }
  }
  cp_async_wait<0>();
  __syncthreads();
  for (int j = tid; j < cnt; j += NT) {
    float4 out;
    if constexpr (kLN) {
      // warp qq's elements: columns [from + 64 E qq - c, + 64 E) of the row
      // within [0, len)
      const int c = L.cls[j];
      const int rl = L.len[j];
      RowStat a = {0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int qq = 0; qq < NW; ++qq) {
        const float4 u = wsa[j][qq];
        stat_merge(a, RowStat{static_cast<float>(stat_warp_count<E>(from, rl, c, qq)), u.x, u.y,
                              u.z, u.w});
      }
      out = make_float4(a.m, a.M2, a.St, a.Stx);
    } else {
      float s2 = wsa[j][0].y, s4 = wsa[j][0].w;
#pragma unroll
      for (int qq = 1; qq < NW; ++qq) {
        s2 = __fadd_rn(s2, wsa[j][qq].y);
        s4 = __fadd_rn(s4, wsa[j][qq].w);
      }
      out = make_float4(0.f, s2, 0.f, s4);
    }
    p.psum[static_cast<int64_t>(L.row[j]) * p.ns1 + s] = out;
  }
}

// Index of column `local` of a stripe in the padded shared partial row: one
// word of padding every 32, so that lanes E columns apart hit distinct banks.
__device__ __forceinline__ int stripe_pad(int local) { return local + (local >> 5); }

// dx of one chunk from its pairs and the row's coefficients {rstd, -mean,
// -mean(t) rstd, -mean(t xhat) rstd} (t = dy gamma), adding dy xhat (and
// dy) to the lane's column sums when wanted.  xhat = (x - mean) rstd: x -
// mean is exact near the mean, where x rstd - mean rstd would carry the
// rounding of mean rstd.
template <bool kLN, int NP>
__device__ __forceinline__ void stripe_dx(const f2 (&xv)[NP], const f2 (&dv)[NP],
                                          const f2 (&gam)[NP], const float4 &cf, bool want,
                                          f2 (&o)[NP], f2 (&accg)[NP], f2 (&accb)[NP]) {
  const f2 C0 = f2_bcast(cf.x), NMU = f2_bcast(cf.y), NA = f2_bcast(cf.z), NB = f2_bcast(cf.w);
#pragma unroll
  for (int i = 0; i < NP; ++i) {
    const f2 xh = kLN ? f2_mul(f2_add(xv[i], NMU), C0) : f2_mul(xv[i], C0);
    const f2 t = f2_mul(dv[i], gam[i]);
    o[i] = f2_fma(t, C0, f2_fma(xh, NB, NA));
    if (want) {
      accg[i] = f2_fma(dv[i], xh, accg[i]);
      if constexpr (kLN) accb[i] = f2_add(accb[i], dv[i]);
    }
  }
}

// ---------------------------------------------------------------------------
// dx and the column sums.  Lane t owns window chunk t of the stripe.  Per
// batch of up to 256 rows of the group: sort, then each listed row's
// statistics, merged from the stats kernel's stripes in stripe order, then the
// rows in list order with the lane's chunks of x and dy of the next
// kDxDepth - 1 rows in flight (cp.async into the lane's own ring slots): the
// lane writes its dx chunk and adds dy xhat (and dy) to its register sums.
// When the head class changes the lane adds those sums into the CTA's
// partial row in shared memory at their columns: the stripe's columns under
// every head class, [from - E, from + W2) for the stripe at window position
// `from`.  A row whose chunks in the warp are all whole takes a path without
// masks; a warp with no element of the row skips it.  The CTA writes its
// partial row to part[g][s] at the end.
// ---------------------------------------------------------------------------
constexpr int kDxDepth = 6;
constexpr size_t kDxRingBytes = static_cast<size_t>(kDxDepth) * 2 * kDxThreads * 16;

template <int OP, typename T>
__global__ void __launch_bounds__(kDxThreads, 3) bwd_stripe_dx_kernel(const StripeParams p) {
  static_assert(OP == kLayerNorm || OP == kRmsNorm, "norm backward passes");
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  constexpr int NP = E / 2;
  constexpr int NT = kDxThreads;
  constexpr int D = kDxDepth;
  constexpr int W = E * NT;                             // window positions of a stripe
  constexpr int W1 = E * kStatThreads * kStatChunks;    // ... of a stats stripe
  constexpr bool kLN = OP == kLayerNorm;
  constexpr int NA = kLN ? 2 : 1;
  constexpr int kSeg = W + E;  // the partial row: E columns of halo, then the stripe's W
  constexpr int kPadW = kSeg + kSeg / 32 + 1;
  __shared__ StripeRows<kDxBatch> L;
  __shared__ float4 coef[kDxBatch];
  __shared__ float spart[NA][kPadW];
  extern __shared__ __align__(16) unsigned char ring[];
  const int tid = threadIdx.x;
  const int64_t s = static_cast<int64_t>(blockIdx.x) / p.ng2;  // heavy stripes first
  const int64_t g = static_cast<int64_t>(blockIdx.x) % p.ng2;
  const int from = static_cast<int>(s) * W;  // the stripe's first window position
  const int cols = static_cast<int>(p.max_len);
  const T *x = static_cast<const T *>(p.x);
  const T *dy = static_cast<const T *>(p.dy);
  T *dx = static_cast<T *>(p.dx);
  const T *gamma = static_cast<const T *>(p.gamma);
  const bool want = p.part != nullptr;
  const uint32_t rbase = smem_addr(ring) + 16u * tid;
  // the lane's bytes of tensor t (0 x, 1 dy) in ring slot sl (list entry j
  // takes slot j mod D, counted as the list is walked)
  const auto slot = [&](int sl, int t) -> uint32_t {
    return rbase + static_cast<uint32_t>(sl) * (2 * NT * 16) + static_cast<uint32_t>(t * NT * 16);
  };
  for (int i = tid; i < NA * kPadW; i += NT) (&spart[0][0])[i] = 0.f;

  f2 accg[NP], accb[NP];
#pragma unroll
  for (int i = 0; i < NP; ++i) accg[i] = accb[i] = f2_bcast(0.f);
  // the class's sums into the partial row at their columns (class c):
  // entry E t + e - c + E is column from - E + E t + e - c
  const auto flush = [&](int c) {
    if (want) {
#pragma unroll
      for (int e = 0; e < E; ++e) {
        const int qq = stripe_pad(E * tid + e - c + E);
        spart[0][qq] = __fadd_rn(spart[0][qq], pair_elem(accg, e));
        if constexpr (kLN) spart[NA - 1][qq] = __fadd_rn(spart[NA - 1][qq], pair_elem(accb, e));
      }
#pragma unroll
      for (int i = 0; i < NP; ++i) accg[i] = accb[i] = f2_bcast(0.f);
    }
    __syncthreads();  // the next flush may add to the same columns
  };
  const int64_t gr0 = g * p.g2;
  const int64_t gr1 = min(gr0 + p.g2, p.rows);
  bool waited = false;
  for (int64_t r0 = gr0; r0 < gr1; r0 += kDxBatch) {
    const int n = static_cast<int>(min(static_cast<int64_t>(kDxBatch), gr1 - r0));
    (void)stripe_sort<T, NT>(L, p.offsets, r0, n, from, p.max_len, p.hb);
    if (!waited) {
      // launched as a programmatic dependent of the stats kernel: its sums
      // are read, and dx (which may be x or dy) written, only past this
      asm volatile("griddepcontrol.wait;" ::: "memory");
      waited = true;
    }
    const int cnt = L.seg[E];
    // list entry j's chunk into the ring (a group per entry, empty or not)
    const auto issue = [&](int j, int sl) {
      if (j < cnt) {
        const int c = L.cls[j];
        const int len = L.len[j];
        const int dc = from + E * tid - c;
        const int lo = max(0, -dc);
        if (lo < min(E, len - dc)) {
          const int64_t o = L.off[j];
          const uint32_t nb = stripe_bytes<SZ>(dc, len);
          cp_async16(slot(sl, 0), x + o + dc, nb);
          cp_async16(slot(sl, 1), dy + o + dc, nb);
        }
      }
      cp_async_commit();
    };
#pragma unroll
    for (int j = 0; j < D - 1; ++j) issue(j, j);
    if (tid < cnt) {
      // the row's statistics: its stripes' in stripe order (stats stripe q
      // holds its columns [W1 q - c, W1 (q + 1) - c) within [0, len))
      const int64_t r = L.row[tid];
      const int len = L.len[tid];
      const int cr = L.cls[tid];
      const int nst = (len + cr + W1 - 1) / W1;
      const float4 *ps = p.psum + r * p.ns1;
      const float inv_n = __frcp_rn(static_cast<float>(len));
      float4 cf;
      if constexpr (kLN) {
        RowStat a = {0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
        for (int qq = 0; qq < nst; ++qq) {
          const float4 u = ps[qq];
          const int nq = min(len, W1 * (qq + 1) - cr) - max(0, W1 * qq - cr);
          stat_merge(a, RowStat{static_cast<float>(nq), u.x, u.y, u.z, u.w});
        }
        const float c0 = rsqrtf(__fadd_rn(__fmul_rn(a.M2, inv_n), p.eps));  // rstd
        const float am = __fmul_rn(a.St, inv_n);                           // mean(t)
        const float bm = __fmul_rn(__fmul_rn(a.Stx, c0), inv_n);           // mean(t xhat)
        cf = make_float4(c0, -a.m, -__fmul_rn(am, c0), -__fmul_rn(bm, c0));
      } else {
        float s2 = 0.f, s4 = 0.f;
#pragma unroll 4
        for (int qq = 0; qq < nst; ++qq) {
          const float4 u = ps[qq];
          s2 = __fadd_rn(s2, u.y);
          s4 = __fadd_rn(s4, u.w);
        }
        const float c0 = rsqrtf(__fmaf_rn(s2, inv_n, p.eps));   // rstd
        const float bm = __fmul_rn(__fmul_rn(s4, c0), inv_n);   // mean(t xhat)
        cf = make_float4(c0, 0.f, 0.f, -__fmul_rn(bm, c0));
      }
      coef[tid] = cf;
    }
    __syncthreads();
    int cur = -1, dc = 0, lo = 0;
    f2 gam[1][NP];
    // sc: entry j's slot; si: the slot entry j + D - 1 is issued into
    for (int j = 0, sc = 0, si = D - 1; j < cnt;
         ++j, sc = sc + 1 == D ? 0 : sc + 1, si = si + 1 == D ? 0 : si + 1) {
      issue(j + D - 1, si);
      const int c = L.cls[j];
      if (c != cur) {  // a new head class: the lane's columns and gamma there
        if (cur >= 0) flush(cur);
        cur = c;
        dc = from + E * tid - c;
        lo = max(0, -dc);
        const int dc1[1] = {dc};
        stripe_gamma<T, 1>(gam, gamma, 0, cols, dc1);
      }
      const int len = L.len[j];
      const int hi = min(E, len - dc);
      const bool full = hi == E && lo == 0;
      cp_async_wait<D - 1>();  // entry j's copies have landed
      if (__all_sync(kFullMask, full)) {
        f2 xv[NP], dv[NP], ov[NP];
        chunk_to_pairs<T>(lds128(slot(sc, 0)), xv);
        chunk_to_pairs<T>(lds128(slot(sc, 1)), dv);
        stripe_dx<kLN, NP>(xv, dv, gam[0], coef[j], want, ov, accg, accb);
        stg_stream(dx + L.off[j] + dc, pairs_to_chunk<T>(ov));
      } else if (lo < hi) {
        // elements outside the chunk's valid range read as 0: no dy, so
        // they add nothing to the column sums
        f2 xv[NP], dv[NP], ov[NP];
        stripe_pairs<T>(lds128(slot(sc, 0)), lo, hi, 0.f, xv);
        stripe_pairs<T>(lds128(slot(sc, 1)), lo, hi, 0.f, dv);
        stripe_dx<kLN, NP>(xv, dv, gam[0], coef[j], want, ov, accg, accb);
        T *dst = dx + L.off[j] + dc;
        if (lo == 0 && hi == E) {
          stg_stream(dst, pairs_to_chunk<T>(ov));
        } else {
#pragma unroll
          for (int e = 0; e < E; ++e)
            if (e >= lo && e < hi) dst[e] = from_f32<T>(pair_elem(ov, e));
        }
      }
    }
    cp_async_wait<0>();
    if (cur >= 0) flush(cur);  // ends with a barrier: L and coef may be rewritten
  }
  if (!waited) asm volatile("griddepcontrol.wait;" ::: "memory");
  if (!want) return;
  __syncthreads();
  for (int a = 0; a < NA; ++a) {
    float *prow = p.part + ((g * p.ns2 + s) * NA + a) * kSeg;
    for (int i = tid; i < kSeg; i += NT) prow[i] = spart[a][stripe_pad(i)];
  }
}

// dgamma[j] (dbeta[j]) for j < cols: the sum over the dx kernel's groups
// g = 0, 1, ... of that group's partial rows at column j.  Partial row
// part[g][s][a] holds columns [W2 s - E, W2 s + W2) at entries [0, W2 + E),
// so column j lies in stripe j / W2 and, for the last E columns of that
// stripe, in the halo of the next: a group's two entries are added first,
// then the groups in order.  A block of 256 threads takes 64 columns: warp w
// adds, for column half w & 1, the groups w >> 1, (w >> 1) + 4, ..., eight
// loads ahead; the four slices are then added in slice order.  Launched as
// a programmatic dependent of the dx kernel.
constexpr int kStripeFinThreads = 256;
template <typename T>
__global__ void __launch_bounds__(kStripeFinThreads) bwd_stripe_finalize_kernel(
    const float *part, int64_t ngroups, int64_t nstripes, int w2, int e_halo, int64_t cols,
    int nacc, T *dgamma, T *dbeta) {
  __shared__ float sums[4][64];
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int lane = threadIdx.x & 31;
  const int w = threadIdx.x >> 5;
  const int a = blockIdx.y;
  T *out = a == 0 ? dgamma : dbeta;
  if (out == nullptr) return;  // uniform over the block
  const int col = 32 * (w & 1) + lane;
  const int slice = w >> 1;
  const int j = blockIdx.x * 64 + col;  // cols <= 2^31
  const int64_t seg = w2 + e_halo;
  float sum = 0.f;
  if (j < cols) {
    const int sa = j / w2;
    const int ia = j - sa * w2 + e_halo;  // entry in stripe sa
    const int ib = ia - w2;               // entry in stripe sa + 1 (its halo)
    const bool twob = sa + 1 < nstripes && ib >= 0;
    constexpr int U = 8;
    for (int64_t g0 = slice; g0 < ngroups; g0 += 4 * U) {
      float va[U], vb[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int64_t gg = g0 + 4 * u;
        const bool ok = gg < ngroups;
        const float *pa = part + ((min(gg, ngroups - 1) * nstripes + sa) * nacc + a) * seg;
        va[u] = ok ? __ldcs(pa + ia) : 0.f;
        vb[u] = (ok && twob) ? __ldcs(pa + nacc * seg + ib) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (g0 + 4 * u < ngroups) sum = __fadd_rn(sum, twob ? __fadd_rn(va[u], vb[u]) : va[u]);
    }
  }
  sums[slice][col] = sum;
  __syncthreads();
  if (w < 2 && j < cols) {
    float t = sums[0][col];
#pragma unroll
    for (int q = 1; q < 4; ++q) t = __fadd_rn(t, sums[q][col]);
    out[j] = from_f32<T>(t);
  }
}

}  // namespace rowop
