// bwd_row.cuh -- backward passes of the row-wise operators for sm_103a:
//
//   softmax      dx = y (dy - sum(dy y))                 (from the output y)
//   log-softmax  dx = dy - exp(y) sum(dy)                (from the output y)
//   LayerNorm    dx = rstd (g - mean(g) - xhat mean(g xhat)),  g = dy gamma,
//                dgamma = sum over rows of dy xhat, dbeta = sum over rows of dy
//   RMSNorm      dx = rstd (g - xhat mean(g xhat)),  dgamma = sum of dy xhat
//
// (the derivatives of the forward definitions; the norm statistics are
// recomputed from x, which costs no memory traffic: x is read anyway).
//
// Design.  A team of TPR threads owns one row at a time and holds it in
// registers: each thread loads its CPT 16-byte chunks (or, for rows that are
// not 16-byte congruent, CPT*E single elements) of the input and of dy, all
// loads issued before the first is used.  The team reduces its per-thread
// statistics with a butterfly over its lanes, then (TPR > 32) through shared
// memory in warp order, then (rows longer than one CTA holds) across the CTAs
// of a thread-block cluster through distributed shared memory, in rank
// order; every thread ends with the same row statistics (LayerNorm takes two
// rounds: the mean, then the sums about it).  The thread then writes its dx
// chunks.  A thread owns the same columns in every dense row, so the norms
// keep gamma at those columns and the thread's dgamma / dbeta sums over all
// rows the team processes in shared memory private to the thread; at the
// end the CTA sums its teams in team order and writes one partial row per
// CTA (per cluster), and bwd_param_finalize_kernel sums the partials in index
// order.  Nothing is atomic: the result is bitwise reproducible for a given
// device (the number of partials follows the grid, which follows the
// device's SM count).
//
// Ragged rows: the team walks one bucket's record list of a classify plan,
// and each row's start, length and head offset are set per row.  The norms
// take the element path there: a thread's columns are then counted from the
// row's first element, whatever its alignment, so gamma and the dgamma /
// dbeta sums stay at fixed columns across rows of any start.  The launch
// covers the columns of its bucket's longest row (p.cols); a shorter row's
// missing columns load as zero and add nothing.
#pragma once

#include "common.cuh"
#include "dispatch.h"
#include "rowmath.cuh"

namespace rowop {

constexpr int kBwdMaxThreads = 512;
constexpr int kBwdMaxTeamWarps = kBwdMaxThreads / 32;
constexpr int kBwdSlots = 32;  // elements a thread holds per tensor

struct BwdParams {
  const void *a;   // y (softmax family) or x (norms)
  const void *dy;
  void *dx;
  const void *gamma;  // norms; NULL = ones
  float *part;        // [nparts][nacc][cols] column partials (norms); NULL = not wanted
  int64_t rows, cols, ld;  // ragged: cols = the columns the launch covers
  float eps;
  int tpr;   // threads of one CTA that share a row
  int h;     // VEC: head offset, in elements, of every row (a, dy and dx alike)
  int nc;    // VEC: 16-byte window chunks of a row
  int nacc;  // partial rows per partial index: 2 (dgamma, dbeta) or 1 (dgamma)
  uint64_t timeout_ns;
  unsigned int *status;
  // ragged: the rows of one bucket of a classify plan
  const RowRec *list;           // that bucket's list: classify block b from entry b * rows_per_block
  const int32_t *block_counts;  // [blocks][3] rows per bucket of each classify block
  int blocks;
  int64_t rows_per_block;
  int bucket;
};

// Shared memory of the backward kernel (static part).
struct BwdShared {
  float wres[2][kBwdMaxTeamWarps][4];  // per-warp sums, by reduction parity
  float cres[2][4];                    // this CTA's sums for the cluster peers
  uint64_t ready[2];                   // peers' sums published (cs arrivals)
  uint64_t released[2];                // peers done reading ours (cs * warps arrivals)
  int pref[257];                       // ragged: list start of each classify block, then the total
};

// Where a thread stands in its team, and the state of the team reductions.
struct BwdTeam {
  int tpr, lane, warp, team, wpt, wfirst, cs, tid;
  uint32_t ready0, released0;
  uint32_t red_count;     // reductions done (their parity picks the buffers)
  uint32_t uses0, uses1;  // cluster exchanges done through buffer 0 / 1
};

// Sum of NV values over the team, in a fixed order: a butterfly over the
// team's lanes (fp32 addition is commutative, so both partners form the same
// sum), then the team's warps in warp order through shared memory, then the
// CTAs of the cluster in rank order through distributed shared memory.  Every
// thread of the team (cluster) ends with the same sums.  Returns false, the
// same on every thread of the CTA, when a bounded cluster wait ran out.
template <int NV, bool CLUSTER>
__device__ __forceinline__ bool bwd_team_sum(float (&v)[NV], BwdShared &sh, BwdTeam &t,
                                             uint64_t timeout_ns, unsigned int *status) {
  const int b = static_cast<int>(t.red_count & 1u);
  ++t.red_count;
  const int width = t.tpr < 32 ? t.tpr : 32;
  for (int o = 1; o < width; o <<= 1) {
#pragma unroll
    for (int i = 0; i < NV; ++i) v[i] = __fadd_rn(v[i], __shfl_xor_sync(kFullMask, v[i], o));
  }
  if (t.tpr > 32) {
    if (t.lane == 0) {
#pragma unroll
      for (int i = 0; i < NV; ++i) sh.wres[b][t.warp][i] = v[i];
    }
    if (CLUSTER) {
      __syncthreads();  // a cluster CTA is one team
    } else {
      named_sync(1 + t.team, t.tpr);
    }
#pragma unroll
    for (int i = 0; i < NV; ++i) v[i] = sh.wres[b][t.wfirst][i];
    for (int w = 1; w < t.wpt; ++w) {
#pragma unroll
      for (int i = 0; i < NV; ++i) v[i] = __fadd_rn(v[i], sh.wres[b][t.wfirst + w][i]);
    }
  }
  if constexpr (CLUSTER) {
    const uint32_t uses_b = b ? t.uses1 : t.uses0;
    if (t.tid == 0) {
      // our sums of two exchanges ago must have been read by every peer; if
      // that wait runs out nothing is published and every peer times out too
      if (uses_b == 0 ||
          mbar_wait_cluster_bounded(t.released0 + 8u * b, (uses_b - 1) & 1u, timeout_ns)) {
#pragma unroll
        for (int i = 0; i < NV; ++i) sh.cres[b][i] = v[i];
        for (int q = 0; q < t.cs; ++q) mbar_arrive_remote(t.ready0 + 8u * b, static_cast<uint32_t>(q));
      }
    }
    const bool ok = mbar_wait_cluster_bounded(t.ready0 + 8u * b, uses_b & 1u, timeout_ns);
    if (__syncthreads_or(ok ? 0 : 1)) {
      if (t.tid == 0) atomicOr(status, kStatusTimeout);
      return false;
    }
    const uint32_t mine = smem_addr(&sh.cres[b][0]);
    float acc[NV];
    for (int q = 0; q < t.cs; ++q) {
      const float4 w = ld_dsmem_f4(map_to_rank(mine, static_cast<uint32_t>(q)));
      const float ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int i = 0; i < NV; ++i) acc[i] = q == 0 ? ww[i] : __fadd_rn(acc[i], ww[i]);
    }
#pragma unroll
    for (int i = 0; i < NV; ++i) v[i] = acc[i];
    __syncwarp();
    if (t.lane < t.cs) mbar_arrive_remote(t.released0 + 8u * b, static_cast<uint32_t>(t.lane));
    if (b) {
      ++t.uses1;
    } else {
      ++t.uses0;
    }
  }
  return true;
}

// Ragged norm rows (element path, half the slots) are compiled for two
// 512-thread CTAs per SM: twice the rows in flight per SM.
template <int OP, bool RAGGED>
constexpr int bwd_min_blocks() {
  return (RAGGED && (OP == kLayerNorm || OP == kRmsNorm)) ? 2 : 1;
}

template <int OP, typename T, int CPT, bool VEC, bool CLUSTER, bool RAGGED = false>
__global__ void __launch_bounds__(kBwdMaxThreads, bwd_min_blocks<OP, RAGGED>())
    bwd_row_kernel(const BwdParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  constexpr int S = CPT * E;  // elements per thread per tensor
  constexpr bool kNorm = (OP == kLayerNorm || OP == kRmsNorm);
  constexpr int NA = OP == kLayerNorm ? 2 : 1;
  static_assert(!(RAGGED && kNorm && VEC), "ragged norm rows take the element path");
  __shared__ BwdShared sh;
  // dynamic (norms): gamma at this thread's columns ([CPT][NT] chunks), the
  // thread's dgamma / dbeta sums ([NA][S/4][NT] float4) -- both private to
  // the thread, so no barrier guards them -- and, when a CTA holds several
  // teams, their combined sums ([NA][cols])
  extern __shared__ __align__(16) unsigned char bwd_dyn[];

  const int NT = blockDim.x;
  const int TPR = p.tpr;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int team = tid / TPR;
  const int tt = tid - team * TPR;
  const int teams_cta = NT / TPR;
  const int cs = CLUSTER ? static_cast<int>(cluster_nctarank()) : 1;
  const int rank = CLUSTER ? static_cast<int>(cluster_ctarank()) : 0;
  int64_t gteam, nteams, warp_team0;
  if (CLUSTER) {
    gteam = cluster_id_x();
    nteams = cluster_count_x();
    warp_team0 = gteam;
  } else {
    gteam = static_cast<int64_t>(blockIdx.x) * teams_cta + team;
    nteams = static_cast<int64_t>(gridDim.x) * teams_cta;
    // several teams share a warp when TPR < 32: the warp runs its first
    // team's row count, so shuffles always see every lane
    warp_team0 = static_cast<int64_t>(blockIdx.x) * teams_cta + (TPR < 32 ? (warp * 32) / TPR : team);
  }
  // row geometry: fixed for dense rows, set per row for ragged ones; pcols
  // (the columns gamma and the partial rows cover) stays the launch's
  const int64_t pcols = p.cols;
  int64_t cols = pcols;
  int h = VEC ? p.h : 0;
  int nc = VEC ? p.nc : 0;
  int cf = (VEC && h > 0) ? 1 : 0;                                 // first full chunk
  int cl = (VEC && ((h + cols) % E) != 0) ? nc - 1 : nc;          // end of full chunks
  int hn = h + static_cast<int>(cols);
  float inv_n = __frcp_rn(static_cast<float>(cols));
  int64_t nrows = p.rows;
  if constexpr (RAGGED) {
    // list position where each classify block's rows of this bucket start
    if (warp == 0) {
      int carry = 0;
      for (int b0 = 0; b0 < p.blocks; b0 += 32) {
        const int b = b0 + lane;
        const int v = b < p.blocks ? p.block_counts[3 * b + p.bucket] : 0;
        int x = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(kFullMask, x, o);
          if (lane >= o) x += y;
        }
        if (b < p.blocks) sh.pref[b] = carry + x - v;
        carry += __shfl_sync(kFullMask, x, 31);
      }
      if (lane == 0) sh.pref[p.blocks] = carry;
    }
    __syncthreads();
    nrows = sh.pref[p.blocks];
  }

  BwdTeam tm;
  tm.tpr = TPR;
  tm.lane = lane;
  tm.warp = warp;
  tm.team = team;
  tm.wpt = TPR >= 32 ? TPR / 32 : 1;
  tm.wfirst = TPR >= 32 ? team * tm.wpt : warp;
  tm.cs = cs;
  tm.tid = tid;
  tm.ready0 = smem_addr(&sh.ready[0]);
  tm.released0 = smem_addr(&sh.released[0]);
  tm.red_count = 0;
  tm.uses0 = tm.uses1 = 0;
  if (CLUSTER) {
    if (tid == 0) {
      mbar_init(tm.ready0, cs);
      mbar_init(tm.ready0 + 8, cs);
      mbar_init(tm.released0, cs * (NT / 32));
      mbar_init(tm.released0 + 8, cs * (NT / 32));
      fence_mbar_init();
    }
    cluster_sync();  // every peer's barriers exist before any remote arrive
  }

  // column of element e of this thread's chunk k, or -1 at or past `lim`:
  // the row's length (column), or the launch's cover (pcolumn: gamma and the
  // partial rows)
  auto column_lim = [&](int k, int e, int64_t lim) -> int64_t {
    if constexpr (VEC) {
      const int c = (k * cs + rank) * TPR + tt;
      if (c >= nc) return -1;
      const int64_t j = static_cast<int64_t>(c) * E + e - h;
      return (j >= 0 && j < lim) ? j : -1;
    } else {
      const int64_t j = (static_cast<int64_t>(k * E + e) * cs + rank) * TPR + tt;
      return j < lim ? j : -1;
    }
  };
  auto column = [&](int k, int e) { return column_lim(k, e, cols); };
  auto pcolumn = [&](int k, int e) { return column_lim(k, e, pcols); };

  const bool accum = kNorm && p.part != nullptr;
  uint4 *gsm = reinterpret_cast<uint4 *>(bwd_dyn);
  float4 *acc = reinterpret_cast<float4 *>(bwd_dyn + (kNorm ? CPT * NT * 16 : 0));
  float *red = reinterpret_cast<float *>(bwd_dyn + (kNorm ? CPT * NT * 16 : 0) +
                                         (accum ? NA * S * NT * 4 : 0));  // [NA][pcols]
  if constexpr (kNorm) {
    // gamma at this thread's columns, once for all rows; the sums start at 0
    const T *gamma = static_cast<const T *>(p.gamma);
#pragma unroll
    for (int k = 0; k < CPT; ++k) {
      float g[E];
#pragma unroll
      for (int e = 0; e < E; ++e) {
        const int64_t j = pcolumn(k, e);
        g[e] = (gamma && j >= 0) ? load_elem(gamma + j) : 1.f;
      }
      gsm[k * NT + tid] = pack<T>(g);
    }
    if (accum) {
#pragma unroll
      for (int q = 0; q < NA * S / 4; ++q) acc[q * NT + tid] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }

  const T *abase = static_cast<const T *>(p.a);
  const T *dybase = static_cast<const T *>(p.dy);
  T *dxbase = static_cast<T *>(p.dx);

  for (int64_t r0 = warp_team0; r0 < nrows; r0 += nteams) {
    const int64_t r = r0 + (gteam - warp_team0);
    const bool active = r < nrows;
    int64_t start = r * p.ld;
    if constexpr (RAGGED) {
      // record r of the bucket's list: classify block lo with pref[lo] <= r < pref[lo + 1]
      start = 0;
      cols = 0;
      if (active) {
        int lo = 0, hi = p.blocks;
        while (hi - lo > 1) {
          const int mid = (lo + hi) >> 1;
          if (sh.pref[mid] <= r) {
            lo = mid;
          } else {
            hi = mid;
          }
        }
        const RowRec rec = p.list[static_cast<int64_t>(lo) * p.rows_per_block + (r - sh.pref[lo])];
        start = rec.start;
        cols = rec.n;
      }
      h = VEC ? static_cast<int>((reinterpret_cast<uintptr_t>(abase + start) & 15u) / SZ) : 0;
      hn = h + static_cast<int>(cols);
      nc = VEC ? (hn + E - 1) / E : 0;
      cf = (VEC && h > 0) ? 1 : 0;
      cl = (VEC && (hn % E) != 0) ? nc - 1 : nc;
      inv_n = __frcp_rn(static_cast<float>(cols));
    }
    const T *arow = abase + start;
    const T *dyrow = dybase + start;
    T *dxrow = dxbase + start;

    // ---- loads: every chunk of both tensors in flight before any is used ----
    uint4 av[CPT], dv[CPT];
    uint32_t msk[CPT];
#pragma unroll
    for (int k = 0; k < CPT; ++k) {
      av[k] = make_uint4(0u, 0u, 0u, 0u);
      dv[k] = av[k];
      msk[k] = 0u;
      if (!active) continue;
      if constexpr (VEC) {
        const int c = (k * cs + rank) * TPR + tt;
        if (c >= nc) continue;
        if (c >= cf && c < cl) {
          av[k] = ldg_stream(reinterpret_cast<const char *>(arow) - h * SZ + static_cast<int64_t>(c) * 16);
          dv[k] = ldg_stream(reinterpret_cast<const char *>(dyrow) - h * SZ + static_cast<int64_t>(c) * 16);
          msk[k] = (1u << E) - 1u;
        } else {
          int lo, hi;
          chunk_valid_range(c, nc, h, hn, E, lo, hi);
          av[k] = load_chunk_elems<T>(arow, c, h, cols);
          dv[k] = load_chunk_elems<T>(dyrow, c, h, cols);
          msk[k] = ((1u << hi) - 1u) & ~((1u << lo) - 1u);
        }
      } else {
        float fa[E], fd[E];
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const int64_t j = column(k, e);
          fa[e] = j >= 0 ? load_elem(arow + j) : 0.f;
          fd[e] = j >= 0 ? load_elem(dyrow + j) : 0.f;
          if (j >= 0) msk[k] |= 1u << e;
        }
        av[k] = pack<T>(fa);
        dv[k] = pack<T>(fd);
      }
    }

    // ---- row sums, in packed pairs (masked elements load as zero and add
    // nothing, but for LayerNorm's deviations, which are masked) ----
    constexpr int NP = E / 2;
    float c0 = 0.f, c1 = 0.f, c2 = 0.f, mu = 0.f;
    bool ok = true;
    if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
      f2 s2 = f2_bcast(0.f);
#pragma unroll
      for (int k = 0; k < CPT; ++k) {
        f2 x[NP], d[NP];
        chunk_to_pairs<T>(av[k], x);
        chunk_to_pairs<T>(dv[k], d);
#pragma unroll
        for (int i = 0; i < NP; ++i) s2 = OP == kSoftmax ? f2_fma(d[i], x[i], s2) : f2_add(s2, d[i]);
      }
      float v[1] = {f2_total(s2)};
      ok = bwd_team_sum<1, CLUSTER>(v, sh, tm, p.timeout_ns, p.status);
      c0 = v[0];  // sum dy y, or sum dy
    } else if constexpr (OP == kRmsNorm) {
      f2 sxx = f2_bcast(0.f), sgx = f2_bcast(0.f);
#pragma unroll
      for (int k = 0; k < CPT; ++k) {
        f2 x[NP], d[NP], g[NP];
        chunk_to_pairs<T>(av[k], x);
        chunk_to_pairs<T>(dv[k], d);
        chunk_to_pairs<T>(gsm[k * NT + tid], g);
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          sxx = f2_fma(x[i], x[i], sxx);
          sgx = f2_fma(f2_mul(d[i], g[i]), x[i], sgx);
        }
      }
      float v[2] = {f2_total(sxx), f2_total(sgx)};
      ok = bwd_team_sum<2, CLUSTER>(v, sh, tm, p.timeout_ns, p.status);
      c0 = rsqrtf(__fmaf_rn(v[0], inv_n, p.eps));      // rstd
      c1 = __fmul_rn(__fmul_rn(v[1], c0), inv_n);      // mean(g xhat)
    } else {
      // LayerNorm: the mean first, then the sums about it
      f2 sx = f2_bcast(0.f);
#pragma unroll
      for (int k = 0; k < CPT; ++k) {
        f2 x[NP];
        chunk_to_pairs<T>(av[k], x);
#pragma unroll
        for (int i = 0; i < NP; ++i) sx = f2_add(sx, x[i]);
      }
      float v1[1] = {f2_total(sx)};
      ok = bwd_team_sum<1, CLUSTER>(v1, sh, tm, p.timeout_ns, p.status);
      mu = __fmul_rn(v1[0], inv_n);
      const f2 nmu = f2_bcast(-mu);
      f2 sdd = f2_bcast(0.f), sg = f2_bcast(0.f), sgd = f2_bcast(0.f);
#pragma unroll
      for (int k = 0; k < CPT; ++k) {
        f2 x[NP], d[NP], g[NP];
        chunk_to_pairs<T>(av[k], x);
        chunk_to_pairs<T>(dv[k], d);
        chunk_to_pairs<T>(gsm[k * NT + tid], g);
        const bool full = msk[k] == (1u << E) - 1u;
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          f2 dev = f2_add(x[i], nmu);
          if (!full) dev = f2_select(dev, (msk[k] >> (2 * i)) & 1u, (msk[k] >> (2 * i + 1)) & 1u, 0.f);
          const f2 gg = f2_mul(d[i], g[i]);
          sdd = f2_fma(dev, dev, sdd);
          sg = f2_add(sg, gg);
          sgd = f2_fma(gg, dev, sgd);
        }
      }
      float v[3] = {f2_total(sdd), f2_total(sg), f2_total(sgd)};
      if (ok) ok = bwd_team_sum<3, CLUSTER>(v, sh, tm, p.timeout_ns, p.status);
      c0 = rsqrtf(__fadd_rn(__fmul_rn(v[0], inv_n), p.eps));   // rstd
      c1 = __fmul_rn(v[1], inv_n);                              // mean(g)
      c2 = __fmul_rn(__fmul_rn(v[2], c0), inv_n);               // mean(g xhat)
    }
    if (!ok) break;  // uniform over the CTA (cluster waits only)

    // ---- dx, and this thread's dgamma / dbeta sums ----
    if (!active) continue;
    const f2 C0 = f2_bcast(c0), NC1 = f2_bcast(-c1), NC2 = f2_bcast(-c2);
    // xhat = (x - mu) rstd: x - mu is exact for x near mu, where x rstd -
    // mu rstd would carry the rounding of mu rstd (large for |mu| >> std)
    const f2 NMU = f2_bcast(-mu);
#pragma unroll
    for (int k = 0; k < CPT; ++k) {
      if (msk[k] == 0u) continue;
      f2 x[NP], d[NP], o[NP], ag[NP];
      chunk_to_pairs<T>(av[k], x);
      chunk_to_pairs<T>(dv[k], d);
      if constexpr (OP == kSoftmax) {
        const f2 ns = f2_bcast(-c0);
#pragma unroll
        for (int i = 0; i < NP; ++i) o[i] = f2_mul(x[i], f2_add(d[i], ns));
      } else if constexpr (OP == kLogSoftmax) {
        const f2 ns = f2_bcast(-c0);
        const f2 l2e = f2_bcast(kLog2e);
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          const f2 u = f2_mul(x[i], l2e);
          o[i] = f2_fma(f2_make(ex2_approx(u.x), ex2_approx(u.y)), ns, d[i]);
        }
      } else {
        f2 g[NP];
        chunk_to_pairs<T>(gsm[k * NT + tid], g);
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          f2 xh;
          if constexpr (OP == kRmsNorm) {
            xh = f2_mul(x[i], C0);
          } else {
            xh = f2_mul(f2_add(x[i], NMU), C0);
          }
          // rstd (g - mean(g) - xhat mean(g xhat)); RMSNorm has no mean(g)
          f2 t = OP == kRmsNorm ? f2_mul(d[i], g[i]) : f2_fma(d[i], g[i], NC1);
          t = f2_fma(xh, OP == kRmsNorm ? NC1 : NC2, t);
          o[i] = f2_mul(C0, t);
          ag[i] = f2_mul(d[i], xh);
        }
        if (accum) {
          // masked elements have d = 0: they add exactly zero
          float4 *ap = acc + (k * E / 4) * NT + tid;
#pragma unroll
          for (int q = 0; q < E / 4; ++q) {
            float4 vg = ap[q * NT];
            const f2 lo = f2_add(make_float2(vg.x, vg.y), ag[2 * q]);
            const f2 hi = f2_add(make_float2(vg.z, vg.w), ag[2 * q + 1]);
            ap[q * NT] = make_float4(lo.x, lo.y, hi.x, hi.y);
            if constexpr (NA == 2) {
              float4 vb = ap[(S / 4 + q) * NT];
              const f2 blo = f2_add(make_float2(vb.x, vb.y), d[2 * q]);
              const f2 bhi = f2_add(make_float2(vb.z, vb.w), d[2 * q + 1]);
              ap[(S / 4 + q) * NT] = make_float4(blo.x, blo.y, bhi.x, bhi.y);
            }
          }
        }
      }
      if constexpr (VEC) {
        const int c = (k * cs + rank) * TPR + tt;
        if (msk[k] == (1u << E) - 1u) {
          stg_stream(reinterpret_cast<char *>(dxrow) - h * SZ + static_cast<int64_t>(c) * 16,
                     pairs_to_chunk<T>(o));
        } else {
#pragma unroll
          for (int e = 0; e < E; ++e)
            if ((msk[k] >> e) & 1u)
              dxrow[static_cast<int64_t>(c) * E + e - h] = from_f32<T>(pair_elem(o, e));
        }
      } else {
#pragma unroll
        for (int e = 0; e < E; ++e)
          if ((msk[k] >> e) & 1u) dxrow[column(k, e)] = from_f32<T>(pair_elem(o, e));
      }
    }
  }

  // ---- cluster: no CTA leaves while a peer may still read its sums ----
  if constexpr (CLUSTER) {
    if (tid == 0) {
      if (tm.uses0 > 0) (void)mbar_wait_cluster_bounded(tm.released0, (tm.uses0 - 1) & 1u, p.timeout_ns);
      if (tm.uses1 > 0)
        (void)mbar_wait_cluster_bounded(tm.released0 + 8u, (tm.uses1 - 1) & 1u, p.timeout_ns);
    }
  }

  // ---- norms: one partial row of dgamma (and dbeta) per CTA / cluster ----
  if constexpr (kNorm) {
    if (!accum) return;
    const float *af = reinterpret_cast<const float *>(acc);
    // this thread's sum for slot s of accumulator a
    auto slot_sum = [&](int a, int s) { return af[((a * S + s) / 4 * NT + tid) * 4 + (s & 3)]; };
    if (TPR < 32) {
      // teams of one warp own the same columns: fold them by butterfly (every
      // lane ends with the fold) and keep the fold in the thread's own sums
      float *aw = reinterpret_cast<float *>(acc);
#pragma unroll
      for (int a = 0; a < NA; ++a)
#pragma unroll
        for (int s = 0; s < S; ++s) {
          float v = slot_sum(a, s);
          for (int o = TPR; o < 32; o <<= 1) v = __fadd_rn(v, __shfl_xor_sync(kFullMask, v, o));
          aw[((a * S + s) / 4 * NT + tid) * 4 + (s & 3)] = v;
        }
    }
    const int units = TPR < 32 ? NT / 32 : teams_cta;  // holders of a full column set
    const int unit = TPR < 32 ? warp : team;
    const bool holder = TPR >= 32 || lane < TPR;
    const int64_t pidx = CLUSTER ? static_cast<int64_t>(cluster_id_x()) : static_cast<int64_t>(blockIdx.x);
    float *prow = p.part + pidx * p.nacc * pcols;
    if (units == 1) {
      if (holder) {
#pragma unroll
        for (int k = 0; k < CPT; ++k)
#pragma unroll
          for (int e = 0; e < E; ++e) {
            const int64_t j = pcolumn(k, e);
            if (j < 0) continue;
#pragma unroll
            for (int a = 0; a < NA; ++a) prow[a * pcols + j] = slot_sum(a, k * E + e);
          }
      }
      return;
    }
    // several teams: sum them in team order in shared memory, then write
    for (int u = 0; u < units; ++u) {
      if (unit == u && holder) {
#pragma unroll
        for (int k = 0; k < CPT; ++k)
#pragma unroll
          for (int e = 0; e < E; ++e) {
            const int64_t j = pcolumn(k, e);
            if (j < 0) continue;
#pragma unroll
            for (int a = 0; a < NA; ++a) {
              const float v = slot_sum(a, k * E + e);
              red[a * pcols + j] = u == 0 ? v : __fadd_rn(red[a * pcols + j], v);
            }
          }
      }
      __syncthreads();
    }
    for (int64_t j = tid; j < NA * pcols; j += NT) prow[j] = red[j];
  }
}

// Partial rows to be summed into dgamma / dbeta: segment i holds nparts[i]
// partials of nacc rows of cover[i] floats each (a dense call has one
// segment; a ragged call one per row bucket, covering that bucket's longest
// row).
constexpr int kMaxBwdSegments = 3;
struct BwdSegments {
  const float *part[kMaxBwdSegments];
  int64_t nparts[kMaxBwdSegments];
  int64_t cover[kMaxBwdSegments];
  int n;
};

// dgamma[j] (dbeta[j]) for j < cols = the sum over the segments in order of
// each segment's sum over its partials q = 0, 1, ... of part[q][0 (1)][j]
// (zero where j is past the segment's cover): a block per 32 columns, one
// column per lane; warp w adds q = w, w + 32, ... in that order, U loads
// ahead, then the 32 warp sums are added in warp order.
constexpr int kFinThreads = 1024;
constexpr int kFinWarps = kFinThreads / 32;
template <typename T>
__global__ void __launch_bounds__(kFinThreads) bwd_param_finalize_kernel(const BwdSegments sg,
                                                                         int64_t cols, int nacc,
                                                                         T *dgamma, T *dbeta) {
  __shared__ float sums[kFinWarps][32];
  // launched as a programmatic dependent of the kernel that wrote the
  // partials: its blocks may start while that kernel drains, and wait here
  // until it has finished and its writes are visible (a no-op otherwise)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int a = blockIdx.y;
  T *out = a == 0 ? dgamma : dbeta;
  if (out == nullptr) return;  // uniform over the block
  const int64_t j = static_cast<int64_t>(blockIdx.x) * 32 + lane;
  float total = 0.f;
  bool first = true;
  for (int i = 0; i < sg.n; ++i) {
    const int64_t cover = sg.cover[i];
    if (static_cast<int64_t>(blockIdx.x) * 32 >= cover) continue;  // uniform over the block
    const float *part = sg.part[i];
    const int64_t nparts = sg.nparts[i];
    float s = 0.f;
    if (j < cover) {
      constexpr int U = 8;
      for (int64_t q0 = warp; q0 < nparts; q0 += kFinWarps * U) {
        float x[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const int64_t q = q0 + u * kFinWarps;
          x[u] = q < nparts ? __ldcs(part + (q * nacc + a) * cover + j) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < U; ++u)
          if (q0 + u * kFinWarps < nparts) s = __fadd_rn(s, x[u]);
      }
    }
    __syncthreads();  // the previous segment's sums have been read
    sums[warp][lane] = s;
    __syncthreads();
    if (warp == 0) {
      float t = sums[0][lane];
      for (int w = 1; w < kFinWarps; ++w) t = __fadd_rn(t, sums[w][lane]);
      total = first ? t : __fadd_rn(total, t);
      first = false;
    }
  }
  if (warp == 0 && j < cols) out[j] = from_f32<T>(total);
}

}  // namespace rowop
