// tile_row.cuh -- the MEDIUM and LARGE buckets (medium_row_kernel and
// large_row_kernel of §2.1) and the fused ragged kernel.
//
// One persistent kernel serves all three uses:
//   * dense MEDIUM (no cluster): each CTA owns whole rows;
//   * dense LARGE (cluster of cs CTAs): the CTAs of a cluster split a row's
//     tiles into cs contiguous portions, each CTA reduces its portion to tile
//     partials in its shared memory, one cluster barrier later every CTA reads
//     all K partials through distributed shared memory and combines them in
//     the same fixed order, then normalises its own portion -- the row is read
//     from HBM once;
//   * ragged: the LARGE rows (cluster-split, assigned round-robin to
//     clusters), then the MEDIUM rows (whole rows, pulled from a device
//     counter), then the SMALL rows (one per warp, pulled from a counter) of
//     one classify pass, in a single launch.
// Rows are staged into shared memory by bulk copies (cp.async.bulk, TMA)
// through an S-stage ring of stage buffers guarded by mbarriers; thread 0
// prefetches S items ahead.  The 16-byte chunks at the two row ends that the
// row only partly covers are read element by element (never outside the row)
// and written into the stage by thread 0 one step later, so their load
// latency overlaps the step in between.  Outputs leave registers through
// 128-bit streaming stores.
#pragma once

#include "common.cuh"
#include "small_row.cuh"

namespace rowop {

enum ItemKind : int { kItemEnd = 0, kItemLarge = 1, kItemMedium = 2 };

struct TileParams {
  const void *in;
  void *out;
  const void *gamma;
  const void *beta;
  int64_t glen;
  int64_t rows;  // dense
  int64_t cols;  // dense
  int64_t ld;    // dense
  float eps;
  uint32_t stage_bytes;  // multiple of kTileBytes
  int stages;
  int max_tiles;  // tiles a stage holds (= stage_bytes / kTileBytes)
  int out_vec;
  int gvec;
  uint64_t timeout_ns;
  unsigned int *status;
  // ragged
  const int64_t *offsets;
  const int32_t *list_small;
  const int32_t *list_medium;
  const int32_t *list_large;
  const int32_t *counts;     // [3]: SMALL, MEDIUM, LARGE
  unsigned int *counters;    // [3]: next MEDIUM, next SMALL, CTAs finished
};

struct ItemMeta {
  int64_t row;
  int32_t kind;
  int32_t pad;
};

// Shared-memory layout of the tile kernel (host and device agree on it).
struct TileSmemLayout {
  uint32_t partials, meta, stats, scratch, bars, flags, total;
  __host__ __device__ TileSmemLayout(uint32_t stage_bytes, int stages, int max_tiles) {
    uint32_t off = stage_bytes * stages;
    partials = off;
    off += 2u * max_tiles * 16u;
    meta = off;
    off += stages * 16u;
    stats = off;
    off += 16u;
    scratch = off;
    off += kCtaWarps * 16u;
    bars = off;
    off += stages * 8u;
    flags = off;
    off += 16u;
    total = off;
  }
};

template <typename T>
struct RowGeo {
  const T *in_row;
  T *out_row;
  int64_t n;
  int h;
  int64_t nc;
  int64_t K;
  int64_t t0, t1;  // this CTA's tiles
};

template <typename T, bool EXACT, bool RAGGED>
__device__ __forceinline__ RowGeo<T> make_geo(const TileParams &p, int kind, int64_t row,
                                              int rank, int cs) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  RowGeo<T> g;
  int64_t start;
  if (RAGGED) {
    start = p.offsets[row];
    g.n = p.offsets[row + 1] - start;
  } else {
    start = row * p.ld;
    g.n = p.cols;
  }
  g.in_row = static_cast<const T *>(p.in) + start;
  g.out_row = static_cast<T *>(p.out) + start;
  g.h = EXACT ? 0 : static_cast<int>((reinterpret_cast<uintptr_t>(g.in_row) & 15) / SZ);
  g.nc = (g.h + g.n + E - 1) / E;
  g.K = (g.nc + kTileChunks - 1) / kTileChunks;
  if (kind == kItemLarge && cs > 1) {
    const int64_t tpc = (g.K + cs - 1) / cs;
    g.t0 = min(g.K, rank * tpc);
    g.t1 = min(g.K, g.t0 + tpc);
  } else {
    g.t0 = 0;
    g.t1 = g.K;
  }
  return g;
}

// Head/tail chunks whose element loads were issued by the producer and whose
// shared-memory write and mbarrier arrival are still to come.
struct PendingEdges {
  int count;  // 0, 1 or 2 chunks; -1 = nothing pending
  uint32_t bar;
  uint32_t dst[2];
  uint4 val[2];
};

__device__ __forceinline__ uint32_t ld_u16_issue(const void *p) {
  unsigned short v;
  asm volatile("ld.global.u16 %0, [%1];" : "=h"(v) : "l"(p));
  return v;
}
__device__ __forceinline__ uint32_t ld_u32_issue(const void *p) {
  uint32_t v;
  asm volatile("ld.global.u32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}

// Chunk image of window chunk c with only the row's own elements loaded.
template <typename T>
__device__ __forceinline__ uint4 load_edge_chunk(const T *in_row, int64_t c, int h, int64_t n) {
  constexpr int E = Elem<T>::kPerChunk;
  uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int64_t j = c * E + e - h;
    if (j >= 0 && j < n) {
      if (sizeof(T) == 2) {
        w[e >> 1] |= ld_u16_issue(in_row + j) << ((e & 1) * 16);
      } else {
        w[e] = ld_u32_issue(in_row + j);
      }
    }
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

__device__ __forceinline__ void complete_pending(PendingEdges &pe) {
  if (pe.count < 0) return;
  for (int i = 0; i < pe.count; ++i) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(pe.dst[i]), "r"(pe.val[i].x),
                 "r"(pe.val[i].y), "r"(pe.val[i].z), "r"(pe.val[i].w)
                 : "memory");
  }
  mbar_arrive(pe.bar);
  pe.count = -1;
}

// Valid element range [lo, hi) of window chunk c.
__device__ __forceinline__ void chunk_range(int64_t c, int64_t nc, int h, int64_t n, int E,
                                            int &lo, int &hi) {
  lo = (c == 0) ? h : 0;
  hi = (c == nc - 1) ? static_cast<int>(h + n - c * E) : E;
}

template <int OP, typename T, bool EXACT, bool CLUSTER, bool RAGGED>
__global__ void __launch_bounds__(kCtaThreads, 2) tile_row_kernel(const TileParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  extern __shared__ __align__(128) unsigned char smem[];
  const TileSmemLayout L(p.stage_bytes, p.stages, p.max_tiles);
  const int S = p.stages;
  float4 *partials = reinterpret_cast<float4 *>(smem + L.partials);
  ItemMeta *meta = reinterpret_cast<ItemMeta *>(smem + L.meta);
  float *stats = reinterpret_cast<float *>(smem + L.stats);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + L.flags);
  const uint32_t bar0 = smem_addr(smem + L.bars);
  const uint32_t stage0 = smem_addr(smem);
  const uint32_t partials_addr = smem_addr(partials);

  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int cs = CLUSTER ? static_cast<int>(cluster_nctarank()) : 1;
  const int rank = CLUSTER ? static_cast<int>(cluster_ctarank()) : 0;
  const int64_t cid = CLUSTER ? cluster_id_x() : blockIdx.x;
  const int64_t ncl = CLUSTER ? cluster_count_x() : gridDim.x;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) mbar_init(bar0 + 8u * s, 1);
    flags[0] = 0;  // aborted
    fence_mbar_init();
  }
  __syncthreads();

  // ---------------- producer state (thread 0 only) ----------------
  int64_t prod_large = 0;   // LARGE items taken by this cluster
  int64_t prod_dense = 0;   // dense items taken
  bool prod_done = false;   // END produced
  PendingEdges pend;
  pend.count = -1;
  uint32_t inflight_mask = 0;   // stages with a bulk copy not yet waited on
  uint32_t inflight_parity = 0;
  const uint64_t policy = l2_evict_first_policy();

  auto next_item = [&](int64_t &row) -> int {
    if (RAGGED) {
      if (!flags[0]) {
        const int64_t li = cid + prod_large * ncl;
        if (li < p.counts[2]) {
          ++prod_large;
          row = p.list_large[li];
          return kItemLarge;
        }
        const unsigned int m = atomicAdd(&p.counters[0], 1u);
        if (m < static_cast<unsigned int>(p.counts[1])) {
          row = p.list_medium[m];
          return kItemMedium;
        }
      } else {
        // aborted: keep the cluster's LARGE sequence (barriers), stop there
        const int64_t li = cid + prod_large * ncl;
        if (li < p.counts[2]) {
          ++prod_large;
          row = p.list_large[li];
          return kItemLarge;
        }
      }
      return kItemEnd;
    } else {
      const int64_t r = cid + prod_dense * ncl;
      if (r < p.rows) {
        ++prod_dense;
        row = r;
        return CLUSTER ? kItemLarge : kItemMedium;
      }
      return kItemEnd;
    }
  };

  auto fill = [&](int s, int64_t item_idx) {
    int64_t row = 0;
    const int kind = prod_done ? kItemEnd : next_item(row);
    if (kind == kItemEnd) prod_done = true;
    meta[s].row = row;
    meta[s].kind = kind;
    const uint32_t bar = bar0 + 8u * s;
    const uint32_t parity = static_cast<uint32_t>((item_idx / S) & 1);
    if (flags[0]) return;  // aborted: no copies, no arrivals
    if (kind == kItemEnd) {
      mbar_arrive(bar);
      return;
    }
    const RowGeo<T> g = make_geo<T, EXACT, RAGGED>(p, kind, row, rank, cs);
    const int64_t c0 = g.t0 * kTileChunks;
    const int64_t c1 = min(g.nc, g.t1 * kTileChunks);
    if (c0 >= c1) {
      mbar_arrive(bar);
      return;
    }
    const int64_t cf = (g.h > 0) ? 1 : 0;
    const int64_t cl = (((g.h + g.n) % E) != 0) ? g.nc - 1 : g.nc;
    const int64_t b0 = max(c0, cf);
    const int64_t b1 = min(c1, cl);
    const uint32_t sbase = stage0 + static_cast<uint32_t>(s) * p.stage_bytes;
    if (b1 > b0) {
      const char *win = reinterpret_cast<const char *>(g.in_row) - g.h * Elem<T>::kSize;
      uint32_t bytes = static_cast<uint32_t>((b1 - b0) * kChunkBytes);
      mbar_expect_tx(bar, bytes);
      fence_proxy_async_smem();
      uint32_t done = 0;
      while (done < bytes) {
        const uint32_t piece = min(bytes - done, 16384u);
        bulk_g2s(sbase + static_cast<uint32_t>((b0 - c0) * kChunkBytes) + done,
                 win + b0 * kChunkBytes + done, piece, bar, policy);
        done += piece;
      }
      inflight_mask |= 1u << s;
      inflight_parity = (inflight_parity & ~(1u << s)) | (parity << s);
    }
    // partly covered chunks at the row ends
    PendingEdges pe;
    pe.count = 0;
    pe.bar = bar;
    int64_t cand[2] = {c0, c1 - 1};
    for (int i = 0; i < 2; ++i) {
      const int64_t c = cand[i];
      if (i == 1 && c == cand[0]) break;
      if (c < cf || c >= cl) {
        pe.dst[pe.count] = sbase + static_cast<uint32_t>((c - c0) * kChunkBytes);
        pe.val[pe.count] = load_edge_chunk<T>(g.in_row, c, g.h, g.n);
        ++pe.count;
      }
    }
    if (pe.count == 0) {
      mbar_arrive(bar);
    } else {
      pend = pe;
      if (S < 2) complete_pending(pend);
    }
  };

  // ---------------- prologue ----------------
  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      complete_pending(pend);
      fill(s, s);
    }
  }

  bool in_cluster_phase = CLUSTER;
  const T *gamma = static_cast<const T *>(p.gamma);
  const T *beta = static_cast<const T *>(p.beta);
  const int64_t glen_g = p.gamma ? p.glen : 0;
  const int64_t glen_b = p.beta ? p.glen : 0;

  for (int64_t j = 0;; ++j) {
    const int s = static_cast<int>(j % S);
    const uint32_t parity = static_cast<uint32_t>((j / S) & 1);
    const uint32_t bar = bar0 + 8u * s;
    const bool aborted_before = flags[0] != 0;
    bool landed = false;
    if (!aborted_before) {
      landed = mbar_wait_bounded(bar, parity, p.timeout_ns);
      if (!landed) {
        atomicOr(p.status, kStatusTimeout);
        flags[0] = 1;
      }
    }
    if (tid == 0 && landed) inflight_mask &= ~(1u << s);
    const int kind = meta[s].kind;
    const int64_t row = meta[s].row;
    if (CLUSTER && in_cluster_phase && kind != kItemLarge) {
      cluster_sync();  // nobody reads our partials any more
      in_cluster_phase = false;
    }
    if (kind == kItemEnd) break;

    const RowGeo<T> g = make_geo<T, EXACT, RAGGED>(p, kind, row, rank, cs);
    const int64_t c0 = g.t0 * kTileChunks;
    const int buf = static_cast<int>(j & 1);
    const unsigned char *stage = smem + static_cast<size_t>(s) * p.stage_bytes;
    const int64_t ntl = g.t1 - g.t0;

    // ---- pass 1: one warp per tile -> tile partial ----
    for (int64_t lt = warp; lt < ntl; lt += kCtaWarps) {
      const int64_t t = g.t0 + lt;
      float x[2][E];
      int lo[2], hi[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int64_t c = t * kTileChunks + lane + 32 * u;
        if (c < g.nc) {
          const uint4 raw = *reinterpret_cast<const uint4 *>(stage + (c - c0) * kChunkBytes);
          unpack(raw, x[u]);
          if (EXACT) {
            lo[u] = 0;
            hi[u] = E;
          } else {
            chunk_range(c, g.nc, g.h, g.n, E, lo[u], hi[u]);
          }
        } else {
          lo[u] = 0;
          hi[u] = 0;
#pragma unroll
          for (int e = 0; e < E; ++e) x[u][e] = 0.f;
        }
      }
      float4 part = make_float4(0.f, 0.f, 0.f, 0.f);
      if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
        float m = -INFINITY;
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
          for (int e = 0; e < E; ++e)
            if (e >= lo[u] && e < hi[u]) m = fmaxf(m, x[u][e]);
        m = warp_max(m);
        float sum = 0.f;
        if (m != -INFINITY) {
#pragma unroll
          for (int u = 0; u < 2; ++u)
#pragma unroll
            for (int e = 0; e < E; ++e)
              if (e >= lo[u] && e < hi[u]) sum = __fadd_rn(sum, expf(__fsub_rn(x[u][e], m)));
        }
        sum = warp_sum(sum);
        part = make_float4(m, sum, 0.f, 0.f);
      } else if constexpr (OP == kLayerNorm) {
        float sum = 0.f;
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
          for (int e = 0; e < E; ++e)
            if (e >= lo[u] && e < hi[u]) sum = __fadd_rn(sum, x[u][e]);
        sum = warp_sum(sum);
        const int64_t w0 = t * kTileChunks * E;
        const int64_t w1 = min(g.nc, (t + 1) * kTileChunks) * E;
        const int64_t nt = max(static_cast<int64_t>(0),
                                 min(static_cast<int64_t>(g.h) + g.n, w1) - max(static_cast<int64_t>(g.h), w0));
        const float ntf = static_cast<float>(nt);
        const float mean = nt > 0 ? __fdiv_rn(sum, ntf) : 0.f;
        float q = 0.f;
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
          for (int e = 0; e < E; ++e)
            if (e >= lo[u] && e < hi[u]) {
              const float d = __fsub_rn(x[u][e], mean);
              q = __fmaf_rn(d, d, q);
            }
        q = warp_sum(q);
        part = make_float4(sum, mean, q, ntf);
      } else {
        float q = 0.f;
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
          for (int e = 0; e < E; ++e)
            if (e >= lo[u] && e < hi[u]) q = __fmaf_rn(x[u][e], x[u][e], q);
        q = warp_sum(q);
        part = make_float4(q, 0.f, 0.f, 0.f);
      }
      if (lane == 0) partials[buf * p.max_tiles + lt] = part;
    }

    const bool cluster_item = CLUSTER && kind == kItemLarge;
    if (cluster_item) {
      cluster_sync();
    } else {
      __syncthreads();
    }

    // ---- combine: warp 0, fixed order over the K tiles of the row ----
    if (warp == 0) {
      const int64_t tpc = cluster_item ? (g.K + cs - 1) / cs : g.K;
      auto read_part = [&](int64_t t) -> float4 {
        if (cluster_item) {
          const int64_t r = t / tpc;
          const int64_t i = t - r * tpc;
          const uint32_t local = partials_addr + static_cast<uint32_t>((buf * p.max_tiles + i) * 16);
          return ld_dsmem_f4(map_to_rank(local, static_cast<uint32_t>(r)));
        }
        return partials[buf * p.max_tiles + t];
      };
      if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
        float m = -INFINITY, sum = 0.f;
        for (int64_t t = lane; t < g.K; t += 32) {
          const float4 pt = read_part(t);
          softmax_merge(m, sum, pt.x, pt.y);
        }
        warp_softmax_merge(m, sum);
        if (lane == 0) {
          stats[0] = m;
          stats[1] = (OP == kSoftmax) ? __frcp_rn(sum) : logf(sum);
        }
      } else if constexpr (OP == kLayerNorm) {
        float sum = 0.f;
        for (int64_t t = lane; t < g.K; t += 32) sum = __fadd_rn(sum, read_part(t).x);
        sum = warp_sum(sum);
        const float nf = static_cast<float>(g.n);
        const float mean = __fdiv_rn(sum, nf);
        float v = 0.f;
        for (int64_t t = lane; t < g.K; t += 32) {
          const float4 pt = read_part(t);
          const float d = __fsub_rn(pt.y, mean);
          v = __fadd_rn(v, __fmaf_rn(__fmul_rn(pt.w, d), d, pt.z));
        }
        v = warp_sum(v);
        if (lane == 0) {
          stats[0] = mean;
          stats[1] = __frsqrt_rn(__fadd_rn(__fdiv_rn(v, nf), p.eps));
        }
      } else {
        float q = 0.f;
        for (int64_t t = lane; t < g.K; t += 32) q = __fadd_rn(q, read_part(t).x);
        q = warp_sum(q);
        if (lane == 0) {
          stats[0] = 0.f;
          stats[1] = __frsqrt_rn(__fadd_rn(__fdiv_rn(q, static_cast<float>(g.n)), p.eps));
        }
      }
    }
    __syncthreads();
    const float st0 = stats[0];
    const float st1 = stats[1];
    const bool aborted = flags[0] != 0;

    // ---- pass 2: normalise this CTA's tiles and store ----
    if (!aborted) {
      char *owin = reinterpret_cast<char *>(g.out_row) - g.h * Elem<T>::kSize;
      for (int64_t lt = warp; lt < ntl; lt += kCtaWarps) {
        const int64_t t = g.t0 + lt;
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int64_t c = t * kTileChunks + lane + 32 * u;
          if (c >= g.nc) continue;
          float x[E], y[E];
          unpack(*reinterpret_cast<const uint4 *>(stage + (c - c0) * kChunkBytes), x);
          int lo = 0, hi = E;
          if (!EXACT) chunk_range(c, g.nc, g.h, g.n, E, lo, hi);
          if constexpr (OP == kSoftmax) {
#pragma unroll
            for (int e = 0; e < E; ++e) y[e] = __fmul_rn(expf(__fsub_rn(x[e], st0)), st1);
          } else if constexpr (OP == kLogSoftmax) {
#pragma unroll
            for (int e = 0; e < E; ++e) y[e] = __fsub_rn(__fsub_rn(x[e], st0), st1);
          } else if constexpr (OP == kLayerNorm) {
            float gg[E], bb[E];
            load_param_chunk<T>(gamma, glen_g, c, g.h, p.gvec != 0, 1.f, gg);
            load_param_chunk<T>(beta, glen_b, c, g.h, p.gvec != 0, 0.f, bb);
#pragma unroll
            for (int e = 0; e < E; ++e)
              y[e] = __fmaf_rn(__fmul_rn(__fsub_rn(x[e], st0), st1), gg[e], bb[e]);
          } else {
            float gg[E];
            load_param_chunk<T>(gamma, glen_g, c, g.h, p.gvec != 0, 1.f, gg);
#pragma unroll
            for (int e = 0; e < E; ++e) y[e] = __fmul_rn(__fmul_rn(x[e], st1), gg[e]);
          }
          if (lo == 0 && hi == E && p.out_vec) {
            stg_stream(owin + c * kChunkBytes, pack(y));
          } else {
#pragma unroll
            for (int e = 0; e < E; ++e)
              if (e >= lo && e < hi) g.out_row[c * E + e - g.h] = from_f32<T>(y[e]);
          }
        }
      }
    }
    __syncthreads();  // stage s is free
    if (tid == 0) {
      complete_pending(pend);
      if (!prod_done) fill(s, j + S);
    }
  }

  // ---- ragged: the SMALL rows, one per warp ----
  if (RAGGED && !flags[0]) {
    SmallRowArgs sa;
    sa.gamma = p.gamma;
    sa.beta = p.beta;
    sa.glen = p.glen;
    sa.eps = p.eps;
    sa.gvec = p.gvec;
    sa.out_vec = p.out_vec;
    constexpr int SZ = Elem<T>::kSize;
    const T *in = static_cast<const T *>(p.in);
    T *out = static_cast<T *>(p.out);
    for (;;) {
      unsigned int idx = 0;
      if (lane == 0) idx = atomicAdd(&p.counters[1], 1u);
      idx = __shfl_sync(kFullMask, idx, 0);
      if (idx >= static_cast<unsigned int>(p.counts[0])) break;
      const int64_t row = p.list_small[idx];
      const int64_t start = p.offsets[row];
      const int64_t n = p.offsets[row + 1] - start;
      const int G = small_group_lanes(n, SZ);
      const int cpl = small_cpl_class((n + E - 1) / E + 1, G);
      const bool active = lane < G;
      if (cpl == 4) {
        small_row<OP, T, 4, false>(in + start, out + start, n, G, lane & (G - 1), active, sa);
      } else if (cpl == 8) {
        small_row<OP, T, 8, false>(in + start, out + start, n, G, lane & (G - 1), active, sa);
      } else {
        small_row<OP, T, 9, false>(in + start, out + start, n, G, lane & (G - 1), active, sa);
      }
    }
  }

  // ---- a CTA that gave up waiting still must not leave copies in flight ----
  if (tid == 0 && inflight_mask) {
    for (int s = 0; s < S; ++s)
      if (inflight_mask >> s & 1u)
        (void)mbar_wait_bounded(bar0 + 8u * s, inflight_parity >> s & 1u, p.timeout_ns);
  }

  // ---- ragged: the last CTA to finish resets the work counters, so a
  // classification can be reused by the next call without a host step ----
  if (RAGGED) {
    __syncthreads();  // every warp of this CTA is done pulling work
    if (tid == 0) {
      __threadfence();
      const unsigned int done = atomicAdd(&p.counters[2], 1u);
      if (done == gridDim.x - 1) {
        atomicExch(&p.counters[0], 0u);
        atomicExch(&p.counters[1], 0u);
        atomicExch(&p.counters[2], 0u);
      }
    }
  }
}

}  // namespace rowop
