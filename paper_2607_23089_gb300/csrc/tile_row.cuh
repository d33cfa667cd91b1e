// tile_row.cuh -- the MEDIUM and LARGE buckets (medium_row_kernel and
// large_row_kernel of §2.1) and the fused ragged kernel.
//
// One persistent, warp-specialised kernel serves all uses.  Each CTA has a
// producer warp and 8 consumer warps:
//   * the producer (one lane) walks the CTA's items (a whole row, or this
//     CTA's portion of a cluster-split row), stages each item into the next
//     free buffer of an S-stage ring with bulk copies (cp.async.bulk, TMA) --
//     one mbarrier per 16 KiB piece so consumers start on the first piece
//     while later ones land -- and reads the at most two 16-byte chunks the
//     row only partly covers element by element (never outside the row),
//     writing them into the stage one item later so their latency overlaps;
//   * consumers reduce one 1 KiB tile per warp to a tile partial, meet at one
//     named barrier per item, combine the K tile partials of the row in a
//     fixed order (every warp redundantly, so no broadcast is needed),
//     normalise their tiles from the stage, store with 128-bit streaming
//     stores and release the stage to the producer.
// Dense MEDIUM rows: one CTA per row.  LARGE rows: the cs CTAs of a cluster
// split the row's tiles into contiguous portions resident in shared memory;
// after pass 1 every CTA signals the others with remote mbarrier arrives,
// gathers all K partials through distributed shared memory and combines them
// exactly like the MEDIUM path -- the row is read from HBM once and the result
// does not depend on cs.  Ragged: the LARGE rows (cluster-split, round-robin
// over clusters), then the MEDIUM rows (pulled from a device counter), then
// the SMALL rows (one per warp, staged through the then idle stage memory).
#pragma once

#include "rowmath.cuh"
#include "small_row.cuh"

namespace rowop {

enum ItemKind : int { kItemEnd = 0, kItemLarge = 1, kItemMedium = 2 };

constexpr int kConsumerWarps = 8;
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kTileThreads = kConsumerThreads + 32;  // + the producer warp
constexpr int kPieceTiles = 16;                      // tiles per piece barrier (16 KiB)
constexpr uint32_t kBarConsumers = 1;                // named barrier of the consumer warps
constexpr int kSmallSliceBytes = 4096 + 128;         // per-warp staging of a ragged SMALL row

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
  uint32_t stage_bytes;  // = max_tiles * kTileBytes
  int stages;
  int max_tiles;     // tiles one stage holds
  int gather_tiles;  // partials the gather buffer holds (cluster launches)
  int out_vec;
  int gvec;
  uint64_t timeout_ns;
  unsigned int *status;
  // ragged
  const RowRec *rec_small;
  const RowRec *rec_medium;
  const RowRec *rec_large;
  const int32_t *counts;   // [3]: SMALL, MEDIUM, LARGE
  unsigned int *counters;  // [3]: next MEDIUM, next SMALL, CTAs finished
};

struct ItemMeta {
  int64_t start;
  int64_t n;
  int32_t kind;
  int32_t pad[3];
};

// Shared-memory layout of the tile kernel (host and device agree on it).
struct TileSmemLayout {
  uint32_t part_c, part_m, gather, meta, bar_meta, bar_piece, bar_empty, bar_ready,
      bar_released, flags, total;
  int pieces;
  __host__ __device__ TileSmemLayout(uint32_t stage_bytes, int stages, int max_tiles,
                                     int gather_tiles) {
    pieces = (max_tiles + kPieceTiles - 1) / kPieceTiles;
    uint32_t off = stage_bytes * stages;
    part_c = off;
    off += 2u * max_tiles * 16u;
    part_m = off;
    off += 2u * max_tiles * 16u;
    gather = off;
    off += static_cast<uint32_t>(gather_tiles) * 16u;
    meta = off;
    off += stages * 32u;
    bar_meta = off;
    off += stages * 8u;
    bar_piece = off;
    off += stages * pieces * 8u;
    bar_empty = off;
    off += stages * 8u;
    bar_ready = off;
    off += 16u;
    bar_released = off;
    off += 16u;
    flags = off;
    off += 16u;
    total = off;
  }
};

struct ItemGeo {
  int64_t start, n;
  int h;
  int64_t nc, K, t0, t1;
  int64_t cf, cl;  // chunks [cf, cl) are entirely the row's
};

template <typename T, bool EXACT>
__device__ __forceinline__ ItemGeo item_geo(const void *in, int64_t start, int64_t n, bool split,
                                            int rank, int cs) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  ItemGeo g;
  g.start = start;
  g.n = n;
  const uintptr_t a = reinterpret_cast<uintptr_t>(static_cast<const T *>(in) + start);
  g.h = EXACT ? 0 : static_cast<int>((a & 15) / SZ);
  g.nc = (g.h + n + E - 1) / E;
  g.K = (g.nc + kTileChunks - 1) / kTileChunks;
  if (split) {
    const int64_t tpc = (g.K + cs - 1) / cs;
    g.t0 = min(g.K, rank * tpc);
    g.t1 = min(g.K, g.t0 + tpc);
  } else {
    g.t0 = 0;
    g.t1 = g.K;
  }
  g.cf = (g.h > 0) ? 1 : 0;
  g.cl = (((g.h + n) % E) != 0) ? g.nc - 1 : g.nc;
  return g;
}

__device__ __forceinline__ bool tile_is_full(int64_t t, const ItemGeo &g) {
  return t * kTileChunks >= g.cf && (t + 1) * kTileChunks <= g.cl;
}

// ---------------------------------------------------------------------------
// pass 1: one warp reduces tile t (its 64 chunks at `tsm`) to a tile partial
//   softmax / log-softmax (m_t, s_t = sum exp(x - m_t)), LayerNorm (sum,
//   mean_t, sum (x - mean_t)^2, n_t), RMSNorm (sum x^2).
// ---------------------------------------------------------------------------
template <int OP, typename T, bool EXACT>
__device__ __forceinline__ float4 tile_partial(const unsigned char *tsm, int64_t t,
                                               const ItemGeo &g, int lane) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  const bool full = tile_is_full(t, g);  // the row's last tile may hold < 64 chunks
  f2 p0[NP], p1[NP];
  chunk_to_pairs(*reinterpret_cast<const uint4 *>(tsm + lane * kChunkBytes), p0);
  chunk_to_pairs(*reinterpret_cast<const uint4 *>(tsm + (lane + 32) * kChunkBytes), p1);
  int lo0 = 0, hi0 = E, lo1 = 0, hi1 = E;
  const int64_t hn = g.h + g.n;
  if (!full) {
    const int64_t c0 = t * kTileChunks + lane;
    const int64_t c1 = c0 + 32;
    if (c0 < g.nc) chunk_valid_range(c0, g.nc, g.h, hn, E, lo0, hi0); else lo0 = hi0 = 0;
    if (c1 < g.nc) chunk_valid_range(c1, g.nc, g.h, hn, E, lo1, hi1); else lo1 = hi1 = 0;
  }
  if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
    float m = chunk_max<NP>(p0, -INFINITY, lo0, hi0);
    m = warp_max(chunk_max<NP>(p1, m, lo1, hi1));
    f2 acc = f2_bcast(0.f);
    if (m != -INFINITY) {
      const f2 m2 = f2_bcast(m);
      acc = chunk_sum_exp<NP>(p0, m2, acc, lo0, hi0);
      acc = chunk_sum_exp<NP>(p1, m2, acc, lo1, hi1);
    }
    return make_float4(m, warp_sum(f2_total(acc)), 0.f, 0.f);
  } else if constexpr (OP == kLayerNorm) {
    f2 acc = chunk_sum<NP>(p0, f2_bcast(0.f), lo0, hi0);
    acc = chunk_sum<NP>(p1, acc, lo1, hi1);
    const float sum = warp_sum(f2_total(acc));
    float mean, ntf;
    if (full) {
      ntf = static_cast<float>(kTileChunks * E);
      mean = __fmul_rn(sum, 1.f / static_cast<float>(kTileChunks * E));  // exact: power of 2
    } else {
      const int64_t w0 = t * kTileChunks * E;
      const int64_t w1 = min(g.nc, (t + 1) * kTileChunks) * E;
      const int64_t nt = max(static_cast<int64_t>(0),
                             min(hn, w1) - max(static_cast<int64_t>(g.h), w0));
      ntf = static_cast<float>(nt);
      mean = nt > 0 ? __fdiv_rn(sum, ntf) : 0.f;
    }
    const f2 mean2 = f2_bcast(mean);
    acc = chunk_sum_sqdev<NP>(p0, mean2, f2_bcast(0.f), lo0, hi0);
    acc = chunk_sum_sqdev<NP>(p1, mean2, acc, lo1, hi1);
    return make_float4(sum, mean, warp_sum(f2_total(acc)), ntf);
  } else {
    f2 acc = chunk_sum_sq<NP>(p0, f2_bcast(0.f), lo0, hi0);
    acc = chunk_sum_sq<NP>(p1, acc, lo1, hi1);
    return make_float4(warp_sum(f2_total(acc)), 0.f, 0.f, 0.f);
  }
}

// ---------------------------------------------------------------------------
// combine: the row statistics from its K tile partials (part[t], t < K), in
// the fixed order lane l: t = l, l+32, ..., then a 5-level butterfly.  Every
// lane of the calling warp ends with the same (s0, s1).
// ---------------------------------------------------------------------------
template <int OP>
__device__ __forceinline__ void combine_stats(const float4 *part, int64_t K, int64_t n,
                                              float eps, int lane, float &s0, float &s1) {
  if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
    float m = -INFINITY;
    for (int64_t t = lane; t < K; t += 32) m = fmaxf(m, part[t].x);
    const float M = warp_max(m);
    float s = 0.f;
    for (int64_t t = lane; t < K; t += 32) {
      const float4 pt = part[t];
      if (pt.x != -INFINITY) s = __fadd_rn(s, __fmul_rn(pt.y, exp_shifted(pt.x, M)));
    }
    const float S = warp_sum(s);
    s0 = M;
    s1 = (OP == kSoftmax) ? __frcp_rn(S) : logf(S);
  } else if constexpr (OP == kLayerNorm) {
    float s = 0.f;
    for (int64_t t = lane; t < K; t += 32) s = __fadd_rn(s, part[t].x);
    const float nf = static_cast<float>(n);
    const float mean = __fdiv_rn(warp_sum(s), nf);
    float v = 0.f;
    for (int64_t t = lane; t < K; t += 32) {
      const float4 pt = part[t];
      const float d = __fsub_rn(pt.y, mean);
      v = __fadd_rn(v, __fmaf_rn(__fmul_rn(pt.w, d), d, pt.z));
    }
    s0 = mean;
    s1 = __frsqrt_rn(__fadd_rn(__fdiv_rn(warp_sum(v), nf), eps));
  } else {
    float q = 0.f;
    for (int64_t t = lane; t < K; t += 32) q = __fadd_rn(q, part[t].x);
    s0 = 0.f;
    s1 = __frsqrt_rn(__fadd_rn(__fdiv_rn(warp_sum(q), static_cast<float>(n)), eps));
  }
}

// pass 2: normalise tile t from the stage and store it
template <int OP, typename T, bool EXACT>
__device__ __forceinline__ void tile_store(const unsigned char *tsm, int64_t t, const ItemGeo &g,
                                           int lane, float s0, float s1, const TileParams &p,
                                           char *owin, T *out_row) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  const bool full = tile_is_full(t, g);  // the row's last tile may hold < 64 chunks
  const int64_t hn = g.h + g.n;
  const T *gamma = static_cast<const T *>(p.gamma);
  const T *beta = static_cast<const T *>(p.beta);
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int64_t c = t * kTileChunks + lane + 32 * u;
    if (!full && c >= g.nc) continue;
    f2 v[NP];
    chunk_to_pairs(*reinterpret_cast<const uint4 *>(tsm + (lane + 32 * u) * kChunkBytes), v);
    int lo = 0, hi = E;
    if (!full) chunk_valid_range(c, g.nc, g.h, hn, E, lo, hi);
    chunk_normalize<OP, T>(v, s0, s1, gamma, gamma ? p.glen : 0, beta, beta ? p.glen : 0, c,
                           g.h, p.gvec != 0);
    store_chunk<T>(v, owin, out_row, c, g.h, lo, hi, p.out_vec != 0);
  }
}

// ---------------------------------------------------------------------------
// producer: edge chunks loaded now, written into the stage one item later
// ---------------------------------------------------------------------------
struct PendingEdges {
  int count;  // chunks pending; -1 = nothing pending
  int nbars;
  uint32_t dst[2];
  uint4 val[2];
  uint32_t bar[2];
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
// Chunk image of window chunk c with only the row's elements (issued loads).
template <typename T>
__device__ __forceinline__ uint4 issue_edge_chunk(const T *in_row, int64_t c, int h, int64_t n) {
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
  for (int i = 0; i < pe.nbars; ++i) mbar_arrive(pe.bar[i]);
  pe.count = -1;
}

template <typename T, bool EXACT, bool CLUSTER, bool RAGGED>
__device__ __forceinline__ void tile_producer(const TileParams &p, const TileSmemLayout &L,
                                              unsigned char *smem, int cs, int rank, int64_t cid,
                                              int64_t ncl) {
  constexpr int SZ = Elem<T>::kSize;
  const int S = p.stages;
  const uint32_t sbase = smem_addr(smem);
  ItemMeta *meta = reinterpret_cast<ItemMeta *>(smem + L.meta);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + L.flags);
  const uint64_t pol = l2_evict_first_policy();
  int64_t k_large = 0, k_dense = 0;
  bool medium_phase = false;
  PendingEdges pend;
  pend.count = -1;
  uint32_t fill_mask = 0, fill_parity = 0;

  for (int64_t it = 0;; ++it) {
    const int s = static_cast<int>(it % S);
    if (it >= S) {
      if (!mbar_wait_bounded(sbase + L.bar_empty + 8u * s,
                             static_cast<uint32_t>(((it / S) - 1) & 1), p.timeout_ns)) {
        atomicOr(p.status, kStatusTimeout);
        flags[0] = 1;
        break;
      }
      fill_mask &= ~(1u << s);
    }
    if (flags[0]) break;
    complete_pending(pend);

    int kind = kItemEnd;
    int64_t start = 0, n = 0;
    if (RAGGED) {
      if (!medium_phase) {
        const int64_t li = cid + k_large * ncl;
        if (li < p.counts[2]) {
          const RowRec r = p.rec_large[li];
          ++k_large;
          kind = kItemLarge;
          start = r.start;
          n = r.n;
        } else {
          medium_phase = true;
        }
      }
      if (medium_phase) {
        const unsigned int m = atomicAdd(&p.counters[0], 1u);
        if (m < static_cast<unsigned int>(p.counts[1])) {
          const RowRec r = p.rec_medium[m];
          kind = kItemMedium;
          start = r.start;
          n = r.n;
        }
      }
    } else {
      const int64_t r = cid + k_dense * ncl;
      if (r < p.rows) {
        ++k_dense;
        kind = CLUSTER ? kItemLarge : kItemMedium;
        start = r * p.ld;
        n = p.cols;
      }
    }
    meta[s].start = start;
    meta[s].n = n;
    meta[s].kind = kind;
    mbar_arrive(sbase + L.bar_meta + 8u * s);
    if (kind == kItemEnd) break;

    const bool split = CLUSTER && kind == kItemLarge;
    const ItemGeo g = item_geo<T, EXACT>(p.in, start, n, split, rank, cs);
    const int64_t c0 = g.t0 * kTileChunks;
    const int64_t c1 = min(g.nc, g.t1 * kTileChunks);
    const T *in_row = static_cast<const T *>(p.in) + start;
    const char *win = reinterpret_cast<const char *>(in_row) - g.h * SZ;
    const uint32_t stage = sbase + static_cast<uint32_t>(s) * p.stage_bytes;
    const bool head = c0 < c1 && g.cf > 0 && c0 == 0;
    const bool tail = c0 < c1 && g.cl < g.nc && c1 == g.nc && !(head && g.nc == 1);
    const int head_pc = 0;
    const int tail_pc = tail ? static_cast<int>((g.nc - 1 - c0) / (kPieceTiles * kTileChunks)) : -1;
    bool any_copy = false;
    for (int pc = 0; pc < L.pieces; ++pc) {
      const uint32_t bar = sbase + L.bar_piece + 8u * (s * L.pieces + pc);
      const int64_t q0 = c0 + static_cast<int64_t>(pc) * kPieceTiles * kTileChunks;
      const int64_t q1 = min(c1, q0 + kPieceTiles * kTileChunks);
      const int64_t b0 = max(q0, g.cf);
      const int64_t b1 = min(q1, g.cl);
      const uint32_t bytes = (q0 < c1 && b1 > b0) ? static_cast<uint32_t>((b1 - b0) * kChunkBytes)
                                                  : 0u;
      const bool edge = (head && pc == head_pc) || (tail && pc == tail_pc);
      if (edge) {
        if (bytes) mbar_expect_tx(bar, bytes);
      } else if (bytes) {
        mbar_arrive_expect_tx(bar, bytes);
      } else {
        mbar_arrive(bar);
      }
      if (bytes) {
        fence_proxy_async_smem();
        bulk_g2s(stage + static_cast<uint32_t>((b0 - c0) * kChunkBytes), win + b0 * kChunkBytes,
                 bytes, bar, pol);
        any_copy = true;
      }
    }
    if (any_copy) {
      fill_mask |= 1u << s;
      fill_parity = (fill_parity & ~(1u << s)) | (static_cast<uint32_t>((it / S) & 1) << s);
    }
    if (head || tail) {
      PendingEdges pe;
      pe.count = 0;
      pe.nbars = 0;
      if (head) {
        pe.dst[pe.count] = stage;
        pe.val[pe.count] = issue_edge_chunk<T>(in_row, 0, g.h, g.n);
        ++pe.count;
        pe.bar[pe.nbars++] = sbase + L.bar_piece + 8u * (s * L.pieces + head_pc);
      }
      if (tail) {
        pe.dst[pe.count] = stage + static_cast<uint32_t>((g.nc - 1 - c0) * kChunkBytes);
        pe.val[pe.count] = issue_edge_chunk<T>(in_row, g.nc - 1, g.h, g.n);
        ++pe.count;
        if (!(head && tail_pc == head_pc))
          pe.bar[pe.nbars++] = sbase + L.bar_piece + 8u * (s * L.pieces + tail_pc);
      }
      pend = pe;
      if (S == 1) complete_pending(pend);
    }
  }
  complete_pending(pend);
  // a producer that gave up must not leave copies in flight into its stages
  if (flags[0]) {
    for (int s = 0; s < S; ++s)
      if (fill_mask >> s & 1u)
        for (int pc = 0; pc < L.pieces; ++pc)
          (void)mbar_wait_bounded(sbase + L.bar_piece + 8u * (s * L.pieces + pc),
                                  fill_parity >> s & 1u, p.timeout_ns);
  }
}

template <int OP, typename T, bool EXACT, bool CLUSTER, bool RAGGED>
__global__ void __launch_bounds__(kTileThreads, 3) tile_row_kernel(const TileParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  extern __shared__ __align__(1024) unsigned char smem[];
  const TileSmemLayout L(p.stage_bytes, p.stages, p.max_tiles, p.gather_tiles);
  const int S = p.stages;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int cs = CLUSTER ? static_cast<int>(cluster_nctarank()) : 1;
  const int rank = CLUSTER ? static_cast<int>(cluster_ctarank()) : 0;
  const int64_t cid = CLUSTER ? cluster_id_x() : blockIdx.x;
  const int64_t ncl = CLUSTER ? cluster_count_x() : gridDim.x;
  const uint32_t sbase = smem_addr(smem);
  float4 *part_c = reinterpret_cast<float4 *>(smem + L.part_c);
  float4 *part_m = reinterpret_cast<float4 *>(smem + L.part_m);
  float4 *gather = reinterpret_cast<float4 *>(smem + L.gather);
  const ItemMeta *meta = reinterpret_cast<const ItemMeta *>(smem + L.meta);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + L.flags);

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(sbase + L.bar_meta + 8u * s, 1);
      mbar_init(sbase + L.bar_empty + 8u * s, kConsumerWarps);
      for (int pc = 0; pc < L.pieces; ++pc) mbar_init(sbase + L.bar_piece + 8u * (s * L.pieces + pc), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(sbase + L.bar_ready + 8u * b, cs);
      mbar_init(sbase + L.bar_released + 8u * b, cs);
    }
    flags[0] = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (CLUSTER) cluster_sync();  // every peer's barriers exist before any remote arrive

  if (warp == kConsumerWarps) {
    if (lane == 0) tile_producer<T, EXACT, CLUSTER, RAGGED>(p, L, smem, cs, rank, cid, ncl);
    return;
  }

  // ------------------------------ consumers ------------------------------
  int64_t uses[2] = {0, 0};  // cluster items that used part_c[b]
  bool ended = false;
  for (int64_t it = 0;; ++it) {
    const int s = static_cast<int>(it % S);
    const uint32_t par = static_cast<uint32_t>((it / S) & 1);
    const int b = static_cast<int>(it & 1);
    bool bad = !mbar_wait_bounded(sbase + L.bar_meta + 8u * s, par, p.timeout_ns);
    int kind = kItemEnd;
    ItemGeo g;
    g.K = 0;
    g.t0 = g.t1 = 0;
    if (!bad) {
      kind = meta[s].kind;
      if (kind != kItemEnd) {
        const bool split = CLUSTER && kind == kItemLarge;
        g = item_geo<T, EXACT>(p.in, meta[s].start, meta[s].n, split, rank, cs);
        if (split && uses[b] > 0)
          bad = !mbar_wait_cluster_bounded(sbase + L.bar_released + 8u * b,
                                           static_cast<uint32_t>((uses[b] - 1) & 1), p.timeout_ns);
      }
    }
    const bool split = CLUSTER && kind == kItemLarge;
    const unsigned char *stage = smem + static_cast<size_t>(s) * p.stage_bytes;
    const int64_t ntl = g.t1 - g.t0;
    float4 *part = (split ? part_c : part_m) + static_cast<size_t>(b) * p.max_tiles;

    // ---- pass 1 ----
    if (!bad && kind != kItemEnd) {
      int waited = -1;
      for (int64_t lt = warp; lt < ntl; lt += kConsumerWarps) {
        const int pc = static_cast<int>(lt / kPieceTiles);
        if (pc != waited) {
          if (!mbar_wait_bounded(sbase + L.bar_piece + 8u * (s * L.pieces + pc), par,
                                 p.timeout_ns)) {
            bad = true;
            break;
          }
          waited = pc;
        }
        const float4 pt = tile_partial<OP, T, EXACT>(stage + lt * kTileBytes, g.t0 + lt, g, lane);
        if (lane == 0) part[lt] = pt;
      }
    }
    if (named_sync_or(kBarConsumers, kConsumerThreads, bad)) {
      if (tid == 0) {
        atomicOr(p.status, kStatusTimeout);
        flags[0] = 1;
      }
      break;
    }
    if (kind == kItemEnd) {
      ended = true;
      break;
    }

    // ---- combine ----
    const float4 *src = part;
    if (split) {
      const uint32_t ready = sbase + L.bar_ready + 8u * b;
      if (tid == 0)
        for (int r = 0; r < cs; ++r) mbar_arrive_remote(ready, static_cast<uint32_t>(r));
      bool ok = mbar_wait_cluster_bounded(ready, static_cast<uint32_t>(uses[b] & 1), p.timeout_ns);
      if (ok) {
        const int64_t tpc = (g.K + cs - 1) / cs;
        const uint32_t mine = smem_addr(part_c + static_cast<size_t>(b) * p.max_tiles);
        for (int64_t t = tid; t < g.K; t += kConsumerThreads) {
          const int64_t r = t / tpc;
          gather[t] = ld_dsmem_f4(map_to_rank(mine + static_cast<uint32_t>((t - r * tpc) * 16),
                                              static_cast<uint32_t>(r)));
        }
      }
      if (named_sync_or(kBarConsumers, kConsumerThreads, !ok)) {
        if (tid == 0) {
          atomicOr(p.status, kStatusTimeout);
          flags[0] = 1;
        }
        break;
      }
      if (tid == 0)
        for (int r = 0; r < cs; ++r)
          mbar_arrive_remote(sbase + L.bar_released + 8u * b, static_cast<uint32_t>(r));
      ++uses[b];
      src = gather;
    }
    float s0, s1;
    combine_stats<OP>(src, g.K, g.n, p.eps, lane, s0, s1);

    // ---- pass 2 ----
    T *out_row = static_cast<T *>(p.out) + g.start;
    char *owin = reinterpret_cast<char *>(out_row) - g.h * SZ;
    for (int64_t lt = warp; lt < ntl; lt += kConsumerWarps)
      tile_store<OP, T, EXACT>(stage + lt * kTileBytes, g.t0 + lt, g, lane, s0, s1, p, owin,
                               out_row);
    __syncwarp();
    if (lane == 0) mbar_arrive(sbase + L.bar_empty + 8u * s);
  }

  // ---- ragged: the SMALL rows, one per warp, staged in a slice of the stages ----
  if (RAGGED && ended) {
    named_sync(kBarConsumers, kConsumerThreads);  // no warp reads the stages any more
    SmallRowArgs sa;
    sa.gamma = p.gamma;
    sa.beta = p.beta;
    sa.glen = p.glen;
    sa.eps = p.eps;
    sa.gvec = p.gvec;
    sa.out_vec = p.out_vec;
    unsigned char *slice = smem + static_cast<size_t>(warp) * kSmallSliceBytes;
    const T *in = static_cast<const T *>(p.in);
    T *out = static_cast<T *>(p.out);
    for (;;) {
      unsigned int idx = 0;
      if (lane == 0) idx = atomicAdd(&p.counters[1], 1u);
      idx = __shfl_sync(kFullMask, idx, 0);
      if (idx >= static_cast<unsigned int>(p.counts[0])) break;
      const RowRec rec = p.rec_small[idx];
      const T *in_row = in + rec.start;
      const uintptr_t ia = reinterpret_cast<uintptr_t>(in_row);
      const int h = static_cast<int>((ia & 15) / SZ);
      const int64_t nc = (h + rec.n + E - 1) / E;
      const char *win = reinterpret_cast<const char *>(ia - (ia & 15));
      for (int64_t c = lane; c < nc; c += 32) {
        int lo, hi;
        chunk_valid_range(c, nc, h, h + rec.n, E, lo, hi);
        *reinterpret_cast<uint4 *>(slice + c * kChunkBytes) =
            (lo == 0 && hi == E) ? ldg_stream(win + c * kChunkBytes)
                                 : load_chunk_elems<T>(in_row, c, h, rec.n);
      }
      __syncwarp();
      const int G = small_group_lanes(rec.n, SZ);
      const int sub = lane & (G - 1);
      const int64_t ncg = lane < G ? nc : 0;
      auto get = [&](int k) {
        return *reinterpret_cast<const uint4 *>(slice + (sub + static_cast<int64_t>(k) * G) *
                                                            kChunkBytes);
      };
      const int cpl = small_cpl_class((rec.n + E - 1) / E + 1, G);
      if (cpl == 4) {
        small_row_core<OP, T, 4, false>(get, out + rec.start, rec.n, h, ncg, G, sub, sa);
      } else if (cpl == 8) {
        small_row_core<OP, T, 8, false>(get, out + rec.start, rec.n, h, ncg, G, sub, sa);
      } else {
        small_row_core<OP, T, 9, false>(get, out + rec.start, rec.n, h, ncg, G, sub, sa);
      }
      __syncwarp();
    }
  }

  // ---- no CTA leaves while a peer may still read its partials ----
  if (CLUSTER) {
    for (int bb = 0; bb < 2; ++bb)
      if (uses[bb] > 0)
        (void)mbar_wait_cluster_bounded(sbase + L.bar_released + 8u * bb,
                                        static_cast<uint32_t>((uses[bb] - 1) & 1), p.timeout_ns);
  }

  // ---- ragged: the last CTA to finish resets the work counters, so a plan
  // can be reused by the next call without a host step ----
  if (RAGGED) {
    named_sync(kBarConsumers, kConsumerThreads);
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
