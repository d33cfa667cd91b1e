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
//   * the 8 consumer warps form 8/W groups of W warps (W = 1, 2, 4 or 8,
//     chosen per launch from the item size); item `it` goes to group
//     it mod (8/W), so groups work on different items at the same time and
//     one group's waits (its loads, the cluster exchange) overlap the others'
//     work.  In a group, each warp reduces its 1 KiB tiles to tile partials,
//     the warps meet at one named barrier per item, combine the K tile
//     partials of the row in a fixed order (every warp redundantly, so no
//     broadcast is needed), normalise their tiles from the stage, store with
//     128-bit streaming stores and release the stage to the producer.  Which
//     warp handles which tile never changes the arithmetic, so the result
//     does not depend on W.
// Dense MEDIUM rows: one CTA per row.  LARGE rows: the cs CTAs of a cluster
// split the row's tiles into contiguous portions resident in shared memory;
// after pass 1 every CTA signals the others with remote mbarrier arrives,
// reads all K partials through distributed shared memory and combines them
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
constexpr uint32_t kBarConsumers = 1;                // named barrier of all consumer warps
constexpr uint32_t kBarGroup0 = 2;                   // named barrier of consumer group g: 2 + g
constexpr int kSmallSliceBytes = 4096 + 128;         // per-warp staging of a ragged SMALL row
constexpr int kShortCombineTiles = 64;  // rows of up to this many tiles: every warp combines

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
  int group_warps;   // W: consumer warps that share one item (1, 2, 4 or 8)
  int out_vec;
  int gvec;
  uint64_t timeout_ns;
  unsigned int *status;
  // ragged
  const RowRec *rec_small;
  const RowRec *rec_medium;
  const RowRec *rec_large;
  const int32_t *block_counts;  // [blocks][3] rows per bucket of each classify block
  int blocks;                   // classify blocks (0: dense launch)
  int64_t rows_per_block;       // classify block b lists from entry b * rows_per_block on
  unsigned int *counters;       // [3]: next MEDIUM, next SMALL, CTAs finished
  // fused residual add (dense norms): sum_out = in + resid, same layout
  const void *resid;
  void *sum_out;
  int rvec;  // resid and sum_out 16-byte congruent to in
};

struct ItemMeta {
  int64_t start;
  int64_t n;
  int32_t kind;
  int32_t pad[3];
};

// Shared-memory layout of the tile kernel (host and device agree on it).
// Per consumer group: tile partials of split items (part_c) and of items a
// CTA handles alone (part_m), both double-buffered by the parity of the
// group's item count; the two halves of the cooperative combine's scratch
// (blk: the block partials of a long row); the partials of a short split row
// gathered from the peers (gather);
// the cluster barriers ready / released, one per buffer.
struct TileSmemLayout {
  uint32_t part_c, part_m, gather, meta, xw, pref, bar_meta, bar_piece, bar_empty, bar_ready,
      bar_released, flags, total;
  int pieces;
  __host__ __device__ TileSmemLayout(uint32_t stage_bytes, int stages, int max_tiles, int groups,
                                     bool split_items, bool local_items, int blocks) {
    pieces = (max_tiles + kPieceTiles - 1) / kPieceTiles;
    const uint32_t part_bytes = static_cast<uint32_t>(groups) * 2u * max_tiles * 16u;
    uint32_t off = stage_bytes * stages;
    part_c = off;
    off += split_items ? part_bytes : 0u;
    part_m = off;
    off += local_items ? part_bytes : 0u;
    gather = off;
    off += split_items ? static_cast<uint32_t>(groups) * kShortCombineTiles * 16u : 0u;
    meta = off;
    off += stages * 32u;
    xw = off;
    off += static_cast<uint32_t>(groups) * kShortCombineTiles * 16u;
    pref = off;  // ragged: [3][blocks + 1] list position where each classify block starts
    off += (3u * (blocks + 1) * 4u + 15u) & ~15u;
    bar_meta = off;
    off += stages * 8u;
    bar_piece = off;
    off += stages * pieces * 8u;
    bar_empty = off;
    off += stages * 8u;
    bar_ready = off;
    off += static_cast<uint32_t>(groups) * 16u;
    bar_released = off;
    off += static_cast<uint32_t>(groups) * 16u;
    flags = off;
    off += 16u;
    total = off;
  }
};

// Row geometry in chunks and tiles.  Rows are at most rowop_max_row_len()
// elements, so every per-row chunk and tile index fits in 32 bits.
struct ItemGeo {
  int64_t start, n;
  int h;
  int nc, K, t0, t1;
  int cf, cl;  // chunks [cf, cl) are entirely the row's
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
  const int hn = g.h + static_cast<int>(n);
  g.nc = (hn + E - 1) / E;
  g.K = (g.nc + kTileChunks - 1) / kTileChunks;
  if (split) {
    const int tpc = (g.K + cs - 1) / cs;
    g.t0 = min(g.K, rank * tpc);
    g.t1 = min(g.K, g.t0 + tpc);
  } else {
    g.t0 = 0;
    g.t1 = g.K;
  }
  g.cf = (g.h > 0) ? 1 : 0;
  g.cl = ((hn % E) != 0) ? g.nc - 1 : g.nc;
  return g;
}

__device__ __forceinline__ bool tile_is_full(int t, const ItemGeo &g) {
  return t * kTileChunks >= g.cf && (t + 1) * kTileChunks <= g.cl;
}

// ---------------------------------------------------------------------------
// pass 1: tile partials.  One warp reduces tile t (its 64 chunks; lane l
// holds chunks l and l+32) to a tile partial:
//   softmax / log-softmax  (m_t, s_t = sum exp(x - m_t))
//   LayerNorm              (sum_t, mean_t, sum (x - mean_t)^2, n_t)
//   RMSNorm                (sum x^2)
// A warp takes up to PB (4 or 2) of its tiles at once, so several
// independent shuffle chains are in flight.
// ---------------------------------------------------------------------------

struct TileMask {
  int lo0, hi0, lo1, hi1;  // valid element ranges of the lane's two chunks
};

template <typename T>
__device__ __forceinline__ TileMask tile_mask(int t, const ItemGeo &g, int lane, bool full) {
  constexpr int E = Elem<T>::kPerChunk;
  TileMask m{0, E, 0, E};
  if (!full) {
    const int hn = g.h + static_cast<int>(g.n);
    const int c0 = t * kTileChunks + lane;
    const int c1 = c0 + 32;
    if (c0 < g.nc) chunk_valid_range(c0, g.nc, g.h, hn, E, m.lo0, m.hi0); else m.lo0 = m.hi0 = 0;
    if (c1 < g.nc) chunk_valid_range(c1, g.nc, g.h, hn, E, m.lo1, m.hi1); else m.lo1 = m.hi1 = 0;
  }
  return m;
}

// first lane-level statistic of a tile from the lane's two chunks (chunk l,
// then chunk l+32) as fp32 pairs: max (softmax family), sum (LayerNorm), sum
// of squares (RMSNorm)
template <int OP, int NP>
__device__ __forceinline__ float tile_pairs_first(const f2 (&p0)[NP], const f2 (&p1)[NP],
                                                  const TileMask &m) {
  if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
    return chunk_max<NP>(p1, chunk_max<NP>(p0, -INFINITY, m.lo0, m.hi0), m.lo1, m.hi1);
  } else if constexpr (OP == kLayerNorm) {
    return f2_total(chunk_sum<NP>(p1, chunk_sum<NP>(p0, f2_bcast(0.f), m.lo0, m.hi0), m.lo1, m.hi1));
  } else {
    return f2_total(
        chunk_sum_sq<NP>(p1, chunk_sum_sq<NP>(p0, f2_bcast(0.f), m.lo0, m.hi0), m.lo1, m.hi1));
  }
}

// second lane-level statistic: sum exp(x - ref) (softmax family, ref = m_t)
// or sum (x - ref)^2 (LayerNorm, ref = mean_t)
template <int OP, int NP>
__device__ __forceinline__ float tile_pairs_second(const f2 (&p0)[NP], const f2 (&p1)[NP],
                                                   const TileMask &m, float ref) {
  const f2 r2 = f2_bcast(ref);
  if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
    if (ref == -INFINITY) return 0.f;  // no element of the tile is above -inf
    return f2_total(chunk_sum_exp<NP>(p1, r2, chunk_sum_exp<NP>(p0, r2, f2_bcast(0.f), m.lo0, m.hi0),
                                      m.lo1, m.hi1));
  } else {
    return f2_total(chunk_sum_sqdev<NP>(p1, r2, chunk_sum_sqdev<NP>(p0, r2, f2_bcast(0.f), m.lo0, m.hi0),
                                        m.lo1, m.hi1));
  }
}

// The lane's two chunks of a staged tile as fp32 pairs.
template <typename T>
__device__ __forceinline__ void tile_lane_pairs(const unsigned char *tsm, int lane,
                                                f2 (&p0)[Elem<T>::kPerChunk / 2],
                                                f2 (&p1)[Elem<T>::kPerChunk / 2]) {
  chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(tsm + lane * kChunkBytes), p0);
  chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(tsm + (lane + 32) * kChunkBytes), p1);
}

template <int OP, typename T>
__device__ __forceinline__ float tile_lane_first(const unsigned char *tsm, const TileMask &m,
                                                 int lane) {
  constexpr int NP = Elem<T>::kPerChunk / 2;
  f2 p0[NP], p1[NP];
  tile_lane_pairs<T>(tsm, lane, p0, p1);
  return tile_pairs_first<OP, NP>(p0, p1, m);
}

template <int OP, typename T>
__device__ __forceinline__ float tile_lane_second(const unsigned char *tsm, const TileMask &m,
                                                  int lane, float ref) {
  constexpr int NP = Elem<T>::kPerChunk / 2;
  f2 p0[NP], p1[NP];
  tile_lane_pairs<T>(tsm, lane, p0, p1);
  return tile_pairs_second<OP, NP>(p0, p1, m, ref);
}

// B tiles of one warp, lt0, lt0 + W, ..., lt0 + W(B-1), all below the item's
// tile count (W = warps of the group): lane-level sums of all of them first,
// then their butterflies interleaved.  FULL: the caller checked that every
// one of them lies entirely in the row, so no element masks are evaluated
// (same arithmetic: the masks of a full tile keep every element).  Waits on
// each stage piece before the first tile read from it (`waited` is the last
// piece waited for); returns false when such a wait ran out.
// Fused residual add for this lane's two chunks of tile t, in the stage:
// each becomes the stored sum x + r (written to sum_out too), so the
// statistics and pass 2 read the sum as stored.
template <typename T>
__device__ __forceinline__ void residual_tile(unsigned char *tsm, int t, const ItemGeo &g,
                                              int lane, const TileParams &p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  const T *r_row = static_cast<const T *>(p.resid) + g.start;
  T *s_row = static_cast<T *>(p.sum_out) + g.start;
  const char *rwin = reinterpret_cast<const char *>(r_row) - g.h * SZ;
  char *swin = reinterpret_cast<char *>(s_row) - g.h * SZ;
  const int hn = g.h + static_cast<int>(g.n);
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int c = t * kTileChunks + lane + 32 * u;
    if (c >= g.nc) continue;
    uint4 *slot = reinterpret_cast<uint4 *>(tsm + (lane + 32 * u) * kChunkBytes);
    int lo, hi;
    chunk_valid_range(c, g.nc, g.h, hn, E, lo, hi);
    *slot = residual_chunk<T>(*slot, r_row, s_row, rwin, swin, c, g.h, lo, hi, g.n, p.rvec != 0);
  }
}

template <int OP, typename T, int B, bool FULL, bool RESID, bool ONLINE = false>
__device__ __forceinline__ bool pass1_batch(const unsigned char *stage, const ItemGeo &g, int lt0,
                                            int W, int lane, float4 *part, uint32_t piece_bar0,
                                            uint32_t par, uint64_t timeout_ns, int &waited,
                                            const TileParams &p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr bool kMaxFirst = (OP == kSoftmax || OP == kLogSoftmax);
  float a[B], b[B];
  static_assert(!(RESID && ONLINE), "the residual add serves the norms only");
  if constexpr (kMaxFirst && ONLINE) {
    // Online statistics: each lane reads its two chunks of the tile from the
    // stage once, forms their maximum and the sum of exp about it from those
    // registers, and the lanes merge their (m, s) pairs by the rescaling
    // butterfly -- one sweep over shared memory instead of two.
    constexpr int NP = E / 2;
#pragma unroll
    for (int q = 0; q < B; ++q) {
      const int lt = lt0 + q * W;
      const int pc = lt / kPieceTiles;
      if (pc != waited) {
        if (!mbar_wait_bounded(piece_bar0 + 8u * pc, par, timeout_ns)) return false;
        waited = pc;
      }
      const int t = g.t0 + lt;
      const TileMask m = FULL ? TileMask{0, E, 0, E} : tile_mask<T>(t, g, lane, tile_is_full(t, g));
      const unsigned char *tsm = stage + lt * kTileBytes;
      f2 p0[NP], p1[NP];
      chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(tsm + lane * kChunkBytes), p0);
      chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(tsm + (lane + 32) * kChunkBytes), p1);
      a[q] = chunk_max<NP>(p1, chunk_max<NP>(p0, -INFINITY, m.lo0, m.hi0), m.lo1, m.hi1);
      const f2 r2 = f2_bcast(a[q]);
      b[q] = a[q] == -INFINITY
                 ? 0.f
                 : f2_total(chunk_sum_exp<NP>(p1, r2, chunk_sum_exp<NP>(p0, r2, f2_bcast(0.f), m.lo0, m.hi0),
                                              m.lo1, m.hi1));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
      for (int q = 0; q < B; ++q) {
        const float m2 = __shfl_xor_sync(kFullMask, a[q], o);
        const float s2 = __shfl_xor_sync(kFullMask, b[q], o);
        online_merge(a[q], b[q], m2, s2);
      }
    }
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < B; ++q) part[lt0 + q * W] = make_float4(a[q], b[q], 0.f, 0.f);
    }
    return true;
  }
  // one tile at a time (the fused ragged kernel): the lane's pairs stay in
  // registers for the second sweep; larger batches read the stage again
  // (keeping them would spill)
  constexpr int NP = E / 2;
  constexpr bool kKeep = (OP != kRmsNorm) && B == 1;
  f2 kp0[kKeep ? B : 1][NP], kp1[kKeep ? B : 1][NP];
#pragma unroll
  for (int q = 0; q < B; ++q) {
    const int lt = lt0 + q * W;
    const int pc = lt / kPieceTiles;
    if (pc != waited) {
      if (!mbar_wait_bounded(piece_bar0 + 8u * pc, par, timeout_ns)) return false;
      waited = pc;
    }
    const int t = g.t0 + lt;
    if constexpr (RESID)
      residual_tile<T>(const_cast<unsigned char *>(stage) + lt * kTileBytes, t, g, lane, p);
    const TileMask m = FULL ? TileMask{0, E, 0, E} : tile_mask<T>(t, g, lane, tile_is_full(t, g));
    if constexpr (kKeep) {
      tile_lane_pairs<T>(stage + lt * kTileBytes, lane, kp0[q], kp1[q]);
      a[q] = tile_pairs_first<OP, NP>(kp0[q], kp1[q], m);
    } else {
      a[q] = tile_lane_first<OP, T>(stage + lt * kTileBytes, m, lane);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
    for (int q = 0; q < B; ++q) {
      const float y = __shfl_xor_sync(kFullMask, a[q], o);
      a[q] = kMaxFirst ? fmaxf(a[q], y) : __fadd_rn(a[q], y);
    }
  }
  if constexpr (OP == kRmsNorm) {
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < B; ++q) part[lt0 + q * W] = make_float4(a[q], 0.f, 0.f, 0.f);
    }
  } else {
    float ref[B], ntf[B];
#pragma unroll
    for (int q = 0; q < B; ++q) {
      const int lt = lt0 + q * W;
      const int t = g.t0 + lt;
      const bool full = FULL || tile_is_full(t, g);
      ref[q] = a[q];
      ntf[q] = 0.f;
      if constexpr (OP == kLayerNorm) {
        if (full) {
          ntf[q] = static_cast<float>(kTileChunks * E);
          ref[q] = __fmul_rn(a[q], 1.f / static_cast<float>(kTileChunks * E));  // exact
        } else {
          const int hn = g.h + static_cast<int>(g.n);
          const int w0 = t * kTileChunks * E;
          const int w1 = min(g.nc, (t + 1) * kTileChunks) * E;
          const int nt = max(0, min(hn, w1) - max(g.h, w0));
          ntf[q] = static_cast<float>(nt);
          ref[q] = nt > 0 ? __fdiv_rn(a[q], ntf[q]) : 0.f;
        }
      }
      const TileMask m = FULL ? TileMask{0, E, 0, E} : tile_mask<T>(t, g, lane, full);
      if constexpr (kKeep) {
        b[q] = tile_pairs_second<OP, NP>(kp0[q], kp1[q], m, ref[q]);
      } else {
        b[q] = tile_lane_second<OP, T>(stage + lt * kTileBytes, m, lane, ref[q]);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
      for (int q = 0; q < B; ++q) b[q] = __fadd_rn(b[q], __shfl_xor_sync(kFullMask, b[q], o));
    }
  if (lane == 0) {
#pragma unroll
      for (int q = 0; q < B; ++q)
        part[lt0 + q * W] = (OP == kLayerNorm) ? make_float4(a[q], ref[q], b[q], ntf[q])
                                                            : make_float4(a[q], b[q], 0.f, 0.f);
    }
  }
  return true;
}

// Pass 1 of an item for warp `wig` of a group of W warps: part[lt] for its
// tiles lt = wig, wig + W, ..., taken PB at a time while that many remain,
// then in a batch of two and one.  Each tile's arithmetic (and its butterfly
// order) is the same whatever batch it falls in.
template <int OP, typename T, int PB, bool RESID, bool ONLINE = false>
__device__ __forceinline__ bool pass1_warp(const unsigned char *stage, const ItemGeo &g, int wig,
                                           int W, int lane, float4 *part, uint32_t piece_bar0,
                                           uint32_t par, uint64_t timeout_ns, const TileParams &p) {
  const int ntl = g.t1 - g.t0;
  // tiles [full0, full1) of the row lie entirely in it (all but its ends)
  const int full0 = g.cf > 0 ? 1 : 0;
  const int full1 = g.cl / kTileChunks;
  int waited = -1;
  int lt0 = wig;
  while (lt0 < ntl) {
    const int left = (ntl - lt0 + W - 1) >> (31 - __clz(W));  // W is a power of two
    const int bsz = left >= PB ? PB : (left >= 2 ? 2 : 1);
    const int ta = g.t0 + lt0, tb = ta + (bsz - 1) * W;
    const bool full = ta >= full0 && tb < full1;
    bool ok;
    if (PB > 2 && bsz == PB) {
      ok = full ? pass1_batch<OP, T, PB, true, RESID, ONLINE>(stage, g, lt0, W, lane, part, piece_bar0, par,
                                               timeout_ns, waited, p)
                : pass1_batch<OP, T, PB, false, RESID, ONLINE>(stage, g, lt0, W, lane, part, piece_bar0, par,
                                                timeout_ns, waited, p);
    } else if (bsz == 2) {
      ok = full ? pass1_batch<OP, T, 2, true, RESID, ONLINE>(stage, g, lt0, W, lane, part, piece_bar0, par,
                                              timeout_ns, waited, p)
                : pass1_batch<OP, T, 2, false, RESID, ONLINE>(stage, g, lt0, W, lane, part, piece_bar0, par,
                                               timeout_ns, waited, p);
    } else {
      ok = full ? pass1_batch<OP, T, 1, true, RESID, ONLINE>(stage, g, lt0, W, lane, part, piece_bar0, par,
                                              timeout_ns, waited, p)
                : pass1_batch<OP, T, 1, false, RESID, ONLINE>(stage, g, lt0, W, lane, part, piece_bar0, par,
                                               timeout_ns, waited, p);
    }
    if (!ok) return false;
    lt0 += bsz * W;
  }
  return true;
}

// ---------------------------------------------------------------------------
// combine: the row statistics from its K tile partials part[0..K), in a fixed
// order that depends on K only.
//   K <= 64: lane l of a warp takes t = l, l+32 in turn, then a 5-level
//            butterfly; every warp computes it, so nothing is broadcast.
//   K > 64:  blocks of 64 consecutive tiles: each block's partial as for
//            K <= 64 (the group's warps share the blocks), then the block
//            partials the same way (combine_blocks).
// (s0, s1): softmax (M, 1/S), log-softmax (M, log S), LayerNorm (mu, rstd),
// RMSNorm (-, rstd).
// ---------------------------------------------------------------------------
template <int OP>
__device__ __forceinline__ void finish_stats(float first, float second, float inv_n, float eps,
                                             float &s0, float &s1) {
  if constexpr (OP == kSoftmax) {
    s0 = first;
    s1 = __frcp_rn(second);
  } else if constexpr (OP == kLogSoftmax) {
    s0 = first;
    s1 = logf(second);
  } else if constexpr (OP == kLayerNorm) {
    s0 = first;  // the mean
    s1 = rsqrtf(__fadd_rn(__fmul_rn(second, inv_n), eps));
  } else {
    s0 = 0.f;
    s1 = rsqrtf(__fadd_rn(__fmul_rn(first, inv_n), eps));
  }
}

// per-partial terms of the second sweep
template <int OP>
__device__ __forceinline__ float second_term(const float4 &pt, float first) {
  if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
    return pt.x == -INFINITY ? 0.f : __fmul_rn(pt.y, exp_shifted(pt.x, first));
  } else {
    const float d = __fsub_rn(pt.y, first);
    return __fmaf_rn(__fmul_rn(pt.w, d), d, pt.z);
  }
}

// `get(t)` returns tile partial t (from this CTA's shared memory, or from a
// peer's through distributed shared memory).
template <int OP, class Get>
__device__ __forceinline__ void combine_short(Get get, int K, float inv_n, float eps, int lane,
                                              float &s0, float &s1) {
  constexpr bool kMax = (OP == kSoftmax || OP == kLogSoftmax);
  const float4 z = make_float4(kMax ? -INFINITY : 0.f, 0.f, 0.f, 0.f);
  const float4 p0 = lane < K ? get(lane) : z;
  const float4 p1 = lane + 32 < K ? get(lane + 32) : z;
  float first;
  if constexpr (kMax) {
    first = warp_max(fmaxf(p0.x, p1.x));
  } else {
    first = warp_sum(__fadd_rn(p0.x, p1.x));
    if constexpr (OP == kLayerNorm) first = __fmul_rn(first, inv_n);
  }
  float second = 0.f;
  if constexpr (OP != kRmsNorm) {
    float v = lane < K ? second_term<OP>(p0, first) : 0.f;
    if (lane + 32 < K) v = __fadd_rn(v, second_term<OP>(p1, first));
    second = warp_sum(v);
  }
  finish_stats<OP>(first, second, inv_n, eps, s0, s1);
}

// Rows of more than 64 tiles: the tiles fall into blocks of 64 consecutive
// tiles.  Level 1: each block's partial is formed from its tile partials the
// way a short row's statistics are (lane l takes the block's tiles l and
// l+32, then butterflies): softmax (M_b, S_b), LayerNorm (sum_b, mean_b, Q_b,
// n_b) with Q_b = sum over the block's tiles of Q_t + n_t (mu_t - mean_b)^2
// (Chan's merge), RMSNorm the block's sum of squares.  The W warps of the
// group take blocks wig, wig + W, ... (two at a time, so their partials are
// fetched together) and leave the block partials in blk[].  Level 2: after
// the group's named barrier `bar`, every warp combines the block partials as
// combine_short combines tile partials.  The order depends on K only.
template <int OP>
__device__ __forceinline__ float4 block_partial(const float4 &p0, const float4 &p1, bool h0,
                                                bool h1) {
  constexpr bool kMax = (OP == kSoftmax || OP == kLogSoftmax);
  float first;
  if constexpr (kMax) {
    first = warp_max(fmaxf(p0.x, p1.x));
  } else {
    first = warp_sum(__fadd_rn(p0.x, p1.x));
  }
  if constexpr (OP == kRmsNorm) {
    return make_float4(first, 0.f, 0.f, 0.f);
  } else if constexpr (OP == kLayerNorm) {
    const float nb = warp_sum(__fadd_rn(p0.w, p1.w));  // element count: exact
    const float mean = nb > 0.f ? __fdiv_rn(first, nb) : 0.f;
    float v = h0 ? second_term<OP>(p0, mean) : 0.f;
    if (h1) v = __fadd_rn(v, second_term<OP>(p1, mean));
    return make_float4(first, mean, warp_sum(v), nb);
  } else {
    float v = h0 ? second_term<OP>(p0, first) : 0.f;
    if (h1) v = __fadd_rn(v, second_term<OP>(p1, first));
    return make_float4(first, warp_sum(v), 0.f, 0.f);
  }
}

template <int OP, class Get>
__device__ __forceinline__ void combine_blocks(Get get, int K, float inv_n, float eps, int lane,
                                               int wig, int W, uint32_t bar, float4 *blk,
                                               float &s0, float &s1) {
  constexpr bool kMax = (OP == kSoftmax || OP == kLogSoftmax);
  const float4 z = make_float4(kMax ? -INFINITY : 0.f, 0.f, 0.f, 0.f);
  const int nb = (K + kShortCombineTiles - 1) / kShortCombineTiles;
  for (int b0 = wig; b0 < nb; b0 += 2 * W) {
    float4 q[2][2];
    bool h[2][2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int bb = b0 + u * W;
      const int kb = bb < nb ? min(kShortCombineTiles, K - kShortCombineTiles * bb) : 0;
      h[u][0] = lane < kb;
      h[u][1] = lane + 32 < kb;
      q[u][0] = h[u][0] ? get(kShortCombineTiles * bb + lane) : z;
      q[u][1] = h[u][1] ? get(kShortCombineTiles * bb + lane + 32) : z;
    }
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int bb = b0 + u * W;
      if (bb < nb) {  // the same for every lane of the warp
        const float4 r = block_partial<OP>(q[u][0], q[u][1], h[u][0], h[u][1]);
        if (lane == 0) blk[bb] = r;
      }
    }
  }
  named_sync(bar, static_cast<uint32_t>(W) * 32u);
  combine_short<OP>([&](int t) { return blk[t]; }, nb, inv_n, eps, lane, s0, s1);
}

// gamma/beta chunk for window chunk c of a row with compile-time head offset
// H; every column it covers is inside [0, glen) and the vector is 16-byte
// aligned (the caller checked).
template <typename T, int H>
__device__ __forceinline__ uint4 param_chunk_fixed(const T *__restrict__ g, int c) {
  constexpr int E = Elem<T>::kPerChunk;
  const uint4 *v = reinterpret_cast<const uint4 *>(g);
  if constexpr (H == 0) {
    return __ldg(v + c);
  } else {
    const uint4 A = __ldg(v + (c - 1));
    const uint4 B = __ldg(v + c);
    if constexpr (E == 4) {
      return shift_words<H>(A, B);
    } else if constexpr ((H & 1) == 0) {
      return shift_words<H / 2>(A, B);
    } else {
      return shift_half<(H + 1) / 2>(A, B);
    }
  }
}

// pass 2 fast path for one chunk: entirely the row's, output 16-byte
// congruent to the input, gamma/beta aligned and covering its columns.  Same
// arithmetic as chunk_store_edge.
template <int OP, typename T, int H, bool P>
__device__ __forceinline__ void chunk_store_fast(const unsigned char *csm, int c, float s0,
                                                 float s1, const T *gamma, const T *beta,
                                                 char *owin) {
  constexpr int NP = Elem<T>::kPerChunk / 2;
  f2 v[NP], g[NP], b[NP];
  chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(csm), v);
  if constexpr (!P) {
#pragma unroll
    for (int i = 0; i < NP; ++i) {
      g[i] = f2_bcast(1.f);
      b[i] = f2_bcast(0.f);
    }
  } else {
    if constexpr (OP == kLayerNorm || OP == kRmsNorm)
      chunk_to_pairs<T>(param_chunk_fixed<T, H>(gamma, c), g);
    if constexpr (OP == kLayerNorm) chunk_to_pairs<T>(param_chunk_fixed<T, H>(beta, c), b);
  }
  normalize_pairs<OP, NP>(v, s0, s1, g, b);
  stg_stream(owin + static_cast<int64_t>(c) * kChunkBytes, pairs_to_chunk<T>(v));
}

// pass 2, one chunk the fast path does not take: a row end the row only
// partly covers, output not 16-byte congruent to the input, or gamma/beta
// unaligned, absent or ending inside the chunk's window.  Elements outside
// the row are masked and stored element by element.  Parameters come as
// aligned vectors realigned for the compile-time head offset H (columns
// before 0 read as zero and are masked) whenever they are aligned and reach
// past the chunk, else element by element.
template <int OP, typename T, int H>
__device__ __forceinline__ void chunk_store_edge(const unsigned char *csm, int c, const ItemGeo &g,
                                                 float s0, float s1, const TileParams &p,
                                                 char *owin, T *out_row) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr bool kAffine = (OP == kLayerNorm || OP == kRmsNorm);
  const int hn = g.h + static_cast<int>(g.n);
  const T *gamma = static_cast<const T *>(p.gamma);
  const T *beta = static_cast<const T *>(p.beta);
  f2 v[NP], gp[NP], bp[NP];
  chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(csm), v);
  int lo, hi;
  chunk_valid_range(c, g.nc, g.h, hn, E, lo, hi);
  if constexpr (kAffine) {
    const bool vec = p.gvec && gamma && (OP == kRmsNorm || beta) && g.h == H &&
                     static_cast<int64_t>(c + 1) * E <= p.glen;
    if (vec) {
      auto realigned = [&](const T *a) {
        const uint4 *w = reinterpret_cast<const uint4 *>(a);
        if constexpr (H == 0) {
          return __ldg(w + c);
        } else {
          const uint4 A = c > 0 ? __ldg(w + (c - 1)) : make_uint4(0u, 0u, 0u, 0u);
          const uint4 B = __ldg(w + c);
          if constexpr (E == 4) {
            return shift_words<H>(A, B);
          } else if constexpr ((H & 1) == 0) {
            return shift_words<H / 2>(A, B);
          } else {
            return shift_half<(H + 1) / 2>(A, B);
          }
        }
      };
      chunk_to_pairs<T>(realigned(gamma), gp);
      if constexpr (OP == kLayerNorm) chunk_to_pairs<T>(realigned(beta), bp);
    } else {
      load_param_pairs<T>(gamma, gamma ? p.glen : 0, c, g.h, p.gvec != 0, 1.f, gp);
      if constexpr (OP == kLayerNorm)
        load_param_pairs<T>(beta, beta ? p.glen : 0, c, g.h, p.gvec != 0, 0.f, bp);
    }
  }
  normalize_pairs<OP, NP>(v, s0, s1, gp, bp);
  store_chunk<T>(v, owin, out_row, c, g.h, lo, hi, p.out_vec != 0);
}

// gamma/beta chunk at v (16-byte aligned vectors, v = chunk c of the
// parameter array) realigned for head offset H: columns c E - H .. c E - H +
// E - 1, from chunks c - 1 and c.
template <typename T, int H>
__device__ __forceinline__ uint4 param_chunk_at(const uint4 *__restrict__ v) {
  constexpr int E = Elem<T>::kPerChunk;
  if constexpr (H == 0) {
    return __ldg(v);
  } else {
    const uint4 A = __ldg(v - 1);
    const uint4 B = __ldg(v);
    if constexpr (E == 4) {
      return shift_words<H>(A, B);
    } else if constexpr ((H & 1) == 0) {
      return shift_words<H / 2>(A, B);
    } else {
      return shift_half<(H + 1) / 2>(A, B);
    }
  }
}

// Both chunks of a lane in a tile made only of fast chunks (see
// chunk_store_fast), c0 the lane's first chunk: every address is formed once
// for the tile and the second chunk (c0 + 32) is reached by a fixed offset.
// P: gamma (and beta) are present; without them (P false) the norms take
// gamma = 1 and beta = 0, as the general path does.
template <int OP, typename T, int H, bool P>
__device__ __forceinline__ void tile_store_fast(const unsigned char *lsm, int c0, float s0,
                                                float s1, const T *gamma, const T *beta,
                                                char *owin) {
  constexpr int NP = Elem<T>::kPerChunk / 2;
  const uint4 *gv = reinterpret_cast<const uint4 *>(gamma) + c0;
  const uint4 *bv = reinterpret_cast<const uint4 *>(beta) + c0;
  uint4 *ov = reinterpret_cast<uint4 *>(owin) + c0;
  f2 v[2][NP], g[2][NP], b[2][NP];
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(lsm + 32 * u * kChunkBytes), v[u]);
    if constexpr (!P) {
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        g[u][i] = f2_bcast(1.f);
        b[u][i] = f2_bcast(0.f);
      }
    } else {
      if constexpr (OP == kLayerNorm || OP == kRmsNorm)
        chunk_to_pairs<T>(param_chunk_at<T, H>(gv + 32 * u), g[u]);
      if constexpr (OP == kLayerNorm) chunk_to_pairs<T>(param_chunk_at<T, H>(bv + 32 * u), b[u]);
    }
  }
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    normalize_pairs<OP, NP>(v[u], s0, s1, g[u], b[u]);
    stg_stream(ov + 32 * u, pairs_to_chunk<T>(v[u]));
  }
}

// pass 2 over this warp's tiles (wig, wig + W, ...) of an item whose head
// offset is H.  Chunks [g.cf, cfast) take the fast path, the row's other
// chunks the general one: tiles made only of fast chunks (all but the row's
// ends, as a rule) run first with both chunks of a lane issued together, then
// the remaining tiles chunk by chunk.
template <int OP, typename T, int H, bool P>
__device__ __forceinline__ void pass2_tiles(const unsigned char *stage, const ItemGeo &g, int wig,
                                            int W, int lane, float s0, float s1,
                                            const TileParams &p, char *owin, T *out_row,
                                            int cfast) {
  const T *gamma = static_cast<const T *>(p.gamma);
  const T *beta = static_cast<const T *>(p.beta);
  const int ntl = g.t1 - g.t0;
  // tiles [fa, fb) of the row hold only fast chunks
  const int fa = (g.cf + kTileChunks - 1) / kTileChunks;
  const int fb = cfast / kTileChunks;
  for (int lt = wig; lt < ntl; lt += W) {
    const int t = g.t0 + lt;
    if (t < fa || t >= fb) continue;
    tile_store_fast<OP, T, H, P>(stage + lt * kTileBytes + lane * kChunkBytes,
                                 t * kTileChunks + lane, s0, s1, gamma, beta, owin);
  }
  for (int lt = wig; lt < ntl; lt += W) {
    const int t = g.t0 + lt;
    if (t >= fa && t < fb) continue;
    for (int u = 0; u < 2; ++u) {
      const int c = t * kTileChunks + lane + 32 * u;
      const unsigned char *csm = stage + lt * kTileBytes + (lane + 32 * u) * kChunkBytes;
      if (c >= g.cf && c < cfast) {
        chunk_store_fast<OP, T, H, P>(csm, c, s0, s1, gamma, beta, owin);
      } else if (c < g.nc) {
        chunk_store_edge<OP, T, H>(csm, c, g, s0, s1, p, owin, out_row);
      }
    }
  }
}

// pass 2 of an item, with the gamma/beta realignment compiled for the item's
// head offset (one dispatch per item, not per chunk).
template <int OP, typename T, bool EXACT>
__device__ __forceinline__ void pass2_item(const unsigned char *stage, const ItemGeo &g, int wig,
                                           int W, int lane, float s0, float s1,
                                           const TileParams &p, char *owin, T *out_row) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr bool kAffine = (OP == kLayerNorm || OP == kRmsNorm);
  // no parameters at all: gamma = 1 and beta = 0 without loads
  const bool none = kAffine && !p.gamma && !p.beta;
  const bool params_ok =
      !kAffine || none || (p.gvec && p.gamma && (OP == kRmsNorm || p.beta != nullptr));
  // fast chunks end where the row's full chunks end, or where the vector
  // parameter loads would reach past gamma/beta (they read up to column
  // (c + 1) * E - 1 for chunk c)
  int cfast = g.cf;
  if (p.out_vec && params_ok)
    cfast = (kAffine && !none) ? static_cast<int>(min(static_cast<int64_t>(g.cl), p.glen / E))
                               : g.cl;
  if (!kAffine || none) {
    pass2_tiles<OP, T, 0, false>(stage, g, wig, W, lane, s0, s1, p, owin, out_row, cfast);
  } else if constexpr (EXACT) {
    pass2_tiles<OP, T, 0, true>(stage, g, wig, W, lane, s0, s1, p, owin, out_row, cfast);
  } else {
    switch (g.h) {
      case 0: pass2_tiles<OP, T, 0, true>(stage, g, wig, W, lane, s0, s1, p, owin, out_row, cfast); break;
      case 1: pass2_tiles<OP, T, 1, true>(stage, g, wig, W, lane, s0, s1, p, owin, out_row, cfast); break;
      case 2: pass2_tiles<OP, T, 2, true>(stage, g, wig, W, lane, s0, s1, p, owin, out_row, cfast); break;
      case 3: pass2_tiles<OP, T, 3, true>(stage, g, wig, W, lane, s0, s1, p, owin, out_row, cfast); break;
      default:
        if constexpr (E == 8) {
          switch (g.h) {
            case 4: pass2_tiles<OP, T, 4, true>(stage, g, wig, W, lane, s0, s1, p, owin, out_row, cfast); break;
            case 5: pass2_tiles<OP, T, 5, true>(stage, g, wig, W, lane, s0, s1, p, owin, out_row, cfast); break;
            case 6: pass2_tiles<OP, T, 6, true>(stage, g, wig, W, lane, s0, s1, p, owin, out_row, cfast); break;
            default: pass2_tiles<OP, T, 7, true>(stage, g, wig, W, lane, s0, s1, p, owin, out_row, cfast); break;
          }
        }
        break;
    }
  }
}

// ---------------------------------------------------------------------------
// producer: one warp.  Lane 0 owns the ring (stage barriers, item records);
// the lanes share the per-item work so that no step waits on another:
//   * ragged records are claimed in batches and looked up one per lane (the
//     LARGE rows of this CTA up to 32 at a time, the MEDIUM rows
//     kFetchBatch per work-counter step), so one round trip serves several
//     items;
//   * lane pc issues piece pc's bulk copy;
//   * the at most two 16-byte chunks a row only partly covers are read one
//     element per lane (all loads in flight together) and written into the
//     stage after the next item's record is in hand, so their latency
//     overlaps that lookup.
// ---------------------------------------------------------------------------
constexpr int kFetchBatch = 4;  // MEDIUM rows one work-counter step claims

// Record `idx` of a bucket's list: the classify block b with
// pref[b] <= idx < pref[b + 1] wrote it at entry b * rows_per_block +
// (idx - pref[b]) of the list (pref: that bucket's [blocks + 1] starts).
__device__ __forceinline__ RowRec ragged_record(const TileParams &p, const int *pref,
                                                const RowRec *list, int64_t idx) {
  int lo = 0, hi = p.blocks;  // pref[lo] <= idx < pref[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (pref[mid] <= idx) {
      lo = mid;
    } else {
      hi = mid;
    }
  }
  return list[static_cast<int64_t>(lo) * p.rows_per_block + (idx - pref[lo])];
}

// A record taken from bucket b's list fits the call that uses it: a row of
// at least one and at most glen elements whose bucket, for this call's
// element type, is b.  A plan made by rowop_ragged_plan for another element
// type or a longer max_len than the planned call's fails this for some rows;
// they are skipped (left untouched) and flagged as rejected rows, and never
// staged past a buffer sized for this call.
template <typename T>
__device__ __forceinline__ bool ragged_record_fits(const RowRec &r, int b, int64_t glen) {
  return r.n >= 1 && r.n <= glen && bucket_of(r.n, Elem<T>::kSize) == b;
}

// The edge elements of an item, one per lane: lanes [0, E) the head chunk
// (window chunk 0), lanes [E, 2E) the tail chunk (the last one), each
// element read only when it lies in the row (zero otherwise), written into
// the stage later.  The chunks' pieces are complete when lane 0 arrives on
// their barriers after the writes.
struct EdgeLanes {
  bool active;              // (uniform) an item's edges are still to be written
  bool mine;                // this lane writes an element
  bool head, tail, tail_own_bar;  // (uniform)
  uint32_t dst;             // this lane's element in the stage
  uint32_t val;             // its bits
  uint32_t head_bar, tail_bar;    // (uniform)
};

template <typename T>
__device__ __forceinline__ void edges_write(EdgeLanes &e, int lane) {
  if (!e.active) return;
  if (e.mine) {
    if constexpr (sizeof(T) == 2) {
      asm volatile("st.shared.u16 [%0], %1;" ::"r"(e.dst), "h"(static_cast<unsigned short>(e.val))
                   : "memory");
    } else {
      asm volatile("st.shared.u32 [%0], %1;" ::"r"(e.dst), "r"(e.val) : "memory");
    }
  }
  __syncwarp();
  if (lane == 0) {
    if (e.head) mbar_arrive(e.head_bar);
    if (e.tail && (e.tail_own_bar || !e.head)) mbar_arrive(e.tail_bar);
  }
  e.active = false;
}

template <typename T, bool EXACT, bool CLUSTER, bool RAGGED>
__device__ __forceinline__ void tile_producer(const TileParams &p, const TileSmemLayout &L,
                                              unsigned char *smem, int cs, int rank, int64_t cid,
                                              int64_t ncl, int lane) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  const int S = p.stages;
  const int G = kConsumerWarps / p.group_warps;  // every group gets an end-of-work item
  int ends = 0;
  const uint32_t sbase = smem_addr(smem);
  ItemMeta *meta = reinterpret_cast<ItemMeta *>(smem + L.meta);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + L.flags);
  const uint64_t pol = l2_evict_first_policy();
  const int *pref = reinterpret_cast<const int *>(smem + L.pref);
  const int nb1 = p.blocks + 1;
  int64_t k_large = 0, k_dense = 0;
  bool medium_phase = false;
  EdgeLanes edges;
  edges.active = false;
  uint32_t fill_mask = 0, fill_parity = 0;

  // the current batch of ragged records: lane k holds record k
  RowRec mine;
  mine.start = 0;
  mine.n = 0;
  int qn = 0, qi = 0, qkind = kItemEnd;
  auto refill = [&]() {
    qn = 0;
    qi = 0;
    if (!medium_phase) {
      const int64_t nl = pref[2 * nb1 + p.blocks];
      const int64_t li0 = cid + k_large * ncl;
      if (li0 < nl) {
        const int cnt = static_cast<int>(min(static_cast<int64_t>(32), (nl - li0 + ncl - 1) / ncl));
        if (lane < cnt) mine = ragged_record(p, pref + 2 * nb1, p.rec_large, li0 + lane * ncl);
        k_large += cnt;
        qn = cnt;
        qkind = kItemLarge;
        return;
      }
      medium_phase = true;
    }
    const int64_t nm = pref[nb1 + p.blocks];
    unsigned int m = 0;
    if (lane == 0) m = atomicAdd(&p.counters[0], static_cast<unsigned int>(kFetchBatch));
    const int64_t m0 = __shfl_sync(kFullMask, m, 0);
    if (m0 >= nm) return;  // no rows left: the end of this CTA's work
    const int cnt = static_cast<int>(min(static_cast<int64_t>(kFetchBatch), nm - m0));
    if (lane < cnt) mine = ragged_record(p, pref + nb1, p.rec_medium, m0 + lane);
    qn = cnt;
    qkind = kItemMedium;
  };
  // The next item of this CTA (the same on every lane).
  auto fetch = [&](int &kind, int64_t &start, int64_t &n) {
    kind = kItemEnd;
    start = 0;
    n = 0;
    if (RAGGED) {
      for (;;) {
        if (qi == qn) {
          refill();
          if (qn == 0) return;
        }
        RowRec r;
        r.start = __shfl_sync(kFullMask, mine.start, qi);
        r.n = __shfl_sync(kFullMask, mine.n, qi);
        ++qi;
        if (!ragged_record_fits<T>(r, qkind == kItemLarge ? kLarge : kMedium, p.glen)) {
          if (lane == 0) atomicOr(p.status, kStatusBadOffsets);
          continue;
        }
        kind = qkind;
        start = r.start;
        n = r.n;
        return;
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
  };
  int next_kind;
  int64_t next_start, next_n;
  fetch(next_kind, next_start, next_n);

  for (int64_t it = 0;; ++it) {
    const int s = static_cast<int>(it % S);
    const int kind = next_kind;
    const int64_t start = next_start, n = next_n;
    bool stop = false;
    if (lane == 0) {
      if (it >= S &&
          !mbar_wait_bounded(sbase + L.bar_empty + 8u * s,
                             static_cast<uint32_t>(((it / S) - 1) & 1), p.timeout_ns)) {
        atomicOr(p.status, kStatusTimeout);
        flags[0] = 1;
      }
      stop = flags[0] != 0;
    }
    if (__shfl_sync(kFullMask, stop ? 1 : 0, 0)) break;
    if (it >= S) fill_mask &= ~(1u << s);
    // (dense, several stages) the previous item's edges, whose loads had the
    // wait above to land
    edges_write<T>(edges, lane);

    if (lane == 0) {
      meta[s].start = start;
      meta[s].n = n;
      meta[s].kind = kind;
      mbar_arrive(sbase + L.bar_meta + 8u * s);
    }
    if (kind == kItemEnd) {
      if (++ends == G) break;
      continue;
    }

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
    // generic writes of this lane into the stage (an earlier item's edges)
    // are ordered before the bulk copies that overwrite it
    fence_proxy_async_smem();
    __syncwarp();
    bool copied = false;
    if (lane < L.pieces) {
      const int pc = lane;
      const uint32_t bar = sbase + L.bar_piece + 8u * (s * L.pieces + pc);
      const int64_t q0 = c0 + static_cast<int64_t>(pc) * kPieceTiles * kTileChunks;
      const int64_t q1 = min(c1, q0 + kPieceTiles * kTileChunks);
      const int64_t b0 = max(q0, static_cast<int64_t>(g.cf));
      const int64_t b1 = min(q1, static_cast<int64_t>(g.cl));
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
        bulk_g2s(stage + static_cast<uint32_t>((b0 - c0) * kChunkBytes), win + b0 * kChunkBytes,
                 bytes, bar, pol);
        copied = true;
      }
    }
    if (__any_sync(kFullMask, copied)) {
      fill_mask |= 1u << s;
      fill_parity = (fill_parity & ~(1u << s)) | (static_cast<uint32_t>((it / S) & 1) << s);
    }
    if (head || tail) {
      // lane l < E: element l of the head chunk; E <= l < 2E: element l - E
      // of the tail chunk
      edges.active = true;
      edges.head = head;
      edges.tail = tail;
      edges.tail_own_bar = tail && !(head && tail_pc == head_pc);
      edges.head_bar = sbase + L.bar_piece + 8u * (s * L.pieces + head_pc);
      edges.tail_bar = sbase + L.bar_piece + 8u * (s * L.pieces + (tail ? tail_pc : 0));
      const bool is_tail = lane >= E;
      const int e = is_tail ? lane - E : lane;
      const int64_t c = is_tail ? g.nc - 1 : 0;
      edges.mine = lane < 2 * E && (is_tail ? tail : head);
      edges.dst = stage + static_cast<uint32_t>((c - c0) * kChunkBytes) + static_cast<uint32_t>(e * SZ);
      edges.val = 0u;
      if (edges.mine) {
        const int64_t j = c * E + e - g.h;
        if (j >= 0 && j < g.n) {
          if constexpr (SZ == 2) {
            edges.val = *reinterpret_cast<const volatile unsigned short *>(in_row + j);
          } else {
            edges.val = *reinterpret_cast<const volatile uint32_t *>(in_row + j);
          }
        }
      }
    }
    // the next item while this one's edge loads are in flight; then its
    // edges (ragged, whose lookups take the round trips, or one stage), or
    // (dense) after the next stage's wait
    fetch(next_kind, next_start, next_n);
    if (RAGGED || S == 1) edges_write<T>(edges, lane);
  }
  edges_write<T>(edges, lane);
  // a producer that gave up must not leave copies in flight into its stages
  if (lane == 0 && flags[0]) {
    for (int s = 0; s < S; ++s)
      if (fill_mask >> s & 1u)
        for (int pc = 0; pc < L.pieces; ++pc)
          (void)mbar_wait_bounded(sbase + L.bar_piece + 8u * (s * L.pieces + pc),
                                  fill_parity >> s & 1u, p.timeout_ns);
  }
}

template <int OP, typename T, bool EXACT, bool CLUSTER, bool RAGGED, bool RESID = false,
          bool ONLINE = false>
__global__ void __launch_bounds__(kTileThreads, 3) tile_row_kernel(const TileParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int SZ = Elem<T>::kSize;
  extern __shared__ __align__(1024) unsigned char smem[];
  // pass-1 batch: four tiles for dense one-CTA rows (groups of two warps, few
  // tiles each), two with the cluster exchange, one in the ragged kernel,
  // whose 72 registers also carry the edge paths and the SMALL phase: larger
  // batches spill there (ragged bf16 LayerNorm 0.58 / 0.40 / 0.32 ms with
  // batches of 4 / 2 / 1)
  constexpr int kPass1Batch = RAGGED ? 1 : (CLUSTER ? 2 : 4);
  const int W = p.group_warps;
  const int G = kConsumerWarps / W;
  const TileSmemLayout L(p.stage_bytes, p.stages, p.max_tiles, G, CLUSTER, !CLUSTER || RAGGED,
                         RAGGED ? p.blocks : 0);
  const int S = p.stages;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int cs = CLUSTER ? static_cast<int>(cluster_nctarank()) : 1;
  const int rank = CLUSTER ? static_cast<int>(cluster_ctarank()) : 0;
  const int64_t cid = CLUSTER ? cluster_id_x() : blockIdx.x;
  const int64_t ncl = CLUSTER ? cluster_count_x() : gridDim.x;
  const uint32_t sbase = smem_addr(smem);
  const ItemMeta *meta = reinterpret_cast<const ItemMeta *>(smem + L.meta);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + L.flags);

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(sbase + L.bar_meta + 8u * s, 1);
      mbar_init(sbase + L.bar_empty + 8u * s, W);
      for (int pc = 0; pc < L.pieces; ++pc) mbar_init(sbase + L.bar_piece + 8u * (s * L.pieces + pc), 1);
    }
    for (int i = 0; i < 2 * G; ++i) {
      mbar_init(sbase + L.bar_ready + 8u * i, cs);           // one arrive per CTA
      mbar_init(sbase + L.bar_released + 8u * i, cs * W);    // one per warp of the group
    }
    flags[0] = 0;
    fence_mbar_init();
  }
  // (ragged) launched as a programmatic dependent of the classify kernel:
  // the barriers above were set up meanwhile; the plan is read below, once
  // that kernel has finished and its writes are visible (a no-op otherwise)
  if constexpr (RAGGED) asm volatile("griddepcontrol.wait;" ::: "memory");
  if (RAGGED && warp < 3) {
    // warp k: exclusive scan of bucket k's row counts over the classify blocks
    int *pref = reinterpret_cast<int *>(smem + L.pref) + warp * (p.blocks + 1);
    int carry = 0;
    for (int b0 = 0; b0 < p.blocks; b0 += 32) {
      const int b = b0 + lane;
      const int v = b < p.blocks ? p.block_counts[3 * b + warp] : 0;
      int x = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFullMask, x, o);
        if (lane >= o) x += y;
      }
      if (b < p.blocks) pref[b] = carry + x - v;
      carry += __shfl_sync(kFullMask, x, 31);
    }
    if (lane == 0) pref[p.blocks] = carry;
  }
  __syncthreads();
  if (CLUSTER) cluster_sync();  // every peer's barriers exist before any remote arrive

  if (warp == kConsumerWarps) {
    tile_producer<T, EXACT, CLUSTER, RAGGED>(p, L, smem, cs, rank, cid, ncl, lane);
    return;
  }

  // ------------------------------ consumers ------------------------------
  const int grp = warp / W;       // this warp's group
  const int wig = warp - grp * W; // its index in the group
  const int gtid = tid - grp * W * 32;
  const uint32_t gthreads = static_cast<uint32_t>(W) * 32u;
  const uint32_t gbar = kBarGroup0 + static_cast<uint32_t>(grp);
  float4 *part_c = reinterpret_cast<float4 *>(smem + L.part_c) + static_cast<size_t>(grp) * 2 * p.max_tiles;
  float4 *part_m = reinterpret_cast<float4 *>(smem + L.part_m) + static_cast<size_t>(grp) * 2 * p.max_tiles;
  float4 *blk = reinterpret_cast<float4 *>(smem + L.xw) + grp * kShortCombineTiles;
  float4 *gather = reinterpret_cast<float4 *>(smem + L.gather) + grp * kShortCombineTiles;
  const uint32_t bar_ready = sbase + L.bar_ready + 16u * grp;        // + 8 b
  const uint32_t bar_released = sbase + L.bar_released + 16u * grp;  // + 8 b
  // split items of this group that used part_c[0] / part_c[1] (kept as
  // scalars: a runtime-indexed array would live in local memory)
  uint32_t uses0 = 0, uses1 = 0;
  bool ended = false;
  for (int64_t j = 0;; ++j) {
    const int64_t it = grp + j * G;  // the group's j-th item
    const int s = static_cast<int>(it % S);
    const uint32_t par = static_cast<uint32_t>((it / S) & 1);
    const int b = static_cast<int>(j & 1);
    const uint32_t uses_b = b ? uses1 : uses0;
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
        if (split && uses_b > 0)
          bad = !mbar_wait_cluster_bounded(bar_released + 8u * b, (uses_b - 1) & 1, p.timeout_ns);
      }
    }
    const bool split = CLUSTER && kind == kItemLarge;
    const unsigned char *stage = smem + static_cast<size_t>(s) * p.stage_bytes;
    float4 *part = (split ? part_c : part_m) + static_cast<size_t>(b) * p.max_tiles;

    // ---- pass 1 ----
    if (!bad && kind != kItemEnd)
      bad = !pass1_warp<OP, T, kPass1Batch, RESID, ONLINE>(stage, g, wig, W, lane, part,
                                                  sbase + L.bar_piece + 8u * (s * L.pieces), par,
                                                  p.timeout_ns, p);
    if (named_sync_or(gbar, gthreads, bad)) {
      if (gtid == 0) {
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
    float s0, s1;
    const float inv_n = __frcp_rn(static_cast<float>(g.n));
    if (split) {
      const uint32_t ready = bar_ready + 8u * b;
      const int tpc = (g.K + cs - 1) / cs;
      // portions of whole 64-tile blocks: each CTA forms its own blocks'
      // partials (the same arithmetic as combine_blocks' level 1) and
      // publishes those, in place of its blocks' first tile partials
      const bool own_blocks = g.K > kShortCombineTiles && tpc % kShortCombineTiles == 0;
      if (own_blocks) {
        const int ntl = g.t1 - g.t0;
        for (int lb = wig; lb * kShortCombineTiles < ntl; lb += W) {
          const int kb = min(kShortCombineTiles, ntl - kShortCombineTiles * lb);
          const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
          const float4 q0 = lane < kb ? part[kShortCombineTiles * lb + lane] : z;
          const float4 q1 = lane + 32 < kb ? part[kShortCombineTiles * lb + lane + 32] : z;
          const float4 r = block_partial<OP>(q0, q1, lane < kb, lane + 32 < kb);
          __syncwarp();
          if (lane == 0) part[kShortCombineTiles * lb] = r;
        }
        named_sync(gbar, gthreads);
      }
      // thread r signals rank r; the named barrier above already ordered
      // every warp's partial writes before these releases
      if (gtid < cs) mbar_arrive_remote(ready, static_cast<uint32_t>(gtid));
      const bool ok = mbar_wait_cluster_bounded(ready, uses_b & 1, p.timeout_ns);
      if (named_sync_or(gbar, gthreads, !ok)) {
        if (gtid == 0) {
          atomicOr(p.status, kStatusTimeout);
          flags[0] = 1;
        }
        break;
      }
      // partial t lives in rank t / tpc at the same offset of its part_c
      const uint32_t mine = smem_addr(part);
      auto peer = [&](int t) {
        const int r = t / tpc;
        return ld_dsmem_f4(map_to_rank(mine + static_cast<uint32_t>((t - r * tpc) * 16),
                                       static_cast<uint32_t>(r)));
      };
      if (own_blocks) {
        // block partial t: rank t / (tpc / 64), first slot of its block there
        const int bpc = tpc / kShortCombineTiles;
        const int nb = (g.K + kShortCombineTiles - 1) / kShortCombineTiles;
        auto peer_block = [&](int t) {
          const int r = t / bpc;
          return ld_dsmem_f4(map_to_rank(
              mine + static_cast<uint32_t>((t - r * bpc) * kShortCombineTiles * 16),
              static_cast<uint32_t>(r)));
        };
        combine_short<OP>(peer_block, nb, inv_n, p.eps, lane, s0, s1);
        __syncwarp();
        if (lane < cs) mbar_arrive_remote(bar_released + 8u * b, static_cast<uint32_t>(lane));
      } else if (g.K <= kShortCombineTiles) {
        // every warp combines all K partials: copy them here once, then
        // combine from local shared memory
        for (int t = gtid; t < g.K; t += static_cast<int>(gthreads)) gather[t] = peer(t);
        named_sync(gbar, gthreads);
        __syncwarp();
        if (lane < cs) mbar_arrive_remote(bar_released + 8u * b, static_cast<uint32_t>(lane));
        combine_short<OP>([&](int t) { return gather[t]; }, g.K, inv_n, p.eps, lane, s0, s1);
      } else {
        combine_blocks<OP>(peer, g.K, inv_n, p.eps, lane, wig, W, gbar, blk, s0, s1);
        // this warp has read every peer partial it needs: let the peers reuse them
        __syncwarp();
        if (lane < cs) mbar_arrive_remote(bar_released + 8u * b, static_cast<uint32_t>(lane));
      }
      if (b) {
        ++uses1;
      } else {
        ++uses0;
      }
    } else {
      auto local = [&](int t) { return part[t]; };
      if (g.K <= kShortCombineTiles) {
        combine_short<OP>(local, g.K, inv_n, p.eps, lane, s0, s1);
      } else {
        combine_blocks<OP>(local, g.K, inv_n, p.eps, lane, wig, W, gbar, blk, s0, s1);
      }
    }

    // ---- pass 2 ----
    T *out_row = static_cast<T *>(p.out) + g.start;
    char *owin = reinterpret_cast<char *>(out_row) - g.h * SZ;
    pass2_item<OP, T, EXACT>(stage, g, wig, W, lane, s0, s1, p, owin, out_row);
    // the stage was written through the generic proxy (the residual sums):
    // order that before the producer's next bulk copies into it
    if constexpr (RESID) fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(sbase + L.bar_empty + 8u * s);
  }

  // ---- ragged: the SMALL rows, one per warp, staged in a slice of the stages ----
  // (every group has left its loop: no warp reads the stages any more)
  if (RAGGED && !named_sync_or(kBarConsumers, kConsumerThreads, !ended)) {
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
      const int *pref = reinterpret_cast<const int *>(smem + L.pref);  // SMALL: bucket 0
      if (idx >= static_cast<unsigned int>(pref[p.blocks])) break;
      const RowRec rec = ragged_record(p, pref, p.rec_small, idx);
      if (!ragged_record_fits<T>(rec, kSmall, p.glen)) {
        if (lane == 0) atomicOr(p.status, kStatusBadOffsets);
        continue;
      }
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
      small_row_core<OP, T, 9, false, false>(get, out + rec.start, rec.n, h, ncg, G, sub, sa);
      __syncwarp();
    }
  }

  // ---- no CTA leaves while a peer may still read its partials ----
  if (CLUSTER) {
    if (uses0 > 0) (void)mbar_wait_cluster_bounded(bar_released, (uses0 - 1) & 1, p.timeout_ns);
    if (uses1 > 0) (void)mbar_wait_cluster_bounded(bar_released + 8u, (uses1 - 1) & 1, p.timeout_ns);
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
