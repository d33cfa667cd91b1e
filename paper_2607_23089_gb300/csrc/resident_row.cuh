// resident_row.cuh -- the register-resident tile design of the MEDIUM and
// LARGE buckets (medium_row_kernel / large_row_kernel of §2.1) and of the
// fused ragged launch.
//
// Same row decomposition and the same arithmetic as tile_row.cuh (1 KiB tiles
// of 64 chunks, lane l of a tile's warp holding chunks l and l+32, tile
// partials combined in a fixed order), so its results equal the staged tile
// design bit for bit.  What differs is where the data lives while the row is
// worked on:
//   * each item (a row, or this CTA's portion of a cluster-split row) is
//     staged into the next buffer of a stage ring with one bulk copy
//     (cp.async.bulk, TMA), issued by one lane of the CTA;
//   * the CTA's 8 warps share each item: warp w owns the item's tiles
//     w, w+8, ... (at most R of them).  A lane reads its 2R chunks from the
//     stage once, converts them to fp32 pairs and keeps them in registers;
//     after the item's barrier every warp holds its chunks, and the issuing
//     lane refills that stage with a later item while the row's statistics,
//     the cluster exchange and the normalisation run from registers.  The at
//     most two chunks a row only partly covers are read from global memory,
//     element by element, by the lanes that own them;
//   * dense rows whose every row starts at the same offset modulo 16 bytes
//     keep gamma/beta of the lane's columns in registers for the whole
//     launch (the lane owns the same columns in every row).
// One shared-memory read and one conversion per element, against three of
// each when pass 1's two sweeps and pass 2 re-read the stage, and no
// separate producer warp: 8-warp CTAs, two per SM, 128 registers a thread.
#pragma once

#include "tile_row.cuh"

namespace rowop {

constexpr int kResWarps = 8;                       // warps of a CTA, one group
constexpr int kResThreads = kResWarps * 32;
constexpr uint32_t kResBar = 1;                    // named barrier of the consumer warps

// Shared-memory layout of the resident kernel (host and device agree on it):
// the stage ring, tile partials of split items (part_c, read by the peers)
// and of items a CTA handles alone (part_m), both double-buffered by the
// parity of the item count, the partials of a short split row gathered from
// the peers, ragged item records, the long combine's scratch, the ragged
// list starts, and the barriers.
struct ResSmemLayout {
  uint32_t part_c, part_m, gather, meta, xw, pref, bar_full, bar_ready, bar_released, flags,
      total;
  __host__ __device__ ResSmemLayout(uint32_t stage_bytes, int stages, int max_tiles, bool split,
                                    int blocks) {
    uint32_t off = stage_bytes * static_cast<uint32_t>(stages);
    const uint32_t part_bytes = 2u * static_cast<uint32_t>(max_tiles) * 16u;
    part_c = off;
    off += split ? part_bytes : 0u;
    part_m = off;
    off += part_bytes;
    gather = off;
    off += split ? kShortCombineTiles * 16u : 0u;
    meta = off;
    off += static_cast<uint32_t>(stages) * 32u;
    xw = off;
    off += 2u * kConsumerWarps * 4u;
    pref = off;  // ragged: [3][blocks + 1] list position where each classify block starts
    off += (3u * static_cast<uint32_t>(blocks + 1) * 4u + 15u) & ~15u;
    bar_full = off;
    off += static_cast<uint32_t>(stages) * 8u;
    bar_ready = off;
    off += 16u;
    bar_released = off;
    off += 16u;
    flags = off;
    off += 16u;
    total = off;
  }
};

// Chunk c (window index) of a lane's slot k: slot k belongs to local tile
// w + 8 (k / 2) of the item and holds that tile's chunk lane + 32 (k % 2).
__device__ __forceinline__ int res_slot_chunk(int t0, int w, int lane, int k) {
  return (t0 + w + kResWarps * (k >> 1)) * kTileChunks + lane + 32 * (k & 1);
}

// Identity of the first row statistic: what an element outside the row
// contributes (nothing: -inf to a maximum, 0 to a sum).
template <int OP>
__device__ __forceinline__ float res_identity() {
  return (OP == kSoftmax || OP == kLogSoftmax) ? -INFINITY : 0.f;
}

// The lane's slots converted to fp32 pairs; elements outside the row (the
// head and tail of the row's end chunks, chunks past the portion) hold the
// identity of the first statistic.
template <int OP, typename T>
__device__ __forceinline__ void res_unpack(const uint4 &raw, bool exists, int lo, int hi,
                                           f2 (&x)[Elem<T>::kPerChunk / 2]) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  const float id = res_identity<OP>();
  chunk_to_pairs<T>(raw, x);
  if (!exists) {
#pragma unroll
    for (int i = 0; i < NP; ++i) x[i] = f2_bcast(id);
  } else if (lo != 0 || hi != E) {
#pragma unroll
    for (int i = 0; i < NP; ++i)
      x[i] = f2_select(x[i], in_range(2 * i, lo, hi), in_range(2 * i + 1, lo, hi), id);
  }
}

// Pass 1 from registers: the tile partials of the lane's R tiles, in the
// order tile_lane_first / tile_lane_second and the butterflies of
// pass1_batch use (chunk l before chunk l+32, pairs in order, even and odd
// halves added last; xor offsets 16 .. 1).  Lane 0 writes part[lt] for the
// tiles that exist.
template <int OP, typename T, int R>
__device__ __forceinline__ void res_pass1(const f2 (&x)[2 * R][Elem<T>::kPerChunk / 2],
                                          const bool (&ex)[2 * R], const int (&lo)[2 * R],
                                          const int (&hi)[2 * R], const ItemGeo &g, int w,
                                          int lane, float4 *part) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr bool kMaxFirst = (OP == kSoftmax || OP == kLogSoftmax);
  const int ntl = g.t1 - g.t0;
  float a[R];
#pragma unroll
  for (int q = 0; q < R; ++q) {
    if constexpr (kMaxFirst) {
      float m = -INFINITY;
#pragma unroll
      for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int i = 0; i < NP; ++i) m = fmaxf(m, fmaxf(f2_lo(x[2 * q + u][i]), f2_hi(x[2 * q + u][i])));
      a[q] = m;
    } else {
      f2 acc = f2_bcast(0.f);
#pragma unroll
      for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int i = 0; i < NP; ++i)
          acc = (OP == kLayerNorm) ? f2_add(acc, x[2 * q + u][i])
                                   : f2_fma(x[2 * q + u][i], x[2 * q + u][i], acc);
      a[q] = f2_total(acc);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
    for (int q = 0; q < R; ++q) {
      const float y = __shfl_xor_sync(kFullMask, a[q], o);
      a[q] = kMaxFirst ? fmaxf(a[q], y) : __fadd_rn(a[q], y);
    }
  }
  if constexpr (OP == kRmsNorm) {
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < R; ++q)
        if (w + kResWarps * q < ntl) part[w + kResWarps * q] = make_float4(a[q], 0.f, 0.f, 0.f);
    }
  } else {
    float ref[R], ntf[R], b[R];
#pragma unroll
    for (int q = 0; q < R; ++q) {
      const int t = g.t0 + w + kResWarps * q;
      ref[q] = a[q];
      ntf[q] = 0.f;
      if constexpr (OP == kLayerNorm) {
        if (tile_is_full(t, g)) {
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
        const f2 nr = f2_bcast(-ref[q]);
        f2 acc = f2_bcast(0.f);
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int k = 2 * q + u;
          const bool full = ex[k] && lo[k] == 0 && hi[k] == E;
#pragma unroll
          for (int i = 0; i < NP; ++i) {
            f2 d = f2_add(x[k][i], nr);
            if (!full) d = f2_select(d, ex[k] && in_range(2 * i, lo[k], hi[k]),
                                     ex[k] && in_range(2 * i + 1, lo[k], hi[k]), 0.f);
            acc = f2_fma(d, d, acc);
          }
        }
        b[q] = f2_total(acc);
      } else {
        // softmax family: sum exp(x - m_t); elements outside the row hold
        // -inf and add exp(-inf) = +0, as the masked sum adds +0
        if (ref[q] == -INFINITY) {
          b[q] = 0.f;
        } else {
          const f2 nm = f2_neg(f2_bcast(ref[q]));
          f2 acc = f2_bcast(0.f);
#pragma unroll
          for (int u = 0; u < 2; ++u)
#pragma unroll
            for (int i = 0; i < NP; ++i) acc = f2_add(acc, f2_exp_shifted(x[2 * q + u][i], nm));
          b[q] = f2_total(acc);
        }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
      for (int q = 0; q < R; ++q) b[q] = __fadd_rn(b[q], __shfl_xor_sync(kFullMask, b[q], o));
    }
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < R; ++q)
        if (w + kResWarps * q < ntl)
          part[w + kResWarps * q] = (OP == kLayerNorm) ? make_float4(a[q], ref[q], b[q], ntf[q])
                                                       : make_float4(a[q], b[q], 0.f, 0.f);
    }
  }
}

// Pass 2 from registers for an item with head offset H: gamma/beta read per
// chunk (realigned vectors for chunks [cf, cfast), the general loader for
// the others), or taken from the lane's cached copies (GC); 128-bit stores
// for the row's full chunks, element stores for its end chunks.
template <int OP, typename T, int R, int H, bool GC>
__device__ __forceinline__ void res_pass2(f2 (&x)[2 * R][Elem<T>::kPerChunk / 2],
                                          const bool (&ex)[2 * R], const int (&lo)[2 * R],
                                          const int (&hi)[2 * R], const int (&cc)[2 * R],
                                          const ItemGeo &g, float s0, float s1,
                                          const TileParams &p, int cfast,
                                          const f2 (&gc)[GC ? 2 * R : 1][Elem<T>::kPerChunk / 2],
                                          const f2 (&bc)[GC ? 2 * R : 1][Elem<T>::kPerChunk / 2]) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr int SZ = Elem<T>::kSize;
  constexpr bool kAffine = (OP == kLayerNorm || OP == kRmsNorm);
  const T *gamma = static_cast<const T *>(p.gamma);
  const T *beta = static_cast<const T *>(p.beta);
  T *out_row = static_cast<T *>(p.out) + g.start;
  char *owin = reinterpret_cast<char *>(out_row) - g.h * SZ;
#pragma unroll
  for (int k = 0; k < 2 * R; ++k) {
    if (!ex[k]) continue;
    const int c = cc[k];
    const bool full = lo[k] == 0 && hi[k] == E;
    f2 gp[NP], bp[NP];
    if constexpr (kAffine) {
      if constexpr (GC) {
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          gp[i] = gc[k][i];
          bp[i] = bc[k][i];
        }
      } else if (c >= g.cf && c < cfast) {
        chunk_to_pairs<T>(param_chunk_fixed<T, H>(gamma, c), gp);
        if constexpr (OP == kLayerNorm) chunk_to_pairs<T>(param_chunk_fixed<T, H>(beta, c), bp);
      } else {
        load_param_pairs<T>(gamma, gamma ? p.glen : 0, c, g.h, p.gvec != 0, 1.f, gp);
        if constexpr (OP == kLayerNorm)
          load_param_pairs<T>(beta, beta ? p.glen : 0, c, g.h, p.gvec != 0, 0.f, bp);
      }
    }
    normalize_pairs<OP, NP>(x[k], s0, s1, gp, bp);
    if (full) {
      stg_stream(owin + static_cast<int64_t>(c) * kChunkBytes, pairs_to_chunk<T>(x[k]));
    } else {
      store_chunk<T>(x[k], owin, out_row, c, g.h, lo[k], hi[k], false);
    }
  }
}

// Pass 2 with the gamma/beta realignment compiled for the item's head offset.
template <int OP, typename T, int R, bool GC>
__device__ __forceinline__ void res_pass2_item(f2 (&x)[2 * R][Elem<T>::kPerChunk / 2],
                                               const bool (&ex)[2 * R], const int (&lo)[2 * R],
                                               const int (&hi)[2 * R], const int (&cc)[2 * R],
                                               const ItemGeo &g, float s0, float s1,
                                               const TileParams &p,
                                               const f2 (&gc)[GC ? 2 * R : 1][Elem<T>::kPerChunk / 2],
                                               const f2 (&bc)[GC ? 2 * R : 1][Elem<T>::kPerChunk / 2]) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr bool kAffine = (OP == kLayerNorm || OP == kRmsNorm);
  if constexpr (!kAffine || GC) {
    res_pass2<OP, T, R, 0, GC>(x, ex, lo, hi, cc, g, s0, s1, p, 0, gc, bc);
  } else {
    // fast parameter chunks: within the row's full chunks and not reaching
    // past gamma/beta (the realigned load of chunk c reads up to column
    // (c + 1) E - 1)
    const bool params_ok = p.gvec && p.gamma && (OP == kRmsNorm || p.beta != nullptr);
    const int cfast = params_ok ? static_cast<int>(min(static_cast<int64_t>(g.cl), p.glen / E)) : g.cf;
    switch (g.h) {
      case 0: res_pass2<OP, T, R, 0, GC>(x, ex, lo, hi, cc, g, s0, s1, p, cfast, gc, bc); break;
      case 1: res_pass2<OP, T, R, 1, GC>(x, ex, lo, hi, cc, g, s0, s1, p, cfast, gc, bc); break;
      case 2: res_pass2<OP, T, R, 2, GC>(x, ex, lo, hi, cc, g, s0, s1, p, cfast, gc, bc); break;
      case 3: res_pass2<OP, T, R, 3, GC>(x, ex, lo, hi, cc, g, s0, s1, p, cfast, gc, bc); break;
      default:
        if constexpr (E == 8) {
          switch (g.h) {
            case 4: res_pass2<OP, T, R, 4, GC>(x, ex, lo, hi, cc, g, s0, s1, p, cfast, gc, bc); break;
            case 5: res_pass2<OP, T, R, 5, GC>(x, ex, lo, hi, cc, g, s0, s1, p, cfast, gc, bc); break;
            case 6: res_pass2<OP, T, R, 6, GC>(x, ex, lo, hi, cc, g, s0, s1, p, cfast, gc, bc); break;
            default: res_pass2<OP, T, R, 7, GC>(x, ex, lo, hi, cc, g, s0, s1, p, cfast, gc, bc); break;
          }
        }
        break;
    }
  }
}

// ---------------------------------------------------------------------------
// The issuing lane (lane 0 of warp 0): it walks the CTA's items and stages
// each with one bulk copy.  Items 0 .. S-1 are issued before the loop; item
// j + S goes into item j's stage right after item j's barrier, when every
// warp has its chunks of item j in registers -- so no stage is ever waited
// for.  Ragged items: the records come from the LARGE list (static
// round-robin over clusters), then the MEDIUM list (device counter); the
// next record is fetched one item ahead so its loads overlap the row's work.
// ---------------------------------------------------------------------------
struct ResIssuer {
  int64_t k_large;      // LARGE records taken
  int64_t next_item;    // items issued so far
  unsigned int pend;    // MEDIUM list index taken for the record after the fetched one
  bool medium_phase;
  bool done;            // the end-of-work record was issued
  int kind;             // the fetched next record
  int64_t start, n;
  uint32_t fill_mask, fill_parity;  // stages with a copy in flight, and its phase
};

// Fetches the record of the next item.  MEDIUM records are pipelined: the
// list index taken from the device counter on one fetch is resolved into its
// record on the next, so neither the counter's round trip nor the record's
// load stalls the issuing warp (an index past the list means the end of
// work, and every later index is past it too).
template <typename T, bool RAGGED, bool CLUSTER>
__device__ __forceinline__ void res_fetch(ResIssuer &q, const TileParams &p, const int *pref,
                                          int64_t cid, int64_t ncl) {
  q.kind = kItemEnd;
  q.start = 0;
  q.n = 0;
  if (RAGGED) {
    const int nb1 = p.blocks + 1;
    for (;;) {
      if (!q.medium_phase) {
        const int64_t li = cid + q.k_large * ncl;
        if (li < pref[2 * nb1 + p.blocks]) {
          const RowRec r = ragged_record(p, pref + 2 * nb1, p.rec_large, li);
          ++q.k_large;
          if (!ragged_record_fits<T>(r, kLarge, p.glen)) {
            atomicOr(p.status, kStatusBadOffsets);
            continue;
          }
          q.kind = kItemLarge;
          q.start = r.start;
          q.n = r.n;
          return;
        }
        q.medium_phase = true;
        q.pend = atomicAdd(&p.counters[0], 1u);
      }
      const unsigned int m = q.pend;
      q.pend = atomicAdd(&p.counters[0], 1u);
      if (m >= static_cast<unsigned int>(pref[nb1 + p.blocks])) return;
      const RowRec r = ragged_record(p, pref + nb1, p.rec_medium, m);
      if (!ragged_record_fits<T>(r, kMedium, p.glen)) {
        atomicOr(p.status, kStatusBadOffsets);
        continue;
      }
      q.kind = kItemMedium;
      q.start = r.start;
      q.n = r.n;
      return;
    }
  } else {
    const int64_t r = cid + q.next_item * ncl;
    if (r < p.rows) {
      q.kind = CLUSTER ? kItemLarge : kItemMedium;
      q.start = r * p.ld;
      q.n = p.cols;
    }
  }
}

// Issues the fetched record as item q.next_item into its stage, then
// fetches the next one.  Ragged records (and the end of work) go to the
// stage's record slot, which the consumers read at least one item barrier
// later.
template <typename T, bool CLUSTER, bool RAGGED>
__device__ __forceinline__ void res_issue(ResIssuer &q, const TileParams &p,
                                          const ResSmemLayout &L, unsigned char *smem, int cs,
                                          int rank, int64_t cid, int64_t ncl, uint64_t pol) {
  if (q.done) return;
  const int S = p.stages;
  const int s = static_cast<int>(q.next_item % S);
  const uint32_t sbase = smem_addr(smem);
  const uint32_t bar = sbase + L.bar_full + 8u * s;
  if (RAGGED) {
    ItemMeta *meta = reinterpret_cast<ItemMeta *>(smem + L.meta);
    meta[s].start = q.start;
    meta[s].n = q.n;
    meta[s].kind = q.kind;
  }
  if (q.kind == kItemEnd) {
    q.done = true;
    return;
  }
  const bool split = CLUSTER && q.kind == kItemLarge;
  const ItemGeo g = item_geo<T, false>(p.in, q.start, q.n, split, rank, cs);
  const int64_t c0 = static_cast<int64_t>(g.t0) * kTileChunks;
  const int64_t c1 = min(static_cast<int64_t>(g.nc), static_cast<int64_t>(g.t1) * kTileChunks);
  const int64_t b0 = max(c0, static_cast<int64_t>(g.cf));
  const int64_t b1 = min(c1, static_cast<int64_t>(g.cl));
  if (b1 > b0) {
    const uint32_t bytes = static_cast<uint32_t>((b1 - b0) * kChunkBytes);
    const char *win = reinterpret_cast<const char *>(static_cast<const T *>(p.in) + q.start) -
                      g.h * Elem<T>::kSize;
    mbar_arrive_expect_tx(bar, bytes);
    fence_proxy_async_smem();
    bulk_g2s(sbase + static_cast<uint32_t>(s) * p.stage_bytes +
                 static_cast<uint32_t>((b0 - c0) * kChunkBytes),
             win + b0 * kChunkBytes, bytes, bar, pol);
    q.fill_mask |= 1u << s;
    q.fill_parity = (q.fill_parity & ~(1u << s)) |
                    (static_cast<uint32_t>((q.next_item / S) & 1) << s);
  } else {
    mbar_arrive(bar);
  }
  ++q.next_item;
}

template <int OP, typename T, int R, bool CLUSTER, bool RAGGED, bool GC>
__global__ void __launch_bounds__(kResThreads, 2) resident_row_kernel(const TileParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr int SZ = Elem<T>::kSize;
  constexpr int NS = 2 * R;
  constexpr bool kAffine = (OP == kLayerNorm || OP == kRmsNorm);
  static_assert(!GC || (kAffine && !RAGGED), "cached parameters: dense norms only");
  extern __shared__ __align__(1024) unsigned char smem[];
  const ResSmemLayout L(p.stage_bytes, p.stages, p.max_tiles, CLUSTER, RAGGED ? p.blocks : 0);
  const int S = p.stages;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int w = tid >> 5;
  const int cs = CLUSTER ? static_cast<int>(cluster_nctarank()) : 1;
  const int rank = CLUSTER ? static_cast<int>(cluster_ctarank()) : 0;
  const int64_t cid = CLUSTER ? cluster_id_x() : blockIdx.x;
  const int64_t ncl = CLUSTER ? cluster_count_x() : gridDim.x;
  const uint32_t sbase = smem_addr(smem);
  const ItemMeta *meta = reinterpret_cast<const ItemMeta *>(smem + L.meta);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + L.flags);
  const int *pref = reinterpret_cast<const int *>(smem + L.pref);
  const bool issuer = tid == 0;
  constexpr uint32_t kThreads = kResThreads;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) mbar_init(sbase + L.bar_full + 8u * s, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(sbase + L.bar_ready + 8u * i, cs);                 // one arrive per CTA
      mbar_init(sbase + L.bar_released + 8u * i, cs * kResWarps);  // one per warp
    }
    flags[0] = 0;
    fence_mbar_init();
  }
  if (RAGGED && w < 3) {
    // warp k: exclusive scan of bucket k's row counts over the classify blocks
    int *pw = reinterpret_cast<int *>(smem + L.pref) + w * (p.blocks + 1);
    int carry = 0;
    for (int b0 = 0; b0 < p.blocks; b0 += 32) {
      const int b = b0 + lane;
      const int v = b < p.blocks ? p.block_counts[3 * b + w] : 0;
      int x = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFullMask, x, o);
        if (lane >= o) x += y;
      }
      if (b < p.blocks) pw[b] = carry + x - v;
      carry += __shfl_sync(kFullMask, x, 31);
    }
    if (lane == 0) pw[p.blocks] = carry;
  }
  __syncthreads();

  // the first S items (their records reach the other warps through the
  // barrier below)
  ResIssuer q;
  q.k_large = 0;
  q.next_item = 0;
  q.pend = 0;
  q.medium_phase = false;
  q.done = false;
  q.fill_mask = 0;
  q.fill_parity = 0;
  const uint64_t pol = issuer ? l2_evict_first_policy() : 0;
  if (issuer) {
    res_fetch<T, RAGGED, CLUSTER>(q, p, pref, cid, ncl);
    for (int s = 0; s < S && !q.done; ++s) {
      res_issue<T, CLUSTER, RAGGED>(q, p, L, smem, cs, rank, cid, ncl, pol);
      if (!q.done) res_fetch<T, RAGGED, CLUSTER>(q, p, pref, cid, ncl);
    }
  }
  __syncthreads();
  if (CLUSTER) cluster_sync();  // every peer's barriers exist before any remote arrive

  float4 *part_c = reinterpret_cast<float4 *>(smem + L.part_c);
  float4 *part_m = reinterpret_cast<float4 *>(smem + L.part_m);
  volatile float *xw = reinterpret_cast<volatile float *>(smem + L.xw);
  float4 *gather = reinterpret_cast<float4 *>(smem + L.gather);
  const uint32_t bar_ready = sbase + L.bar_ready;
  const uint32_t bar_released = sbase + L.bar_released;

  // cached gamma/beta of the lane's columns (dense rows at one head offset,
  // so every row puts the same columns in the same slots)
  f2 gc[GC ? NS : 1][NP], bc[GC ? NS : 1][NP];
  if constexpr (GC) {
    const ItemGeo g0 = item_geo<T, false>(p.in, 0, p.cols, CLUSTER, rank, cs);
#pragma unroll
    for (int k = 0; k < NS; ++k) {
      const int c = res_slot_chunk(g0.t0, w, lane, k);
      load_param_pairs<T>(static_cast<const T *>(p.gamma), p.gamma ? p.glen : 0, c, g0.h,
                          p.gvec != 0, 1.f, gc[k]);
      if constexpr (OP == kLayerNorm)
        load_param_pairs<T>(static_cast<const T *>(p.beta), p.beta ? p.glen : 0, c, g0.h,
                            p.gvec != 0, 0.f, bc[k]);
    }
  }

  uint32_t uses0 = 0, uses1 = 0;
  bool ended = false;
  for (int64_t j = 0;; ++j) {
    const int s = static_cast<int>(j % S);
    const uint32_t par = static_cast<uint32_t>((j / S) & 1);
    const int b = static_cast<int>(j & 1);
    const uint32_t uses_b = b ? uses1 : uses0;
    bool bad = false;
    int kind = kItemEnd;
    int64_t start = 0, n = 0;
    if constexpr (RAGGED) {
      kind = meta[s].kind;
      start = meta[s].start;
      n = meta[s].n;
    } else {
      const int64_t r = cid + j * ncl;
      if (r < p.rows) {
        kind = CLUSTER ? kItemLarge : kItemMedium;
        start = r * p.ld;
        n = p.cols;
      }
    }
    const bool split = CLUSTER && kind == kItemLarge;
    ItemGeo g;
    g.start = start;
    g.n = n;
    g.h = 0;
    g.nc = g.K = g.t0 = g.t1 = g.cf = g.cl = 0;
    if (kind != kItemEnd) {
      g = item_geo<T, false>(p.in, start, n, split, rank, cs);
      if (split && uses_b > 0)
        bad = !mbar_wait_cluster_bounded(bar_released + 8u * b, (uses_b - 1) & 1, p.timeout_ns);
    }
    float4 *part = (split ? part_c : part_m) + static_cast<size_t>(b) * p.max_tiles;

    // ---- the lane's chunks: row ends from global memory, the rest from the stage ----
    const int ntl = g.t1 - g.t0;
    const int hn = g.h + static_cast<int>(n);
    const T *in_row = static_cast<const T *>(p.in) + start;
    bool ex[NS], edge[NS];
    int lo[NS], hi[NS], cc[NS];
    uint4 raw[NS];
#pragma unroll
    for (int k = 0; k < NS; ++k) {
      const int lt = w + kResWarps * (k >> 1);
      cc[k] = res_slot_chunk(g.t0, w, lane, k);
      ex[k] = lt < ntl && cc[k] < g.nc;
      edge[k] = ex[k] && (cc[k] < g.cf || cc[k] >= g.cl);
      lo[k] = 0;
      hi[k] = E;
      if (ex[k]) chunk_valid_range(cc[k], g.nc, g.h, hn, E, lo[k], hi[k]);
      raw[k] = edge[k] ? load_chunk_elems<T>(in_row, cc[k], g.h, n) : make_uint4(0u, 0u, 0u, 0u);
    }
    if (kind != kItemEnd && !bad) {
      bad = !mbar_wait_bounded(sbase + L.bar_full + 8u * s, par, p.timeout_ns);
      if (!bad) {
        const unsigned char *stage = smem + static_cast<size_t>(s) * p.stage_bytes;
        const int c0 = g.t0 * kTileChunks;
#pragma unroll
        for (int k = 0; k < NS; ++k)
          if (ex[k] && !edge[k])
            raw[k] = *reinterpret_cast<const uint4 *>(stage + (cc[k] - c0) * kChunkBytes);
      }
    }
    f2 x[NS][NP];
#pragma unroll
    for (int k = 0; k < NS; ++k) res_unpack<OP, T>(raw[k], ex[k], lo[k], hi[k], x[k]);

    // ---- pass 1 ----
    if (kind != kItemEnd && !bad) res_pass1<OP, T, R>(x, ex, lo, hi, g, w, lane, part);
    // every warp has its chunks of this item in registers past this barrier
    if (named_sync_or(kResBar, kThreads, bad)) {
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
    // the stage of item j is free: refill it with item j + S
    if (issuer) {
      fence_proxy_async_smem();
      res_issue<T, CLUSTER, RAGGED>(q, p, L, smem, cs, rank, cid, ncl, pol);
      if (!q.done) res_fetch<T, RAGGED, CLUSTER>(q, p, pref, cid, ncl);
    }

    // ---- combine ----
    float s0, s1;
    const float inv_n = __frcp_rn(static_cast<float>(n));
    if (split) {
      const uint32_t ready = bar_ready + 8u * b;
      if (tid < cs) mbar_arrive_remote(ready, static_cast<uint32_t>(tid));
      const bool ok = mbar_wait_cluster_bounded(ready, uses_b & 1, p.timeout_ns);
      if (named_sync_or(kResBar, kThreads, !ok)) {
        if (tid == 0) {
          atomicOr(p.status, kStatusTimeout);
          flags[0] = 1;
        }
        break;
      }
      const int tpc = (g.K + cs - 1) / cs;
      const uint32_t mine = smem_addr(part);
      auto peer = [&](int t) {
        const int r = t / tpc;
        return ld_dsmem_f4(map_to_rank(mine + static_cast<uint32_t>((t - r * tpc) * 16),
                                       static_cast<uint32_t>(r)));
      };
      if (g.K <= kShortCombineTiles) {
        for (int t = tid; t < g.K; t += static_cast<int>(kThreads)) gather[t] = peer(t);
        named_sync(kResBar, kThreads);
        __syncwarp();
        if (lane < cs) mbar_arrive_remote(bar_released + 8u * b, static_cast<uint32_t>(lane));
        combine_short<OP>([&](int t) { return gather[t]; }, g.K, inv_n, p.eps, lane, s0, s1);
      } else {
        combine_long<OP>(peer, g.K, inv_n, p.eps, lane, w, kResWarps, kResBar, xw, s0, s1);
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
        combine_long<OP>(local, g.K, inv_n, p.eps, lane, w, kResWarps, kResBar, xw, s0, s1);
      }
    }

    // ---- pass 2 ----
    res_pass2_item<OP, T, R, GC>(x, ex, lo, hi, cc, g, s0, s1, p, gc, bc);
  }

  // a CTA that gave up must not leave copies in flight into its stages
  if (issuer && flags[0]) {
    for (int s = 0; s < S; ++s)
      if (q.fill_mask >> s & 1u)
        (void)mbar_wait_bounded(sbase + L.bar_full + 8u * s, q.fill_parity >> s & 1u,
                                p.timeout_ns);
  }

  // ---- ragged: the SMALL rows, one per warp, staged in a slice of the stages ----
  // (every warp has left its loop at the end-of-work record: every copy
  // into the stages has landed and been read)
  if (RAGGED && !named_sync_or(kResBar, kThreads, !ended)) {
    SmallRowArgs sa;
    sa.gamma = p.gamma;
    sa.beta = p.beta;
    sa.glen = p.glen;
    sa.eps = p.eps;
    sa.gvec = p.gvec;
    sa.out_vec = p.out_vec;
    unsigned char *slice = smem + static_cast<size_t>(w) * kSmallSliceBytes;
    const T *in = static_cast<const T *>(p.in);
    T *out = static_cast<T *>(p.out);
    for (;;) {
      unsigned int idx = 0;
      if (lane == 0) idx = atomicAdd(&p.counters[1], 1u);
      idx = __shfl_sync(kFullMask, idx, 0);
      if (idx >= static_cast<unsigned int>(pref[p.blocks])) break;  // SMALL: bucket 0
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
        int l0, h0;
        chunk_valid_range(c, nc, h, h + rec.n, E, l0, h0);
        *reinterpret_cast<uint4 *>(slice + c * kChunkBytes) =
            (l0 == 0 && h0 == E) ? ldg_stream(win + c * kChunkBytes)
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

  // ---- ragged: the last CTA to finish resets the work counters ----
  if (RAGGED) {
    named_sync(kResBar, kThreads);
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

// ---------------------------------------------------------------------------
// Whole-tile rows: the resident design specialised for dense rows that are a
// whole number of tiles, 16-byte aligned, and split so that every warp owns
// exactly R tiles of every item (one CTA: K = 8R; a cluster of cs CTAs:
// K = 8R cs).  Every slot of every lane is then a full chunk of the row at a
// fixed offset, so no element is masked, nothing is read element by element,
// and the per-lane geometry is computed once for the launch.  The arithmetic
// is the general resident kernel's (and the staged kernel's) with every mask
// known to keep everything.
// ---------------------------------------------------------------------------
template <int OP, typename T, int R>
__device__ __forceinline__ void full_pass1(const f2 (&x)[2 * R][Elem<T>::kPerChunk / 2], int w,
                                           int lane, float4 *part) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr bool kMaxFirst = (OP == kSoftmax || OP == kLogSoftmax);
  float a[R];
#pragma unroll
  for (int q = 0; q < R; ++q) {
    if constexpr (kMaxFirst) {
      float m = -INFINITY;
#pragma unroll
      for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int i = 0; i < NP; ++i)
          m = fmaxf(m, fmaxf(f2_lo(x[2 * q + u][i]), f2_hi(x[2 * q + u][i])));
      a[q] = m;
    } else {
      f2 acc = f2_bcast(0.f);
#pragma unroll
      for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int i = 0; i < NP; ++i)
          acc = (OP == kLayerNorm) ? f2_add(acc, x[2 * q + u][i])
                                   : f2_fma(x[2 * q + u][i], x[2 * q + u][i], acc);
      a[q] = f2_total(acc);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
    for (int q = 0; q < R; ++q) {
      const float y = __shfl_xor_sync(kFullMask, a[q], o);
      a[q] = kMaxFirst ? fmaxf(a[q], y) : __fadd_rn(a[q], y);
    }
  }
  if constexpr (OP == kRmsNorm) {
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < R; ++q) part[w + kResWarps * q] = make_float4(a[q], 0.f, 0.f, 0.f);
    }
  } else {
    constexpr float kTileElems = static_cast<float>(kTileChunks * E);
    float ref[R], b[R];
#pragma unroll
    for (int q = 0; q < R; ++q) {
      ref[q] = (OP == kLayerNorm) ? __fmul_rn(a[q], 1.f / kTileElems) : a[q];  // exact
      f2 acc = f2_bcast(0.f);
      if constexpr (OP == kLayerNorm) {
        const f2 nr = f2_bcast(-ref[q]);
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
          for (int i = 0; i < NP; ++i) {
            const f2 d = f2_add(x[2 * q + u][i], nr);
            acc = f2_fma(d, d, acc);
          }
        b[q] = f2_total(acc);
      } else if (ref[q] == -INFINITY) {
        b[q] = 0.f;  // no element of the tile is above -inf
      } else {
        const f2 nm = f2_neg(f2_bcast(ref[q]));
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
          for (int i = 0; i < NP; ++i) acc = f2_add(acc, f2_exp_shifted(x[2 * q + u][i], nm));
        b[q] = f2_total(acc);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
      for (int q = 0; q < R; ++q) b[q] = __fadd_rn(b[q], __shfl_xor_sync(kFullMask, b[q], o));
    }
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < R; ++q)
        part[w + kResWarps * q] = (OP == kLayerNorm) ? make_float4(a[q], ref[q], b[q], kTileElems)
                                                     : make_float4(a[q], b[q], 0.f, 0.f);
    }
  }
}

// MINB: CTAs per SM the kernel is compiled for (its register budget).
template <int OP, typename T, int R, bool CLUSTER, bool GC, int MINB>
__global__ void __launch_bounds__(kResThreads, MINB) resident_full_kernel(const TileParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr int SZ = Elem<T>::kSize;
  constexpr int NS = 2 * R;
  constexpr int kPortionTiles = kResWarps * R;
  constexpr uint32_t kPortionBytes = kPortionTiles * kTileBytes;
  constexpr bool kAffine = (OP == kLayerNorm || OP == kRmsNorm);
  static_assert(!GC || kAffine, "cached parameters: norms only");
  extern __shared__ __align__(1024) unsigned char smem[];
  const ResSmemLayout L(p.stage_bytes, p.stages, p.max_tiles, CLUSTER, 0);
  const int S = p.stages;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int w = tid >> 5;
  const int cs = CLUSTER ? static_cast<int>(cluster_nctarank()) : 1;
  const int rank = CLUSTER ? static_cast<int>(cluster_ctarank()) : 0;
  const int64_t cid = CLUSTER ? cluster_id_x() : blockIdx.x;
  const int64_t ncl = CLUSTER ? cluster_count_x() : gridDim.x;
  const uint32_t sbase = smem_addr(smem);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + L.flags);
  const bool issuer = tid == 0;
  constexpr uint32_t kThreads = kResThreads;
  const int K = kPortionTiles * cs;  // tiles of a row
  const int t0 = kPortionTiles * rank;
  const int64_t row_bytes = p.ld * SZ;
  const char *in_portion = static_cast<const char *>(p.in) + static_cast<int64_t>(t0) * kTileBytes;
  char *out_portion = static_cast<char *>(p.out) + static_cast<int64_t>(t0) * kTileBytes;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) mbar_init(sbase + L.bar_full + 8u * s, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(sbase + L.bar_ready + 8u * i, cs);
      mbar_init(sbase + L.bar_released + 8u * i, cs * kResWarps);
    }
    flags[0] = 0;
    fence_mbar_init();
  }
  __syncthreads();
  // the first S rows
  const uint64_t pol = issuer ? l2_evict_first_policy() : 0;
  uint32_t fill_mask = 0;
  if (issuer) {
    for (int s = 0; s < S; ++s) {
      const int64_t r = cid + s * ncl;
      if (r >= p.rows) break;
      const uint32_t bar = sbase + L.bar_full + 8u * s;
      mbar_arrive_expect_tx(bar, kPortionBytes);
      bulk_g2s(sbase + static_cast<uint32_t>(s) * p.stage_bytes, in_portion + r * row_bytes,
               kPortionBytes, bar, pol);
      fill_mask |= 1u << s;
    }
  }
  __syncthreads();
  if (CLUSTER) cluster_sync();  // every peer's barriers exist before any remote arrive

  float4 *part_c = reinterpret_cast<float4 *>(smem + L.part_c);
  float4 *part_m = reinterpret_cast<float4 *>(smem + L.part_m);
  volatile float *xw = reinterpret_cast<volatile float *>(smem + L.xw);
  float4 *gather = reinterpret_cast<float4 *>(smem + L.gather);
  const uint32_t bar_ready = sbase + L.bar_ready;
  const uint32_t bar_released = sbase + L.bar_released;

  // byte offset of each slot in the portion (stage and row alike)
  uint32_t off[NS];
#pragma unroll
  for (int k = 0; k < NS; ++k)
    off[k] = static_cast<uint32_t>(((w + kResWarps * (k >> 1)) * kTileChunks + lane + 32 * (k & 1)) *
                                   kChunkBytes);
  f2 gc[GC ? NS : 1][NP], bc[GC ? NS : 1][NP];
  if constexpr (GC) {
#pragma unroll
    for (int k = 0; k < NS; ++k) {
      const int c = t0 * kTileChunks + static_cast<int>(off[k] / kChunkBytes);
      load_param_pairs<T>(static_cast<const T *>(p.gamma), p.gamma ? p.glen : 0, c, 0,
                          p.gvec != 0, 1.f, gc[k]);
      if constexpr (OP == kLayerNorm)
        load_param_pairs<T>(static_cast<const T *>(p.beta), p.beta ? p.glen : 0, c, 0,
                            p.gvec != 0, 0.f, bc[k]);
    }
  }
  const float inv_n = __frcp_rn(static_cast<float>(p.cols));

  uint32_t uses0 = 0, uses1 = 0;
  int s = 0;
  uint32_t par = 0;
  for (int64_t j = 0;; ++j) {
    const int64_t r = cid + j * ncl;
    if (r >= p.rows) break;
    const int b = static_cast<int>(j & 1);
    const uint32_t uses_b = b ? uses1 : uses0;
    bool bad = false;
    if (CLUSTER && uses_b > 0)
      bad = !mbar_wait_cluster_bounded(bar_released + 8u * b, (uses_b - 1) & 1, p.timeout_ns);
    float4 *part = (CLUSTER ? part_c : part_m) + static_cast<size_t>(b) * p.max_tiles;
    f2 x[NS][NP];
    if (!bad) bad = !mbar_wait_bounded(sbase + L.bar_full + 8u * s, par, p.timeout_ns);
    if (!bad) {
      const unsigned char *stage = smem + static_cast<size_t>(s) * p.stage_bytes;
#pragma unroll
      for (int k = 0; k < NS; ++k)
        chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(stage + off[k]), x[k]);
      full_pass1<OP, T, R>(x, w, lane, part);
    }
    // every warp has its chunks of row r in registers past this barrier
    if (named_sync_or(kResBar, kThreads, bad)) {
      if (tid == 0) {
        atomicOr(p.status, kStatusTimeout);
        flags[0] = 1;
      }
      break;
    }
    if (issuer) {  // refill the stage with row r + S ncl
      const int64_t rn = r + static_cast<int64_t>(S) * ncl;
      if (rn < p.rows) {
        const uint32_t bar = sbase + L.bar_full + 8u * s;
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(bar, kPortionBytes);
        bulk_g2s(sbase + static_cast<uint32_t>(s) * p.stage_bytes, in_portion + rn * row_bytes,
                 kPortionBytes, bar, pol);
      } else {
        fill_mask &= ~(1u << s);
      }
    }
    if (++s == S) {
      s = 0;
      par ^= 1u;
    }

    // ---- combine ----
    float s0, s1;
    if (CLUSTER) {
      const uint32_t ready = bar_ready + 8u * b;
      if (tid < cs) mbar_arrive_remote(ready, static_cast<uint32_t>(tid));
      const bool ok = mbar_wait_cluster_bounded(ready, uses_b & 1, p.timeout_ns);
      if (named_sync_or(kResBar, kThreads, !ok)) {
        if (tid == 0) {
          atomicOr(p.status, kStatusTimeout);
          flags[0] = 1;
        }
        break;
      }
      const uint32_t mine = smem_addr(part);
      auto peer = [&](int t) {
        const int rk = t / kPortionTiles;
        return ld_dsmem_f4(map_to_rank(mine + static_cast<uint32_t>((t - rk * kPortionTiles) * 16),
                                       static_cast<uint32_t>(rk)));
      };
      if (K <= kShortCombineTiles) {
        for (int t = tid; t < K; t += static_cast<int>(kThreads)) gather[t] = peer(t);
        named_sync(kResBar, kThreads);
        __syncwarp();
        if (lane < cs) mbar_arrive_remote(bar_released + 8u * b, static_cast<uint32_t>(lane));
        combine_short<OP>([&](int t) { return gather[t]; }, K, inv_n, p.eps, lane, s0, s1);
      } else {
        combine_long<OP>(peer, K, inv_n, p.eps, lane, w, kResWarps, kResBar, xw, s0, s1);
        __syncwarp();
        if (lane < cs) mbar_arrive_remote(bar_released + 8u * b, static_cast<uint32_t>(lane));
      }
      if (b) {
        ++uses1;
      } else {
        ++uses0;
      }
    } else {
      combine_short<OP>([&](int t) { return part[t]; }, K, inv_n, p.eps, lane, s0, s1);
    }

    // ---- pass 2 ----
    char *orow = out_portion + r * row_bytes;
#pragma unroll
    for (int k = 0; k < NS; ++k) {
      f2 gp[NP], bp[NP];
      if constexpr (kAffine) {
        if constexpr (GC) {
#pragma unroll
          for (int i = 0; i < NP; ++i) {
            gp[i] = gc[k][i];
            bp[i] = bc[k][i];
          }
        } else {
          const int c = t0 * kTileChunks + static_cast<int>(off[k] / kChunkBytes);
          load_param_pairs<T>(static_cast<const T *>(p.gamma), p.gamma ? p.glen : 0, c, 0,
                              p.gvec != 0, 1.f, gp);
          if constexpr (OP == kLayerNorm)
            load_param_pairs<T>(static_cast<const T *>(p.beta), p.beta ? p.glen : 0, c, 0,
                                p.gvec != 0, 0.f, bp);
        }
      }
      normalize_pairs<OP, NP>(x[k], s0, s1, gp, bp);
      stg_stream(orow + off[k], pairs_to_chunk<T>(x[k]));
    }
  }

  // a CTA that gave up must not leave copies in flight into its stages
  if (issuer && flags[0]) {
    // stage s holds the next unconsumed row: its phase is par, the ones
    // after it (in ring order) were issued one round earlier or later
    for (int i = 0; i < S; ++i) {
      const int si = (s + i) % S;
      if (fill_mask >> si & 1u)
        (void)mbar_wait_bounded(sbase + L.bar_full + 8u * si, si >= s ? par : par ^ 1u,
                                p.timeout_ns);
    }
  }
  // no CTA leaves while a peer may still read its partials
  if (CLUSTER) {
    if (uses0 > 0) (void)mbar_wait_cluster_bounded(bar_released, (uses0 - 1) & 1, p.timeout_ns);
    if (uses1 > 0) (void)mbar_wait_cluster_bounded(bar_released + 8u, (uses1 - 1) & 1, p.timeout_ns);
  }
}

}  // namespace rowop
