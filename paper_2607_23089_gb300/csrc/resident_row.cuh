// resident_row.cuh -- the register-resident tile design of the MEDIUM and
// LARGE buckets (medium_row_kernel / large_row_kernel of §2.1) for dense rows
// that are a whole number of tiles.
//
// Same row decomposition and the same arithmetic as tile_row.cuh (1 KiB tiles
// of 64 chunks, lane l of a tile's warp holding chunks l and l+32, tile
// partials combined in a fixed order), so its results equal the staged tile
// design bit for bit.  What differs is where the data lives while the row is
// worked on:
//   * each row (or this CTA's portion of a cluster-split row) is staged into
//     the next buffer of a stage ring with one bulk copy (cp.async.bulk,
//     TMA), issued by one lane of the CTA;
//   * each of the CTA's NW warps owns R tiles of every row.  A lane reads its
//     2R chunks from the stage once, converts them to fp32 pairs and keeps
//     them in registers; after the row's barrier every warp holds its
//     chunks, and the issuing lane refills that stage with a later row while
//     the row's statistics, the cluster exchange and the normalisation run
//     from registers;
//   * gamma/beta of the lane's columns stay in registers for the whole launch
//     where they fit (the lane owns the same columns in every row).
// One shared-memory read and one conversion per element, against three of
// each when pass 1's two sweeps and pass 2 re-read the stage, no masks, and
// no separate producer warp.
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
    xw = off;  // block partials of a long row
    off += kShortCombineTiles * 16u;
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
template <int OP, typename T, int R, int NW>
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
      for (int q = 0; q < R; ++q) part[w + NW * q] = make_float4(a[q], 0.f, 0.f, 0.f);
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
        part[w + NW * q] = (OP == kLayerNorm) ? make_float4(a[q], ref[q], b[q], kTileElems)
                                                     : make_float4(a[q], b[q], 0.f, 0.f);
    }
  }
}

// NW: warps of a CTA (4 or 8); MINB: CTAs per SM the kernel is compiled for
// (its register budget).
template <int OP, typename T, int R, int NW, bool CLUSTER, bool GC, int MINB>
__global__ void __launch_bounds__(NW * 32, MINB) resident_full_kernel(const TileParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr int SZ = Elem<T>::kSize;
  constexpr int NS = 2 * R;
  constexpr int kPortionTiles = NW * R;
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
  constexpr uint32_t kThreads = NW * 32;
  const int K = kPortionTiles * cs;  // tiles of a row
  const int t0 = kPortionTiles * rank;
  const int64_t row_bytes = p.ld * SZ;
  const char *in_portion = static_cast<const char *>(p.in) + static_cast<int64_t>(t0) * kTileBytes;
  char *out_portion = static_cast<char *>(p.out) + static_cast<int64_t>(t0) * kTileBytes;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) mbar_init(sbase + L.bar_full + 8u * s, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(sbase + L.bar_ready + 8u * i, cs);
      mbar_init(sbase + L.bar_released + 8u * i, cs * NW);
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
  float4 *blk = reinterpret_cast<float4 *>(smem + L.xw);
  float4 *gather = reinterpret_cast<float4 *>(smem + L.gather);
  const uint32_t bar_ready = sbase + L.bar_ready;
  const uint32_t bar_released = sbase + L.bar_released;

  // byte offset of each slot in the portion (stage and row alike): the
  // lane's base plus a compile-time offset per slot
  const uint32_t obase = static_cast<uint32_t>((w * kTileChunks + lane) * kChunkBytes);
  auto off = [&](int k) -> uint32_t {
    return obase + static_cast<uint32_t>((NW * (k >> 1) * kTileChunks + 32 * (k & 1)) * kChunkBytes);
  };
  f2 gc[GC ? NS : 1][NP], bc[GC ? NS : 1][NP];
  if constexpr (GC) {
#pragma unroll
    for (int k = 0; k < NS; ++k) {
      const int c = t0 * kTileChunks + static_cast<int>(off(k) / kChunkBytes);
      load_param_pairs<T>(static_cast<const T *>(p.gamma), p.gamma ? p.glen : 0, c, 0,
                          p.gvec != 0, 1.f, gc[k]);
      if constexpr (OP == kLayerNorm)
        load_param_pairs<T>(static_cast<const T *>(p.beta), p.beta ? p.glen : 0, c, 0,
                            p.gvec != 0, 0.f, bc[k]);
    }
  }
  const float inv_n = __frcp_rn(static_cast<float>(p.cols));
  // gamma/beta read as vectors: present, 16-byte aligned (the row's columns
  // are whole chunks, all below glen)
  const bool pvec = kAffine && p.gvec && p.gamma && (OP == kRmsNorm || p.beta != nullptr);
  const uint4 *gv = reinterpret_cast<const uint4 *>(p.gamma) + t0 * kTileChunks;
  const uint4 *bv = reinterpret_cast<const uint4 *>(p.beta) + t0 * kTileChunks;

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
        chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(stage + off(k)), x[k]);
      full_pass1<OP, T, R, NW>(x, w, lane, part);
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
    // portions of whole 64-tile blocks: each CTA forms its own blocks'
    // partials (combine_blocks' level 1) and publishes those in place of its
    // blocks' first tile partials
    constexpr bool kOwnBlocks = kPortionTiles % kShortCombineTiles == 0;
    if (CLUSTER) {
      const uint32_t ready = bar_ready + 8u * b;
      if (kOwnBlocks && K > kShortCombineTiles) {
        for (int lb = w; lb * kShortCombineTiles < kPortionTiles; lb += NW) {
          const float4 r = block_partial<OP>(part[kShortCombineTiles * lb + lane],
                                             part[kShortCombineTiles * lb + lane + 32], true, true);
          __syncwarp();
          if (lane == 0) part[kShortCombineTiles * lb] = r;
        }
        named_sync(kResBar, kThreads);
      }
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
      if (kOwnBlocks && K > kShortCombineTiles) {
        constexpr int bpc = kPortionTiles / kShortCombineTiles;
        auto peer_block = [&](int t) {
          const int rk = t / bpc;
          return ld_dsmem_f4(map_to_rank(
              mine + static_cast<uint32_t>((t - rk * bpc) * kShortCombineTiles * 16),
              static_cast<uint32_t>(rk)));
        };
        combine_short<OP>(peer_block, K / kShortCombineTiles, inv_n, p.eps, lane, s0, s1);
        __syncwarp();
        if (lane < cs) mbar_arrive_remote(bar_released + 8u * b, static_cast<uint32_t>(lane));
      } else if (K <= kShortCombineTiles) {
        for (int t = tid; t < K; t += static_cast<int>(kThreads)) gather[t] = peer(t);
        named_sync(kResBar, kThreads);
        __syncwarp();
        if (lane < cs) mbar_arrive_remote(bar_released + 8u * b, static_cast<uint32_t>(lane));
        combine_short<OP>([&](int t) { return gather[t]; }, K, inv_n, p.eps, lane, s0, s1);
      } else {
        combine_blocks<OP>(peer, K, inv_n, p.eps, lane, w, NW, kResBar, blk, s0, s1);
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
        } else if (pvec) {
          // aligned gamma/beta covering the row: one vector load each
          chunk_to_pairs<T>(__ldg(gv + off(k) / kChunkBytes), gp);
          if constexpr (OP == kLayerNorm) chunk_to_pairs<T>(__ldg(bv + off(k) / kChunkBytes), bp);
        } else {
          const int c = t0 * kTileChunks + static_cast<int>(off(k) / kChunkBytes);
          load_param_pairs<T>(static_cast<const T *>(p.gamma), p.gamma ? p.glen : 0, c, 0,
                              p.gvec != 0, 1.f, gp);
          if constexpr (OP == kLayerNorm)
            load_param_pairs<T>(static_cast<const T *>(p.beta), p.beta ? p.glen : 0, c, 0,
                                p.gvec != 0, 0.f, bp);
        }
      }
      normalize_pairs<OP, NP>(x[k], s0, s1, gp, bp);
      stg_stream(orow + off(k), pairs_to_chunk<T>(x[k]));
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
