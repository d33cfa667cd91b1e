// stream_row.cuh -- the LARGE bucket (large_row_kernel of §2.1) for dense
// rows that are a whole number of 64-tile blocks per cluster CTA: the row is
// streamed twice instead of held in shared memory.
//
// A cluster of cs CTAs splits each row into cs portions of whole 64-tile
// blocks, as the staged split does, but a CTA keeps only a ring of 16 KiB
// pieces, not its whole portion:
//   * pass 1 streams the portion through the ring (bulk copies with an L2
//     evict-last hint) and reduces each tile to its tile partial;
//   * the CTA forms its blocks' partials and the cluster combines all of
//     them through distributed shared memory, exactly as the staged split
//     does, so every CTA has the row statistics;
//   * pass 2 streams the portion again (evict-first: the bytes of pass 1 are
//     still in L2), normalises and stores it with streaming stores.
// The producer warp runs up to the ring's depth ahead of the consumers, so
// pass 2's pieces load while the cluster exchanges partials and the next
// row's pass-1 pieces load while pass 2 runs: HBM sees one read and one
// write per element, and the loads never stop for the exchange.  The tile
// partials, block partials and combine are the staged design's, so the
// results equal it bit for bit.
#pragma once

#include "resident_row.cuh"

namespace rowop {

constexpr int kStreamPieceTiles = 16;  // tiles of one ring piece (16 KiB)
constexpr uint32_t kStreamPieceBytes = kStreamPieceTiles * kTileBytes;
constexpr int kStreamWarps = 8;        // consumer warps
constexpr int kStreamThreads = kStreamWarps * 32 + 32;
constexpr uint32_t kStreamBar = 1;     // named barrier of the consumer warps

struct StreamParams {
  const void *in;
  void *out;
  const void *gamma;
  const void *beta;
  int64_t rows, cols, ld;
  float eps;
  int pieces;     // ring depth
  int portion;    // tiles of one CTA's portion (a multiple of 64)
  int gvec;       // gamma / beta present and 16-byte aligned
  uint64_t timeout_ns;
  unsigned int *status;
};

// Shared memory (host and device agree on it): the ring, the tile partials
// of the portion double-buffered by the row's parity (the peers read them),
// the ring and cluster barriers and the abort flag.
struct StreamSmem {
  uint32_t part, bar_full, bar_empty, bar_ready, bar_released, flags, total;
  __host__ __device__ StreamSmem(int pieces, int portion) {
    uint32_t off = static_cast<uint32_t>(pieces) * kStreamPieceBytes;
    part = off;
    off += 2u * static_cast<uint32_t>(portion) * 16u;
    bar_full = off;
    off += static_cast<uint32_t>(pieces) * 8u;
    bar_empty = off;
    off += static_cast<uint32_t>(pieces) * 8u;
    bar_ready = off;
    off += 16u;
    bar_released = off;
    off += 16u;
    flags = off;
    off += 16u;
    total = off;
  }
};

__device__ __forceinline__ uint64_t l2_evict_last_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

template <int OP, typename T>
__global__ void __launch_bounds__(kStreamThreads, 2) stream_row_kernel(const StreamParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NPAIR = E / 2;
  constexpr int SZ = Elem<T>::kSize;
  constexpr bool kAffine = (OP == kLayerNorm || OP == kRmsNorm);
  constexpr uint32_t kThreads = kStreamWarps * 32;
  extern __shared__ __align__(1024) unsigned char smem[];
  const StreamSmem L(p.pieces, p.portion);
  const int NP = p.pieces;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int w = tid >> 5;
  const int cs = static_cast<int>(cluster_nctarank());
  const int rank = static_cast<int>(cluster_ctarank());
  const int64_t cid = cluster_id_x();
  const int64_t ncl = cluster_count_x();
  const uint32_t sbase = smem_addr(smem);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + L.flags);
  const int PT = p.portion;
  const int npc = PT / kStreamPieceTiles;  // pieces per pass
  const int K = PT * cs;                   // tiles of a row
  const int64_t row_bytes = p.ld * SZ;
  const int64_t t0 = static_cast<int64_t>(PT) * rank;  // first tile of this CTA's portion

  if (tid == 0) {
    for (int s = 0; s < NP; ++s) {
      mbar_init(sbase + L.bar_full + 8u * s, 1);
      mbar_init(sbase + L.bar_empty + 8u * s, kStreamWarps);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(sbase + L.bar_ready + 8u * i, cs);
      mbar_init(sbase + L.bar_released + 8u * i, cs * kStreamWarps);
    }
    flags[0] = 0;
    fence_mbar_init();
  }
  __syncthreads();
  cluster_sync();  // every peer's barriers exist before any remote arrive

  if (w == kStreamWarps) {
    // ------------------------------ producer ------------------------------
    if (lane != 0) return;
    const uint64_t keep = l2_evict_last_policy();
    const uint64_t drop = l2_evict_first_policy();
    const char *in = static_cast<const char *>(p.in) + t0 * kTileBytes;
    int64_t seq = 0;
    uint32_t fill_mask = 0, fill_parity = 0;
    bool stop = false;
    for (int64_t r = cid; r < p.rows && !stop; r += ncl) {
      for (int pass = 0; pass < 2 && !stop; ++pass) {
        for (int q = 0; q < npc; ++q, ++seq) {
          const int s = static_cast<int>(seq % NP);
          if (seq >= NP) {
            if (!mbar_wait_bounded(sbase + L.bar_empty + 8u * s,
                                   static_cast<uint32_t>(((seq / NP) - 1) & 1), p.timeout_ns)) {
              atomicOr(p.status, kStatusTimeout);
              flags[0] = 1;
            }
            fill_mask &= ~(1u << s);
          }
          if (flags[0]) {
            stop = true;
            break;
          }
          const uint32_t bar = sbase + L.bar_full + 8u * s;
          mbar_arrive_expect_tx(bar, kStreamPieceBytes);
          bulk_g2s(sbase + static_cast<uint32_t>(s) * kStreamPieceBytes,
                   in + r * row_bytes + static_cast<int64_t>(q) * kStreamPieceBytes,
                   kStreamPieceBytes, bar, pass == 0 ? keep : drop);
          fill_mask |= 1u << s;
          fill_parity = (fill_parity & ~(1u << s)) | (static_cast<uint32_t>((seq / NP) & 1) << s);
        }
      }
    }
    // a producer that gave up must not leave copies in flight into the ring
    if (flags[0]) {
      for (int s = 0; s < NP; ++s)
        if (fill_mask >> s & 1u)
          (void)mbar_wait_bounded(sbase + L.bar_full + 8u * s, fill_parity >> s & 1u,
                                  p.timeout_ns);
    }
    return;
  }

  // ------------------------------ consumers ------------------------------
  float4 *part_base = reinterpret_cast<float4 *>(smem + L.part);
  const uint32_t bar_ready = sbase + L.bar_ready;
  const uint32_t bar_released = sbase + L.bar_released;
  const float inv_n = __frcp_rn(static_cast<float>(p.cols));
  const int nb = K / kShortCombineTiles;           // blocks of the row
  const int bpc = PT / kShortCombineTiles;          // blocks of a portion
  // byte offset of a lane's chunk u (0..3) in a piece: tiles w and w + 8,
  // chunks lane and lane + 32 of each
  auto poff = [&](int u) -> uint32_t {
    return static_cast<uint32_t>((((w + kStreamWarps * (u >> 1)) * kTileChunks) + lane + 32 * (u & 1)) *
                                 kChunkBytes);
  };
  const bool pvec = kAffine && p.gvec;
  uint32_t uses0 = 0, uses1 = 0;
  int64_t seq = 0;
  bool bad = false;
  for (int64_t j = 0;; ++j) {
    const int64_t r = cid + j * ncl;
    if (r >= p.rows) break;
    const int b = static_cast<int>(j & 1);
    const uint32_t uses_b = b ? uses1 : uses0;
    float4 *part = part_base + static_cast<size_t>(b) * PT;
    // the peers are done with this buffer's partials of two rows ago
    if (uses_b > 0)
      bad = !mbar_wait_cluster_bounded(bar_released + 8u * b, (uses_b - 1) & 1, p.timeout_ns);

    // ---- pass 1: tile partials ----
    for (int q = 0; q < npc; ++q, ++seq) {
      const int s = static_cast<int>(seq % NP);
      if (!bad) bad = !mbar_wait_bounded(sbase + L.bar_full + 8u * s,
                                         static_cast<uint32_t>((seq / NP) & 1), p.timeout_ns);
      if (!bad) {
        const unsigned char *piece = smem + static_cast<size_t>(s) * kStreamPieceBytes;
        f2 x[4][NPAIR];
#pragma unroll
        for (int u = 0; u < 4; ++u)
          chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(piece + poff(u)), x[u]);
        full_pass1<OP, T, 2, kStreamWarps>(x, w, lane, part + q * kStreamPieceTiles);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(sbase + L.bar_empty + 8u * s);
    }
    if (named_sync_or(kStreamBar, kThreads, bad)) {
      bad = true;
      break;
    }

    // ---- this CTA's block partials, then the cluster's combine ----
    for (int lb = w; lb < bpc; lb += kStreamWarps) {
      const float4 rb = block_partial<OP>(part[kShortCombineTiles * lb + lane],
                                          part[kShortCombineTiles * lb + lane + 32], true, true);
      __syncwarp();
      if (lane == 0) part[kShortCombineTiles * lb] = rb;
    }
    named_sync(kStreamBar, kThreads);
    const uint32_t ready = bar_ready + 8u * b;
    if (tid < cs) mbar_arrive_remote(ready, static_cast<uint32_t>(tid));
    const bool ok = mbar_wait_cluster_bounded(ready, uses_b & 1, p.timeout_ns);
    if (named_sync_or(kStreamBar, kThreads, !ok)) {
      bad = true;
      break;
    }
    const uint32_t mine = smem_addr(part);
    auto peer_block = [&](int t) {
      const int rk = t / bpc;
      return ld_dsmem_f4(map_to_rank(
          mine + static_cast<uint32_t>((t - rk * bpc) * kShortCombineTiles * 16),
          static_cast<uint32_t>(rk)));
    };
    float s0, s1;
    combine_short<OP>(peer_block, nb, inv_n, p.eps, lane, s0, s1);
    __syncwarp();
    if (lane < cs) mbar_arrive_remote(bar_released + 8u * b, static_cast<uint32_t>(lane));
    if (b) {
      ++uses1;
    } else {
      ++uses0;
    }

    // ---- pass 2: normalise and store ----
    char *orow = static_cast<char *>(p.out) + r * row_bytes + t0 * kTileBytes;
    for (int q = 0; q < npc; ++q, ++seq) {
      const int s = static_cast<int>(seq % NP);
      if (!bad) bad = !mbar_wait_bounded(sbase + L.bar_full + 8u * s,
                                         static_cast<uint32_t>((seq / NP) & 1), p.timeout_ns);
      if (!bad) {
        const unsigned char *piece = smem + static_cast<size_t>(s) * kStreamPieceBytes;
        char *opiece = orow + static_cast<int64_t>(q) * kStreamPieceBytes;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          f2 x[NPAIR], gp[NPAIR], bp[NPAIR];
          chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(piece + poff(u)), x);
          if constexpr (kAffine) {
            // column chunk of this element chunk: the row's chunks are columns
            const int64_t c = (t0 + static_cast<int64_t>(q) * kStreamPieceTiles) * kTileChunks +
                              poff(u) / kChunkBytes;
            if (pvec) {
              chunk_to_pairs<T>(__ldg(reinterpret_cast<const uint4 *>(p.gamma) + c), gp);
              if constexpr (OP == kLayerNorm)
                chunk_to_pairs<T>(__ldg(reinterpret_cast<const uint4 *>(p.beta) + c), bp);
            } else {
              load_param_pairs<T>(static_cast<const T *>(p.gamma), p.gamma ? p.cols : 0, c, 0,
                                  false, 1.f, gp);
              if constexpr (OP == kLayerNorm)
                load_param_pairs<T>(static_cast<const T *>(p.beta), p.beta ? p.cols : 0, c, 0,
                                    false, 0.f, bp);
            }
          }
          normalize_pairs<OP, NPAIR>(x, s0, s1, gp, bp);
          stg_stream(opiece + poff(u), pairs_to_chunk<T>(x));
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(sbase + L.bar_empty + 8u * s);
    }
    if (named_sync_or(kStreamBar, kThreads, bad)) {
      bad = true;
      break;
    }
  }
  if (bad && tid == 0) {
    atomicOr(p.status, kStatusTimeout);
    flags[0] = 1;
  }
  // no CTA leaves while a peer may still read its partials
  if (uses0 > 0) (void)mbar_wait_cluster_bounded(bar_released, (uses0 - 1) & 1, p.timeout_ns);
  if (uses1 > 0) (void)mbar_wait_cluster_bounded(bar_released + 8u, (uses1 - 1) & 1, p.timeout_ns);
}

}  // namespace rowop
