// launchers.cuh -- host side of launch_by_rows (§2.1): picks the bucket design
// for a call, sizes the stage ring, the cluster and the persistent grid, and
// launches.  Included by one translation unit per operator (ops_*.cu), which
// instantiates launch_dense<OP> and launch_ragged<OP>.
#pragma once

#include "launch_util.cuh"
#include "stream_row.cuh"
#include "small_row.cuh"
#include "tile_row.cuh"

namespace rowop {

// ---------------------------------------------------------------------------
// SMALL: register-resident rows, G lanes per row
// ---------------------------------------------------------------------------
template <int OP, typename T, int CPL, bool EXACT, bool RESID>
cudaError_t launch_small_k(const SmallParams &p, const DeviceInfo &d, cudaStream_t stream) {
  auto kern = small_row_kernel<OP, T, CPL, EXACT, RESID>;
  if constexpr (OP == kSoftmax || OP == kLogSoftmax) {
    if (read_knobs().softmax_online) kern = small_row_kernel<OP, T, CPL, EXACT, RESID, true>;
  }
  const int bps = cached_occupancy(reinterpret_cast<const void *>(kern), kCtaThreads, 0, 1,
                                   nullptr);
  const int64_t rows_per_cta = static_cast<int64_t>(kCtaWarps) * (32 / p.G);
  const int64_t want = ceil_div(p.rows, rows_per_cta);
  const int64_t cap = static_cast<int64_t>(std::max(bps, 1)) * d.sm_count;
  const int grid = static_cast<int>(std::max<int64_t>(1, std::min(want, cap)));
  kern<<<grid, kCtaThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

template <int OP, typename T, bool RESID>
cudaError_t launch_small(const DenseCall &c, const DeviceInfo &d, bool exact, bool out_vec,
                         bool gvec) {
  constexpr int SZ = sizeof(T);
  constexpr int E = 16 / SZ;
  SmallParams p;
  p.in = c.in;
  p.out = c.out;
  p.rows = c.rows;
  p.cols = c.cols;
  p.ld = c.ld;
  p.G = small_group_lanes(c.cols, SZ);
  p.a.gamma = c.gamma;
  p.a.beta = c.beta;
  p.a.glen = c.cols;
  p.a.eps = c.eps;
  p.a.gvec = gvec;
  p.a.out_vec = out_vec;
  p.resid = c.resid;
  p.sum_out = c.sum_out;
  p.rvec = RESID && congruent16(c.in, c.resid) && congruent16(c.in, c.sum_out);
  const int64_t max_chunks = ceil_div(c.cols, E) + (exact ? 0 : 1);
  const int cpl = small_cpl_class(max_chunks, p.G);
  if (exact) {
    if (cpl == 4) return launch_small_k<OP, T, 4, true, RESID>(p, d, c.stream);
    if (cpl == 8) return launch_small_k<OP, T, 8, true, RESID>(p, d, c.stream);
    return launch_small_k<OP, T, 9, true, RESID>(p, d, c.stream);
  }
  if (cpl == 4) return launch_small_k<OP, T, 4, false, RESID>(p, d, c.stream);
  if (cpl == 8) return launch_small_k<OP, T, 8, false, RESID>(p, d, c.stream);
  return launch_small_k<OP, T, 9, false, RESID>(p, d, c.stream);
}

// ---------------------------------------------------------------------------
// MEDIUM / LARGE / ragged: the tile kernel
// ---------------------------------------------------------------------------
// group_warps: consumer warps per item group (W); the stage ring holds at
// least one item per group.  min_stage_area: bytes the stages must span
// together (ragged SMALL staging).
template <int OP, typename T, bool EXACT, bool CLUSTER, bool RAGGED, bool RESID = false,
          bool ONLINE = false>
cudaError_t launch_tile_k(TileParams p, int cs, int stages, int stage_tiles, int group_warps,
                          int64_t items, const DeviceInfo &d, cudaStream_t stream,
                          uint32_t min_stage_area = 0) {
  auto kern = tile_row_kernel<OP, T, EXACT, CLUSTER, RAGGED, RESID, ONLINE>;
  const void *kp = reinterpret_cast<const void *>(kern);
  const int max_ctas_per_sm = read_knobs().ctas_per_sm;
  p.stage_bytes = static_cast<uint32_t>(stage_tiles) * kTileBytes;
  p.max_tiles = stage_tiles;
  while (static_cast<uint64_t>(stages) * p.stage_bytes < min_stage_area) ++stages;
  const auto total = [&](int s, int w) {
    return TileSmemLayout(p.stage_bytes, s, stage_tiles, kConsumerWarps / w, CLUSTER,
                          !CLUSTER || RAGGED, RAGGED ? p.blocks : 0).total;
  };
  // as many of the wanted stages as fit in the CTA's shared memory, at least
  // one per group: fewer, larger groups when even that does not fit
  const uint32_t optin = static_cast<uint32_t>(d.max_smem_optin);
  int W = group_warps;
  stages = std::max(stages, kConsumerWarps / W);
  for (;;) {
    const int G = kConsumerWarps / W;
    while (stages > G && total(stages, W) > optin) --stages;
    if (total(stages, W) <= optin) break;
    if (W == kConsumerWarps) return cudaErrorInvalidConfiguration;
    W *= 2;
  }
  if (static_cast<uint64_t>(stages) * p.stage_bytes < min_stage_area)
    return cudaErrorInvalidConfiguration;
  p.stages = stages;
  p.group_warps = W;
  const size_t smem = total(stages, W);
  if (smem > static_cast<size_t>(d.max_smem_optin)) return cudaErrorInvalidConfiguration;
  cudaError_t e = prepare_kernel(kp, d, CLUSTER);
  if (e != cudaSuccess) return e;

  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  cfg.blockDim = dim3(kTileThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  int grid;
  cfg.attrs = attr;
  cfg.numAttrs = 0;
  if (CLUSTER) {
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(cs * std::max(1, d.sm_count / cs), 1, 1);
    int ncl = cached_occupancy(kp, kTileThreads, smem, cs, &cfg);
    if (max_ctas_per_sm > 0) ncl = std::min(ncl, max_ctas_per_sm * d.sm_count / cs);
    if (ncl < 1) ncl = 1;
    grid = static_cast<int>(cs * std::max<int64_t>(1, std::min<int64_t>(items, ncl)));
  } else {
    int bps = std::max(1, cached_occupancy(kp, kTileThreads, smem, 1, nullptr));
    if (max_ctas_per_sm > 0) bps = std::min(bps, max_ctas_per_sm);
    grid = static_cast<int>(std::max<int64_t>(
        1, std::min<int64_t>(items, static_cast<int64_t>(bps) * d.sm_count)));
  }
  cfg.gridDim = dim3(grid, 1, 1);
  if (RAGGED) {
    // a programmatic dependent of the classify launch before it: the fused
    // kernel's launch and set-up overlap the classify tail, and its threads
    // wait on the device for the classify results
    attr[cfg.numAttrs].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[cfg.numAttrs].val.programmaticStreamSerializationAllowed = 1;
    ++cfg.numAttrs;
  }
  e = cudaLaunchKernelEx(&cfg, kern, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// MEDIUM / LARGE dense rows of whole tiles: the register-resident tile kernel
// ---------------------------------------------------------------------------
// Tiles a warp keeps in registers: 64 fp32 values of row data per lane
// (eight 1 KiB tiles of fp32, four of 16-bit elements).
template <typename T>
constexpr int res_max_r() {
  return (sizeof(T) == 4 ? kResMaxTilesF32 : kResMaxTiles16) / kResWarps;
}
// Whole-tile dense rows on the specialised resident kernel: each of the NW
// warps of a CTA owns exactly R tiles of each row (or of this CTA's portion
// of it).  4-warp CTAs are compiled for four CTAs an SM when they cache
// gamma/beta in registers and six when they do not, 8-warp CTAs with one tile
// a warp for three, the others for two.
template <int OP, typename T, int R, int NW, bool CLUSTER, bool GC>
cudaError_t launch_res_full_k(TileParams p, int cs, const DenseCall &c, const DeviceInfo &d) {
  constexpr int MINB = NW == 4 ? (GC ? 4 : 6) : (R == 1 ? 3 : 2);
  auto kern = resident_full_kernel<OP, T, R, NW, CLUSTER, GC, MINB>;
  const void *kp = reinterpret_cast<const void *>(kern);
  const Knobs kn = read_knobs();
  const int stage_tiles = NW * R;
  p.stage_bytes = static_cast<uint32_t>(stage_tiles) * kTileBytes;
  p.max_tiles = stage_tiles;
  p.group_warps = NW;
  const int64_t budget = res_stage_budget(MINB);
  int stages = kn.stages > 0 ? std::min(kn.stages, 32)
                             : static_cast<int>(std::max<int64_t>(
                                   1, std::min<int64_t>(16, budget / p.stage_bytes)));
  const auto total = [&](int st) {
    return ResSmemLayout(p.stage_bytes, st, stage_tiles, CLUSTER, 0).total;
  };
  const uint32_t optin = static_cast<uint32_t>(d.max_smem_optin);
  while (stages > 1 && total(stages) > optin) --stages;
  if (total(stages) > optin) return cudaErrorInvalidConfiguration;
  p.stages = stages;
  const size_t smem = total(stages);
  cudaError_t e = prepare_kernel(kp, d, CLUSTER);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  cfg.blockDim = dim3(NW * 32, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = c.stream;
  int grid;
  if (CLUSTER) {
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(cs * std::max(1, d.sm_count / cs), 1, 1);
    int ncl = cached_occupancy(kp, NW * 32, smem, cs, &cfg);
    if (kn.ctas_per_sm > 0) ncl = std::min(ncl, kn.ctas_per_sm * d.sm_count / cs);
    if (ncl < 1) ncl = 1;
    grid = static_cast<int>(cs * std::max<int64_t>(1, std::min<int64_t>(c.rows, ncl)));
  } else {
    int bps = std::max(1, cached_occupancy(kp, NW * 32, smem, 1, nullptr));
    if (kn.ctas_per_sm > 0) bps = std::min(bps, kn.ctas_per_sm);
    grid = static_cast<int>(std::max<int64_t>(
        1, std::min<int64_t>(c.rows, static_cast<int64_t>(bps) * d.sm_count)));
  }
  cfg.gridDim = dim3(grid, 1, 1);
  e = cudaLaunchKernelEx(&cfg, kern, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// Tries the whole-tile resident kernel for a dense call: rows a whole number
// of tiles, 16-byte aligned in and out, every row at a 16-byte boundary.
// One CTA per row when the row is MEDIUM and 8, 16 or 32 tiles long; a
// cluster of cs CTAs of R tiles a warp (the largest R that splits the row
// into 2..16 equal portions) when it is LARGE.  Returns false when the call
// does not qualify (the caller takes another design).
// LARGE dense rows whose cluster portions are whole 64-tile blocks: the
// streamed split (stream_row.cuh).  Portions of at most 128 tiles (the
// smallest such cluster) and a ring of 4 pieces, so three CTAs share an SM
// (measured on 256 x 262144 fp32 log-softmax: clusters of 8 with 4 pieces
// 106 us; 3 / 6 pieces 108 / 114 us; clusters of 4 / 16 118 / 132 us);
// ROWOP_CLUSTER and ROWOP_STAGES override.  Returns false, launching
// nothing, for any other shape.
template <int OP, typename T>
bool try_stream(const DenseCall &c, const DeviceInfo &d, const Knobs &kn, cudaError_t *err) {
  constexpr int SZ = sizeof(T);
  constexpr int E = 16 / SZ;
  constexpr bool kAffine = (OP == kLayerNorm || OP == kRmsNorm);
  if (kn.stream == 0 || c.rows <= 0) return false;
  if (!aligned16(c.in) || !aligned16(c.out) || (c.ld * SZ) % 16 != 0) return false;
  if (c.cols % (kTileChunks * E) != 0) return false;
  const int64_t K = c.cols / (kTileChunks * E);
  int cs = 2;
  if (kn.cluster > 1) {
    cs = kn.cluster;
  } else {
    while (cs < kMaxCluster && K / cs > 128) cs <<= 1;
  }
  if (K % (static_cast<int64_t>(cs) * kShortCombineTiles) != 0) return false;
  const int PT = static_cast<int>(K / cs);
  const int NP = kn.stages > 0 ? std::min(kn.stages, 16) : 4;
  const StreamSmem L(NP, PT);
  if (L.total > static_cast<uint32_t>(d.max_smem_optin)) return false;
  auto kern = stream_row_kernel<OP, T>;
  const void *kp = reinterpret_cast<const void *>(kern);
  cudaError_t e = prepare_kernel(kp, d, true);
  if (e != cudaSuccess) {
    *err = e;
    return true;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.blockDim = dim3(kStreamThreads, 1, 1);
  cfg.dynamicSmemBytes = L.total;
  cfg.stream = c.stream;
  cfg.gridDim = dim3(cs * std::max(1, d.sm_count / cs), 1, 1);
  int ncl = cached_occupancy(kp, kStreamThreads, L.total, cs, &cfg);
  if (kn.ctas_per_sm > 0) ncl = std::min(ncl, kn.ctas_per_sm * d.sm_count / cs);
  ncl = std::max(1, ncl);
  cfg.gridDim = dim3(static_cast<unsigned>(cs * std::min<int64_t>(c.rows, ncl)), 1, 1);
  StreamParams sp = {};
  sp.in = c.in;
  sp.out = c.out;
  sp.gamma = c.gamma;
  sp.beta = c.beta;
  sp.rows = c.rows;
  sp.cols = c.cols;
  sp.ld = c.ld;
  sp.eps = c.eps;
  sp.pieces = NP;
  sp.portion = PT;
  sp.gvec = kAffine && c.gamma && aligned16(c.gamma) &&
            (OP == kRmsNorm || (c.beta && aligned16(c.beta)));
  sp.timeout_ns = kWaitLimitNs;
  sp.status = d.status;
  e = cudaLaunchKernelEx(&cfg, kern, sp);
  *err = e != cudaSuccess ? e : cudaGetLastError();
  return true;
}

template <int OP, typename T>
bool try_res_full(const TileParams &p, const DenseCall &c, const DeviceInfo &d, int bucket,
                  const Knobs &kn, cudaError_t *err) {
  constexpr int SZ = sizeof(T);
  constexpr int E = 16 / SZ;
  constexpr bool kAffine = (OP == kLayerNorm || OP == kRmsNorm);
  if (!aligned16(c.in) || !aligned16(c.out) || (c.ld * SZ) % 16 != 0) return false;
  if (c.cols % (kTileChunks * E) != 0) return false;
  const int64_t K = c.cols / (kTileChunks * E);
  if (bucket == kMedium) {
    if (kn.cluster > 1) return false;
    if (K == 8) {  // four warps of two tiles: more of each row per lane
      *err = (kAffine && kn.res_gc) ? launch_res_full_k<OP, T, 2, 4, false, kAffine>(p, 1, c, d)
                                    : launch_res_full_k<OP, T, 2, 4, false, false>(p, 1, c, d);
      return true;
    }
    if (K == 16) {
      if constexpr (kAffine && SZ == 4) {
        *err = launch_res_full_k<OP, T, 2, 8, false, true>(p, 1, c, d);
      } else {
        *err = launch_res_full_k<OP, T, 2, 8, false, false>(p, 1, c, d);
      }
      return true;
    }
    if (K == 32) {
      *err = launch_res_full_k<OP, T, 4, 8, false, false>(p, 1, c, d);
      return true;
    }
    return false;
  }
  // LARGE: equal portions of R tiles a warp over a cluster of 2..16 CTAs --
  // on request only: two CTAs an SM fit fewer 16-CTA clusters than the
  // staged design's three (1 MiB fp32 rows: 155 us against 148 us)
  if (kn.resident < 2) return false;
  for (int R = res_max_r<T>(); R >= 2; R /= 2) {
    if (K % (kResWarps * R) != 0) continue;
    const int64_t cs = K / (kResWarps * R);
    if (cs < 2 || cs > kMaxCluster || (cs & (cs - 1)) != 0) continue;
    if (kn.cluster > 0 && kn.cluster != cs) continue;
    if (R == 2) {
      *err = launch_res_full_k<OP, T, 2, 8, true, false>(p, static_cast<int>(cs), c, d);
    } else if (R == 4) {
      *err = launch_res_full_k<OP, T, 4, 8, true, false>(p, static_cast<int>(cs), c, d);
    } else {
      if constexpr (SZ == 4) *err = launch_res_full_k<OP, T, 8, 8, true, false>(p, static_cast<int>(cs), c, d);
    }
    return true;
  }
  return false;
}

// Consumer warps per item group.  Items of a few tiles (dense rows of up to
// 16 KiB): groups of 2 warps, so several items are in work per CTA and one
// group's waits overlap the others' work.  Larger items: one group of all 8
// warps and a single stage, which keeps three CTAs on every SM -- measured
// faster than fewer CTAs that stage ahead (workloads 4 and 5).
inline int pick_group_warps(int64_t stage_tiles, bool ragged, int knob) {
  if (knob == 1 || knob == 2 || knob == 4 || knob == 8) return knob;
  if (!ragged && stage_tiles <= 16) return 2;
  return 8;
}


// Stages: one per group and up to one and a half per group within the
// three-CTA budget (a ragged launch, one group, gets a single stage: three
// CTAs with one large stage each beat fewer CTAs with two, as measured);
// stages too large for that budget get two per group (launch_tile_k then
// keeps as many as fit the CTA's shared memory).
inline int pick_stages(int64_t stage_tiles, int group_warps, int knob) {
  if (knob > 0) return std::min(knob, 32);
  const int G = kConsumerWarps / group_warps;
  const int64_t fit = kStageBudgetBytes / (stage_tiles * kTileBytes);
  if (fit >= G) return static_cast<int>(std::min<int64_t>(G + G / 2, fit));
  return 2 * G;
}

// Smallest cluster (power of two, >= 2) whose portions of a K-tile row hold
// at most `cap` tiles; 16 if none does.
inline int pick_cluster(int64_t K, int64_t cap, int knob) {
  if (knob == 1 || knob == 2 || knob == 4 || knob == 8 || knob == 16) return knob;
  int cs = 2;
  while (cs < kMaxCluster && ceil_div(K, cs) > cap) cs <<= 1;
  return cs;
}

template <int OP, typename T, bool RESID>
cudaError_t launch_dense_impl(const DenseCall &c, const DeviceInfo &d) {
  constexpr int SZ = sizeof(T);
  constexpr int E = 16 / SZ;
  const Knobs kn = read_knobs();
  const bool exact = aligned16(c.in) && aligned16(c.out) && ((c.ld * SZ) % 16 == 0) &&
                     (c.cols % E == 0);
  const bool out_vec = congruent16(c.in, c.out);
  const bool gvec = (!c.gamma || aligned16(c.gamma)) && (!c.beta || aligned16(c.beta));
  int bucket = bucket_of(c.cols, SZ);
  const int64_t nc_max = ceil_div(c.cols + (exact ? 0 : E - 1), E);
  const int64_t K = ceil_div(nc_max, kTileChunks);
  if (kn.force_bucket == kSmall && nc_max <= 9 * 32) bucket = kSmall;
  if (kn.force_bucket == kMedium && K <= kMaxPortionTiles) bucket = kMedium;
  if (kn.force_bucket == kLarge) bucket = kLarge;
  if (bucket == kMedium && K > kMaxPortionTiles) bucket = kLarge;

  if (bucket == kSmall) return launch_small<OP, T, RESID>(c, d, exact, out_vec, gvec);
  // LARGE rows of whole 64-tile blocks per cluster CTA: the streamed split
  // (not the online softmax statistics, another arithmetic)
  if (!RESID && out_vec && bucket == kLarge &&
      !((OP == kSoftmax || OP == kLogSoftmax) && kn.softmax_online)) {
    cudaError_t err = cudaSuccess;
    if (try_stream<OP, T>(c, d, kn, &err)) return err;
  }

  TileParams p = {};
  p.in = c.in;
  p.out = c.out;
  p.gamma = c.gamma;
  p.beta = c.beta;
  p.glen = c.cols;
  p.rows = c.rows;
  p.cols = c.cols;
  p.ld = c.ld;
  p.eps = c.eps;
  p.out_vec = out_vec;
  p.gvec = gvec;
  p.timeout_ns = kWaitLimitNs;
  p.status = d.status;
  p.resid = c.resid;
  p.sum_out = c.sum_out;
  p.rvec = RESID && congruent16(c.in, c.resid) && congruent16(c.in, c.sum_out);
  // portions within the three-CTA stage budget: a 1 MiB fp32 row goes to
  // clusters of 16 with 64 KiB per CTA, three CTAs per SM (0.17 ms on
  // workload 4 against 0.23 ms for clusters of 8 with 128 KiB, one per SM)
  const int cs = bucket == kMedium ? 1 : pick_cluster(K, kStageBudgetBytes / kTileBytes, kn.cluster);
  const int st = static_cast<int>(ceil_div(K, cs));
  if (st > kMaxPortionTiles) return cudaErrorInvalidValue;
  const int W = pick_group_warps(st, false, kn.group_warps);
  const int S = pick_stages(st, W, kn.stages);
  if constexpr ((OP == kSoftmax || OP == kLogSoftmax) && !RESID) {
    // the online one-pass tile statistics (a comparison variant, see Knobs)
    if (kn.softmax_online) {
      if (cs == 1) {
        if (exact)
          return launch_tile_k<OP, T, true, false, false, false, true>(p, 1, S, st, W, c.rows, d,
                                                                       c.stream);
        return launch_tile_k<OP, T, false, false, false, false, true>(p, 1, S, st, W, c.rows, d,
                                                                      c.stream);
      }
      if (exact)
        return launch_tile_k<OP, T, true, true, false, false, true>(p, cs, S, st, W, c.rows, d,
                                                                    c.stream);
      return launch_tile_k<OP, T, false, true, false, false, true>(p, cs, S, st, W, c.rows, d,
                                                                   c.stream);
    }
  }
  // the register-resident design: rows, or cluster portions, that the
  // consumer warps can hold in registers (one CTA: up to 32 tiles), output
  // 16-byte congruent to the input
  if (!RESID && kn.resident != 0 && out_vec) {
    cudaError_t err = cudaSuccess;
    if (try_res_full<OP, T>(p, c, d, bucket, kn, &err)) return err;
  }
  if (cs == 1) {
    if (exact)
      return launch_tile_k<OP, T, true, false, false, RESID>(p, 1, S, st, W, c.rows, d, c.stream);
    return launch_tile_k<OP, T, false, false, false, RESID>(p, 1, S, st, W, c.rows, d, c.stream);
  }
  if (exact)
    return launch_tile_k<OP, T, true, true, false, RESID>(p, cs, S, st, W, c.rows, d, c.stream);
  return launch_tile_k<OP, T, false, true, false, RESID>(p, cs, S, st, W, c.rows, d, c.stream);
}

// The dense launch path of one operator and type; the norms also serve the
// fused residual add when the call carries a residual.
template <int OP, typename T>
cudaError_t launch_dense_t(const DenseCall &c, const DeviceInfo &d) {
  if constexpr (OP == kLayerNorm || OP == kRmsNorm) {
    if (c.resid) return launch_dense_impl<OP, T, true>(c, d);
  }
  return launch_dense_impl<OP, T, false>(c, d);
}


template <int OP, typename T>
cudaError_t launch_ragged_t(const RaggedCall &c, const DeviceInfo &d) {
  constexpr int SZ = sizeof(T);
  constexpr int E = 16 / SZ;
  const Knobs kn = read_knobs();
  unsigned char *ws = static_cast<unsigned char *>(c.ws);
  const RowRec *list0 = reinterpret_cast<const RowRec *>(ws + ragged_lists_offset(c.rows));
  if (c.classify) {
    const cudaError_t e = launch_classify(c, d);
    if (e != cudaSuccess) return e;
  }
  if (c.max_len == 0) return cudaSuccess;

  TileParams p = {};
  p.in = c.in;
  p.out = c.out;
  p.gamma = c.gamma;
  p.beta = c.beta;
  p.glen = c.max_len;
  p.eps = c.eps;
  p.out_vec = congruent16(c.in, c.out);
  p.gvec = (!c.gamma || aligned16(c.gamma)) && (!c.beta || aligned16(c.beta));
  p.timeout_ns = kWaitLimitNs;
  p.status = d.status;
  p.rec_small = list0;
  p.rec_medium = list0 + c.rows;
  p.rec_large = list0 + 2 * c.rows;
  p.block_counts = reinterpret_cast<const int32_t *>(ws + ragged_counts_offset(c.rows));
  p.blocks = static_cast<int>(ragged_blocks(c.rows));
  p.rows_per_block = ragged_rows_per_block(c.rows);
  p.counters = reinterpret_cast<unsigned int *>(ws + kWsCounters);

  const int64_t kmax = ceil_div(ceil_div(c.max_len + E - 1, E), kTileChunks);
  const int64_t med_len = std::min<int64_t>(c.max_len, kMediumMaxBytes / SZ);
  const int64_t kmed = ceil_div(ceil_div(med_len + E - 1, E), kTileChunks);
  const bool has_large = bucket_of(c.max_len, SZ) == kLarge;
  int cs = 1;
  int64_t st = std::max<int64_t>(1, kmed);
  if (has_large) {
    // rows that fit one CTA's stage budget run whole on one CTA: the
    // cluster exchange costs more than it saves on them (measured); longer
    // ones are split over the smallest cluster that brings the portions
    // within that budget
    const int64_t budget = kStageBudgetBytes / kTileBytes;
    cs = (kn.cluster == 0 && kmax <= budget) ? 1
                                              : pick_cluster(kmax, std::max(kmed, budget), kn.cluster);
    st = std::max<int64_t>(st, ceil_div(kmax, cs));
  }
  const uint32_t small_area = kConsumerWarps * kSmallSliceBytes;
  if (st > kMaxPortionTiles) return cudaErrorInvalidValue;
  const int W = pick_group_warps(st, true, kn.group_warps);
  const int S = pick_stages(st, W, kn.stages);
  if (cs > 1)
    return launch_tile_k<OP, T, false, true, true>(p, cs, S, static_cast<int>(st), W, c.rows, d,
                                                   c.stream, small_area);
  return launch_tile_k<OP, T, false, false, true>(p, 1, S, static_cast<int>(st), W, c.rows, d,
                                                  c.stream, small_area);
}


}  // namespace rowop
