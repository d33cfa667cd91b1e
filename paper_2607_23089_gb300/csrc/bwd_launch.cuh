// bwd_launch.cuh -- host side of the backward passes: the team shape for the
// row length, the grid, and the dgamma / dbeta finalize launch.  Included by
// one translation unit per (operator, type) pair (bwd_instance.cu).
#pragma once

#include "bwd_call.h"
#include "bwd_row.cuh"
#include "bwd_stripe.cuh"
#include "bwd_tile.cuh"
#include "launch_util.cuh"

namespace rowop {

struct BwdShape {
  int tpr;  // threads of one CTA per row
  int nt;   // threads per CTA
  int cs;   // CTAs per row (cluster size)
};

// Team shape for rows of `units` chunk slots (16-byte window chunks, or
// groups of E elements) held CPT per thread: lane groups of a power of two up
// to a warp, whole warps up to 512 threads in one CTA, else a cluster of a
// power of two CTAs (up to 16).  CTAs of lane groups or small teams hold
// several teams: `small_cta` threads (256 for the softmax family; 128 for the
// norms, whose per-thread shared memory grows with the CTA).  `force_cs`
// (2..16) splits every row.
inline bool bwd_shape(int64_t units, int cpt, int force_cs, int small_cta, BwdShape &s) {
  const int64_t need = std::max<int64_t>(1, ceil_div(units, cpt));
  const auto warps32 = [](int64_t n) { return static_cast<int>(ceil_div(n, 32) * 32); };
  if (force_cs == 2 || force_cs == 4 || force_cs == 8 || force_cs == 16) {
    const int64_t per = ceil_div(need, force_cs);
    if (per <= kBwdMaxThreads) {
      s = {warps32(per), warps32(per), force_cs};
      return true;
    }
  }
  if (need <= 32) {
    int t = 1;
    while (t < need) t <<= 1;
    s = {t, small_cta, 1};
  } else if (need <= small_cta) {
    const int t = warps32(need);
    s = {t, t * (small_cta / t), 1};
  } else if (need <= kBwdMaxThreads) {
    const int t = warps32(need);
    s = {t, t, 1};
  } else {
    int cs = 2;
    while (cs < kMaxCluster && ceil_div(need, cs) > kBwdMaxThreads) cs <<= 1;
    if (ceil_div(need, cs) > kBwdMaxThreads) return false;
    const int t = warps32(ceil_div(need, cs));
    s = {t, t, cs};
  }
  return true;
}

template <typename T>
cudaError_t launch_bwd_finalize(const BwdSegments &sg, int64_t cols, int nacc, void *dgamma,
                                void *dbeta, cudaStream_t stream) {
  if (cols <= 0) return cudaSuccess;
  // a block per 32 columns, so many SMs share the reads, and 32 warps per
  // block over the partials, so each warp's chain of loads is short
  // a programmatic dependent launch: the finalize's launch overlaps the
  // tail of the kernel before it, whose results it waits for on the device
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(static_cast<unsigned>(ceil_div(cols, 32)), static_cast<unsigned>(nacc), 1);
  cfg.blockDim = dim3(kFinThreads, 1, 1);
  cfg.stream = stream;
  cudaError_t e = cudaLaunchKernelEx(&cfg, bwd_param_finalize_kernel<T>, sg, cols, nacc,
                                     static_cast<T *>(dgamma), static_cast<T *>(dbeta));
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// One segment of nparts partials covering all `cols` columns (a dense call).
inline BwdSegments one_segment(const float *part, int64_t nparts, int64_t cols) {
  BwdSegments sg = {};
  sg.part[0] = part;
  sg.nparts[0] = nparts;
  sg.cover[0] = cols;
  sg.n = 1;
  return sg;
}

// Launches the team kernel; with partials wanted (p.part), either adds them
// up into c.dgamma / c.dbeta (nparts_out NULL) or reports how many the
// launch writes (nparts_out) for the caller to add up.
template <int OP, typename T, int CPT, bool VEC, bool CLUSTER, bool RAGGED = false>
cudaError_t launch_bwd_k(const BwdParams &p, const BwdShape &s, const BwdCall &c,
                         const DeviceInfo &d, int64_t *nparts_out = nullptr) {
  auto kern = bwd_row_kernel<OP, T, CPT, VEC, CLUSTER, RAGGED>;
  const void *kp = reinterpret_cast<const void *>(kern);
  constexpr bool kNorm = (OP == kLayerNorm || OP == kRmsNorm);
  const int teams_cta = s.nt / s.tpr;
  // CTAs that hold several teams sum their dgamma / dbeta in shared memory
  const bool multi = !CLUSTER && (s.tpr < 32 || teams_cta > 1);
  constexpr int S = CPT * Elem<T>::kPerChunk;
  const size_t na = static_cast<size_t>(p.nacc);
  const size_t smem = (kNorm ? static_cast<size_t>(CPT) * s.nt * 16 : 0) +
                      ((kNorm && p.part) ? na * S * s.nt * sizeof(float) : 0) +
                      ((kNorm && p.part && multi) ? na * static_cast<size_t>(c.cols) * sizeof(float)
                                                  : 0);
  if (smem > static_cast<size_t>(d.max_smem_optin)) return cudaErrorInvalidConfiguration;
  {
    static std::mutex mu;
    static std::map<std::pair<const void *, int>, bool> done;
    std::lock_guard<std::mutex> lk(mu);
    const auto key = std::make_pair(kp, d.device);
    if (!done.count(key)) {
      cudaFuncAttributes fa;
      cudaError_t e = cudaFuncGetAttributes(&fa, kp);
      if (e != cudaSuccess) return e;
      e = cudaFuncSetAttribute(kp, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               d.max_smem_optin - static_cast<int>(fa.sharedSizeBytes));
      if (e != cudaSuccess) return e;
      if (CLUSTER) {
        e = cudaFuncSetAttribute(kp, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
      }
      done[key] = true;
    }
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  cfg.blockDim = dim3(s.nt, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = c.stream;
  const int64_t part_cap = static_cast<int64_t>(kBwdMaxPartsPerSm) * d.sm_count;
  int64_t grid, nparts;
  if (CLUSTER) {
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = s.cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(s.cs * std::max(1, d.sm_count / s.cs), 1, 1);
    int64_t ncl = std::max(1, cached_occupancy(kp, s.nt, smem, s.cs, &cfg));
    ncl = std::min<int64_t>(ncl, std::max<int64_t>(1, part_cap / s.cs));
    nparts = std::max<int64_t>(1, std::min<int64_t>(c.rows, ncl));
    grid = nparts * s.cs;
  } else {
    const int bps = std::max(1, cached_occupancy(kp, s.nt, smem, 1, nullptr));
    grid = std::max<int64_t>(1, std::min<int64_t>({ceil_div(c.rows, teams_cta),
                                                   static_cast<int64_t>(bps) * d.sm_count,
                                                   part_cap}));
    nparts = grid;
  }
  cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, p);
  if (e != cudaSuccess) return e;
  e = cudaGetLastError();
  if (e != cudaSuccess || !p.part) return e;
  if (nparts_out) {
    *nparts_out = nparts;
    return cudaSuccess;
  }
  return launch_bwd_finalize<T>(one_segment(p.part, nparts, c.cols), c.cols, p.nacc, c.dgamma,
                                c.dbeta, c.stream);
}

// The whole-tile norm kernel (bwd_tile.cuh) on rows of NW R tiles: compiled
// for 16 warps an SM, as many stages as the CTA's share of shared memory
// holds (up to kBwdTileMaxStages), a grid of at most the resident CTAs and
// at most one CTA per row, and the finalize over the grid's partial rows.
template <int OP, typename T, int R, int NW>
cudaError_t launch_bwd_tile_k(const BwdCall &c, const DeviceInfo &d) {
  constexpr int MINB = 16 / NW;
  auto kern = bwd_tile_kernel<OP, T, R, NW, MINB>;
  const void *kp = reinterpret_cast<const void *>(kern);
  cudaError_t e = prepare_kernel(kp, d, false);
  if (e != cudaSuccess) return e;
  constexpr uint32_t stage_bytes = 2u * NW * R * kTileBytes;
  const int stages = static_cast<int>(std::max<int64_t>(
      1, std::min<int64_t>(kBwdTileMaxStages, res_stage_budget(MINB) / stage_bytes)));
  const BwdTileSmem L(stage_bytes, stages, NW);
  const int occ = std::max(1, cached_occupancy(kp, NW * 32, L.total, 1, nullptr));
  const int64_t grid = std::max<int64_t>(
      1, std::min<int64_t>({c.rows, static_cast<int64_t>(occ) * d.sm_count,
                            static_cast<int64_t>(kBwdMaxPartsPerSm) * d.sm_count}));
  const bool want_params = c.dgamma || c.dbeta;
  BwdTileParams p = {};
  p.x = c.a;
  p.dy = c.dy;
  p.dx = c.dx;
  p.gamma = c.gamma;
  p.part = want_params ? static_cast<float *>(c.ws) : nullptr;
  p.rows = c.rows;
  p.cols = c.cols;
  p.ld = c.ld;
  p.eps = c.eps;
  p.stages = stages;
  p.stage_bytes = stage_bytes;
  p.timeout_ns = kWaitLimitNs;
  p.status = d.status;
  kern<<<static_cast<unsigned>(grid), NW * 32, L.total, c.stream>>>(p);
  e = cudaGetLastError();
  if (e != cudaSuccess || !want_params) return e;
  return launch_bwd_finalize<T>(one_segment(p.part, grid, c.cols), c.cols,
                                OP == kLayerNorm ? 2 : 1, c.dgamma, c.dbeta, c.stream);
}

// Dense norm rows the whole-tile kernel takes: x, dy and dx 16-byte aligned,
// a row stride of whole chunks, and rows of 4, 8 or 16 warps' tiles (one
// tile a warp for 16-bit types, two for fp32: 16 elements a lane per
// tensor).  Returns false, launching nothing, for any other shape.
template <int OP, typename T>
bool try_bwd_tile(const BwdCall &c, const DeviceInfo &d, cudaError_t *err) {
  constexpr int SZ = sizeof(T);
  constexpr int E = 16 / SZ;
  constexpr int R = SZ == 4 ? 2 : 1;
  if (c.rows <= 0 || !aligned16(c.a) || !aligned16(c.dy) || !aligned16(c.dx) ||
      (c.ld * SZ) % 16 != 0 || c.cols % (kTileChunks * E * R) != 0)
    return false;
  switch (c.cols / (kTileChunks * E * R)) {
    case 4:
      *err = launch_bwd_tile_k<OP, T, R, 4>(c, d);
      return true;
    case 8:
      *err = launch_bwd_tile_k<OP, T, R, 8>(c, d);
      return true;
    case 16:
      *err = launch_bwd_tile_k<OP, T, R, 16>(c, d);
      return true;
    default:
      return false;
  }
}

template <int OP, typename T>
cudaError_t launch_bwd_t(const BwdCall &c, const DeviceInfo &d) {
  constexpr int SZ = sizeof(T);
  constexpr int E = 16 / SZ;
  constexpr bool kNorm = (OP == kLayerNorm || OP == kRmsNorm);
  constexpr int CPT = kBwdSlots / E;
  const int small_cta = kNorm ? 128 : 256;
  const int nacc = OP == kLayerNorm ? 2 : 1;
  const bool want_params = kNorm && (c.dgamma || c.dbeta);
  if (c.rows == 0) {  // the parameter gradients of no rows are zero
    if (!want_params) return cudaSuccess;
    return launch_bwd_finalize<T>(one_segment(nullptr, 0, c.cols), c.cols, nacc, c.dgamma,
                                  c.dbeta, c.stream);
  }
  const Knobs kn = read_knobs();
  const int force_cs = kn.bwd_cluster;
  if constexpr (kNorm) {
    cudaError_t err = cudaSuccess;
    if (kn.bwd_tile != 0 && force_cs == 0 && try_bwd_tile<OP, T>(c, d, &err)) return err;
  }
  bool vec = ((c.ld * SZ) % 16 == 0) && congruent16(c.a, c.dy) && congruent16(c.a, c.dx);
  int h = vec ? static_cast<int>((reinterpret_cast<uintptr_t>(c.a) & 15u) / SZ) : 0;
  int64_t units = vec ? ceil_div(h + c.cols, E) : ceil_div(c.cols, E);
  BwdShape s;
  if (!bwd_shape(units, CPT, force_cs, small_cta, s)) {
    // a row of the longest length that starts mid-chunk needs one window
    // chunk more than the largest cluster holds: take the element path
    vec = false;
    h = 0;
    units = ceil_div(c.cols, E);
    if (!bwd_shape(units, CPT, force_cs, small_cta, s)) return cudaErrorInvalidValue;
  }
  BwdParams p = {};
  p.a = c.a;
  p.dy = c.dy;
  p.dx = c.dx;
  p.gamma = c.gamma;
  p.part = want_params ? static_cast<float *>(c.ws) : nullptr;
  p.rows = c.rows;
  p.cols = c.cols;
  p.ld = c.ld;
  p.eps = c.eps;
  p.tpr = s.tpr;
  p.h = h;
  p.nc = static_cast<int>(units);
  p.nacc = nacc;
  p.timeout_ns = kWaitLimitNs;
  p.status = d.status;
  if (s.cs > 1) {
    if (vec) return launch_bwd_k<OP, T, CPT, true, true>(p, s, c, d);
    return launch_bwd_k<OP, T, CPT, false, true>(p, s, c, d);
  }
  if (vec) return launch_bwd_k<OP, T, CPT, true, false>(p, s, c, d);
  return launch_bwd_k<OP, T, CPT, false, false>(p, s, c, d);
}

// Ragged norm rows by column stripes (bwd_stripe.cuh: the stats kernel, the
// dx kernel, then its own finalize over the group partial rows): x, dy and dx
// congruent modulo 16 bytes and, unless forced (mode 2), max_len of at
// least kStripeMinCols.  Returns false, launching nothing, otherwise.
template <int OP, typename T>
bool try_bwd_stripe(const BwdRaggedCall &c, const DeviceInfo &d, int mode, cudaError_t *err) {
  constexpr int SZ = sizeof(T);
  if (mode == 0 || c.rows <= 0 || c.max_len <= 0) return false;
  if (mode != 2 && c.max_len < kStripeMinCols) return false;
  if (!congruent16(c.a, c.dy) || !congruent16(c.a, c.dx)) return false;
  const int nacc = OP == kLayerNorm ? 2 : 1;
  const bool want_params = c.dgamma || c.dbeta;
  const StripeLayout L = stripe_layout(c.rows, c.max_len, SZ, nacc);
  unsigned char *ws = static_cast<unsigned char *>(c.ws);
  StripeParams p = {};
  p.x = c.a;
  p.dy = c.dy;
  p.dx = c.dx;
  p.gamma = c.gamma;
  p.offsets = c.offsets;
  p.rows = c.rows;
  p.max_len = c.max_len;
  p.eps = c.eps;
  p.hb = static_cast<int>((reinterpret_cast<uintptr_t>(c.a) & 15u) / SZ);
  p.psum = reinterpret_cast<float4 *>(ws + L.psum);
  p.part = want_params ? reinterpret_cast<float *>(ws + L.part) : nullptr;
  p.ns1 = L.ns1;
  p.ng1 = L.ng1;
  p.ns2 = L.ns2;
  p.ng2 = L.ng2;
  p.g2 = L.g2;
  p.status = d.status;
  const void *k1 = reinterpret_cast<const void *>(bwd_stripe_stats_kernel<OP, T>);
  const void *k2 = reinterpret_cast<const void *>(bwd_stripe_dx_kernel<OP, T>);
  cudaError_t e = reserve_dynamic_smem(k1, d, kStatRingBytes);
  if (e == cudaSuccess) e = reserve_dynamic_smem(k2, d, kDxRingBytes);
  if (e != cudaSuccess) {
    *err = e;
    return true;
  }
  bwd_stripe_stats_kernel<OP, T>
      <<<static_cast<unsigned>(L.ns1 * L.ng1), kStatThreads, kStatRingBytes, c.stream>>>(p);
  e = cudaGetLastError();
  if (e == cudaSuccess) {
    // a programmatic dependent launch: the dx kernel's CTAs sort their rows
    // while the stats kernel drains, and wait for it on the device
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(static_cast<unsigned>(L.ns2 * L.ng2), 1, 1);
    cfg.blockDim = dim3(kDxThreads, 1, 1);
    cfg.dynamicSmemBytes = kDxRingBytes;
    cfg.stream = c.stream;
    e = cudaLaunchKernelEx(&cfg, bwd_stripe_dx_kernel<OP, T>, p);
    if (e == cudaSuccess) e = cudaGetLastError();
  }
  if (e == cudaSuccess && want_params) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(static_cast<unsigned>(ceil_div(c.max_len, 64)), static_cast<unsigned>(nacc), 1);
    cfg.blockDim = dim3(kStripeFinThreads, 1, 1);
    cfg.stream = c.stream;
    e = cudaLaunchKernelEx(&cfg, bwd_stripe_finalize_kernel<T>, static_cast<const float *>(p.part),
                           L.ng2, L.ns2, static_cast<int>(stripe_dx_width(SZ)), 16 / SZ,
                           c.max_len, nacc, static_cast<T *>(c.dgamma), static_cast<T *>(c.dbeta));
    if (e == cudaSuccess) e = cudaGetLastError();
  }
  *err = e;
  return true;
}

// Ragged backward: the forward's classify pass sorts the rows into three
// buckets by byte length; each bucket that max_len allows gets one launch of
// the team kernel, shaped for the bucket's longest row, which walks that
// bucket's list.  Rows are independent, so each row's dx depends only on its
// values, length and alignment and on the shape of its bucket's teams.  The
// norms (element path) write each bucket's dgamma / dbeta partial rows into
// that bucket's workspace segment, covering its longest row, and one
// finalize adds the segments up in bucket order: the result depends on the
// rows' lengths and the device, not on their order in memory.
template <int OP, typename T>
cudaError_t launch_bwd_ragged_t(const BwdRaggedCall &c, const DeviceInfo &d) {
  constexpr int SZ = sizeof(T);
  constexpr int E = 16 / SZ;
  constexpr int CPT = kBwdSlots / E;
  constexpr bool kNorm = (OP == kLayerNorm || OP == kRmsNorm);
  // the norms' element path holds half the slots: one register per element
  // in flight (not one per two, as 16-byte chunks of 16-bit types take)
  constexpr int kCptN = CPT / 2;
  static_assert(static_cast<int64_t>(kCptN) * E * kBwdMaxThreads * kMaxCluster ==
                    kBwdMaxColsNormRagged,
                "the longest ragged norm row one team can hold");
  const int nacc = OP == kLayerNorm ? 2 : 1;
  const bool want_params = kNorm && (c.dgamma || c.dbeta);
  if constexpr (kNorm) {
    cudaError_t err = cudaSuccess;
    if (try_bwd_stripe<OP, T>(c, d, read_knobs().bwd_stripe, &err)) return err;
  }
  unsigned char *ws = static_cast<unsigned char *>(c.ws);
  size_t seg_off[3] = {0, 0, 0};
  if (kNorm) (void)bwd_ragged_layout(c.rows, c.max_len, SZ, nacc, d.sm_count, seg_off);
  int64_t cover[3];
  bwd_ragged_covers(c.max_len, SZ, cover);
  BwdSegments sg = {};
  if (c.rows > 0) {
    RaggedCall rc = {};
    rc.dtype = c.dtype;
    rc.offsets = c.offsets;
    rc.rows = c.rows;
    rc.max_len = c.max_len;
    rc.ws = c.ws;
    rc.stream = c.stream;
    rc.classify = true;
    cudaError_t e = launch_classify(rc, d);
    if (e != cudaSuccess) return e;
  }
  if (c.rows > 0 && c.max_len > 0) {
    const RowRec *list0 = reinterpret_cast<const RowRec *>(ws + ragged_lists_offset(c.rows));
    const bool vec = !kNorm && congruent16(c.a, c.dy) && congruent16(c.a, c.dx);
    BwdParams p = {};
    p.a = c.a;
    p.dy = c.dy;
    p.dx = c.dx;
    p.gamma = kNorm ? c.gamma : nullptr;
    p.rows = c.rows;  // an upper bound on every bucket's rows: sizes the grid
    p.ld = 0;
    p.eps = kNorm ? c.eps : 0.f;
    p.nacc = nacc;
    p.timeout_ns = kWaitLimitNs;
    p.status = d.status;
    p.block_counts = reinterpret_cast<const int32_t *>(ws + ragged_counts_offset(c.rows));
    p.blocks = static_cast<int>(ragged_blocks(c.rows));
    p.rows_per_block = ragged_rows_per_block(c.rows);
    const int small_cta = kNorm ? 128 : 256;
    for (int b = kSmall; b <= kLarge; ++b) {
      if (cover[b] == 0) continue;  // no row can be this long
      const int64_t longest = cover[b];
      bool bvec = vec;
      BwdShape s;
      const int cpt = kNorm ? kCptN : CPT;
      if (!bwd_shape(bvec ? ceil_div(longest + E - 1, E) : ceil_div(longest, E), cpt, 0,
                     small_cta, s)) {
        // the longest row, starting mid-chunk, needs a chunk more than the
        // largest cluster holds: this bucket takes the element path
        bvec = false;
        if (!bwd_shape(ceil_div(longest, E), cpt, 0, small_cta, s)) return cudaErrorInvalidValue;
      }
      p.list = list0 + static_cast<int64_t>(b) * c.rows;
      p.bucket = b;
      p.tpr = s.tpr;
      p.cols = longest;
      p.part = want_params ? reinterpret_cast<float *>(ws + seg_off[b]) : nullptr;
      BwdCall bc = {};
      bc.dtype = c.dtype;
      bc.a = c.a;
      bc.dy = c.dy;
      bc.dx = c.dx;
      bc.rows = c.rows;
      bc.cols = longest;
      bc.stream = c.stream;
      int64_t np = 0;
      cudaError_t e;
      if constexpr (kNorm) {
        e = s.cs > 1 ? launch_bwd_k<OP, T, kCptN, false, true, true>(p, s, bc, d, &np)
                     : launch_bwd_k<OP, T, kCptN, false, false, true>(p, s, bc, d, &np);
      } else if (s.cs > 1) {
        e = bvec ? launch_bwd_k<OP, T, CPT, true, true, true>(p, s, bc, d)
                 : launch_bwd_k<OP, T, CPT, false, true, true>(p, s, bc, d);
      } else {
        e = bvec ? launch_bwd_k<OP, T, CPT, true, false, true>(p, s, bc, d)
                 : launch_bwd_k<OP, T, CPT, false, false, true>(p, s, bc, d);
      }
      if (e != cudaSuccess) return e;
      if (want_params) {
        sg.part[sg.n] = p.part;
        sg.nparts[sg.n] = np;
        sg.cover[sg.n] = longest;
        ++sg.n;
      }
    }
  }
  if (!want_params) return cudaSuccess;
  return launch_bwd_finalize<T>(sg, c.max_len, nacc, c.dgamma, c.dbeta, c.stream);
}

}  // namespace rowop
