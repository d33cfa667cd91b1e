// bwd_tile.cuh -- the LayerNorm / RMSNorm backward passes (the derivatives
// of §2.1's row-wise norms, as in bwd_row.cuh) for dense rows that are a
// whole number of 1 KiB tiles, 16-byte aligned.
//
// The forward's whole-tile design, applied to two input tensors:
//   * one lane of the CTA stages each row of x and of dy into the next
//     buffer of a stage ring, two bulk copies (cp.async.bulk, TMA) on one
//     mbarrier, S rows ahead;
//   * warp w of the CTA's NW warps owns tiles w, w + NW, ... (R of them) of
//     every row, and lane l of the warp chunks l and l + 32 of each: a lane
//     reads its 2R chunks of x and dy from the stage once and keeps them in
//     registers as fp32 pairs; after the row's first barrier every warp holds
//     its chunks and the issuing lane refills that stage with a later row;
//   * a lane owns the same columns in every row, so gamma at its columns is
//     loaded once per launch and its dgamma / dbeta sums over all of the
//     CTA's rows stay in registers.  At the end the CTA writes them as one
//     partial row; bwd_param_finalize_kernel sums the partial rows in index
//     order.
// Row sums: per lane in packed pairs, a butterfly over the warp, then the NW
// warps' values in warp order through shared memory at one named barrier
// per row.  LayerNorm: each warp first takes the mean of its own 512
// elements (a butterfly) and forms its sums about it from the registers;
// the warps' statistics are then merged (equal counts: the mean of the
// means, M2 plus 512 times the squared offsets of the means).
// Nothing is atomic and the order of every sum is fixed by the shape, so the
// result is bitwise reproducible.
#pragma once

#include "bwd_row.cuh"
#include "common.cuh"

namespace rowop {

constexpr uint32_t kBwdTileBar = 1;  // named barrier of the CTA's warps
constexpr int kBwdTileMaxStages = 8;

struct BwdTileParams {
  const void *x;
  const void *dy;
  void *dx;
  const void *gamma;  // NULL = ones
  float *part;        // [grid][nacc][cols] partial rows; NULL = not wanted
  int64_t rows, cols, ld;
  float eps;
  int stages;
  uint32_t stage_bytes;  // one row of x, then one row of dy
  uint64_t timeout_ns;
  unsigned int *status;
};

// Shared memory of the kernel (host and device agree on it): the stage ring,
// the per-warp sums of the two reduction rounds, the stage barriers and the
// abort flag.
struct BwdTileSmem {
  uint32_t red, bar_full, flags, total;
  __host__ __device__ BwdTileSmem(uint32_t stage_bytes, int stages, int nw) {
    uint32_t off = stage_bytes * static_cast<uint32_t>(stages);
    red = off;
    off += 2u * static_cast<uint32_t>(nw) * 16u;
    bar_full = off;
    off += static_cast<uint32_t>(stages) * 8u;
    flags = off;
    off += 16u;
    total = off;
  }
};

// Sum over the CTA's NW warps of NV lane values: a butterfly over the warp,
// lane 0 writes the warp's sums to red[w], a named barrier, then every thread
// adds the NW entries in warp order.  `bad` is or-ed over the CTA through the
// barrier; returns true when any thread passed bad.
template <int NV, int NW>
__device__ __forceinline__ bool bwd_cta_sum(float (&v)[NV], float4 *red, int w, int lane,
                                            bool bad) {
  static_assert(NV <= 4, "four sums per round");
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
    for (int i = 0; i < NV; ++i) v[i] = __fadd_rn(v[i], __shfl_xor_sync(kFullMask, v[i], o));
  }
  if (lane == 0) {
    float u[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int i = 0; i < NV; ++i) u[i] = v[i];
    red[w] = make_float4(u[0], u[1], u[2], u[3]);
  }
  if (named_sync_or(kBwdTileBar, NW * 32, bad)) return true;
  float4 t = red[0];
#pragma unroll
  for (int q = 1; q < NW; ++q) {
    const float4 u = red[q];
    t.x = __fadd_rn(t.x, u.x);
    t.y = __fadd_rn(t.y, u.y);
    t.z = __fadd_rn(t.z, u.z);
    t.w = __fadd_rn(t.w, u.w);
  }
  const float tt[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
  for (int i = 0; i < NV; ++i) v[i] = tt[i];
  return false;
}

// NW warps of R tiles each: rows of K = NW R tiles.  MINB: CTAs per SM the
// kernel is compiled for (its register budget).
template <int OP, typename T, int R, int NW, int MINB>
__global__ void __launch_bounds__(NW * 32, MINB) bwd_tile_kernel(const BwdTileParams p) {
  static_assert(OP == kLayerNorm || OP == kRmsNorm, "norm backward passes");
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int NP = E / 2;
  constexpr int SZ = Elem<T>::kSize;
  constexpr int NS = 2 * R;
  constexpr uint32_t kRowBytes = NW * R * kTileBytes;
  constexpr bool kLN = OP == kLayerNorm;
  constexpr int kWarpElems = NS * Elem<T>::kPerChunk * 32;  // elements a warp holds: 512
  static_assert((kWarpElems & (kWarpElems - 1)) == 0 && (NW & (NW - 1)) == 0, "exact scalings");
  extern __shared__ __align__(1024) unsigned char smem[];
  const BwdTileSmem L(p.stage_bytes, p.stages, NW);
  const int S = p.stages;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int w = tid >> 5;
  const int64_t cid = blockIdx.x;
  const int64_t ncta = gridDim.x;
  const uint32_t sbase = smem_addr(smem);
  volatile int *flags = reinterpret_cast<volatile int *>(smem + L.flags);
  float4 *red = reinterpret_cast<float4 *>(smem + L.red);
  const bool issuer = tid == 0;
  const int64_t row_bytes = p.ld * SZ;
  const char *xbase = static_cast<const char *>(p.x);
  const char *dybase = static_cast<const char *>(p.dy);
  char *dxbase = static_cast<char *>(p.dx);

  if (issuer) {
    for (int s = 0; s < S; ++s) mbar_init(sbase + L.bar_full + 8u * s, 1);
    flags[0] = 0;
    fence_mbar_init();
  }
  __syncthreads();
  const uint64_t pol = issuer ? l2_evict_first_policy() : 0;
  uint32_t fill_mask = 0;
  auto issue = [&](int s, int64_t r) {
    const uint32_t bar = sbase + L.bar_full + 8u * s;
    const uint32_t dst = sbase + static_cast<uint32_t>(s) * p.stage_bytes;
    mbar_arrive_expect_tx(bar, 2u * kRowBytes);
    bulk_g2s(dst, xbase + r * row_bytes, kRowBytes, bar, pol);
    bulk_g2s(dst + kRowBytes, dybase + r * row_bytes, kRowBytes, bar, pol);
  };
  if (issuer) {
    for (int s = 0; s < S; ++s) {
      const int64_t r = cid + s * ncta;
      if (r >= p.rows) break;
      issue(s, r);
      fill_mask |= 1u << s;
    }
  }

  // byte offset of each slot in the row (stage and global row alike)
  const uint32_t obase = static_cast<uint32_t>((w * kTileChunks + lane) * kChunkBytes);
  auto off = [&](int k) -> uint32_t {
    return obase + static_cast<uint32_t>((NW * (k >> 1) * kTileChunks + 32 * (k & 1)) * kChunkBytes);
  };
  // gamma at the lane's columns, once for all rows; the sums start at zero
  f2 gam[NS][NP], sg_acc[NS][NP], sb_acc[kLN ? NS : 1][NP];
  {
    const T *gamma = static_cast<const T *>(p.gamma);
    const bool gvec = gamma && (reinterpret_cast<uintptr_t>(gamma) & 15u) == 0;
#pragma unroll
    for (int k = 0; k < NS; ++k) {
      const int64_t c = off(k) / kChunkBytes;  // the slot's chunk of the row
      if (gvec) {
        chunk_to_pairs<T>(__ldg(reinterpret_cast<const uint4 *>(gamma) + c), gam[k]);
      } else {
        float g[E];
#pragma unroll
        for (int e = 0; e < E; ++e) g[e] = gamma ? load_elem(gamma + c * E + e) : 1.f;
#pragma unroll
        for (int i = 0; i < NP; ++i) gam[k][i] = f2_make(g[2 * i], g[2 * i + 1]);
      }
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        sg_acc[k][i] = f2_bcast(0.f);
        if constexpr (kLN) sb_acc[k][i] = f2_bcast(0.f);
      }
    }
  }
  const float inv_n = __frcp_rn(static_cast<float>(p.cols));

  int s = 0;
  uint32_t par = 0;
  for (int64_t j = 0;; ++j) {
    const int64_t r = cid + j * ncta;
    if (r >= p.rows) break;
    f2 x[NS][NP], d[NS][NP];
    bool bad = !mbar_wait_bounded(sbase + L.bar_full + 8u * s, par, p.timeout_ns);
    if (!bad) {
      const unsigned char *stage = smem + static_cast<size_t>(s) * p.stage_bytes;
#pragma unroll
      for (int k = 0; k < NS; ++k) {
        chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(stage + off(k)), x[k]);
        chunk_to_pairs<T>(*reinterpret_cast<const uint4 *>(stage + kRowBytes + off(k)), d[k]);
      }
    } else {
#pragma unroll
      for (int k = 0; k < NS; ++k)
#pragma unroll
        for (int i = 0; i < NP; ++i) x[k][i] = d[k][i] = f2_bcast(0.f);
    }
    // ---- the row's sums, one round through shared memory; past its
    // barrier every warp holds its chunks of row r, so the stage is
    // refilled ----
    float c0, c1, c2 = 0.f, sh = 0.f;
    bool stop;
    float4 *redj = red + NW * static_cast<int>(j & 1);
    if constexpr (kLN) {
      // each warp holds kWarpElems of the row: its own mean (a butterfly),
      // then its sums about that mean from the registers: sum (x - m_w)^2,
      // sum g, sum g (x - m_w), g = dy gamma
      f2 sx = f2_bcast(0.f);
#pragma unroll
      for (int k = 0; k < NS; ++k)
#pragma unroll
        for (int i = 0; i < NP; ++i) sx = f2_add(sx, x[k][i]);
      float t = f2_total(sx);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) t = __fadd_rn(t, __shfl_xor_sync(kFullMask, t, o));
      const float mw = __fmul_rn(t, 1.f / kWarpElems);  // a power of two: exact
      const f2 nmw = f2_bcast(-mw);
      f2 sdd = f2_bcast(0.f), sg = f2_bcast(0.f), sgd = f2_bcast(0.f);
#pragma unroll
      for (int k = 0; k < NS; ++k)
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          x[k][i] = f2_add(x[k][i], nmw);  // x - m_w from here on
          const f2 gg = f2_mul(d[k][i], gam[k][i]);
          sdd = f2_fma(x[k][i], x[k][i], sdd);
          sg = f2_add(sg, gg);
          sgd = f2_fma(gg, x[k][i], sgd);
        }
      float v[3] = {f2_total(sdd), f2_total(sg), f2_total(sgd)};
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
        for (int q = 0; q < 3; ++q) v[q] = __fadd_rn(v[q], __shfl_xor_sync(kFullMask, v[q], o));
      }
      if (lane == 0) redj[w] = make_float4(mw, v[0], v[1], v[2]);
      stop = named_sync_or(kBwdTileBar, NW * 32, bad);
      if (!stop) {
        // the warps' statistics merged (equal counts), in warp order: the
        // mean of the means, M2 = sum M2_w + n_w sum (m_w - mean)^2,
        // sum g (x - mean) = sum (sum g (x - m_w) + sum g (m_w - mean))
        float sm = redj[0].x;
#pragma unroll 4
        for (int q = 1; q < NW; ++q) sm = __fadd_rn(sm, redj[q].x);
        const float mean = __fmul_rn(sm, 1.f / NW);  // a power of two: exact
        float m2 = 0.f, dd = 0.f, st = 0.f, stx = 0.f;
#pragma unroll 2
        for (int q = 0; q < NW; ++q) {
          const float4 u = redj[q];
          const float dm = __fsub_rn(u.x, mean);
          m2 = __fadd_rn(m2, u.y);
          dd = __fmaf_rn(dm, dm, dd);
          st = __fadd_rn(st, u.z);
          stx = __fadd_rn(stx, __fmaf_rn(u.z, dm, u.w));
        }
        m2 = __fmaf_rn(static_cast<float>(kWarpElems), dd, m2);
        c0 = rsqrtf(__fmaf_rn(m2, inv_n, p.eps));     // rstd
        c1 = __fmul_rn(st, inv_n);                    // mean(g)
        c2 = __fmul_rn(__fmul_rn(stx, c0), inv_n);    // mean(g xhat)
        sh = __fmul_rn(__fsub_rn(mw, mean), c0);      // (m_w - mean) rstd
      }
    } else {
      f2 sxx = f2_bcast(0.f), sgx = f2_bcast(0.f);
#pragma unroll
      for (int k = 0; k < NS; ++k)
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          sxx = f2_fma(x[k][i], x[k][i], sxx);
          sgx = f2_fma(f2_mul(d[k][i], gam[k][i]), x[k][i], sgx);
        }
      float v[2] = {f2_total(sxx), f2_total(sgx)};
      stop = bwd_cta_sum<2, NW>(v, redj, w, lane, bad);
      c0 = rsqrtf(__fmaf_rn(v[0], inv_n, p.eps));  // rstd
      c1 = __fmul_rn(__fmul_rn(v[1], c0), inv_n);  // mean(g xhat)
    }
    if (stop) {
      if (issuer) {
        atomicOr(p.status, kStatusTimeout);
        flags[0] = 1;
      }
      break;
    }
    if (issuer) {  // refill the stage with row r + S ncta
      const int64_t rn = r + static_cast<int64_t>(S) * ncta;
      if (rn < p.rows) {
        fence_proxy_async_smem();
        issue(s, rn);
      } else {
        fill_mask &= ~(1u << s);
      }
    }
    if (++s == S) {
      s = 0;
      par ^= 1u;
    }
    // ---- dx = rstd (g - mean(g) - xhat mean(g xhat)), and the lane's
    // dgamma (dy xhat) and dbeta (dy) sums ----
    const f2 C0 = f2_bcast(c0), NC1 = f2_bcast(-c1), NC2 = f2_bcast(-c2), SH = f2_bcast(sh);
    char *dxrow = dxbase + r * row_bytes;
#pragma unroll
    for (int k = 0; k < NS; ++k) {
      f2 o[NP];
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        // LayerNorm: x holds x - m_w; xhat = (x - m_w) rstd + (m_w - mean) rstd
        const f2 xh = kLN ? f2_fma(x[k][i], C0, SH) : f2_mul(x[k][i], C0);
        f2 t = kLN ? f2_fma(d[k][i], gam[k][i], NC1) : f2_mul(d[k][i], gam[k][i]);
        t = f2_fma(xh, kLN ? NC2 : NC1, t);
        o[i] = f2_mul(C0, t);
        sg_acc[k][i] = f2_fma(d[k][i], xh, sg_acc[k][i]);
        if constexpr (kLN) sb_acc[k][i] = f2_add(sb_acc[k][i], d[k][i]);
      }
      stg_stream(dxrow + off(k), pairs_to_chunk<T>(o));
    }
  }

  // a CTA that gave up must not leave copies in flight into its stages
  if (issuer && flags[0]) {
    for (int i = 0; i < S; ++i) {
      const int si = (s + i) % S;
      if (fill_mask >> si & 1u)
        (void)mbar_wait_bounded(sbase + L.bar_full + 8u * si, si >= s ? par : par ^ 1u,
                                p.timeout_ns);
    }
  }
  // ---- this CTA's partial row(s) ----
  if (p.part) {
    constexpr int NA = kLN ? 2 : 1;
    float *prow = p.part + cid * NA * p.cols;
#pragma unroll
    for (int k = 0; k < NS; ++k) {
      const int64_t c0i = static_cast<int64_t>(off(k) / kChunkBytes) * E;
#pragma unroll
      for (int q = 0; q < NP / 2; ++q) {
        reinterpret_cast<float4 *>(prow + c0i)[q] =
            make_float4(sg_acc[k][2 * q].x, sg_acc[k][2 * q].y, sg_acc[k][2 * q + 1].x,
                        sg_acc[k][2 * q + 1].y);
        if constexpr (kLN)
          reinterpret_cast<float4 *>(prow + p.cols + c0i)[q] =
              make_float4(sb_acc[k][2 * q].x, sb_acc[k][2 * q].y, sb_acc[k][2 * q + 1].x,
                          sb_acc[k][2 * q + 1].y);
      }
    }
  }
}

}  // namespace rowop
