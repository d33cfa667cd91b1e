// pad_moe.cu -- two more row-wise operators the paper traces, as HBM-bound
// streaming kernels for sm_103a:
//
//   * the Hyena FFT-size padding operator (§6, "Representative cross-layer
//     trace"): out[r][c] = scale * in[r][c] for c < seqlen, 0 up to fft_size;
//   * the MoE group score (§2.1, "A Running Example"): for every group of 32
//     consecutive expert scores, the largest sum of two distinct members,
//     i.e. the sum of the two largest values with a tied maximum counted
//     twice.
//
// Both work on a two-dimensional decomposition (rows x 16-byte chunks), so no
// element index is ever divided or reduced modulo a row length.
#include "common.cuh"
#include "dispatch.h"

namespace rowop {

constexpr int kPadThreads = 256;
constexpr int kPadWarps = kPadThreads / 32;
constexpr int kPadSegChunks = 512;  // 16-byte output chunks per work item
constexpr int kPadUnroll = 4;       // chunks each lane has in flight

struct PadParams {
  const void *in;
  void *out;
  int64_t rows, seqlen, fft, ld_in, ld_out;
  int64_t segs;  // work items per row
  float scale;
};

// One 16-byte output chunk c of a row (window aligned to the row start):
// live columns scaled from the input, columns past seqlen zero.
template <typename T>
__device__ __forceinline__ uint4 pad_chunk(const T *in_row, int64_t c, int64_t seqlen, float scale,
                                           bool full_live, uint4 raw) {
  constexpr int E = Elem<T>::kPerChunk;
  float v[E];
  if (full_live) {
    unpack<T>(raw, v);
#pragma unroll
    for (int e = 0; e < E; ++e) v[e] = __fmul_rn(v[e], scale);
  } else {
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const int64_t j = c * E + e;
      v[e] = j < seqlen ? __fmul_rn(load_elem(in_row + j), scale) : 0.f;
    }
  }
  return pack<T>(v);
}

// VEC: in/out rows 16-byte aligned and fft a whole number of chunks.  Work
// item = (row, segment of kPadSegChunks output chunks), taken round-robin by
// the warps of a persistent grid; each lane keeps kPadUnroll chunk loads in
// flight before it stores.
template <typename T, bool VEC>
__global__ void __launch_bounds__(kPadThreads) pad_scale_kernel(const PadParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  const int lane = threadIdx.x & 31;
  const int64_t warp = static_cast<int64_t>(blockIdx.x) * kPadWarps + (threadIdx.x >> 5);
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kPadWarps;
  const int64_t items = p.rows * p.segs;
  const T *in = static_cast<const T *>(p.in);
  T *out = static_cast<T *>(p.out);
  for (int64_t it = warp; it < items; it += nwarps) {
    const int64_t r = it / p.segs;
    const int64_t sg = it - r * p.segs;
    const T *in_row = in + r * p.ld_in;
    T *out_row = out + r * p.ld_out;
    if constexpr (VEC) {
      const int64_t nout = p.fft / E;
      const int64_t nlive = p.seqlen / E;  // chunks entirely inside seqlen
      const int64_t c_end = min(nout, (sg + 1) * kPadSegChunks);
      for (int64_t c0 = sg * kPadSegChunks; c0 < c_end; c0 += 32 * kPadUnroll) {
        uint4 raw[kPadUnroll];
#pragma unroll
        for (int u = 0; u < kPadUnroll; ++u) {
          const int64_t c = c0 + u * 32 + lane;
          raw[u] = (c < c_end && c < nlive) ? ldg_stream(in_row + c * E) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < kPadUnroll; ++u) {
          const int64_t c = c0 + u * 32 + lane;
          if (c < c_end)
            stg_stream(out_row + c * E, pad_chunk<T>(in_row, c, p.seqlen, p.scale, c < nlive, raw[u]));
        }
      }
    } else {
      const int64_t c_end = min(p.fft, (sg + 1) * kPadSegChunks * E);
      for (int64_t c = sg * kPadSegChunks * E + lane; c < c_end; c += 32)
        out_row[c] = from_f32<T>(c < p.seqlen ? __fmul_rn(load_elem(in_row + c), p.scale) : 0.f);
    }
  }
}

template <typename T>
cudaError_t launch_pad_scale_t(const PadCall &c, const DeviceInfo &d) {
  constexpr int SZ = sizeof(T);
  constexpr int E = 16 / SZ;
  PadParams p;
  p.in = c.in;
  p.out = c.out;
  p.rows = c.rows;
  p.seqlen = c.seqlen;
  p.fft = c.fft;
  p.ld_in = c.ld_in;
  p.ld_out = c.ld_out;
  p.scale = c.scale;
  const bool vec = (reinterpret_cast<uintptr_t>(c.in) % 16 == 0) &&
                   (reinterpret_cast<uintptr_t>(c.out) % 16 == 0) && (c.ld_in * SZ) % 16 == 0 &&
                   (c.ld_out * SZ) % 16 == 0 && c.fft % E == 0;
  const int64_t seg_elems = static_cast<int64_t>(kPadSegChunks) * E;
  p.segs = (c.fft + seg_elems - 1) / seg_elems;
  const int64_t items = p.rows * p.segs;
  auto kern = vec ? pad_scale_kernel<T, true> : pad_scale_kernel<T, false>;
  int bps = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, kern, kPadThreads, 0) != cudaSuccess) {
    cudaGetLastError();
    bps = 4;
  }
  const int64_t want = (items + kPadWarps - 1) / kPadWarps;
  const int grid = static_cast<int>(std::max<int64_t>(
      1, std::min<int64_t>(want, static_cast<int64_t>(std::max(bps, 1)) * d.sm_count)));
  kern<<<grid, kPadThreads, 0, c.stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_pad_scale(const PadCall &c, const DeviceInfo &d) {
  if (c.dtype == 0) return launch_pad_scale_t<float>(c, d);
  if (c.dtype == 2) return launch_pad_scale_t<__half>(c, d);
  return launch_pad_scale_t<__nv_bfloat16>(c, d);
}

// ---------------------------------------------------------------------------
// MoE group score
// ---------------------------------------------------------------------------
constexpr int kMoeGroup = 32;
constexpr int kMoeThreads = 256;
constexpr int kMoeWarps = kMoeThreads / 32;

struct MoeParams {
  const void *scores;
  float *out;
  int64_t tokens, experts, ld, groups;
};

// (t1, t2): the two largest values seen, t1 >= t2, as a multiset (a value
// seen twice fills both).  Merging two such pairs keeps the two largest of
// the four, with no comparison of positions.
__device__ __forceinline__ void top2_add(float &t1, float &t2, float v) {
  t2 = fmaxf(t2, fminf(t1, v));
  t1 = fmaxf(t1, v);
}
__device__ __forceinline__ void top2_merge(float &t1, float &t2, float u1, float u2) {
  t2 = fmaxf(fminf(t1, u1), fmaxf(t2, u2));
  t1 = fmaxf(t1, u1);
}
// butterfly over the `width` lanes of a group (xor offsets below width)
__device__ __forceinline__ void top2_group(float &t1, float &t2, int width) {
  for (int o = 1; o < width; o <<= 1) {
    const float u1 = __shfl_xor_sync(kFullMask, t1, o);
    const float u2 = __shfl_xor_sync(kFullMask, t2, o);
    top2_merge(t1, t2, u1, u2);
  }
}

// VEC: score rows 16-byte aligned; a group's 32 scores are the 32/E
// consecutive 16-byte chunks held by 32/E consecutive lanes.  Otherwise one
// score per lane, a group per warp step.
template <typename T, bool VEC>
__global__ void __launch_bounds__(kMoeThreads) moe_group_top2_kernel(const MoeParams p) {
  constexpr int E = Elem<T>::kPerChunk;
  constexpr int LG = kMoeGroup / E;  // lanes per group (VEC)
  const int lane = threadIdx.x & 31;
  const int64_t warp = static_cast<int64_t>(blockIdx.x) * kMoeWarps + (threadIdx.x >> 5);
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kMoeWarps;
  const T *scores = static_cast<const T *>(p.scores);
  for (int64_t t = warp; t < p.tokens; t += nwarps) {
    const T *row = scores + t * p.ld;
    float *orow = p.out + t * p.groups;
    if constexpr (VEC) {
      const int64_t nchunks = p.experts / E;  // a multiple of LG
      for (int64_t c0 = 0; c0 < nchunks; c0 += 32) {
        const int64_t c = c0 + lane;
        float t1 = -INFINITY, t2 = -INFINITY;
        if (c < nchunks) {
          float v[E];
          unpack<T>(ldg_stream(row + c * E), v);
#pragma unroll
          for (int e = 0; e < E; ++e) top2_add(t1, t2, v[e]);
        }
        top2_group(t1, t2, LG);  // lanes past the row end form whole groups of their own
        if (c < nchunks && (lane & (LG - 1)) == 0) orow[c / LG] = __fadd_rn(t1, t2);
      }
    } else {
      for (int64_t g = 0; g < p.groups; ++g) {
        float t1 = load_elem(row + g * kMoeGroup + lane), t2 = -INFINITY;
        top2_group(t1, t2, 32);
        if (lane == 0) orow[g] = __fadd_rn(t1, t2);
      }
    }
  }
}

template <typename T>
cudaError_t launch_moe_t(const MoeCall &c, const DeviceInfo &d) {
  constexpr int SZ = sizeof(T);
  MoeParams p;
  p.scores = c.scores;
  p.out = c.out;
  p.tokens = c.tokens;
  p.experts = c.experts;
  p.ld = c.ld;
  p.groups = c.experts / kMoeGroup;
  const bool vec = (reinterpret_cast<uintptr_t>(c.scores) % 16 == 0) && (c.ld * SZ) % 16 == 0;
  auto kern = vec ? moe_group_top2_kernel<T, true> : moe_group_top2_kernel<T, false>;
  int bps = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, kern, kMoeThreads, 0) != cudaSuccess) {
    cudaGetLastError();
    bps = 4;
  }
  const int64_t want = (c.tokens + kMoeWarps - 1) / kMoeWarps;
  const int grid = static_cast<int>(std::max<int64_t>(
      1, std::min<int64_t>(want, static_cast<int64_t>(std::max(bps, 1)) * d.sm_count)));
  kern<<<grid, kMoeThreads, 0, c.stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_moe_group_top2(const MoeCall &c, const DeviceInfo &d) {
  if (c.dtype == 0) return launch_moe_t<float>(c, d);
  if (c.dtype == 2) return launch_moe_t<__half>(c, d);
  return launch_moe_t<__nv_bfloat16>(c, d);
}

}  // namespace rowop
