// bwd_call.h -- internal host interface of the ragged backward passes,
// between the C ABI (rowop_api.cu) and their launch code (bwd_launch.cuh).
#pragma once

#include <algorithm>

#include "common.cuh"
#include "dispatch.h"

namespace rowop {

// Backward pass over ragged rows (CSR offsets; the same offsets index a, dy
// and dx); ws holds a classify plan and, for the norms, the dgamma / dbeta
// partial rows of each bucket (bwd_ragged_layout).  a = y (softmax family)
// or x (norms); gamma / dgamma / dbeta / eps serve the norms.
struct BwdRaggedCall {
  int dtype;
  const void *a;
  const void *dy;
  void *dx;
  const void *gamma;
  void *dgamma;
  void *dbeta;
  float eps;
  const int64_t *offsets;
  int64_t rows, max_len;
  void *ws;
  cudaStream_t stream;
};

// Longest ragged row of the norms' backward: the element path holds 16
// elements per thread per tensor, in teams of up to 16 CTAs of 512 threads
// (checked against those constants in bwd_launch.cuh).
constexpr int64_t kBwdMaxColsNormRagged = 131072;

// Columns covered by the launch of each row bucket (SMALL, MEDIUM, LARGE) of
// rows up to max_len elements of esize bytes: the bucket's longest row, or 0
// when no row can fall in the bucket.
inline void bwd_ragged_covers(int64_t max_len, int esize, int64_t cover[3]) {
  const int64_t max_bytes = max_len * esize;
  cover[kSmall] = std::max<int64_t>(1, std::min(max_bytes, kSmallMaxBytes) / esize);
  cover[kMedium] = max_bytes > kSmallMaxBytes ? std::min(max_bytes, kMediumMaxBytes) / esize : 0;
  cover[kLarge] = max_bytes > kMediumMaxBytes ? max_len : 0;
}

// Norm workspace of a ragged backward call: the classify plan of `rows` rows,
// then for each bucket with a cover a segment of at most
// kBwdMaxPartsPerSm * sm partials of nacc rows of cover floats, each segment
// 256-byte aligned.  seg_off (may be NULL) receives the segment offsets;
// returns the total bytes.
inline size_t bwd_ragged_layout(int64_t rows, int64_t max_len, int esize, int nacc, int sm,
                                size_t seg_off[3]) {
  int64_t cover[3];
  bwd_ragged_covers(max_len, esize, cover);
  size_t off = (ragged_ws_bytes(rows) + 255) & ~static_cast<size_t>(255);
  for (int b = 0; b < 3; ++b) {
    if (seg_off) seg_off[b] = off;
    const size_t bytes = static_cast<size_t>(kBwdMaxPartsPerSm) * static_cast<size_t>(sm) *
                         static_cast<size_t>(nacc) * static_cast<size_t>(cover[b]) * sizeof(float);
    off = (off + bytes + 255) & ~static_cast<size_t>(255);
  }
  return off;
}

}  // namespace rowop
