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

// The striped ragged norm backward (bwd_stripe.cuh): each kernel's stripe
// is a range of 16-byte window chunks (one per chunk slot of its CTA), so a
// stripe's columns move with the row's head offset.
constexpr int kStatThreads = 256;  // threads of a stats CTA
constexpr int kStatChunks = 2;     // window chunks a stats lane holds per row
constexpr int kStatRows = 64;      // rows of a stats CTA
constexpr int kDxThreads = 256;    // threads of a dx CTA (one chunk a lane per row)
constexpr int kDxBatch = 256;      // rows a dx CTA sorts at a time
constexpr int kDxMaxGroups = 128;  // dgamma / dbeta partial rows at most
constexpr int kDxMinGroupRows = 32;
// max_len from which the ragged norm backward takes the striped design by
// default (ROWOP_BWD_STRIPE=1; 2 takes it for every max_len, 0 never)
constexpr int64_t kStripeMinCols = 2048;

inline int64_t stripe_stat_width(int esize) {
  return static_cast<int64_t>(16 / esize) * kStatThreads * kStatChunks;
}
inline int64_t stripe_dx_width(int esize) { return static_cast<int64_t>(16 / esize) * kDxThreads; }

// Workspace of the striped design, both parts 256-byte aligned: the
// per-stripe row statistics [rows][ns1] float4, and the dgamma / dbeta
// partial rows [ng2][ns2][nacc][W2 + E] float32 (a dx stripe's columns
// under every head offset).  ns = stripes covering window positions up to
// max_len + E - 1.
struct StripeLayout {
  int64_t ns1, ng1, ns2, ng2, g2;  // stripes and row groups of the two kernels
  size_t psum, part, total;
};

inline StripeLayout stripe_layout(int64_t rows, int64_t max_len, int esize, int nacc) {
  StripeLayout L = {};
  const auto up = [](size_t v) { return (v + 255) & ~static_cast<size_t>(255); };
  const int64_t span = max_len > 0 ? max_len + 16 / esize - 1 : 0;
  L.ns1 = (span + stripe_stat_width(esize) - 1) / stripe_stat_width(esize);
  L.ns2 = (span + stripe_dx_width(esize) - 1) / stripe_dx_width(esize);
  L.ng1 = (rows + kStatRows - 1) / kStatRows;
  L.ng2 = std::max<int64_t>(
      1, std::min<int64_t>((rows + kDxMinGroupRows - 1) / kDxMinGroupRows, kDxMaxGroups));
  L.g2 = (rows + L.ng2 - 1) / L.ng2;
  const size_t r = static_cast<size_t>(std::max<int64_t>(rows, 0));
  L.psum = 0;
  L.part = L.psum + up(r * static_cast<size_t>(L.ns1) * 16u);
  L.total = L.part + up(static_cast<size_t>(L.ng2) * static_cast<size_t>(L.ns2) *
                        static_cast<size_t>(nacc) *
                        static_cast<size_t>(stripe_dx_width(esize) + 16 / esize) * sizeof(float));
  return L;
}

// Workspace bytes of a ragged norm backward call: enough for either design.
inline size_t bwd_ragged_norm_ws(int64_t rows, int64_t max_len, int esize, int nacc, int sm) {
  return std::max(bwd_ragged_layout(rows, max_len, esize, nacc, sm, nullptr),
                  stripe_layout(rows, max_len, esize, nacc).total);
}

}  // namespace rowop
