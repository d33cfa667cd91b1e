// classify.cuh -- device-side launch_by_rows for ragged rows (§2.1): reads the
// int64 CSR offsets, gives every row its bucket, and appends each non-empty
// row's (start, length) record, in increasing row order, to its bucket's list
// by a block-wide prefix scan.  Every block handles its own contiguous range
// of rows and writes into its own segment of each list, plus its per-bucket
// counts, so blocks never wait on one another; the fused kernel that follows
// on the same stream turns the block counts into list positions.  No host
// round trip.
#pragma once

#include "common.cuh"

namespace rowop {

constexpr int kClassifyThreads = 1024;
constexpr int kClassifyPerThread = 8;
constexpr uint8_t kBucketRejected = 255;

struct ClassifyParams {
  const int64_t *offsets;
  int64_t rows;
  int64_t rows_per_block;
  int64_t max_len;
  int esize;
  uint8_t *bucket;          // [rows]
  RowRec *list[3];          // [rows] each: SMALL, MEDIUM, LARGE
  int32_t *block_counts;    // [blocks][3]
  unsigned int *ws_status;  // zeroed before the launch
  unsigned int *status;     // device status word
};

static __global__ void __launch_bounds__(kClassifyThreads)
    ragged_classify_kernel(const ClassifyParams p) {
  __shared__ int warp_tot[kClassifyThreads / 32][3];
  __shared__ int base[3];
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int64_t row0 = static_cast<int64_t>(blockIdx.x) * p.rows_per_block;
  const int64_t row1 = min(p.rows, row0 + p.rows_per_block);
  if (tid < 3) base[tid] = 0;
  __syncthreads();
  int any_bad = 0;
  for (int64_t blk = row0; blk < row1;
       blk += static_cast<int64_t>(kClassifyThreads) * kClassifyPerThread) {
    int b[kClassifyPerThread];
    int64_t st[kClassifyPerThread], ln[kClassifyPerThread];
    int cnt[3] = {0, 0, 0};
    const int64_t r0 = blk + static_cast<int64_t>(tid) * kClassifyPerThread;
#pragma unroll
    for (int i = 0; i < kClassifyPerThread; ++i) {
      const int64_t r = r0 + i;
      b[i] = -1;  // not listed
      st[i] = 0;
      ln[i] = 0;
      if (r < row1) {
        st[i] = p.offsets[r];
        ln[i] = p.offsets[r + 1] - st[i];
        if (ln[i] < 0 || ln[i] > p.max_len) {
          p.bucket[r] = kBucketRejected;
          any_bad = 1;
        } else {
          const int k = bucket_of(ln[i], p.esize);
          p.bucket[r] = static_cast<uint8_t>(k);
          if (ln[i] > 0) {
            b[i] = k;
            ++cnt[k];
          }
        }
      }
    }
    // inclusive warp scan of the three counts
    int inc[3] = {cnt[0], cnt[1], cnt[2]};
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
#pragma unroll
      for (int k = 0; k < 3; ++k) {
        const int v = __shfl_up_sync(kFullMask, inc[k], o);
        if (lane >= o) inc[k] += v;
      }
    }
    if (lane == 31) {
      warp_tot[warp][0] = inc[0];
      warp_tot[warp][1] = inc[1];
      warp_tot[warp][2] = inc[2];
    }
    __syncthreads();
    if (warp == 0) {  // exclusive scan over the 32 warp totals
#pragma unroll
      for (int k = 0; k < 3; ++k) {
        const int t = warp_tot[lane][k];
        int x = t;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int v = __shfl_up_sync(kFullMask, x, o);
          if (lane >= o) x += v;
        }
        warp_tot[lane][k] = x - t;
      }
    }
    __syncthreads();
    int pos[3];
#pragma unroll
    for (int k = 0; k < 3; ++k) pos[k] = base[k] + warp_tot[warp][k] + inc[k] - cnt[k];
#pragma unroll
    for (int i = 0; i < kClassifyPerThread; ++i) {
      if (b[i] >= 0) {
        RowRec rec;
        rec.start = st[i];
        rec.n = ln[i];
        p.list[b[i]][row0 + pos[b[i]]++] = rec;
      }
    }
    __syncthreads();
    if (tid == kClassifyThreads - 1) {
#pragma unroll
      for (int k = 0; k < 3; ++k) base[k] = pos[k];
    }
    __syncthreads();
  }
  any_bad = __syncthreads_or(any_bad);
  if (tid == 0) {
    p.block_counts[3 * blockIdx.x + 0] = base[0];
    p.block_counts[3 * blockIdx.x + 1] = base[1];
    p.block_counts[3 * blockIdx.x + 2] = base[2];
    if (any_bad) {
      atomicOr(p.ws_status, kStatusBadOffsets);
      atomicOr(p.status, kStatusBadOffsets);
    }
  }
}

}  // namespace rowop
