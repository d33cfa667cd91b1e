// dispatch.h -- internal host interface between the C ABI (rowop_api.cu) and
// the per-operator launch code (ops_*.cu).  Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace rowop {

struct DeviceInfo {
  int device;
  int sm_count;
  int max_smem_optin;      // bytes of dynamic shared memory a CTA may opt into
  unsigned int *status;    // device status word of this device
};

struct DenseCall {
  int dtype;  // 0 fp32, 1 bf16
  const void *in;
  void *out;
  const void *gamma;
  const void *beta;
  int64_t rows, cols, ld;
  float eps;
  cudaStream_t stream;
  // fused residual add (norms only): sum_out = in + resid, then the norm of
  // sum_out; both NULL for the plain operator
  const void *resid = nullptr;
  void *sum_out = nullptr;
};

struct RaggedCall {
  int dtype;
  const void *in;
  void *out;
  const void *gamma;
  const void *beta;
  const int64_t *offsets;
  int64_t rows, max_len;
  float eps;
  void *ws;
  cudaStream_t stream;
  bool classify;  // run the classify pass first (false: reuse a plan in ws)
};

// Hyena FFT-size padding: out[r][c] = scale * in[r][c] (c < seqlen), else 0.
struct PadCall {
  int dtype;
  const void *in;
  void *out;
  int64_t rows, seqlen, fft, ld_in, ld_out;
  float scale;
  cudaStream_t stream;
};

// MoE group score over groups of 32 consecutive experts (fp32 output).
struct MoeCall {
  int dtype;
  const void *scores;
  float *out;
  int64_t tokens, experts, ld;
  cudaStream_t stream;
};

// Backward pass of one operator over dense rows: `a` is the forward output y
// (softmax family) or the forward input x (norms); dgamma / dbeta (norms,
// either may be NULL) are column sums over all rows, formed from per-CTA
// partials in `ws`.
struct BwdCall {
  int dtype;
  const void *a;
  const void *dy;
  void *dx;
  const void *gamma;
  void *dgamma;
  void *dbeta;
  int64_t rows, cols, ld;
  float eps;
  void *ws;
  cudaStream_t stream;
};

// Partial rows of dgamma / dbeta: the backward launch never runs more than
// this many CTAs per SM (one partial row each).
constexpr int kBwdMaxPartsPerSm = 8;
// bytes of the partials workspace: nacc = 2 (LayerNorm) or 1 (RMSNorm)
inline size_t bwd_ws_bytes(int nacc, int64_t cols, int sm_count) {
  return static_cast<size_t>(kBwdMaxPartsPerSm) * static_cast<size_t>(sm_count) *
         static_cast<size_t>(nacc) * static_cast<size_t>(cols) * sizeof(float);
}
// Longest backward row: 16 CTAs of 512 threads holding 32 elements each.
constexpr int64_t kBwdMaxColsSoftmax = 16 * 512 * 32;
constexpr int64_t kBwdMaxColsNorm = 16 * 512 * 32;

cudaError_t launch_pad_scale(const PadCall &c, const DeviceInfo &d);
cudaError_t launch_moe_group_top2(const MoeCall &c, const DeviceInfo &d);

// Ragged workspace layout (bytes): [0,4) status bits of the call, [128,140)
// uint32 work counters, [256, 256+rows) uint8 bucket per row, then the int32
// per-bucket row counts of every classify block ([blocks][3], at
// ragged_counts_offset(rows)), then three lists (SMALL, MEDIUM, LARGE) of
// `rows` records {int64 start, int64 length} each, starting at
// ragged_lists_offset(rows).  Classify block b handles rows
// [b*rpb, (b+1)*rpb) (rpb = ragged_rows_per_block(rows)) and writes its
// records, in row order, from entry b*rpb of each list on.
constexpr size_t kWsStatus = 0;
constexpr size_t kWsCounters = 128;
constexpr size_t kWsHeader = 256;  // [0, 256) is zeroed before the classify launch
constexpr size_t kWsBuckets = 256;
constexpr size_t kWsRecordBytes = 16;
constexpr int64_t kClassifyRowsPerBlock = 1024;
constexpr int64_t kClassifyMaxBlocks = 256;
constexpr int64_t ragged_blocks(int64_t rows) {
  return rows <= 0 ? 1
                   : ((rows + kClassifyRowsPerBlock - 1) / kClassifyRowsPerBlock < kClassifyMaxBlocks
                          ? (rows + kClassifyRowsPerBlock - 1) / kClassifyRowsPerBlock
                          : kClassifyMaxBlocks);
}
constexpr int64_t ragged_rows_per_block(int64_t rows) {
  return rows <= 0 ? 1 : (rows + ragged_blocks(rows) - 1) / ragged_blocks(rows);
}
constexpr size_t ragged_counts_offset(int64_t rows) {
  return (kWsBuckets + static_cast<size_t>(rows) + 255) & ~static_cast<size_t>(255);
}
constexpr size_t ragged_lists_offset(int64_t rows) {
  return (ragged_counts_offset(rows) + 12 * static_cast<size_t>(ragged_blocks(rows)) + 255) &
         ~static_cast<size_t>(255);
}
constexpr size_t ragged_ws_bytes(int64_t rows) {
  return ragged_lists_offset(rows) + 3 * kWsRecordBytes * static_cast<size_t>(rows) + 256;
}

// Every bounded device wait gives up after this long.
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s
// Shared memory one CTA of the staged tile design spends on stages, so that
// three CTAs fit an SM.
constexpr int64_t kStageBudgetBytes = 72 * 1024;
// Shared memory one CTA of the register-resident design spends on stages
// when `ctas` CTAs share an SM's 228 KiB (a stage is refilled as soon as its
// row is in registers, so a few stages keep enough bytes in flight).
constexpr int64_t res_stage_budget(int ctas) { return (228 * 1024) / ctas - 8 * 1024; }
// Longest row portion (tiles) one CTA of the register-resident design holds:
// 64 fp32 values of row data per thread, 8 warps of 32 lanes, two 16-byte
// chunks a lane per tile.
constexpr int kResMaxTilesF32 = 64;
constexpr int kResMaxTiles16 = 32;

// Tile budget of one CTA portion: the longest row the resident split-row
// design takes is this many 1 KiB tiles per CTA times the largest cluster.
constexpr int kMaxPortionTiles = 192;
constexpr int kMaxCluster = 16;
inline int64_t max_row_len_elems(int esize) {
  const int64_t e = 16 / esize;
  return static_cast<int64_t>(kMaxPortionTiles) * kMaxCluster * 64 * e - (e - 1);
}

// Test-and-tuning knobs read from the environment (none changes results but
// ROWOP_SOFTMAX_ONLINE, ROWOP_BWD_CLUSTER and ROWOP_BWD_TILE, which select
// another way to round):
//   ROWOP_FORCE_BUCKET  0/1/2 -> dense rows use that design when it can hold
//                       the row (SMALL only for rows of <= 288 chunks)
//   ROWOP_CLUSTER       cluster size for split rows (1, 2, 4, 8, 16)
//   ROWOP_STAGES        stage-ring depth of the tile kernel
//   ROWOP_CTAS_PER_SM   upper bound on resident tile-kernel CTAs per SM
//   ROWOP_GROUP_WARPS   consumer warps per item group of the tile kernel (1, 2, 4, 8)
//   ROWOP_SOFTMAX_ONLINE 1 -> dense softmax / log-softmax use online one-pass
//                       statistics instead of the two-pass ones: SMALL rows
//                       a running maximum over the lane's chunks, MEDIUM /
//                       LARGE tiles one sweep over the stage (a comparison
//                       variant: its results differ by rounding)
//   ROWOP_BWD_CLUSTER   backward passes: split every row over a cluster of
//                       this many CTAs (2, 4, 8, 16); changes rounding order
//   ROWOP_RESIDENT      0 -> dense MEDIUM rows of whole tiles use the staged
//                       tile design instead of the register-resident one;
//                       2 -> LARGE rows of whole tiles use the resident one
//                       too, split over a cluster (all give the same bits)
//   ROWOP_RESIDENT_GC   0 -> the register-resident design reads gamma/beta
//                       per row instead of keeping them in registers (fewer
//                       registers, more CTAs an SM; the same bits)
//   ROWOP_STREAM        0 -> LARGE dense rows whose cluster portions are whole
//                       64-tile blocks are held in shared memory (the staged
//                       split) instead of streamed twice through a ring
//                       (the same bits)
//   ROWOP_BWD_TILE      0 -> dense norm backward rows of whole tiles use the
//                       team design instead of the whole-tile one (another
//                       summation order)
//   ROWOP_BWD_STRIPE    ragged norm backward: 0 -> the bucket launches of the
//                       team design for every max_len; 2 -> the column-stripe
//                       design for every max_len (default 1: from
//                       kStripeMinCols); another summation order
struct Knobs {
  int force_bucket = -1;
  int cluster = 0;
  int stages = 0;
  int ctas_per_sm = 0;
  int group_warps = 0;
  int softmax_online = 0;
  int bwd_cluster = 0;
  int resident = 1;
  int res_gc = 1;
  int bwd_tile = 1;
  int stream = 1;
  int bwd_stripe = 1;
};
Knobs read_knobs();

// Ragged classify pass into the workspace (defined in rowop_api.cu).
cudaError_t launch_classify(const RaggedCall &c, const DeviceInfo &d);



}  // namespace rowop
