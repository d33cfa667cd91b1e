// rowop_api.cu -- the C ABI of librowop (declared in include/rowop.h):
// synchronous argument validation, the per-device status word, and the hand
// off to the per-operator launch paths (launch_by_rows, §2.1).
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "bwd_call.h"
#include "classify.cuh"
#include "common.cuh"
#include "dispatch.h"
#include "rowop.h"

namespace rowop {

// The per-type launch paths, instantiated one (operator, type) pair per
// object file from ops_instance.cu.
template <int OP, typename T>
cudaError_t launch_dense_t(const DenseCall &c, const DeviceInfo &d);
template <int OP, typename T>
cudaError_t launch_ragged_t(const RaggedCall &c, const DeviceInfo &d);

// The backward passes, instantiated one (operator, type) pair per object file
// from bwd_instance.cu.
template <int OP, typename T>
cudaError_t launch_bwd_t(const BwdCall &c, const DeviceInfo &d);

template <int OP, typename T>
cudaError_t launch_bwd_ragged_t(const BwdRaggedCall &c, const DeviceInfo &d);

template <int OP>
static cudaError_t launch_bwd_ragged(const BwdRaggedCall &c, const DeviceInfo &d) {
  if (c.dtype == ROWOP_F32) return launch_bwd_ragged_t<OP, float>(c, d);
  if (c.dtype == ROWOP_F16) return launch_bwd_ragged_t<OP, __half>(c, d);
  return launch_bwd_ragged_t<OP, __nv_bfloat16>(c, d);
}

template <int OP>
static cudaError_t launch_bwd(const BwdCall &c, const DeviceInfo &d) {
  if (c.dtype == ROWOP_F32) return launch_bwd_t<OP, float>(c, d);
  if (c.dtype == ROWOP_F16) return launch_bwd_t<OP, __half>(c, d);
  return launch_bwd_t<OP, __nv_bfloat16>(c, d);
}

template <int OP>
static cudaError_t launch_dense(const DenseCall &c, const DeviceInfo &d) {
  if (c.dtype == ROWOP_F32) return launch_dense_t<OP, float>(c, d);
  if (c.dtype == ROWOP_F16) return launch_dense_t<OP, __half>(c, d);
  return launch_dense_t<OP, __nv_bfloat16>(c, d);
}
template <int OP>
static cudaError_t launch_ragged(const RaggedCall &c, const DeviceInfo &d) {
  if (c.dtype == ROWOP_F32) return launch_ragged_t<OP, float>(c, d);
  if (c.dtype == ROWOP_F16) return launch_ragged_t<OP, __half>(c, d);
  return launch_ragged_t<OP, __nv_bfloat16>(c, d);
}

// Device-side status bits (kStatusTimeout, kStatusBadOffsets), one word per
// device; kernels receive its address.
static __device__ unsigned int g_status_word;

static int env_int(const char *name, int dflt) {
  const char *v = std::getenv(name);
  if (!v || !*v) return dflt;
  return std::atoi(v);
}

Knobs read_knobs() {
  Knobs k;
  k.force_bucket = env_int("ROWOP_FORCE_BUCKET", -1);
  k.cluster = env_int("ROWOP_CLUSTER", 0);
  k.stages = env_int("ROWOP_STAGES", 0);
  k.ctas_per_sm = env_int("ROWOP_CTAS_PER_SM", 0);
  k.group_warps = env_int("ROWOP_GROUP_WARPS", 0);
  k.softmax_online = env_int("ROWOP_SOFTMAX_ONLINE", 0);
  k.bwd_cluster = env_int("ROWOP_BWD_CLUSTER", 0);
  k.resident = env_int("ROWOP_RESIDENT", 1);
  k.res_gc = env_int("ROWOP_RESIDENT_GC", 1);
  k.bwd_tile = env_int("ROWOP_BWD_TILE", 1);
  k.stream = env_int("ROWOP_STREAM", 1);
  k.bwd_stripe = env_int("ROWOP_BWD_STRIPE", 1);
  return k;
}

cudaError_t launch_classify(const RaggedCall &c, const DeviceInfo &d) {
  unsigned char *ws = static_cast<unsigned char *>(c.ws);
  RowRec *list0 = reinterpret_cast<RowRec *>(ws + ragged_lists_offset(c.rows));
  ClassifyParams cp;
  cp.offsets = c.offsets;
  cp.rows = c.rows;
  cp.rows_per_block = ragged_rows_per_block(c.rows);
  cp.max_len = c.max_len;
  cp.esize = c.dtype == 0 ? 4 : 2;
  cp.bucket = ws + kWsBuckets;
  cp.list[0] = list0;
  cp.list[1] = list0 + c.rows;
  cp.list[2] = list0 + 2 * c.rows;
  cp.block_counts = reinterpret_cast<int32_t *>(ws + ragged_counts_offset(c.rows));
  cp.ws_status = reinterpret_cast<unsigned int *>(ws + kWsStatus);
  cp.status = d.status;
  // status bits and work counters start at zero
  cudaError_t e = cudaMemsetAsync(ws, 0, kWsHeader, c.stream);
  if (e != cudaSuccess) return e;
  const int blocks = static_cast<int>(ragged_blocks(c.rows));
  ragged_classify_kernel<<<blocks, kClassifyThreads, 0, c.stream>>>(cp);
  return cudaGetLastError();
}

static int device_info(DeviceInfo *out) {
  static std::mutex mu;
  static DeviceInfo cache[64];
  static bool have[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return ROWOP_ERR_CUDA;
  }
  std::lock_guard<std::mutex> lk(mu);
  if (!have[dev]) {
    DeviceInfo d;
    d.device = dev;
    void *status = nullptr;
    if (cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&d.max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin,
                               dev) != cudaSuccess ||
        cudaGetSymbolAddress(&status, g_status_word) != cudaSuccess) {
      cudaGetLastError();
      return ROWOP_ERR_CUDA;
    }
    d.status = static_cast<unsigned int *>(status);
    cache[dev] = d;
    have[dev] = true;
  }
  *out = cache[dev];
  return ROWOP_OK;
}

// Library-owned ragged workspace of rowop_layernorm_ragged_static: one array
// per device (a __device__ variable has one instance in every device's
// context), sized for ROWOP_STATIC_MAX_ROWS rows.
constexpr size_t kStaticWsBytes = ragged_ws_bytes(ROWOP_STATIC_MAX_ROWS);
static __device__ __align__(256) unsigned char g_static_ws[kStaticWsBytes];

// Address of the current device's g_static_ws, looked up once per device.
static int static_workspace(void **ws) {
  static std::mutex mu;
  static void *addr[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return ROWOP_ERR_CUDA;
  }
  std::lock_guard<std::mutex> lk(mu);
  if (!addr[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_ws) != cudaSuccess || p == nullptr) {
      cudaGetLastError();
      return ROWOP_ERR_CUDA;
    }
    addr[dev] = p;
  }
  *ws = addr[dev];
  return ROWOP_OK;
}

static int esize_of(int dtype) {
  return dtype == ROWOP_F32 ? 4 : ((dtype == ROWOP_BF16 || dtype == ROWOP_F16) ? 2 : 0);
}

static bool elem_aligned(const void *p, int esize) {
  return (reinterpret_cast<uintptr_t>(p) % static_cast<uintptr_t>(esize)) == 0;
}

static bool eps_ok(float eps) { return std::isfinite(eps) && eps >= 0.f; }

// the last CUDA error that a call of this thread turned into ROWOP_ERR_CUDA
static thread_local cudaError_t t_last_cuda_error = cudaSuccess;

static int from_cuda(cudaError_t e) {
  if (e == cudaSuccess) return ROWOP_OK;
  t_last_cuda_error = e;
  cudaGetLastError();
  return ROWOP_ERR_CUDA;
}

// 0 = go on, 1 = valid no-op, else an error code (returned negated)
static int check_dense(const void *in, const void *out, const void *gamma, const void *beta,
                       int64_t rows, int64_t cols, int64_t ld, int dtype, float eps, bool norm) {
  const int es = esize_of(dtype);
  if (es == 0) return -ROWOP_ERR_UNSUPPORTED_DTYPE;
  if (rows < 0) return -ROWOP_ERR_INVALID_ARG;
  if (norm && !eps_ok(eps)) return -ROWOP_ERR_INVALID_ARG;
  if (rows == 0) return 1;
  if (cols <= 0 || ld < cols) return -ROWOP_ERR_INVALID_ARG;
  if (!in || !out) return -ROWOP_ERR_INVALID_ARG;
  if (!elem_aligned(in, es) || !elem_aligned(out, es)) return -ROWOP_ERR_INVALID_ARG;
  if ((gamma && !elem_aligned(gamma, es)) || (beta && !elem_aligned(beta, es)))
    return -ROWOP_ERR_INVALID_ARG;
  if (ld > INT64_MAX / es / rows) return -ROWOP_ERR_INVALID_ARG;
  if (cols > max_row_len_elems(es)) return -ROWOP_ERR_TOO_LONG;
  return 0;
}

static int run_dense(int op, const void *in, void *out, const void *gamma, const void *beta,
                     int64_t rows, int64_t cols, int64_t ld, rowop_dtype_t dtype, float eps,
                     cudaStream_t stream, const void *resid = nullptr, void *sum_out = nullptr) {
  const bool norm = (op == kLayerNorm || op == kRmsNorm);
  const int chk = check_dense(in, out, gamma, beta, rows, cols, ld, dtype, eps, norm);
  if (chk < 0) return -chk;
  if (resid || sum_out) {
    const int es = esize_of(dtype);
    if (!norm || !resid || !sum_out || !elem_aligned(resid, es) || !elem_aligned(sum_out, es))
      return ROWOP_ERR_INVALID_ARG;
  }
  if (chk == 1) return ROWOP_OK;
  DeviceInfo d;
  const int st = device_info(&d);
  if (st != ROWOP_OK) return st;
  DenseCall c;
  c.dtype = dtype;
  c.in = in;
  c.out = out;
  c.gamma = gamma;
  c.beta = beta;
  c.rows = rows;
  c.cols = cols;
  c.ld = ld;
  c.eps = eps;
  c.stream = stream;
  c.resid = resid;
  c.sum_out = sum_out;
  switch (op) {
    case kSoftmax: return from_cuda(launch_dense<kSoftmax>(c, d));
    case kLogSoftmax: return from_cuda(launch_dense<kLogSoftmax>(c, d));
    case kLayerNorm: return from_cuda(launch_dense<kLayerNorm>(c, d));
    default: return from_cuda(launch_dense<kRmsNorm>(c, d));
  }
}

// op < 0: only the classify pass (rowop_ragged_plan)
// Argument checks of a ragged call, everything but the workspace: the
// status the call returns for them, or ROWOP_OK.
static int check_ragged_args(int op, const void *in, const void *out, const void *gamma,
                             const void *beta, const int64_t *offsets, int64_t rows,
                             int64_t max_len, rowop_dtype_t dtype, float eps) {
  const int es = esize_of(dtype);
  const bool norm = (op == kLayerNorm || op == kRmsNorm);
  if (es == 0) return ROWOP_ERR_UNSUPPORTED_DTYPE;
  if (rows < 0 || rows > INT32_MAX - 1 || max_len < 0) return ROWOP_ERR_INVALID_ARG;
  if (norm && !eps_ok(eps)) return ROWOP_ERR_INVALID_ARG;
  if (rows == 0) return ROWOP_OK;
  if (!offsets || !elem_aligned(offsets, 8)) return ROWOP_ERR_INVALID_ARG;
  if (op >= 0 && (!in || !out || !elem_aligned(in, es) || !elem_aligned(out, es)))
    return ROWOP_ERR_INVALID_ARG;
  if ((gamma && !elem_aligned(gamma, es)) || (beta && !elem_aligned(beta, es)))
    return ROWOP_ERR_INVALID_ARG;
  if (max_len > max_row_len_elems(es)) return ROWOP_ERR_TOO_LONG;
  return ROWOP_OK;
}

static int run_ragged(int op, const void *in, void *out, const void *gamma, const void *beta,
                      const int64_t *offsets, int64_t rows, int64_t max_len,
                      rowop_dtype_t dtype, float eps, void *ws, size_t ws_bytes,
                      cudaStream_t stream, bool classify) {
  const int chk = check_ragged_args(op, in, out, gamma, beta, offsets, rows, max_len, dtype, eps);
  if (chk != ROWOP_OK || rows == 0) return chk;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0 ||
      ws_bytes < ragged_ws_bytes(rows))
    return ROWOP_ERR_WORKSPACE;
  DeviceInfo d;
  const int st = device_info(&d);
  if (st != ROWOP_OK) return st;
  RaggedCall c;
  c.dtype = dtype;
  c.in = in;
  c.out = out;
  c.gamma = gamma;
  c.beta = beta;
  c.offsets = offsets;
  c.rows = rows;
  c.max_len = max_len;
  c.eps = eps;
  c.ws = ws;
  c.stream = stream;
  c.classify = classify;
  if (op < 0) return from_cuda(launch_classify(c, d));
  switch (op) {
    case kSoftmax: return from_cuda(launch_ragged<kSoftmax>(c, d));
    case kLogSoftmax: return from_cuda(launch_ragged<kLogSoftmax>(c, d));
    case kLayerNorm: return from_cuda(launch_ragged<kLayerNorm>(c, d));
    default: return from_cuda(launch_ragged<kRmsNorm>(c, d));
  }
}

// Backward passes.  a = y (softmax family) or x (norms).
static int run_bwd(int op, const void *a, const void *dy, void *dx, const void *gamma,
                   void *dgamma, void *dbeta, int64_t rows, int64_t cols, int64_t ld,
                   rowop_dtype_t dtype, float eps, void *ws, size_t ws_bytes,
                   cudaStream_t stream) {
  const int es = esize_of(dtype);
  const bool norm = (op == kLayerNorm || op == kRmsNorm);
  if (es == 0) return ROWOP_ERR_UNSUPPORTED_DTYPE;
  if (rows < 0) return ROWOP_ERR_INVALID_ARG;
  if (norm && !eps_ok(eps)) return ROWOP_ERR_INVALID_ARG;
  const bool want = norm && (dgamma || dbeta);
  if (rows == 0 && !want) return ROWOP_OK;
  if (cols <= 0) return ROWOP_ERR_INVALID_ARG;
  if ((gamma && !elem_aligned(gamma, es)) || (dgamma && !elem_aligned(dgamma, es)) ||
      (dbeta && !elem_aligned(dbeta, es)))
    return ROWOP_ERR_INVALID_ARG;
  if (rows > 0) {
    if (ld < cols || !a || !dy || !dx) return ROWOP_ERR_INVALID_ARG;
    if (!elem_aligned(a, es) || !elem_aligned(dy, es) || !elem_aligned(dx, es))
      return ROWOP_ERR_INVALID_ARG;
    if (ld > INT64_MAX / es / rows) return ROWOP_ERR_INVALID_ARG;
  }
  if (cols > (norm ? kBwdMaxColsNorm : kBwdMaxColsSoftmax)) return ROWOP_ERR_TOO_LONG;
  DeviceInfo d;
  const int st = device_info(&d);
  if (st != ROWOP_OK) return st;
  if (want && rows > 0 &&
      (!ws || (reinterpret_cast<uintptr_t>(ws) & 15u) != 0 ||
       ws_bytes < bwd_ws_bytes(op == kLayerNorm ? 2 : 1, cols, d.sm_count)))
    return ROWOP_ERR_WORKSPACE;
  BwdCall c;
  c.dtype = dtype;
  c.a = a;
  c.dy = dy;
  c.dx = dx;
  c.gamma = gamma;
  c.dgamma = dgamma;
  c.dbeta = dbeta;
  c.rows = rows;
  c.cols = cols;
  c.ld = ld;
  c.eps = eps;
  c.ws = ws;
  c.stream = stream;
  switch (op) {
    case kSoftmax: return from_cuda(launch_bwd<kSoftmax>(c, d));
    case kLogSoftmax: return from_cuda(launch_bwd<kLogSoftmax>(c, d));
    case kLayerNorm: return from_cuda(launch_bwd<kLayerNorm>(c, d));
    default: return from_cuda(launch_bwd<kRmsNorm>(c, d));
  }
}

// Ragged backward passes.  a = y (softmax family) or x (norms).
static int run_bwd_ragged(int op, const void *a, const void *dy, void *dx, const void *gamma,
                          void *dgamma, void *dbeta, const int64_t *offsets, int64_t rows,
                          int64_t max_len, rowop_dtype_t dtype, float eps, void *ws,
                          size_t ws_bytes, cudaStream_t stream) {
  const int es = esize_of(dtype);
  const bool norm = (op == kLayerNorm || op == kRmsNorm);
  if (es == 0) return ROWOP_ERR_UNSUPPORTED_DTYPE;
  if (rows < 0 || rows > INT32_MAX - 1 || max_len < 0) return ROWOP_ERR_INVALID_ARG;
  if (norm && !eps_ok(eps)) return ROWOP_ERR_INVALID_ARG;
  const bool want = norm && (dgamma || dbeta) && max_len > 0;
  if (rows == 0 && !want) return ROWOP_OK;
  if ((gamma && !elem_aligned(gamma, es)) || (dgamma && !elem_aligned(dgamma, es)) ||
      (dbeta && !elem_aligned(dbeta, es)))
    return ROWOP_ERR_INVALID_ARG;
  if (rows > 0) {
    if (!offsets || !elem_aligned(offsets, 8)) return ROWOP_ERR_INVALID_ARG;
    if (!a || !dy || !dx || !elem_aligned(a, es) || !elem_aligned(dy, es) ||
        !elem_aligned(dx, es))
      return ROWOP_ERR_INVALID_ARG;
  }
  if (max_len > (norm ? kBwdMaxColsNormRagged : kBwdMaxColsSoftmax)) return ROWOP_ERR_TOO_LONG;
  // every call holds at least the classify plan; the norms' partial rows
  // follow it, sized by the device's SM count
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < ragged_ws_bytes(rows))
    return ROWOP_ERR_WORKSPACE;
  DeviceInfo d;
  const int st = device_info(&d);
  if (st != ROWOP_OK) return st;
  if (norm && ws_bytes < bwd_ragged_norm_ws(rows, max_len, es, op == kLayerNorm ? 2 : 1,
                                            d.sm_count))
    return ROWOP_ERR_WORKSPACE;
  BwdRaggedCall c;
  c.dtype = dtype;
  c.a = a;
  c.dy = dy;
  c.dx = dx;
  c.gamma = norm ? gamma : nullptr;
  c.dgamma = norm ? dgamma : nullptr;
  c.dbeta = op == kLayerNorm ? dbeta : nullptr;
  c.eps = eps;
  c.offsets = offsets;
  c.rows = rows;
  c.max_len = max_len;
  c.ws = ws;
  c.stream = stream;
  switch (op) {
    case kSoftmax: return from_cuda(launch_bwd_ragged<kSoftmax>(c, d));
    case kLogSoftmax: return from_cuda(launch_bwd_ragged<kLogSoftmax>(c, d));
    case kLayerNorm: return from_cuda(launch_bwd_ragged<kLayerNorm>(c, d));
    default: return from_cuda(launch_bwd_ragged<kRmsNorm>(c, d));
  }
}

static size_t bwd_ragged_workspace_size(int nacc, int64_t rows, int64_t max_len,
                                        rowop_dtype_t dtype) {
  const int es = esize_of(dtype);
  if (es == 0 || rows < 0 || max_len < 0) return 0;
  DeviceInfo d;
  if (device_info(&d) != ROWOP_OK) return 0;
  return bwd_ragged_norm_ws(rows, max_len, es, nacc, d.sm_count);
}

static size_t bwd_workspace_size(int nacc, int64_t cols) {
  if (cols <= 0) return 0;
  DeviceInfo d;
  if (device_info(&d) != ROWOP_OK) return 0;
  return bwd_ws_bytes(nacc, cols, d.sm_count);
}

// Waits on a barrier phase that only half of its expected arrivals reach, so
// the bounded wait must run out; records the timeout and returns.
__global__ void debug_wait_timeout_kernel(uint64_t limit_ns, unsigned int *status) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = smem_addr(&bar);
  if (threadIdx.x == 0) {
    mbar_init(b, 2);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_arrive(b);
  const bool ok = mbar_wait_bounded(b, 0, limit_ns);
  if (!ok && threadIdx.x == 0) atomicOr(status, kStatusTimeout);
  __syncthreads();
  if (threadIdx.x == 0) asm volatile("mbarrier.inval.shared::cta.b64 [%0];" ::"r"(b) : "memory");
}

}  // namespace rowop

using namespace rowop;

extern "C" {

int rowop_softmax(const void *in, void *out, int64_t rows, int64_t cols, int64_t ld,
                  rowop_dtype_t dtype, cudaStream_t stream) {
  return run_dense(kSoftmax, in, out, nullptr, nullptr, rows, cols, ld, dtype, 0.f, stream);
}

int rowop_logsoftmax(const void *in, void *out, int64_t rows, int64_t cols, int64_t ld,
                     rowop_dtype_t dtype, cudaStream_t stream) {
  return run_dense(kLogSoftmax, in, out, nullptr, nullptr, rows, cols, ld, dtype, 0.f, stream);
}

int rowop_layernorm(const void *in, void *out, const void *gamma, const void *beta,
                    int64_t rows, int64_t cols, int64_t ld, rowop_dtype_t dtype, float eps,
                    cudaStream_t stream) {
  return run_dense(kLayerNorm, in, out, gamma, beta, rows, cols, ld, dtype, eps, stream);
}

int rowop_rmsnorm(const void *in, void *out, const void *gamma, int64_t rows, int64_t cols,
                  int64_t ld, rowop_dtype_t dtype, float eps, cudaStream_t stream) {
  return run_dense(kRmsNorm, in, out, gamma, nullptr, rows, cols, ld, dtype, eps, stream);
}

int rowop_add_layernorm(const void *x, const void *r, void *sum_out, void *y,
                        const void *gamma, const void *beta, int64_t rows, int64_t cols,
                        int64_t ld, rowop_dtype_t dtype, float eps, cudaStream_t stream) {
  if (!r || !sum_out) return rows == 0 ? ROWOP_OK : ROWOP_ERR_INVALID_ARG;
  return run_dense(kLayerNorm, x, y, gamma, beta, rows, cols, ld, dtype, eps, stream, r,
                   sum_out);
}

int rowop_add_rmsnorm(const void *x, const void *r, void *sum_out, void *y, const void *gamma,
                      int64_t rows, int64_t cols, int64_t ld, rowop_dtype_t dtype, float eps,
                      cudaStream_t stream) {
  if (!r || !sum_out) return rows == 0 ? ROWOP_OK : ROWOP_ERR_INVALID_ARG;
  return run_dense(kRmsNorm, x, y, gamma, nullptr, rows, cols, ld, dtype, eps, stream, r,
                   sum_out);
}

int rowop_softmax_backward(const void *y, const void *dy, void *dx, int64_t rows, int64_t cols,
                           int64_t ld, rowop_dtype_t dtype, cudaStream_t stream) {
  return run_bwd(kSoftmax, y, dy, dx, nullptr, nullptr, nullptr, rows, cols, ld, dtype, 0.f,
                 nullptr, 0, stream);
}

int rowop_logsoftmax_backward(const void *y, const void *dy, void *dx, int64_t rows,
                              int64_t cols, int64_t ld, rowop_dtype_t dtype,
                              cudaStream_t stream) {
  return run_bwd(kLogSoftmax, y, dy, dx, nullptr, nullptr, nullptr, rows, cols, ld, dtype, 0.f,
                 nullptr, 0, stream);
}

int rowop_layernorm_backward(const void *x, const void *dy, const void *gamma, void *dx,
                             void *dgamma, void *dbeta, int64_t rows, int64_t cols, int64_t ld,
                             rowop_dtype_t dtype, float eps, void *ws, size_t ws_bytes,
                             cudaStream_t stream) {
  return run_bwd(kLayerNorm, x, dy, dx, gamma, dgamma, dbeta, rows, cols, ld, dtype, eps, ws,
                 ws_bytes, stream);
}

int rowop_rmsnorm_backward(const void *x, const void *dy, const void *gamma, void *dx,
                           void *dgamma, int64_t rows, int64_t cols, int64_t ld,
                           rowop_dtype_t dtype, float eps, void *ws, size_t ws_bytes,
                           cudaStream_t stream) {
  return run_bwd(kRmsNorm, x, dy, dx, gamma, dgamma, nullptr, rows, cols, ld, dtype, eps, ws,
                 ws_bytes, stream);
}

int rowop_softmax_backward_ragged(const void *y, const void *dy, void *dx, const int64_t *offsets,
                                  int64_t rows, int64_t max_len, rowop_dtype_t dtype, void *ws,
                                  size_t ws_bytes, cudaStream_t stream) {
  return run_bwd_ragged(kSoftmax, y, dy, dx, nullptr, nullptr, nullptr, offsets, rows, max_len,
                        dtype, 0.f, ws, ws_bytes, stream);
}

int rowop_logsoftmax_backward_ragged(const void *y, const void *dy, void *dx,
                                     const int64_t *offsets, int64_t rows, int64_t max_len,
                                     rowop_dtype_t dtype, void *ws, size_t ws_bytes,
                                     cudaStream_t stream) {
  return run_bwd_ragged(kLogSoftmax, y, dy, dx, nullptr, nullptr, nullptr, offsets, rows,
                        max_len, dtype, 0.f, ws, ws_bytes, stream);
}

int rowop_layernorm_backward_ragged(const void *x, const void *dy, const void *gamma, void *dx,
                                    void *dgamma, void *dbeta, const int64_t *offsets,
                                    int64_t rows, int64_t max_len, rowop_dtype_t dtype,
                                    float eps, void *ws, size_t ws_bytes, cudaStream_t stream) {
  return run_bwd_ragged(kLayerNorm, x, dy, dx, gamma, dgamma, dbeta, offsets, rows, max_len,
                        dtype, eps, ws, ws_bytes, stream);
}

int rowop_rmsnorm_backward_ragged(const void *x, const void *dy, const void *gamma, void *dx,
                                  void *dgamma, const int64_t *offsets, int64_t rows,
                                  int64_t max_len, rowop_dtype_t dtype, float eps, void *ws,
                                  size_t ws_bytes, cudaStream_t stream) {
  return run_bwd_ragged(kRmsNorm, x, dy, dx, gamma, dgamma, nullptr, offsets, rows, max_len,
                        dtype, eps, ws, ws_bytes, stream);
}

size_t rowop_layernorm_backward_ragged_workspace_size(int64_t rows, int64_t max_len,
                                                      rowop_dtype_t dtype) {
  return bwd_ragged_workspace_size(2, rows, max_len, dtype);
}

size_t rowop_rmsnorm_backward_ragged_workspace_size(int64_t rows, int64_t max_len,
                                                    rowop_dtype_t dtype) {
  return bwd_ragged_workspace_size(1, rows, max_len, dtype);
}

size_t rowop_layernorm_backward_workspace_size(int64_t cols) { return bwd_workspace_size(2, cols); }

size_t rowop_rmsnorm_backward_workspace_size(int64_t cols) { return bwd_workspace_size(1, cols); }

size_t rowop_ragged_workspace_size(int64_t rows) {
  return rows <= 0 ? 256 : ragged_ws_bytes(rows);
}

int rowop_softmax_ragged(const void *in, void *out, const int64_t *offsets, int64_t rows,
                         int64_t max_len, rowop_dtype_t dtype, void *ws, size_t ws_bytes,
                         cudaStream_t stream) {
  return run_ragged(kSoftmax, in, out, nullptr, nullptr, offsets, rows, max_len, dtype, 0.f, ws,
                    ws_bytes, stream, true);
}

int rowop_logsoftmax_ragged(const void *in, void *out, const int64_t *offsets, int64_t rows,
                            int64_t max_len, rowop_dtype_t dtype, void *ws, size_t ws_bytes,
                            cudaStream_t stream) {
  return run_ragged(kLogSoftmax, in, out, nullptr, nullptr, offsets, rows, max_len, dtype, 0.f,
                    ws, ws_bytes, stream, true);
}

int rowop_layernorm_ragged(const void *in, void *out, const void *gamma, const void *beta,
                           const int64_t *offsets, int64_t rows, int64_t max_len,
                           rowop_dtype_t dtype, float eps, void *ws, size_t ws_bytes,
                           cudaStream_t stream) {
  return run_ragged(kLayerNorm, in, out, gamma, beta, offsets, rows, max_len, dtype, eps, ws,
                    ws_bytes, stream, true);
}

int rowop_rmsnorm_ragged(const void *in, void *out, const void *gamma, const int64_t *offsets,
                         int64_t rows, int64_t max_len, rowop_dtype_t dtype, float eps,
                         void *ws, size_t ws_bytes, cudaStream_t stream) {
  return run_ragged(kRmsNorm, in, out, gamma, nullptr, offsets, rows, max_len, dtype, eps, ws,
                    ws_bytes, stream, true);
}

int rowop_ragged_plan(const int64_t *offsets, int64_t rows, int64_t max_len,
                      rowop_dtype_t dtype, void *ws, size_t ws_bytes, cudaStream_t stream) {
  return run_ragged(-1, nullptr, nullptr, nullptr, nullptr, offsets, rows, max_len, dtype, 0.f,
                    ws, ws_bytes, stream, true);
}

int rowop_softmax_ragged_planned(const void *in, void *out, const int64_t *offsets,
                                 int64_t rows, int64_t max_len, rowop_dtype_t dtype, void *ws,
                                 size_t ws_bytes, cudaStream_t stream) {
  return run_ragged(kSoftmax, in, out, nullptr, nullptr, offsets, rows, max_len, dtype, 0.f, ws,
                    ws_bytes, stream, false);
}

int rowop_logsoftmax_ragged_planned(const void *in, void *out, const int64_t *offsets,
                                    int64_t rows, int64_t max_len, rowop_dtype_t dtype,
                                    void *ws, size_t ws_bytes, cudaStream_t stream) {
  return run_ragged(kLogSoftmax, in, out, nullptr, nullptr, offsets, rows, max_len, dtype, 0.f,
                    ws, ws_bytes, stream, false);
}

int rowop_layernorm_ragged_planned(const void *in, void *out, const void *gamma,
                                   const void *beta, const int64_t *offsets, int64_t rows,
                                   int64_t max_len, rowop_dtype_t dtype, float eps, void *ws,
                                   size_t ws_bytes, cudaStream_t stream) {
  return run_ragged(kLayerNorm, in, out, gamma, beta, offsets, rows, max_len, dtype, eps, ws,
                    ws_bytes, stream, false);
}

int rowop_rmsnorm_ragged_planned(const void *in, void *out, const void *gamma,
                                 const int64_t *offsets, int64_t rows, int64_t max_len,
                                 rowop_dtype_t dtype, float eps, void *ws, size_t ws_bytes,
                                 cudaStream_t stream) {
  return run_ragged(kRmsNorm, in, out, gamma, nullptr, offsets, rows, max_len, dtype, eps, ws,
                    ws_bytes, stream, false);
}

int rowop_layernorm_ragged_static(const void *in, void *out, const void *gamma,
                                  const void *beta, const int64_t *offsets, int64_t rows,
                                  int64_t max_len, rowop_dtype_t dtype, float eps,
                                  cudaStream_t stream) {
  // argument errors first, as the caller-workspace call reports them; only a
  // call that is otherwise valid is refused for its row count
  const int chk = check_ragged_args(kLayerNorm, in, out, gamma, beta, offsets, rows, max_len,
                                    dtype, eps);
  if (chk != ROWOP_OK || rows == 0) return chk;
  if (rows > ROWOP_STATIC_MAX_ROWS) return ROWOP_ERR_WORKSPACE;
  void *ws = nullptr;
  const int st = static_workspace(&ws);
  if (st != ROWOP_OK) return st;
  return run_ragged(kLayerNorm, in, out, gamma, beta, offsets, rows, max_len, dtype, eps, ws,
                    kStaticWsBytes, stream, true);
}

int rowop_pad_scale(const void *in, void *out, int64_t rows, int64_t seqlen, int64_t fft_size,
                    int64_t ld_in, int64_t ld_out, float scale, rowop_dtype_t dtype,
                    cudaStream_t stream) {
  const int es = esize_of(dtype);
  if (es == 0) return ROWOP_ERR_UNSUPPORTED_DTYPE;
  if (rows < 0 || seqlen < 0 || fft_size < seqlen || !std::isfinite(scale))
    return ROWOP_ERR_INVALID_ARG;
  if (rows == 0 || fft_size == 0) return ROWOP_OK;
  if (!out || ld_out < fft_size || (seqlen > 0 && (!in || ld_in < seqlen)))
    return ROWOP_ERR_INVALID_ARG;
  if (!elem_aligned(out, es) || (in && !elem_aligned(in, es))) return ROWOP_ERR_INVALID_ARG;
  if (ld_out > INT64_MAX / es / rows || (seqlen > 0 && ld_in > INT64_MAX / es / rows))
    return ROWOP_ERR_INVALID_ARG;
  DeviceInfo d;
  const int st = device_info(&d);
  if (st != ROWOP_OK) return st;
  PadCall c;
  c.dtype = dtype;
  c.in = in;
  c.out = out;
  c.rows = rows;
  c.seqlen = seqlen;
  c.fft = fft_size;
  c.ld_in = seqlen > 0 ? ld_in : 0;
  c.ld_out = ld_out;
  c.scale = scale;
  c.stream = stream;
  return from_cuda(launch_pad_scale(c, d));
}

int rowop_moe_group_top2(const void *scores, float *out, int64_t tokens, int64_t experts,
                         int64_t ld, rowop_dtype_t dtype, cudaStream_t stream) {
  const int es = esize_of(dtype);
  if (es == 0) return ROWOP_ERR_UNSUPPORTED_DTYPE;
  if (tokens < 0 || experts <= 0 || experts % 32 != 0 || ld < experts)
    return ROWOP_ERR_INVALID_ARG;
  if (tokens == 0) return ROWOP_OK;
  if (!scores || !out || !elem_aligned(scores, es) || !elem_aligned(out, 4))
    return ROWOP_ERR_INVALID_ARG;
  if (ld > INT64_MAX / es / tokens) return ROWOP_ERR_INVALID_ARG;
  DeviceInfo d;
  const int st = device_info(&d);
  if (st != ROWOP_OK) return st;
  MoeCall c;
  c.dtype = dtype;
  c.scores = scores;
  c.out = out;
  c.tokens = tokens;
  c.experts = experts;
  c.ld = ld;
  c.stream = stream;
  return from_cuda(launch_moe_group_top2(c, d));
}

int rowop_select_bucket(int64_t len, rowop_dtype_t dtype) {
  const int es = esize_of(dtype);
  if (es == 0 || len < 0) return -1;
  return bucket_of(len, es);
}

int64_t rowop_max_row_len(rowop_dtype_t dtype) {
  const int es = esize_of(dtype);
  return es == 0 ? 0 : max_row_len_elems(es);
}

const char *rowop_last_cuda_error(void) { return cudaGetErrorString(t_last_cuda_error); }

const char *rowop_status_string(int status) {
  switch (status) {
    case ROWOP_OK: return "ROWOP_OK";
    case ROWOP_ERR_INVALID_ARG: return "ROWOP_ERR_INVALID_ARG: invalid argument";
    case ROWOP_ERR_UNSUPPORTED_DTYPE: return "ROWOP_ERR_UNSUPPORTED_DTYPE: unsupported dtype";
    case ROWOP_ERR_WORKSPACE: return "ROWOP_ERR_WORKSPACE: workspace missing, misaligned or too small";
    case ROWOP_ERR_CUDA: return "ROWOP_ERR_CUDA: a CUDA call or launch failed";
    case ROWOP_ERR_TIMEOUT: return "ROWOP_ERR_TIMEOUT: a bounded device wait ran out";
    case ROWOP_ERR_BAD_OFFSETS: return "ROWOP_ERR_BAD_OFFSETS: ragged rows rejected (decreasing offsets or len > max_len)";
    case ROWOP_ERR_TOO_LONG: return "ROWOP_ERR_TOO_LONG: row longer than rowop_max_row_len()";
    default: return "ROWOP: unknown status";
  }
}

int rowop_get_config(rowop_config_t *cfg) {
  if (!cfg) return ROWOP_ERR_INVALID_ARG;
  rowop_config_t c;
  std::memset(&c, 0, sizeof(c));
  c.size = sizeof(rowop_config_t);
  c.chunk_bytes = kChunkBytes;
  c.tile_bytes = kTileBytes;
  c.max_cluster = kMaxCluster;
  c.small_max_bytes = kSmallMaxBytes;
  c.medium_max_bytes = kMediumMaxBytes;
  c.max_row_len[ROWOP_F32] = max_row_len_elems(4);
  c.max_row_len[ROWOP_BF16] = max_row_len_elems(2);
  c.max_row_len[ROWOP_F16] = max_row_len_elems(2);
  c.resident_max_tiles[0] = kResMaxTilesF32;
  c.resident_max_tiles[1] = kResMaxTiles16;
  c.staged_max_tiles = kMaxPortionTiles;
  c.stage_budget_bytes[0] = res_stage_budget(2);
  c.stage_budget_bytes[1] = kStageBudgetBytes;
  c.wait_limit_ns = static_cast<int64_t>(kWaitLimitNs);
  c.static_max_rows = ROWOP_STATIC_MAX_ROWS;
  *cfg = c;
  return ROWOP_OK;
}

int rowop_check_status(cudaStream_t stream) {
  DeviceInfo d;
  const int st = device_info(&d);
  if (st != ROWOP_OK) return st;
  unsigned int word = 0;
  if (cudaStreamSynchronize(stream) != cudaSuccess ||
      cudaMemcpyAsync(&word, d.status, sizeof(word), cudaMemcpyDeviceToHost, stream) !=
          cudaSuccess ||
      cudaMemsetAsync(d.status, 0, sizeof(word), stream) != cudaSuccess ||
      cudaStreamSynchronize(stream) != cudaSuccess) {
    cudaGetLastError();
    return ROWOP_ERR_CUDA;
  }
  if (word & kStatusTimeout) return ROWOP_ERR_TIMEOUT;
  if (word & kStatusBadOffsets) return ROWOP_ERR_BAD_OFFSETS;
  return ROWOP_OK;
}

int rowop_debug_wait_timeout(int64_t limit_ns, cudaStream_t stream) {
  if (limit_ns < 1 || limit_ns > 1000000000LL) return ROWOP_ERR_INVALID_ARG;
  DeviceInfo d;
  const int st = device_info(&d);
  if (st != ROWOP_OK) return st;
  debug_wait_timeout_kernel<<<1, 32, 0, stream>>>(static_cast<uint64_t>(limit_ns), d.status);
  return from_cuda(cudaGetLastError());
}

}  // extern "C"
