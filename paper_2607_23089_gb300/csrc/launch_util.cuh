// launch_util.cuh -- host helpers shared by the launch paths: alignment
// tests, cached occupancy queries and one-time kernel attributes.
#pragma once

#include <algorithm>
#include <map>
#include <mutex>
#include <tuple>

#include "dispatch.h"

namespace rowop {


inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline bool congruent16(const void *a, const void *b) {
  return ((reinterpret_cast<uintptr_t>(a) ^ reinterpret_cast<uintptr_t>(b)) & 15u) == 0;
}
inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Occupancy answers are cached per (kernel, block, shared memory, cluster size, device).
inline int cached_occupancy(const void *kernel, int threads, size_t smem, int cluster,
                            const cudaLaunchConfig_t *cfg) {
  static std::mutex mu;
  static std::map<std::tuple<const void *, int, size_t, int, int>, int> cache;
  int dev = 0;
  cudaGetDevice(&dev);
  const auto key = std::make_tuple(kernel, threads, smem, cluster, dev);
  {
    std::lock_guard<std::mutex> lk(mu);
    auto it = cache.find(key);
    if (it != cache.end()) return it->second;
  }
  int n = 0;
  cudaError_t e;
  if (cluster > 1) {
    e = cudaOccupancyMaxActiveClusters(&n, kernel, cfg);
  } else {
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, threads, smem);
  }
  if (e != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  std::lock_guard<std::mutex> lk(mu);
  cache[key] = n;
  return n;
}

// Kernel attributes are raised once per kernel and device: the full opt-in
// shared memory, the shared-memory carveout, and (cluster kernels) clusters
// of up to 16 CTAs.
inline cudaError_t prepare_kernel(const void *kernel, const DeviceInfo &d, bool cluster) {
  static std::mutex mu;
  static std::map<std::pair<const void *, int>, bool> done;
  std::lock_guard<std::mutex> lk(mu);
  const auto key = std::make_pair(kernel, d.device);
  if (done.count(key)) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       d.max_smem_optin);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  if (cluster) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  done[key] = true;
  return cudaSuccess;
}

// A kernel's dynamic shared-memory limit raised to `bytes` (for kernels
// that also hold static shared memory), once per kernel and device.
inline cudaError_t reserve_dynamic_smem(const void *kernel, const DeviceInfo &d, size_t bytes) {
  static std::mutex mu;
  static std::map<std::pair<const void *, int>, size_t> done;
  std::lock_guard<std::mutex> lk(mu);
  const auto key = std::make_pair(kernel, d.device);
  auto it = done.find(key);
  if (it != done.end() && it->second >= bytes) return cudaSuccess;
  const cudaError_t e =
      cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
  if (e != cudaSuccess) return e;
  done[key] = bytes;
  return cudaSuccess;
}

}  // namespace rowop
