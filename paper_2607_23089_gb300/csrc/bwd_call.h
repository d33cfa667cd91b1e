// bwd_call.h -- internal host interface of the ragged backward passes,
// between the C ABI (rowop_api.cu) and their launch code (bwd_launch.cuh).
#pragma once

#include "dispatch.h"

namespace rowop {

// Backward pass of the softmax family over ragged rows (CSR offsets, the
// same offsets index a = y, dy and dx); ws holds a classify plan.
struct BwdRaggedCall {
  int dtype;
  const void *a;
  const void *dy;
  void *dx;
  const int64_t *offsets;
  int64_t rows, max_len;
  void *ws;
  cudaStream_t stream;
};

}  // namespace rowop
