// ops_instance.cu -- instantiates the dense and ragged launch paths (all three
// bucket designs) of one operator for one element type.  The build compiles
// this file once per (operator, type) pair, naming them with
// -DROWOP_INST_OP=<operator> -DROWOP_INST_T=<type>, so the twelve
// instantiations compile in parallel.
#include "launchers.cuh"

#ifndef ROWOP_INST_OP
#error "ROWOP_INST_OP (kSoftmax, kLogSoftmax, kLayerNorm or kRmsNorm) must be defined"
#endif
#ifndef ROWOP_INST_T
#error "ROWOP_INST_T (float, __nv_bfloat16 or __half) must be defined"
#endif

namespace rowop {
template cudaError_t launch_dense_t<ROWOP_INST_OP, ROWOP_INST_T>(const DenseCall &,
                                                                 const DeviceInfo &);
template cudaError_t launch_ragged_t<ROWOP_INST_OP, ROWOP_INST_T>(const RaggedCall &,
                                                                  const DeviceInfo &);
}  // namespace rowop
