// bwd_instance.cu -- instantiates the backward launch path of one operator for
// one element type; the build compiles it once per (operator, type) pair,
// naming them with -DROWOP_INST_OP=<operator> -DROWOP_INST_T=<type>.
#include "bwd_launch.cuh"

#ifndef ROWOP_INST_OP
#error "ROWOP_INST_OP (kSoftmax, kLogSoftmax, kLayerNorm or kRmsNorm) must be defined"
#endif
#ifndef ROWOP_INST_T
#error "ROWOP_INST_T (float, __nv_bfloat16 or __half) must be defined"
#endif

namespace rowop {
template cudaError_t launch_bwd_t<ROWOP_INST_OP, ROWOP_INST_T>(const BwdCall &,
                                                               const DeviceInfo &);
template cudaError_t launch_bwd_ragged_t<ROWOP_INST_OP, ROWOP_INST_T>(const BwdRaggedCall &,
                                                                      const DeviceInfo &);
}  // namespace rowop
