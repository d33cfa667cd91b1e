// ops_logsoftmax.cu -- instantiates the dense and ragged launch paths (all three
// bucket designs, fp32 and bf16) for the logsoftmax operator.  One operator per
// translation unit so the library compiles in parallel.
#include "launchers.cuh"

namespace rowop {
template cudaError_t launch_dense<kLogSoftmax>(const DenseCall &, const DeviceInfo &);
template cudaError_t launch_ragged<kLogSoftmax>(const RaggedCall &, const DeviceInfo &);
}  // namespace rowop
