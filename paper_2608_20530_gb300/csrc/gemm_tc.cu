// Tensor-core (tcgen05) linear layer for the bf16 head. Not enabled yet: every
// product runs on the fp32 CUDA-core kernel.
#include "internal.cuh"

namespace lilicorr {

bool gemm_tc_supported(const GemmArgs& g) {
  (void)g;
  return false;
}

lilicorr_status_t launch_gemm_tc(const GemmArgs& g, cudaStream_t st) {
  (void)g; (void)st;
  return LILICORR_ERR_DTYPE;
}

}  // namespace lilicorr
