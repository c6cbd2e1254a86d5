// lmhead.cu — fused lm_head + acceptance (step a6).  Placeholder until the
// tcgen05 kernel lands: every call reports SSD_ERR_UNSUPPORTED.
#include "kernels.cuh"

namespace ssd {

size_t lmhead_workspace(int32_t rows, int32_t V) { return 256; }

ssd_status lmhead_check(int32_t rows, int32_t V, int32_t K) { return SSD_ERR_UNSUPPORTED; }

cudaError_t launch_lmhead(const LmHeadArgs& a, void* ws, size_t ws_bytes, cudaStream_t stream) {
  return cudaErrorNotSupported;
}

}  // namespace ssd
