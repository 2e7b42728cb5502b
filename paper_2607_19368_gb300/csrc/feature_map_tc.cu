// bf16 feature map on the tcgen05 tensor cores (placeholder until the
// TMA/tcgen05 kernel lands): reports the shape as unsupported so the caller
// takes the SIMT path.
#include "common.cuh"
#include "kernels.cuh"

namespace sls {

int launch_feature_map_tc(const void*, int64_t, int, int64_t, const void*, const float*, int,
                          float*, cudaStream_t) {
  return SLS_ERR_UNSUPPORTED;
}

}  // namespace sls
