// Lanczos kernel instantiations for 4 float4 column groups of Phi per compute
// thread (D <= 4096), for every basis tile count KT.
#include "lanczos_kernel.cuh"

namespace sls {

int launch_lanczos_gpt4(SLS_LZ_LAUNCH_ARGS) {
  switch (kt) {
    case 1: return launch_lanczos_t<4, 1>(bt, scratch, gstride, groups, g, rows_cap, stages, status, smem, stream);
    case 2: return launch_lanczos_t<4, 2>(bt, scratch, gstride, groups, g, rows_cap, stages, status, smem, stream);
    case 4: return launch_lanczos_t<4, 4>(bt, scratch, gstride, groups, g, rows_cap, stages, status, smem, stream);
    default: return SLS_ERR_UNSUPPORTED;
  }
}

}  // namespace sls
