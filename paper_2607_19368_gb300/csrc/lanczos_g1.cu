// Lanczos kernel instantiations for 1 float4 column group(s) of Phi per
// compute thread (D <= 1024), float32 Phi, for every basis tile count KT.
#include "lanczos_kernel.cuh"

namespace sls {

int launch_lanczos_gpt1(SLS_LZ_LAUNCH_ARGS) {
  return launch_lanczos_kt<1, float>(bt, scratch, gstride, groups, g, rows_cap, stages, status,
                                      smem, stream, kt);
}

}  // namespace sls
