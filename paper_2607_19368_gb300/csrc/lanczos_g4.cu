// Lanczos kernel instantiations for 4 float4 column group(s) of Phi per
// compute thread (D <= 4096), float32 Phi, for every basis tile count KT, with
// one team of compute warps.
#include "lanczos_kernel.cuh"

namespace sls {

int launch_lanczos_gpt4(SLS_LZ_LAUNCH_ARGS) {
  if (teams != 1) return SLS_ERR_UNSUPPORTED;
  return launch_lanczos_kt<4, float, 1>(bt, scratch, gstride, groups, g, rows_cap, stages, status,
                                        smem, stream, kt);
}

}  // namespace sls
