// Lanczos kernel instantiations for 4 float4 column group(s) of Phi per
// compute thread (D <= 4096), Phi stored as bfloat16, for every basis tile count KT, with
// one team of compute warps.
#include "lanczos_kernel.cuh"

namespace sls {

int launch_lanczos_bf16_gpt4(SLS_LZ_LAUNCH_ARGS) {
  if (teams != 1) return SLS_ERR_UNSUPPORTED;
  return launch_lanczos_kt<4, uint16_t, 1>(bt, scratch, gstride, groups, g, rows_cap, stages, status,
                                        smem, stream, kt);
}

}  // namespace sls
