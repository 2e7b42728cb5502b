// Lanczos kernel instantiations for 1 float4 column group(s) of Phi per
// compute thread (D <= 1024), float32 Phi, for every basis tile count KT, with
// one team (D < 1024) or two (D = 1024) of compute warps.
#include "lanczos_kernel.cuh"

namespace sls {

int launch_lanczos_gpt1(SLS_LZ_LAUNCH_ARGS) {
  return teams == 2 ? launch_lanczos_kt<1, float, 2>(bt, scratch, gstride, groups, g, rows_cap,
                                                      stages, status, smem, stream, kt)
                    : launch_lanczos_kt<1, float, 1>(bt, scratch, gstride, groups, g, rows_cap,
                                                      stages, status, smem, stream, kt);
}

}  // namespace sls
