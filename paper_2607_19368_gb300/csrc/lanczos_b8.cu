// Lanczos kernel instantiations for 8 four-element column group(s) of Phi
// per compute thread (D <= 8192), Phi stored as bfloat16, for every basis tile
// count KT.
#include "lanczos_kernel.cuh"

namespace sls {

int launch_lanczos_bf16_gpt8(SLS_LZ_LAUNCH_ARGS) {
  return launch_lanczos_kt<8, uint16_t>(bt, scratch, gstride, groups, g, rows_cap, stages,
                                         status, smem, stream, kt);
}

}  // namespace sls
