// The step before the pass: a prompt's input embeddings X = E[ids], one row
// of the model's input embedding table E per token (Sec. 3.1: X comes from the
// LLM's input embedding layer; Fig. 1: prompt tokens -> input embeddings).
//
// A pure copy bound by HBM bandwidth: one warp per token row, grid-stride over
// the rows with a grid of a few CTAs per SM.  When every row start is 16-byte
// aligned (the table and X bases, their row strides and the row length) the
// rows move as 16-byte vectors, otherwise as single elements.  An id outside
// [0, V) gives a zero row and is counted in *bad.
#include <algorithm>

#include "common.cuh"
#include "kernels.cuh"

namespace sls {

namespace {

constexpr int EG_T = 256;
constexpr int EG_WARPS = EG_T / 32;
constexpr int EG_CTAS_PER_SM = 8;

// T is the unit of the copy (uint4, uint32_t or uint16_t); row lengths and
// strides are in units of T.
template <typename T>
__global__ void __launch_bounds__(EG_T)
embed_gather_kernel(const T* __restrict__ table, int64_t V, int64_t ld_table,
                    const int32_t* __restrict__ ids, int64_t N, int64_t row_units,
                    T* __restrict__ X, int64_t ldx, int* __restrict__ bad) {
  const int lane = threadIdx.x & 31;
  const int64_t step = (int64_t)gridDim.x * EG_WARPS;
  for (int64_t i = (int64_t)blockIdx.x * EG_WARPS + (threadIdx.x >> 5); i < N; i += step) {
    const int64_t v = ids[i];
    T* dst = X + i * ldx;
    if (v >= 0 && v < V) {
      const T* src = table + v * ld_table;
#pragma unroll 4
      for (int64_t k = lane; k < row_units; k += 32) dst[k] = src[k];
    } else {
      const T zero{};
      for (int64_t k = lane; k < row_units; k += 32) dst[k] = zero;
      if (lane == 0 && bad) atomicAdd(bad, 1);
    }
  }
}

template <typename T>
int launch_gather(const void* table, int64_t V, int64_t ld_table_b, const int32_t* ids,
                  int64_t N, int64_t row_b, void* X, int64_t ldx_b, int* bad, int grid,
                  cudaStream_t stream) {
  const int64_t u = (int64_t)sizeof(T);
  embed_gather_kernel<T><<<grid, EG_T, 0, stream>>>((const T*)table, V, ld_table_b / u, ids, N,
                                                    row_b / u, (T*)X, ldx_b / u, bad);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

}  // namespace

int launch_embed_gather(const void* table, int x_dtype, int64_t V, int d, int64_t ld_table,
                        const int32_t* ids, int64_t N, void* X, int64_t ldx, int* bad,
                        cudaStream_t stream) {
  if (bad) SLS_CUDA_TRY(cudaMemsetAsync(bad, 0, sizeof(int), stream));
  if (N <= 0) return SLS_OK;
  const int64_t elt = (x_dtype == SLS_BF16) ? 2 : 4;
  const int64_t row_b = (int64_t)d * elt, ldt_b = ld_table * elt, ldx_b = ldx * elt;
  int dev = 0, sms = 0;
  SLS_CUDA_TRY(cudaGetDevice(&dev));
  SLS_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const int64_t want = (N + EG_WARPS - 1) / EG_WARPS;
  const int grid = (int)std::min<int64_t>(want, (int64_t)sms * EG_CTAS_PER_SM);
  const bool vec = ((uintptr_t)table % 16 == 0) && ((uintptr_t)X % 16 == 0) && row_b % 16 == 0 &&
                   ldt_b % 16 == 0 && ldx_b % 16 == 0;
  if (vec) return launch_gather<uint4>(table, V, ldt_b, ids, N, row_b, X, ldx_b, bad, grid, stream);
  if (elt == 4)
    return launch_gather<uint32_t>(table, V, ldt_b, ids, N, row_b, X, ldx_b, bad, grid, stream);
  return launch_gather<uint16_t>(table, V, ldt_b, ids, N, row_b, X, ldx_b, bad, grid, stream);
}

}  // namespace sls
