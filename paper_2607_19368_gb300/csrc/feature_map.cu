// Random Fourier feature map, Sec. 3.2 Eq. rff_map:
//   Phi[i, c] = sqrt(2/D) * cos( X[i, :] . W[c, :] + b[c] ),  W = Omega^T (D x d).
//
// The contraction X W^T is GEMM-shaped (M = tokens, N = features, K = d).
// This file holds the fp32 SIMT kernel (used for float32 embeddings and as
// the reference path for small shapes); the bf16 tcgen05 kernel lives in
// feature_map_tc.cu.  Both fuse the bias, cosine and scale into the epilogue,
// so Phi is written exactly once, as float32 or (opt-in) as bfloat16 rounded
// to nearest even from the float32 value.
#include "common.cuh"
#include "kernels.cuh"

namespace sls {

namespace {

constexpr int FM_BM = 64;   // tokens per CTA tile
constexpr int FM_BN = 64;   // features per CTA tile
constexpr int FM_BK = 16;   // K slice
constexpr int FM_THREADS = 256;

template <typename T>
SLS_DEV float load_elem(const T* p);

template <>
SLS_DEV float load_elem<float>(const float* p) {
  return *p;
}

template <>
SLS_DEV float load_elem<uint16_t>(const uint16_t* p) {
  return __uint_as_float(((unsigned)*p) << 16);
}

// One CTA computes a 64 x 64 tile; each thread a 4 x 4 block.  T: element
// type of X and W; OT: of Phi (float, or uint16_t for bfloat16).
template <typename T, typename OT>
__global__ void __launch_bounds__(FM_THREADS)
feature_map_simt_kernel(const T* __restrict__ X, int64_t N, int d, int64_t ldx,
                        const T* __restrict__ W, const float* __restrict__ bvec,
                        int D, float scale, OT* __restrict__ Phi) {
  __shared__ float As[FM_BK][FM_BM + 4];
  __shared__ float Bs[FM_BK][FM_BN + 4];
  const int tid = threadIdx.x;
  const int64_t row0 = (int64_t)blockIdx.y * FM_BM;
  const int col0 = blockIdx.x * FM_BN;
  const int ty = tid / 16, tx = tid % 16;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < d; k0 += FM_BK) {
    // each thread loads 4 elements of A and 4 of B (64 x 16 each)
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      int e = tid + t * FM_THREADS;  // 0..1023
      int r = e / FM_BK, k = e % FM_BK;
      int64_t gr = row0 + r;
      int gk = k0 + k;
      As[k][r] = (gr < N && gk < d) ? load_elem<T>(X + gr * ldx + gk) : 0.f;
      int c = col0 + r;
      Bs[k][r] = (c < D && gk < d) ? load_elem<T>(W + (int64_t)c * d + gk) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < FM_BK; ++k) {
      float a[4], bb[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[k][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) bb[j] = Bs[k][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], bb[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    int64_t gr = row0 + ty * 4 + i;
    if (gr >= N) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int c = col0 + tx * 4 + j;
      if (c < D) phi_st(Phi + gr * D + c, scale * cosf(acc[i][j] + bvec[c]));
    }
  }
}

template <typename T>
void launch_simt_t(const void* X, int64_t N, int d, int64_t ldx, const void* W, const float* b,
                   int D, float scale, void* Phi, int phi_bf16, dim3 grid, cudaStream_t stream) {
  if (phi_bf16)
    feature_map_simt_kernel<T, uint16_t><<<grid, FM_THREADS, 0, stream>>>(
        (const T*)X, N, d, ldx, (const T*)W, b, D, scale, (uint16_t*)Phi);
  else
    feature_map_simt_kernel<T, float><<<grid, FM_THREADS, 0, stream>>>(
        (const T*)X, N, d, ldx, (const T*)W, b, D, scale, (float*)Phi);
}

}  // namespace

int launch_feature_map_simt(const void* X, int x_dtype, int64_t N, int d, int64_t ldx,
                            const void* W, const float* b, int D, void* Phi,
                            cudaStream_t stream, int phi_bf16) {
  if (N == 0) return SLS_OK;
  const float scale = (float)sqrt(2.0 / (double)D);
  dim3 grid((D + FM_BN - 1) / FM_BN, (unsigned)((N + FM_BM - 1) / FM_BM));
  if (grid.y > 65535u) return SLS_ERR_UNSUPPORTED;
  if (x_dtype == SLS_F32)
    launch_simt_t<float>(X, N, d, ldx, W, b, D, scale, Phi, phi_bf16, grid, stream);
  else
    launch_simt_t<uint16_t>(X, N, d, ldx, W, b, D, scale, Phi, phi_bf16, grid, stream);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

}  // namespace sls
