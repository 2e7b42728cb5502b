// The row-normalised operator of Sec. 3.2: diag(s)^-1 Phi (Phi^T v) with the
// row sums s = Phi (Phi^T 1), run by Lanczos in its symmetric form
// D^{-1/2} Phi Phi^T D^{-1/2} (D = diag(s)), i.e. the unnormalised operator of
// the rows Phi_i / sqrt(s_i); a row with s_i <= 0 is scaled by 0.  For every
// problem (a prompt or a spectral window, rows [row0, row0 + n) of Phi):
//   1. column sums c = Phi^T 1 in double-float, per block of NB_ROWS rows;
//   2. the blocks of a problem added per column;
//   3. one warp per row: s_i = Phi_i . c (exact products, Dot2 sums), then the
//      row scaled in place by 1 / sqrt(s_i), each element rounded once to
//      float32 from its float64 product.
#include "common.cuh"
#include "kernels.cuh"

namespace sls {

namespace {

constexpr int NB_ROWS = 256;  // rows per column-sum block
constexpr int NB_T = 256;

struct NormProblems {
  const int64_t* row0;  // NULL: one problem of n_single rows from row 0
  const int* n;
  int nprob_max;
  const int* nprob_dev;
  int64_t n_single;
};

SLS_DEV bool norm_problem(const NormProblems& P, int p, int64_t& row0, int64_t& n) {
  int np = P.nprob_max;
  if (P.nprob_dev) np = min(np, *P.nprob_dev);
  if (p >= np) return false;
  row0 = P.row0 ? P.row0[p] : 0;
  n = P.n ? (int64_t)P.n[p] : P.n_single;
  return true;
}

// grid (blocks per problem, problems): column sums of one block of rows
__global__ void __launch_bounds__(NB_T)
norm_colsum_kernel(const float* __restrict__ Phi, int D, NormProblems P, int nblk,
                   float2* __restrict__ part) {
  int64_t row0, n;
  if (!norm_problem(P, blockIdx.y, row0, n)) return;
  const int64_t r0 = (int64_t)blockIdx.x * NB_ROWS;
  if (r0 >= n) return;
  const int64_t r1 = min(n, r0 + NB_ROWS);
  float2* out = part + ((size_t)blockIdx.y * nblk + blockIdx.x) * D;
  for (int c = threadIdx.x; c < D; c += NB_T) {
    float sh = 0.f, sl = 0.f;
    for (int64_t i = r0; i < r1; ++i) {
      float s, e;
      two_sum(sh, Phi[(row0 + i) * D + c], s, e);
      sh = s;
      sl = __fadd_rn(sl, e);
    }
    out[c] = f2(df_norm(sh, sl));
  }
}

// grid (column groups, problems): a problem's column sums
__global__ void __launch_bounds__(NB_T)
norm_colreduce_kernel(int D, NormProblems P, int nblk, const float2* __restrict__ part,
                      float2* __restrict__ colsum) {
  int64_t row0, n;
  if (!norm_problem(P, blockIdx.y, row0, n)) return;
  const int c = blockIdx.x * NB_T + threadIdx.x;
  if (c >= D) return;
  const int nb = (int)((n + NB_ROWS - 1) / NB_ROWS);
  const float2* src = part + (size_t)blockIdx.y * nblk * D;
  dfloat acc = df_make(0.f, 0.f);
  for (int b = 0; b < nb; ++b) acc = df_add(acc, dfv(src[(size_t)b * D + c]));
  colsum[(size_t)blockIdx.y * D + c] = f2(acc);
}

// grid (row blocks, problems): s_i = Phi_i . c and the row scaled in place
__global__ void __launch_bounds__(NB_T)
norm_rows_kernel(float* __restrict__ Phi, int D, NormProblems P,
                 const float2* __restrict__ colsum, double* __restrict__ s_out) {
  int64_t row0, n;
  if (!norm_problem(P, blockIdx.y, row0, n)) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float2* cp = colsum + (size_t)blockIdx.y * D;
  const int64_t rb = (int64_t)blockIdx.x * NB_ROWS;
  for (int64_t i = rb + warp; i < min(n, rb + NB_ROWS); i += NB_T / 32) {
    float* row = Phi + (row0 + i) * D;
    float sh = 0.f, sl = 0.f;
    for (int c = lane; c < D; c += 32) {
      const float2 cc = cp[c];
      dot2_acc(sh, sl, row[c], cc.x, cc.y);
    }
    const double s = df_to_double(warp_sum_df(df_norm(sh, sl)));
    const double w = (s > 0.0) ? 1.0 / sqrt(s) : 0.0;
    if (s_out && lane == 0) s_out[row0 + i] = s;
    for (int c = lane; c < D; c += 32) row[c] = (float)((double)row[c] * w);
  }
}

}  // namespace

size_t feature_normalize_scratch_bytes(int64_t nmax, int D, int nprob) {
  const int64_t nblk = (nmax + NB_ROWS - 1) / NB_ROWS;
  return (size_t)nprob * (size_t)(nblk + 1) * (size_t)D * sizeof(float2);
}

int launch_feature_normalize(float* Phi, int D, const int64_t* row0, const int* n,
                             int nprob_max, const int* nprob_dev, int64_t n_single, int64_t nmax,
                             float2* scratch, double* s_out, cudaStream_t stream) {
  if (nprob_max <= 0 || nmax <= 0) return SLS_OK;
  const int64_t nblk = (nmax + NB_ROWS - 1) / NB_ROWS;
  if (nblk > 65535 || nprob_max > 65535) return SLS_ERR_UNSUPPORTED;
  NormProblems P{row0, n, nprob_max, nprob_dev, n_single};
  float2* part = scratch;
  float2* colsum = scratch + (size_t)nprob_max * nblk * D;
  norm_colsum_kernel<<<dim3((unsigned)nblk, nprob_max), NB_T, 0, stream>>>(Phi, D, P, (int)nblk,
                                                                           part);
  SLS_LAUNCH_CHECK();
  norm_colreduce_kernel<<<dim3((D + NB_T - 1) / NB_T, nprob_max), NB_T, 0, stream>>>(
      D, P, (int)nblk, part, colsum);
  SLS_LAUNCH_CHECK();
  norm_rows_kernel<<<dim3((unsigned)nblk, nprob_max), NB_T, 0, stream>>>(Phi, D, P, colsum,
                                                                         s_out);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

}  // namespace sls
