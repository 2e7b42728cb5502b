// The row-normalised operator of Sec. 3.2: diag(s)^-1 Phi (Phi^T v) with the
// row sums s = Phi (Phi^T 1), run by Lanczos in its symmetric form
// D^{-1/2} Phi Phi^T D^{-1/2} (D = diag(s)), i.e. the unnormalised operator of
// the rows Phi_i / sqrt(s_i); a row with s_i <= 0 is scaled by 0.  For every
// problem (a prompt or a spectral window, rows [row0, row0 + n) of Phi):
//   1. column sums c = Phi^T 1 in double-float, per block of NB_ROWS rows
//      (float4 column groups per thread, rows split over thread phases when
//      D is narrow, several rows' loads in flight per thread);
//   2. the blocks of a problem added per column (eight block phases per
//      column, combined in a fixed order);
//   3. one warp per row, the row held in registers: s_i = Phi_i . c (exact
//      products, Dot2 sums), then the row scaled in place by w = 1/sqrt(s_i):
//      each element is x * w to within one float32 rounding, formed from
//      w = wh + wl (two floats) as the exact product x * wh plus x * wl.
// All three kernels are bound by HBM bandwidth: Phi is read twice and written
// once.
#include "common.cuh"
#include "kernels.cuh"

namespace sls {

namespace {

constexpr int NB_ROWS = 64;   // rows per column-sum block
constexpr int NB_T = 256;
constexpr int NB_U = 8;       // rows in flight per thread in the column sums
constexpr int NR_ROWS = 32;   // rows per CTA of the row kernel (4 per warp)

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

SLS_DEV void acc4(float (&h)[4], float (&l)[4], float4 v) {
  const float x[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    float s, e;
    two_sum(h[k], x[k], s, e);
    h[k] = s;
    l[k] = __fadd_rn(l[k], e);
  }
}

// grid (blocks per problem, problems): column sums of one block of rows.
// G = D / 4 float4 groups; Gt = min(G, NB_T) threads per row phase and
// NB_T / Gt phases (phase ph takes rows ph, ph + phases, ...).
__global__ void __launch_bounds__(NB_T)
norm_colsum_kernel(const float* __restrict__ Phi, int D, NormProblems P, int nblk,
                   float2* __restrict__ part) {
  __shared__ float2 red[NB_T * 4];
  int64_t row0, n;
  if (!norm_problem(P, blockIdx.y, row0, n)) return;
  const int64_t r0 = (int64_t)blockIdx.x * NB_ROWS;
  if (r0 >= n) return;
  const int rows = (int)((n - r0) < NB_ROWS ? (n - r0) : NB_ROWS);
  const int G = D / 4;
  const int Gt = min(G, NB_T);
  const int phases = NB_T / Gt;
  const int t = threadIdx.x, ph = t / Gt, gx = t % Gt;
  const float4* base = reinterpret_cast<const float4*>(Phi + (row0 + r0) * D);
  float2* out = part + ((size_t)blockIdx.y * nblk + blockIdx.x) * D;
  for (int g = gx; g < G; g += Gt) {
    float h[4] = {0.f, 0.f, 0.f, 0.f}, l[4] = {0.f, 0.f, 0.f, 0.f};
    if (ph < phases) {
      int i = ph;
      for (; i + (NB_U - 1) * phases < rows; i += NB_U * phases) {
        float4 v[NB_U];
#pragma unroll
        for (int u = 0; u < NB_U; ++u) v[u] = __ldg(base + (size_t)(i + u * phases) * G + g);
#pragma unroll
        for (int u = 0; u < NB_U; ++u) acc4(h, l, v[u]);
      }
      for (; i < rows; i += phases) acc4(h, l, __ldg(base + (size_t)i * G + g));
    }
    if (phases == 1) {
#pragma unroll
      for (int k = 0; k < 4; ++k) out[4 * g + k] = f2(df_norm(h[k], l[k]));
    } else {
      // phases > 1 only when G < NB_T: every thread runs this body once
      if (ph < phases) {
#pragma unroll
        for (int k = 0; k < 4; ++k) red[t * 4 + k] = make_float2(h[k], l[k]);
      }
      __syncthreads();
      if (ph == 0) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          dfloat acc = df_norm(h[k], l[k]);
          for (int p = 1; p < phases; ++p) acc = df_add(acc, dfv(red[(p * Gt + gx) * 4 + k]));
          out[4 * g + k] = f2(acc);
        }
      }
    }
  }
}

// grid (column groups of 32, problems): a problem's column sums; warp w adds
// blocks w, w + 8, ... for column 32 * blockIdx.x + lane, then warp 0 adds the
// eight warp sums in order.
__global__ void __launch_bounds__(NB_T)
norm_colreduce_kernel(int D, NormProblems P, int nblk, const float2* __restrict__ part,
                      float2* __restrict__ colsum) {
  __shared__ float2 red[NB_T / 32][32];
  int64_t row0, n;
  if (!norm_problem(P, blockIdx.y, row0, n)) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int c = blockIdx.x * 32 + lane;
  const int nb = (int)((n + NB_ROWS - 1) / NB_ROWS);
  const float2* src = part + (size_t)blockIdx.y * nblk * D;
  dfloat acc = df_make(0.f, 0.f);
  if (c < D)
    for (int b = warp; b < nb; b += NB_T / 32) acc = df_add(acc, dfv(src[(size_t)b * D + c]));
  red[warp][lane] = f2(acc);
  __syncthreads();
  if (warp == 0 && c < D) {
    dfloat a = dfv(red[0][lane]);
    for (int w = 1; w < NB_T / 32; ++w) a = df_add(a, dfv(red[w][lane]));
    colsum[(size_t)blockIdx.y * D + c] = f2(a);
  }
}

// x * w for w = wh + wl, to within one float32 rounding: the product x * wh
// split exactly (TwoProduct) and x * wl added to its error term.
SLS_DEV float scale_df(float x, float wh, float wl) {
  const float p = __fmul_rn(x, wh);
  const float e = __fmaf_rn(x, wl, __fmaf_rn(x, wh, -p));
  return __fadd_rn(p, e);
}

SLS_DEV float4 scale4(float4 v, double w, float wh, float wl, bool split) {
  if (split) return make_float4(scale_df(v.x, wh, wl), scale_df(v.y, wh, wl),
                                scale_df(v.z, wh, wl), scale_df(v.w, wh, wl));
  return make_float4((float)((double)v.x * w), (float)((double)v.y * w),
                     (float)((double)v.z * w), (float)((double)v.w * w));
}

SLS_DEV void dot4(float& sh, float& sl, float4 v, const float4* __restrict__ c4, int g) {
  const float4 a = __ldg(c4 + 2 * g), b = __ldg(c4 + 2 * g + 1);  // (hi, lo) of 4 columns
  dot2_acc(sh, sl, v.x, a.x, a.y);
  dot2_acc(sh, sl, v.y, a.z, a.w);
  dot2_acc(sh, sl, v.z, b.x, b.y);
  dot2_acc(sh, sl, v.w, b.z, b.w);
}

// grid (row blocks of NR_ROWS, problems): s_i = Phi_i . c and the row scaled
// in place.  VPL float4 groups per lane held in registers (D <= 128 * VPL);
// VPL = 0 streams the row twice for wider D.
template <int VPL>
__global__ void __launch_bounds__(NB_T)
norm_rows_kernel(float* __restrict__ Phi, int D, NormProblems P,
                 const float2* __restrict__ colsum, double* __restrict__ s_out) {
  int64_t row0, n;
  if (!norm_problem(P, blockIdx.y, row0, n)) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int G = D / 4;
  const float4* c4 = reinterpret_cast<const float4*>(colsum + (size_t)blockIdx.y * D);
  const int64_t rb = (int64_t)blockIdx.x * NR_ROWS;
  const int64_t re = min(n, rb + NR_ROWS);
  for (int64_t i = rb + warp; i < re; i += NB_T / 32) {
    float4* row = reinterpret_cast<float4*>(Phi + (row0 + i) * D);
    float sh = 0.f, sl = 0.f;
    float4 v[VPL > 0 ? VPL : 1];
    if (VPL > 0) {
#pragma unroll
      for (int k = 0; k < VPL; ++k) {
        const int g = lane + 32 * k;
        v[k] = g < G ? row[g] : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int k = 0; k < VPL; ++k)
        if (lane + 32 * k < G) dot4(sh, sl, v[k], c4, lane + 32 * k);
    } else {
      for (int g = lane; g < G; g += 32) dot4(sh, sl, row[g], c4, g);
    }
    const double s = df_to_double(warp_sum_df(df_norm(sh, sl)));
    const double w = (s > 0.0) ? 1.0 / sqrt(s) : 0.0;
    // the two-float split needs w (and its low part) inside float range
    const bool split = w < 1e30;
    const float wh = split ? __double2float_rn(w) : 0.f;
    const float wl = split ? __double2float_rn(w - (double)wh) : 0.f;
    if (s_out && lane == 0) s_out[row0 + i] = s;
    if (VPL > 0) {
#pragma unroll
      for (int k = 0; k < VPL; ++k) {
        const int g = lane + 32 * k;
        if (g < G) row[g] = scale4(v[k], w, wh, wl, split);
      }
    } else {
      for (int g = lane; g < G; g += 32) row[g] = scale4(row[g], w, wh, wl, split);
    }
  }
}

template <int VPL>
void launch_rows(float* Phi, int D, const NormProblems& P, int64_t nmax, const float2* colsum,
                 double* s_out, cudaStream_t stream) {
  const int64_t nrb = (nmax + NR_ROWS - 1) / NR_ROWS;
  norm_rows_kernel<VPL><<<dim3((unsigned)nrb, P.nprob_max), NB_T, 0, stream>>>(Phi, D, P,
                                                                              colsum, s_out);
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
  if (D % 4) return SLS_ERR_UNSUPPORTED;
  const int64_t nblk = (nmax + NB_ROWS - 1) / NB_ROWS;
  const int64_t nrb = (nmax + NR_ROWS - 1) / NR_ROWS;
  if (nrb > 0x7fffffffLL || nprob_max > 65535) return SLS_ERR_UNSUPPORTED;
  NormProblems P{row0, n, nprob_max, nprob_dev, n_single};
  float2* part = scratch;
  float2* colsum = scratch + (size_t)nprob_max * nblk * D;
  norm_colsum_kernel<<<dim3((unsigned)nblk, nprob_max), NB_T, 0, stream>>>(Phi, D, P, (int)nblk,
                                                                           part);
  SLS_LAUNCH_CHECK();
  norm_colreduce_kernel<<<dim3((D + 31) / 32, nprob_max), NB_T, 0, stream>>>(D, P, (int)nblk,
                                                                             part, colsum);
  SLS_LAUNCH_CHECK();
  const int vpl = (D / 4 + 31) / 32;
  if (vpl <= 1) launch_rows<1>(Phi, D, P, nmax, colsum, s_out, stream);
  else if (vpl <= 2) launch_rows<2>(Phi, D, P, nmax, colsum, s_out, stream);
  else if (vpl <= 4) launch_rows<4>(Phi, D, P, nmax, colsum, s_out, stream);
  else if (vpl <= 8) launch_rows<8>(Phi, D, P, nmax, colsum, s_out, stream);
  else if (vpl <= 16) launch_rows<16>(Phi, D, P, nmax, colsum, s_out, stream);
  else launch_rows<0>(Phi, D, P, nmax, colsum, s_out, stream);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

}  // namespace sls
