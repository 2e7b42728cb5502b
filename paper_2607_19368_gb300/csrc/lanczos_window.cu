// Algorithm 2 (implicit Lanczos) and the Ritz values of Algorithm 1 for
// batches of small problems: the windows of the local and adaptive backends
// (Sec. 3.5, 3.6) with at most 32 tokens and r <= 32 steps.
//
// One warp per problem.  Every step is Algorithm 2 as written:
//   z = Phi (Phi^T q_j)  (Eq. implicit_matvec),  alpha_j = q_j^T z,
//   z -= alpha_j q_j + beta_{j-1} q_{j-1},  two passes of classical
//   Gram-Schmidt against q_1..q_j,  beta_j = |z|,  and the scale-relative
//   break test beta_j <= tol * max_i(|alpha_i| + beta_i).
// The two products with Phi are double-float on the FP32 pipes (offset
// accumulation against a power of two above twice the bound of every partial
// sum, from the window's max|Phi|; each step's rounding error is formed by an
// FMA and kept in the low part); the
// vector work of a step -- alpha, the recurrence, both Gram-Schmidt passes,
// beta and q_{j+1} = z / beta -- is float64, as in the algorithm's own
// statement: near a breakdown (a window whose Phi has lower rank than r) the
// residual that the break test compares against tol * scale is rounding
// noise amplified by the process, and at double-float precision it lands
// above the threshold where float64 lands below.  That vector work is
// O(n j) per step, so float64 costs little here.  Lane i owns row i of the
// Krylov vectors; lane l owns the columns l, l + 32, ... of Phi^T q_j.
// Phi rows are read through the read-only cache (a window's rows are reused
// by every step).  The Ritz values (Eigh of T) follow in the same warp, one
// lane per eigenvalue, by bisection on double-float Sturm counts of the
// power-of-two-scaled T.  Outputs use the layout of the big-problem kernel
// (alpha, beta, theta at p * r, r_eff, double-float basis rows of Q), so the
// eigenvectors and U = Q S come from the same kernels as there.
#include <cfloat>

#include "kernels.cuh"
#include "tridiag.cuh"

namespace sls {

namespace {

constexpr int LW_MAXN = 32;
constexpr int LW_MAXR = 32;
constexpr int LW_MAX_WARPS = 8;     // launch bound of the kernel
constexpr int LW_LAUNCH_WARPS = 2;  // windows per CTA: small CTAs spread the
                                    // windows evenly over the SMs (measured
                                    // 3.6% faster than 8 on the local pass)
constexpr unsigned FULL = 0xffffffffu;

// Shared memory of one warp, in 8-byte units: y = Phi^T q (D, double-float),
// the broadcast copy of q (32, double-float), Q (nmax x (r + 1), float64), T
// as double-float for the Sturm counts (alpha and beta^2: 2 x 32) and T in
// float64 (alpha, beta: 2 x 32).
__host__ __device__ inline int lw_warp_f2(int nmax, int D, int r) {
  return D + 32 + nmax * (r + 1) + 64 + 64;
}

SLS_DEV dfloat shfl_xor_df(dfloat v, int o) {
  dfloat r;
  r.hi = __shfl_xor_sync(FULL, v.hi, o);
  r.lo = __shfl_xor_sync(FULL, v.lo, o);
  return r;
}

SLS_DEV double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL, v, o);
  return v;
}

// Transposed butterfly on float64: lane l ends with the sum over all lanes of
// v[l % RV] (RV in {16, 32}; RV - 1 exchanges, then one more for RV = 16).
template <int RV>
SLS_DEV double transpose_reduce_d(double (&v)[RV], int lane) {
#pragma unroll
  for (int o = RV / 2; o >= 1; o >>= 1) {
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int t = 0; t < o; ++t) {
      const double send = up ? v[t] : v[t + o];
      const double keep = up ? v[t + o] : v[t];
      v[t] = keep + __shfl_xor_sync(FULL, send, o);
    }
  }
  double r = v[0];
#pragma unroll
  for (int o = RV; o < 32; o <<= 1) r += __shfl_xor_sync(FULL, r, o);
  return r;
}

// Transposed butterfly: lane l ends with the sum over all lanes of v[l % NV]
// (NV in {16, 32}); NV - 1 double-float exchanges instead of NV full sums.
template <int NV>
SLS_DEV dfloat transpose_reduce(dfloat (&v)[NV], int lane) {
#pragma unroll
  for (int o = NV / 2; o >= 1; o >>= 1) {
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int t = 0; t < o; ++t) {
      const dfloat send = up ? v[t] : v[t + o];
      const dfloat keep = up ? v[t + o] : v[t];
      v[t] = df_add(keep, shfl_xor_df(send, o));
    }
  }
  dfloat r = v[0];
#pragma unroll
  for (int o = NV; o < 32; o <<= 1) r = df_add(r, shfl_xor_df(r, o));
  return r;
}

template <int NV, int RV, typename PT>
__global__ void __launch_bounds__(LW_MAX_WARPS * 32)
lanczos_window_kernel(LanczosBatch bt) {
  constexpr int CU = (NV <= 16) ? 2 : 1;  // columns in flight per lane
  extern __shared__ float2 lw_smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int p = blockIdx.x * (blockDim.x >> 5) + warp;
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  if (p >= nprob) return;  // the whole warp leaves; no block-wide barrier follows
  const int D = bt.D, r = bt.r, R1 = r + 1;
  const int nmax = (int)bt.nmax;
  float2* ys = lw_smem + (size_t)warp * lw_warp_f2(nmax, D, r);
  float2* qb = ys + D;
  double* Qs = reinterpret_cast<double*>(qb + 32);
  float2* sa = reinterpret_cast<float2*>(Qs + (size_t)nmax * R1);
  float2* sb2 = sa + 32;
  double* ad = reinterpret_cast<double*>(sb2 + 32);
  double* bd = ad + 32;
  const int64_t row0 = bt.row0 ? bt.row0[p] : 0;
  const int n = bt.n ? bt.n[p] : (int)bt.n_single;
  const int64_t qoff = bt.q1off ? bt.q1off[p] : row0;
  const PT* __restrict__ Phi = reinterpret_cast<const PT*>(bt.Phi) + row0 * D;
  const int rmax = min(r, n);
  const bool mine = lane < n;

  // q_1 = q1 / |q1|
  const double v0 = mine ? bt.q1[qoff + lane] : 0.0;
  const double nrm = sqrt(warp_sum_d(v0 * v0));
  double q = mine ? v0 / nrm : 0.0;
  double qprev = 0.0, bprev = 0.0, scale = 0.0;
  int reff = 0;
  // max |Phi| over the window: the bound behind the offsets of both products
  float pm = 0.f;
  for (int c = lane; c < D; c += 32)
    for (int i = 0; i < n; ++i) pm = fmaxf(pm, fabsf(phi_ld(Phi, (size_t)i * D + c)));
  for (int o = 16; o > 0; o >>= 1) pm = fmaxf(pm, __shfl_xor_sync(FULL, pm, o));
  for (int j = 0; j < rmax; ++j) {
    if (mine) Qs[lane * R1 + j] = q;
    qb[lane] = f2(df_from_double(q));
    __syncwarp();
    // y = Phi^T q_j (all rows of a column are loaded before they are used),
    // offset accumulation against Cy above twice max|Phi| |q_j|_1
    float qa = mine ? fabsf((float)q) : 0.f;
    for (int o = 16; o > 0; o >>= 1) qa += __shfl_xor_sync(FULL, qa, o);
    const float Cy = ofs_pow2(pm * qa);
    float ya = 0.f;  // l1 norm of this lane's columns of y: the bound of its row partials
#pragma unroll CU
    for (int c = lane; c < D; c += 32) {
      float ph[NV];
#pragma unroll
      for (int i = 0; i < NV; ++i) ph[i] = (i < n) ? phi_ld(Phi, (size_t)i * D + c) : 0.f;
      float sh = Cy, sl = 0.f;
#pragma unroll
      for (int i = 0; i < NV; ++i) {
        if (i < n) {
          const float2 qi = qb[i];
          ofs_fma_acc(sh, sl, ph[i], qi.x, qi.y);
        }
      }
      const dfloat yv = df_norm(sh - Cy, sl);  // sh - Cy exact
      ya += fabsf(yv.hi);
      ys[c] = f2(yv);
    }
    __syncwarp();
    // z = Phi y: per-lane partials over its columns for every row, then the
    // transposed butterfly hands row i's sum to lane i
    const float Cz = ofs_pow2(pm * ya);
    dfloat part[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) part[i] = df_make(Cz, 0.f);
#pragma unroll CU
    for (int c = lane; c < D; c += 32) {
      const float2 yc = ys[c];
      float ph[NV];
#pragma unroll
      for (int i = 0; i < NV; ++i) ph[i] = (i < n) ? phi_ld(Phi, (size_t)i * D + c) : 0.f;
#pragma unroll
      for (int i = 0; i < NV; ++i)
        if (i < n) ofs_fma_acc(part[i].hi, part[i].lo, ph[i], yc.x, yc.y);
    }
#pragma unroll
    for (int i = 0; i < NV; ++i) part[i] = df_norm(part[i].hi - Cz, part[i].lo);
    const dfloat zdf = transpose_reduce<NV>(part, lane);
    double z = mine ? df_to_double(zdf) : 0.0;
    // alpha_j and the three-term recurrence
    const double a = warp_sum_d(q * z);
    z = z - a * q - bprev * qprev;
    // full re-orthogonalisation: two classical Gram-Schmidt passes
    for (int pass = 0; pass < 2; ++pass) {
      double pr[RV];
#pragma unroll
      for (int k = 0; k < RV; ++k) pr[k] = (k <= j && mine) ? Qs[lane * R1 + k] * z : 0.0;
      const double c = transpose_reduce_d<RV>(pr, lane);  // lane k (mod RV): (Q^T z)_k
      double corr = 0.0;
      for (int k = 0; k <= j; ++k) {
        const double ck = __shfl_sync(FULL, c, k);
        if (mine) corr = fma(Qs[lane * R1 + k], ck, corr);
      }
      z -= corr;
    }
    // beta = |z| and q = z / beta from one reciprocal square root (float64
    // divides and square roots are long sequences on this GPU's FP64 pipe)
    const double zz = warp_sum_d(z * z);
    const double inv = (zz > 0.0) ? rsqrt(zz) : 0.0;
    const double b = (zz > 0.0) ? zz * inv : 0.0;
    if (lane == 0) ad[j] = a;
    reff = j + 1;
    scale = fmax(scale, fabs(a) + b);
    if (j == rmax - 1 || b <= bt.tol * scale) break;
    if (lane == 0) bd[j] = b;
    qprev = q;
    bprev = b;
    q = z * inv;
  }
  __syncwarp();

  // outputs of the recurrence
  double* alpha = bt.alpha + (size_t)p * r;
  double* beta = bt.beta + (size_t)p * r;
  double* theta = bt.theta + (size_t)p * r;
  for (int k = lane; k < reff; k += 32) {
    alpha[k] = ad[k];
    if (k < reff - 1) beta[k] = bd[k];
  }
  if (lane == 0) bt.r_eff[p] = reff;
  if (mine) {
    const int ldq = q_ld(r);
    float2* Qg = bt.Q + (row0 + lane) * ldq;
    for (int k = 0; k < reff; ++k) Qg[k] = f2(df_from_double(Qs[lane * R1 + k]));
  }

  // Ritz values: Gershgorin interval, an exact power-of-two scale into
  // [-1, 1], then bisection on Sturm counts, lane m for the m-th largest
  const int k = reff;
  double glo = DBL_MAX, ghi = -DBL_MAX;
  if (lane < k) {
    const double bl = (lane > 0) ? fabs(bd[lane - 1]) : 0.0;
    const double br = (lane < k - 1) ? fabs(bd[lane]) : 0.0;
    glo = ad[lane] - bl - br;
    ghi = ad[lane] + bl + br;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    glo = fmin(glo, __shfl_xor_sync(FULL, glo, o));
    ghi = fmax(ghi, __shfl_xor_sync(FULL, ghi, o));
  }
  const double big = fmax(fabs(glo), fabs(ghi));
  int ex = 0;
  frexp(big > 0.0 ? big : 1.0, &ex);
  const double sc = ldexp(1.0, -ex);
  if (lane < k) {
    sa[lane] = f2(df_from_double(ad[lane] * sc));
    if (lane < k - 1) {
      const double bs = bd[lane] * sc;
      sb2[lane] = f2(df_from_double(bs * bs));
    }
  }
  __syncwarp();
  if (lane < k) {
    const double pad = 0x1p-40 * fmax(fabs(glo * sc), fabs(ghi * sc)) + 0x1p-100;
    double lo = glo * sc - pad, hi = ghi * sc + pad;
    const int kasc = k - 1 - lane;  // ascending index of the wanted eigenvalue
    for (int it = 0; it < 160; ++it) {
      // 2^-46 relative, or one float64 unit of the scaled |T| <= 1
      if (hi - lo <= 0x1p-46 * fmax(fabs(lo), fabs(hi)) || hi - lo <= 0x1p-52) break;
      const double x = 0.5 * (lo + hi);
      if (sturm_count(sa, sb2, k, df_from_double(x)) > kasc)
        hi = x;
      else
        lo = x;
    }
    theta[lane] = (0.5 * (lo + hi)) / sc;
  } else if (lane < r) {
    theta[lane] = 0.0;
  }
}

}  // namespace

bool lanczos_window_fits(int64_t nmax, int D, int r) {
  if (nmax < 1 || nmax > LW_MAXN || r < 1 || r > LW_MAXR || D < 1) return false;
  return (size_t)lw_warp_f2((int)nmax, D, r) * sizeof(float2) <= 200 * 1024;
}

int launch_lanczos_window(const LanczosBatch& bt, cudaStream_t stream) {
  if (!lanczos_window_fits(bt.nmax, bt.D, bt.r)) return SLS_ERR_UNSUPPORTED;
  const size_t per_warp = (size_t)lw_warp_f2((int)bt.nmax, bt.D, bt.r) * sizeof(float2);
  int warps = (int)((200 * 1024) / per_warp);
  if (warps > LW_LAUNCH_WARPS) warps = LW_LAUNCH_WARPS;
  if (warps < 1) warps = 1;
  const size_t smem = per_warp * warps;
  const int blocks = (bt.nprob_max + warps - 1) / warps;
#define SLS_LW_LAUNCH_T(NV, RV, PT)                                                         \
  do {                                                                                      \
    SLS_CUDA_TRY(cudaFuncSetAttribute(lanczos_window_kernel<NV, RV, PT>,                    \
                                      cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)); \
    lanczos_window_kernel<NV, RV, PT><<<blocks, warps * 32, smem, stream>>>(bt);             \
  } while (0)
#define SLS_LW_LAUNCH(NV, RV)                                                               \
  do {                                                                                      \
    if (bt.phi_bf16)                                                                        \
      SLS_LW_LAUNCH_T(NV, RV, uint16_t);                                                    \
    else                                                                                    \
      SLS_LW_LAUNCH_T(NV, RV, float);                                                       \
  } while (0)
  if (bt.nmax <= 16 && bt.r <= 16)
    SLS_LW_LAUNCH(16, 16);
  else if (bt.nmax <= 16)
    SLS_LW_LAUNCH(16, 32);
  else if (bt.r <= 16)
    SLS_LW_LAUNCH(32, 16);
  else
    SLS_LW_LAUNCH(32, 32);
#undef SLS_LW_LAUNCH
#undef SLS_LW_LAUNCH_T
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

}  // namespace sls
