// Eigh(T) and Ritz vectors (Algorithm 1) after the implicit Lanczos of
// lanczos_kernel.cuh, plus the planning and launch of the Lanczos kernel.
//
// The r x r (r <= 128) tridiagonal T is solved on the device: Ritz values by
// Sturm-count multisection (a CTA of 256 shifts per eigenvalue when the
// launch has few, one warp of 32 shifts when it has many; double-float
// recurrence), eigenvectors by inverse iteration with
// partial-pivoting LU (double-float), with
// modified Gram-Schmidt inside clusters of nearly equal eigenvalues.  Finally
// U = Q S.
#include "lanczos_kernel.cuh"
#include "tridiag.cuh"

namespace sls {

namespace {

// Lanczos steps kept for problem p, clamped to [0, r]: r_eff is set to -1
// before the Lanczos launch and keeps that value if a device-side wait of the
// kernel gave up, so the later kernels then treat the problem as empty.
SLS_DEV int reff_clamped(const LanczosBatch& bt, int p) {
  return min(bt.r, max(0, bt.r_eff[p]));
}

// ----------------------------------------------------------------------------
// Eigenvalues of T: multisection on Sturm counts.  The arithmetic of the
// recurrences is double-float on the FP32 pipes: float64 on this part has a
// 64-cycle dependent latency (and a divide of several hundred cycles), which
// a serial recurrence pays at every step.
// ----------------------------------------------------------------------------

// Ritz values of few problems: one CTA per eigenvalue, 256 shifts per round
// (fewer, longer rounds: the faster form when the launch has few eigenvalues)
constexpr int EIG_THREADS = 256;  // shifts per multisection round
constexpr float kInvShiftsF = 1.0f / (float)(EIG_THREADS + 1);

__global__ void __launch_bounds__(EIG_THREADS)
tridiag_eigvals_cta_kernel(LanczosBatch bt) {
  __shared__ float2 sa[SLS_MAX_R], sb2[SLS_MAX_R];
  __shared__ int s_first[EIG_THREADS / 32];
  __shared__ double s_sc;
  __shared__ float2 s_lo, s_hi;  // the interval, double-float
  const int m = blockIdx.x, p = blockIdx.y, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  if (p >= nprob) return;
  const int r = bt.r;
  const int n = reff_clamped(bt, p);
  double* theta = bt.theta + (size_t)p * r;
  if (m >= n) {
    if (tid == 0) theta[m] = 0.0;
    return;
  }
  const double* a = bt.alpha + (size_t)p * r;
  const double* b = bt.beta + (size_t)p * r;
  if (warp == 0) {
    // Gershgorin interval, and a power-of-two scale that maps it into [-1, 1]
    double glo = DBL_MAX, ghi = -DBL_MAX;
    for (int i = lane; i < n; i += 32) {
      const double bl = (i > 0) ? fabs(b[i - 1]) : 0.0;
      const double br = (i < n - 1) ? fabs(b[i]) : 0.0;
      glo = fmin(glo, a[i] - bl - br);
      ghi = fmax(ghi, a[i] + bl + br);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      glo = fmin(glo, __shfl_xor_sync(0xffffffffu, glo, o));
      ghi = fmax(ghi, __shfl_xor_sync(0xffffffffu, ghi, o));
    }
    if (lane == 0) {
      const double big = fmax(fabs(glo), fabs(ghi));
      int ex = 0;
      frexp(big > 0.0 ? big : 1.0, &ex);
      const double sc = ldexp(1.0, -ex);  // exact scaling
      double lo = glo * sc, hi = ghi * sc;
      const double pad = 0x1p-40 * fmax(fabs(lo), fabs(hi)) + 0x1p-100;
      s_lo = f2(df_from_double(lo - pad));
      s_hi = f2(df_from_double(hi + pad));
      s_sc = sc;
    }
  }
  __syncthreads();
  const double sc = s_sc;
  for (int i = tid; i < n; i += EIG_THREADS) {
    sa[i] = f2(df_from_double(a[i] * sc));
    if (i < n - 1) {
      const double bs = b[i] * sc;
      sb2[i] = f2(df_from_double(bs * bs));
    }
  }
  __syncthreads();
  const int k = n - 1 - m;  // ascending index of the wanted eigenvalue
  for (int round = 0; round < 40; ++round) {
    const dfloat lo = dfv(s_lo), hi = dfv(s_hi);
    const dfloat w = df_sub(hi, lo);
    // 2^-46 relative, or one float64 unit of the scaled |T| <= 1
    if (w.hi <= 0x1p-46f * fmaxf(fabsf(lo.hi), fabsf(hi.hi)) || w.hi <= 0x1p-52f) break;
    // shift t: lo + (t + 1) (hi - lo) / (EIG_THREADS + 1), in double-float on
    // the float32 pipes (every thread computes one per round)
    const dfloat step = df_mul_f(w, kInvShiftsF);
    const int c = sturm_count(sa, sb2, n, df_add(lo, df_mul_f(step, (float)(tid + 1))));
    const unsigned ball = __ballot_sync(0xffffffffu, c > k);
    if (lane == 0) s_first[warp] = ball ? warp * 32 + __ffs(ball) - 1 : EIG_THREADS;
    __syncthreads();
    if (tid == 0) {
      int f = EIG_THREADS;
      for (int w2 = 0; w2 < EIG_THREADS / 32; ++w2) f = min(f, s_first[w2]);
      // count(x_t) is non-decreasing in t: the eigenvalue lies in (x_{f-1}, x_f]
      if (f < EIG_THREADS) s_hi = f2(df_add(lo, df_mul_f(step, (float)(f + 1))));
      if (f > 0) s_lo = f2(df_add(lo, df_mul_f(step, (float)f)));
    }
    __syncthreads();
  }
  if (tid == 0) theta[m] = (0.5 * df_to_double(df_add(dfv(s_lo), dfv(s_hi)))) / sc;
}

constexpr int EIG_WARPS = 8;  // eigenvalues per CTA (one warp each)

// Ritz values of many problems: one warp per eigenvalue, multisection on
// Sturm counts (32 shifts per round, one per lane; a ballot finds the
// subinterval that holds the wanted eigenvalue), the warps of a CTA sharing
// the problem's scaled T.
__global__ void __launch_bounds__(EIG_WARPS * 32)
tridiag_eigvals_kernel(LanczosBatch bt) {
  __shared__ float2 sa[SLS_MAX_R], sb2[SLS_MAX_R];
  __shared__ double s_glo, s_ghi;
  const int p = blockIdx.y, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  if (p >= nprob) return;
  const int r = bt.r;
  const int n = reff_clamped(bt, p);
  const int m = blockIdx.x * EIG_WARPS + warp;  // descending index of this warp's value
  double* theta = bt.theta + (size_t)p * r;
  const double* a = bt.alpha + (size_t)p * r;
  const double* b = bt.beta + (size_t)p * r;
  if (warp == 0) {
    // Gershgorin interval
    double glo = DBL_MAX, ghi = -DBL_MAX;
    for (int i = lane; i < n; i += 32) {
      const double bl = (i > 0) ? fabs(b[i - 1]) : 0.0;
      const double br = (i < n - 1) ? fabs(b[i]) : 0.0;
      glo = fmin(glo, a[i] - bl - br);
      ghi = fmax(ghi, a[i] + bl + br);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      glo = fmin(glo, __shfl_xor_sync(0xffffffffu, glo, o));
      ghi = fmax(ghi, __shfl_xor_sync(0xffffffffu, ghi, o));
    }
    if (lane == 0) {
      s_glo = glo;
      s_ghi = ghi;
    }
  }
  __syncthreads();
  // a power-of-two scale that maps the interval into [-1, 1] (exact)
  const double glo = s_glo, ghi = s_ghi;
  const double big = fmax(fabs(glo), fabs(ghi));
  int ex = 0;
  frexp(big > 0.0 ? big : 1.0, &ex);
  const double sc = ldexp(1.0, -ex);
  for (int i = tid; i < n; i += EIG_WARPS * 32) {
    sa[i] = f2(df_from_double(a[i] * sc));
    if (i < n - 1) {
      const double bs = b[i] * sc;
      sb2[i] = f2(df_from_double(bs * bs));
    }
  }
  __syncthreads();
  if (m >= r) return;
  if (m >= n) {
    if (lane == 0) theta[m] = 0.0;
    return;
  }
  const double pad = 0x1p-40 * fmax(fabs(glo * sc), fabs(ghi * sc)) + 0x1p-100;
  // the interval in double-float: the shifts and updates of every round run
  // on the float32 pipes (float64 throughput is a small fraction here, and
  // every lane of every warp computes a shift per round)
  dfloat lo = df_from_double(glo * sc - pad), hi = df_from_double(ghi * sc + pad);
  const int k = n - 1 - m;  // ascending index of the wanted eigenvalue
  for (int round = 0; round < 40; ++round) {
    const dfloat w = df_sub(hi, lo);
    if (w.hi <= 0x1p-46f * fmaxf(fabsf(lo.hi), fabsf(hi.hi)) || w.hi <= 0x1p-52f) break;
    const dfloat step = df_mul_f(w, 1.0f / 33.0f);
    const int c = sturm_count(sa, sb2, n, df_add(lo, df_mul_f(step, (float)(lane + 1))));
    // count(x_t) is non-decreasing in t: the eigenvalue lies in (x_{f-1}, x_f]
    const unsigned ball = __ballot_sync(0xffffffffu, c > k);
    const int f = ball ? __ffs(ball) - 1 : 32;
    const dfloat nhi = (f < 32) ? df_add(lo, df_mul_f(step, (float)(f + 1))) : hi;
    const dfloat nlo = (f > 0) ? df_add(lo, df_mul_f(step, (float)f)) : lo;
    lo = nlo;
    hi = nhi;
  }
  if (lane == 0) theta[m] = (0.5 * df_to_double(df_add(lo, hi))) / sc;
}

// ----------------------------------------------------------------------------
// Eigenvectors of T: inverse iteration with partial-pivoting LU (double-float),
// modified Gram-Schmidt within clusters of close eigenvalues
// ----------------------------------------------------------------------------

// Eigenvectors of one cluster [first, last] of nearly equal Ritz values of
// problem p (n = r_eff), written as columns of S: inverse iteration with
// partial-pivoting LU of T - shift I in double-float, two iterations, each
// followed by modified Gram-Schmidt against the cluster members already
// found.  One thread; the work arrays (n entries each) belong to the caller.
// The recurrences carry their running values in registers (the factorisation
// the current pivot row, the solves the last one or two entries), so a step's
// dependent chain holds no memory access, and the back substitution
// multiplies by the pivots' reciprocals, formed during the factorisation off
// that chain; sums over n run as four interleaved partial sums.
SLS_DEV dfloat sum4_df(dfloat (&acc)[4]) {
  return df_add(df_add(acc[0], acc[1]), df_add(acc[2], acc[3]));
}

// A power-of-two scale of T for problem p (the eigenvectors do not change):
// 1 / 2^ceil(log2 |T|), |T| from the extreme Ritz values.
SLS_DEV double eig_scale(const double* th, int n, double* tnorm_out) {
  const double tnorm = fmax(fabs(th[0]), fabs(th[n - 1])) + DBL_MIN;
  int ex = 0;
  frexp(tnorm, &ex);
  *tnorm_out = tnorm;
  return ldexp(1.0, -ex);
}

// The scaled diagonal sa[i] = alpha_i sc and off-diagonal sb[i] = beta_i sc of
// problem p as double-float, entries i = t, t + nt, ... for the nt calling
// threads (t = their index): every eigenvector of the problem starts from
// them, and the float64 products and splits, whose dependent latency is long
// on this part, run once per problem and in parallel.
SLS_DEV void eig_scaled_T(const LanczosBatch& bt, int p, int n, double sc, int t, int nt,
                          float2* __restrict__ sa, float2* __restrict__ sb) {
  const double* a = bt.alpha + (size_t)p * bt.r;
  const double* b = bt.beta + (size_t)p * bt.r;
  for (int i = t; i < n; i += nt) {
    sa[i] = f2(df_from_double(a[i] * sc));
    if (i < n - 1) sb[i] = f2(df_from_double(b[i] * sc));
  }
}

SLS_DEV void eigvec_cluster(const LanczosBatch& bt, int p, int n, int first, int last,
                            double sc, double tnorm, const float2* __restrict__ sa,
                            const float2* __restrict__ sb, float2* __restrict__ d,
                            float2* __restrict__ du, float2* __restrict__ du2,
                            float2* __restrict__ dl, float2* __restrict__ y,
                            unsigned char* __restrict__ piv) {
  const int r = bt.r;
  double* S = bt.S + (size_t)p * r * r;
  const double* th = bt.theta + (size_t)p * r;
  const double pert = 0x1p-44 * tnorm * sc;
  const dfloat pert_df = df_from_double(pert);
  const dfloat one = df_make(1.f, 0.f);
  for (int mm = first; mm <= last; ++mm) {
    // distinct shifts inside a cluster
    const dfloat shift = df_from_double((th[mm] - (double)(mm - first) * 4.0 * (pert / sc)) * sc);
    // the diagonal of T - shift I (d) and the off-diagonal (dl), unfactored
    for (int i = 0; i < n; ++i) {
      d[i] = f2(df_sub(dfv(sa[i]), shift));
      if (i < n - 1) dl[i] = sb[i];
    }
    if (n == 1) {
      y[0] = make_float2(1.f, 0.f);
    } else {
      // LU with partial pivoting of T - shift I; cd, cu: the current pivot
      // row's diagonal and superdiagonal entries as the elimination has left
      // them.  d[i] then holds the reciprocal of pivot i.
      dfloat cd = dfv(d[0]), cu = dfv(dl[0]);
      for (int i = 0; i < n - 1; ++i) {
        const dfloat li = dfv(dl[i]);
        const dfloat dn0 = dfv(d[i + 1]);
        const dfloat un0 = (i < n - 2) ? dfv(dl[i + 1]) : df_make(0.f, 0.f);
        if (fabsf(cd.hi) >= fabsf(li.hi)) {
          if (cd.hi == 0.f) cd = pert_df;
          const dfloat f = df_div(li, cd);
          d[i] = f2(df_div(one, cd));
          dl[i] = f2(f);
          du[i] = f2(cu);
          du2[i] = make_float2(0.f, 0.f);
          cd = df_sub(dn0, df_mul(f, cu));
          cu = un0;
          piv[i] = 0;
        } else {
          const dfloat f = df_div(cd, li);
          d[i] = f2(df_div(one, li));
          dl[i] = f2(f);
          du[i] = f2(dn0);
          du2[i] = f2(un0);
          cd = df_sub(cu, df_mul(f, dn0));
          cu = df_neg(df_mul(f, un0));
          piv[i] = 1;
        }
      }
      if (cd.hi == 0.f) cd = pert_df;
      d[n - 1] = f2(df_div(one, cd));
      // deterministic start vector
      for (int i = 0; i < n; ++i) {
        unsigned h = (unsigned)(i + 1) * 2654435761u ^ (unsigned)(mm + 7) * 40503u;
        h ^= h >> 13;
        h *= 0x5bd1e995u;
        h ^= h >> 15;
        y[i] = make_float2(0.5f + (float)(h & 0xffffu) / 65536.f, 0.f);
      }
      for (int it = 0; it < 2; ++it) {
        // forward substitution with the row interchanges; cy: the running y[i]
        dfloat cy = dfv(y[0]);
        for (int i = 0; i < n - 1; ++i) {
          const dfloat yn = dfv(y[i + 1]);
          const dfloat li = dfv(dl[i]);
          if (!piv[i]) {
            y[i] = f2(cy);
            cy = df_sub(yn, df_mul(li, cy));
          } else {
            y[i] = f2(yn);
            cy = df_sub(cy, df_mul(li, yn));
          }
        }
        // back substitution; c1, c2: y[i + 1], y[i + 2]
        dfloat c1 = df_mul(cy, dfv(d[n - 1]));
        y[n - 1] = f2(c1);
        dfloat c2 = c1;
        c1 = df_mul(df_sub(dfv(y[n - 2]), df_mul(dfv(du[n - 2]), c1)), dfv(d[n - 2]));
        y[n - 2] = f2(c1);
        for (int i = n - 3; i >= 0; --i) {
          const dfloat t = df_sub(df_sub(dfv(y[i]), df_mul(dfv(du[i]), c1)),
                                  df_mul(dfv(du2[i]), c2));
          c2 = c1;
          c1 = df_mul(t, dfv(d[i]));
          y[i] = f2(c1);
        }
        // keep the iterate in range: divide by its largest entry (a power of two)
        float ymax = 0.f;
        for (int i = 0; i < n; ++i) ymax = fmaxf(ymax, fabsf(y[i].x));
        if (ymax > 0.f && isfinite(ymax)) {
          int e2 = 0;
          frexpf(ymax, &e2);
          const float s2 = ldexpf(1.f, -e2);
          for (int i = 0; i < n; ++i) y[i] = f2(df_scale(dfv(y[i]), s2));
        }
        // orthogonalise against the cluster members found so far
        for (int pm = first; pm < mm; ++pm) {
          dfloat acc[4] = {df_make(0.f, 0.f), df_make(0.f, 0.f), df_make(0.f, 0.f),
                           df_make(0.f, 0.f)};
          for (int i = 0; i < n; ++i)
            acc[i & 3] = df_add(acc[i & 3],
                                df_mul(df_from_double(S[(size_t)i * r + pm]), dfv(y[i])));
          const dfloat dot = sum4_df(acc);
          for (int i = 0; i < n; ++i)
            y[i] = f2(df_sub(dfv(y[i]), df_mul(dot, df_from_double(S[(size_t)i * r + pm]))));
        }
        dfloat acc[4] = {df_make(0.f, 0.f), df_make(0.f, 0.f), df_make(0.f, 0.f),
                         df_make(0.f, 0.f)};
        for (int i = 0; i < n; ++i) acc[i & 3] = df_add(acc[i & 3], df_mul(dfv(y[i]), dfv(y[i])));
        const double nr = sqrt(df_to_double(sum4_df(acc)));
        if (!(nr > 0.0) || !isfinite(nr)) {
          for (int i = 0; i < n; ++i) y[i] = make_float2((i == mm) ? 1.f : 0.f, 0.f);
        } else {
          const dfloat inv = df_from_double(1.0 / nr);
          for (int i = 0; i < n; ++i) y[i] = f2(df_mul(dfv(y[i]), inv));
        }
      }
    }
    const double sg = (y[0].x < 0.f) ? -1.0 : 1.0;
#pragma unroll 4
    for (int i = 0; i < n; ++i) S[(size_t)i * r + mm] = sg * df_to_double(dfv(y[i]));
  }
}

// Cluster bounds of eigenvalue m: [first, last] with neighbours closer than
// 1e-7 * |T| merged (the eigenvectors of a cluster are computed together).
SLS_DEV void eig_cluster(const double* th, int n, int m, int& first, int& last) {
  const double tnorm = fmax(fabs(th[0]), fabs(th[n - 1])) + DBL_MIN;
  const double ctol = 1e-7 * tnorm;
  first = m;
  while (first > 0 && th[first - 1] - th[first] <= ctol) --first;
  last = m;
  while (last + 1 < n && th[last] - th[last + 1] <= ctol) ++last;
}

// One CTA (lane 0 working) per Ritz value: the CTA of a cluster's first
// member computes the whole cluster.
__global__ void __launch_bounds__(32)
tridiag_eigvecs_kernel(LanczosBatch bt) {
  __shared__ float2 d[SLS_MAX_R], du[SLS_MAX_R], du2[SLS_MAX_R], dl[SLS_MAX_R];
  __shared__ float2 y[SLS_MAX_R], sa[SLS_MAX_R], sb[SLS_MAX_R];
  __shared__ unsigned char piv[SLS_MAX_R];
  const int m = blockIdx.x, p = blockIdx.y, lane = threadIdx.x;
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  if (p >= nprob) return;
  const int r = bt.r;
  const int n = reff_clamped(bt, p);
  double* S = bt.S + (size_t)p * r * r;
  if (m >= n) {
    for (int k = lane; k < r; k += 32) S[(size_t)k * r + m] = 0.0;
    return;
  }
  int first, last;
  eig_cluster(bt.theta + (size_t)p * r, n, m, first, last);
  if (first != m) return;  // another CTA (the first member of this cluster) writes this column
  for (int k = lane + n; k < r; k += 32)
    for (int mm = first; mm <= last; ++mm) S[(size_t)k * r + mm] = 0.0;
  double tnorm;
  const double sc = eig_scale(bt.theta + (size_t)p * r, n, &tnorm);
  eig_scaled_T(bt, p, n, sc, lane, 32, sa, sb);
  __syncwarp();
  if (lane != 0) return;
  eigvec_cluster(bt, p, n, first, last, sc, tnorm, sa, sb, d, du, du2, dl, y, piv);
}

// Small problems (r <= 32): one warp per problem, one lane per Ritz value;
// the lane of a cluster's first member computes the whole cluster, with its
// work arrays in local memory.
constexpr int EIGW_WARPS = 1;  // one problem per CTA: the fewest idle SMs at the end
constexpr int EIGW_MAXR = 32;

__global__ void __launch_bounds__(EIGW_WARPS * 32)
tridiag_eigvecs_warp_kernel(LanczosBatch bt) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int p = blockIdx.x * EIGW_WARPS + warp;
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  if (p >= nprob) return;
  const int r = bt.r;
  const int n = reff_clamped(bt, p);
  double* S = bt.S + (size_t)p * r * r;
  // S rows and columns beyond r_eff are zero
  for (int e = lane; e < r * r; e += 32) {
    const int i = e / r, m = e % r;
    if (i >= n || m >= n) S[e] = 0.0;
  }
  __shared__ float2 sa[EIGW_WARPS][EIGW_MAXR], sb[EIGW_WARPS][EIGW_MAXR];
  double tnorm = 1.0, sc = 1.0;
  if (n > 0) {
    sc = eig_scale(bt.theta + (size_t)p * r, n, &tnorm);
    eig_scaled_T(bt, p, n, sc, lane, 32, sa[warp], sb[warp]);
  }
  __syncwarp();
  if (lane >= n) return;
  int first, last;
  eig_cluster(bt.theta + (size_t)p * r, n, lane, first, last);
  if (first != lane) return;
  float2 d[EIGW_MAXR], du[EIGW_MAXR], du2[EIGW_MAXR], dl[EIGW_MAXR], y[EIGW_MAXR];
  unsigned char piv[EIGW_MAXR];
  eigvec_cluster(bt, p, n, first, last, sc, tnorm, sa[warp], sb[warp], d, du, du2, dl, y, piv);
}

// ----------------------------------------------------------------------------
// Ritz vectors U = Q S (float32 output): tiles of basis rows in shared memory,
// 4 x 4 outputs per thread
// ----------------------------------------------------------------------------

constexpr int RITZ_THREADS = 256;

__host__ __device__ inline int ritz_tile_rows(int r) {
  const int cg = (r + 3) / 4;
  return (RITZ_THREADS / cg) * 4;
}

__global__ void __launch_bounds__(RITZ_THREADS)
ritz_vectors_kernel(LanczosBatch bt, float* __restrict__ U) {
  extern __shared__ float rsm[];
  const int p = blockIdx.y;
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  if (p >= nprob) return;
  const int r = bt.r, ldq = q_ld(r);
  const int kn = reff_clamped(bt, p);
  const int64_t row0 = bt.row0 ? bt.row0[p] : 0;
  const int64_t n = bt.n ? (int64_t)bt.n[p] : bt.n_single;
  const int cg = (r + 3) / 4, rg = RITZ_THREADS / cg, TR = rg * 4, qs = r + 1;
  float* Ss = rsm;                    // r x r
  float* Qh = Ss + (size_t)r * r;     // TR x (r+1)
  float* Ql = Qh + (size_t)TR * qs;   // TR x (r+1)
  const double* S = bt.S + (size_t)p * r * r;
  for (int e = threadIdx.x; e < r * r; e += RITZ_THREADS) Ss[e] = (float)S[e];
  const int t = threadIdx.x;
  const int rgi = t / cg, cgi = t % cg;
  const bool active = rgi < rg;
  for (int64_t i0 = (int64_t)blockIdx.x * TR; i0 < n; i0 += (int64_t)gridDim.x * TR) {
    const int nt = (int)min((int64_t)TR, n - i0);
    __syncthreads();
    const float2* Qt = bt.Q + (row0 + i0) * ldq;
    for (int e = t; e < nt * kn; e += RITZ_THREADS) {
      const int rr = e / kn, k = e % kn;
      const float2 q = Qt[(size_t)rr * ldq + k];
      Qh[rr * qs + k] = q.x;
      Ql[rr * qs + k] = q.y;
    }
    __syncthreads();
    if (!active) continue;
    float acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[a][c] = 0.f;
    const int rb = rgi * 4, cb = cgi * 4;
    for (int k = 0; k < kn; ++k) {
      float s[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) s[c] = (cb + c < r) ? Ss[k * r + cb + c] : 0.f;
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        const float qh = Qh[(rb + a) * qs + k], ql = Ql[(rb + a) * qs + k];
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[a][c] = fmaf(qh, s[c], fmaf(ql, s[c], acc[a][c]));
      }
    }
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      if (rb + a < nt) {
#pragma unroll
        for (int c = 0; c < 4; ++c)
          if (cb + c < r) U[(row0 + i0 + rb + a) * r + cb + c] = (cb + c < kn) ? acc[a][c] : 0.f;
      }
    }
  }
}

int num_sms() {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && v > 0)
      sms = v;
    else
      return 152;  // no device visible: plan for a GB300 (host-only size queries)
  }
  return sms;
}

}  // namespace

int lanczos_plan(int64_t nmax, int D, int r, int nprob, int* groups, int* ctas_per_group) {
  const int sms = num_sms();
  if (nprob <= 1) {
    // one problem: spread it over the whole GPU, but keep >= 32 rows per CTA
    int64_t g = (nmax + 31) / 32;
    if (g > sms) g = sms;
    if (g < 1) g = 1;
    *groups = 1;
    *ctas_per_group = (int)g;
  } else {
    // a batch: enough CTAs per problem for ~1024 rows each, as many groups as
    // fit (fewer CTAs per problem amortise the per-step barriers over more
    // rows; measured on 512 windows of 2048 rows at D = 1024: 256 rows per CTA
    // 65.7 ms, 512 62.4, 1024 59.5, 2048 66.8 with too few groups per round)
    int64_t g = (nmax + 1023) / 1024;
    if (g < 1) g = 1;
    if (g > sms) g = sms;
    int64_t gr = sms / g;
    if (gr < 1) gr = 1;
    if (gr > nprob) gr = nprob;
    *groups = (int)gr;
    *ctas_per_group = (int)g;
  }
  // rows per CTA must fit the shared-memory staging of u
  const int64_t rows = (nmax + *ctas_per_group - 1) / *ctas_per_group;
  if (rows > 8192) return SLS_ERR_UNSUPPORTED;
  (void)D;
  (void)r;
  return SLS_OK;
}

size_t lanczos_scratch_bytes(int64_t nmax, int D, int r, int groups, int g) {
  return (size_t)groups * lz_layout(nmax, D, r, g).total;
}

int launch_lanczos(const LanczosBatch& bt, void* scratch, size_t scratch_bytes, int* status,
                   int groups, int g, cudaStream_t stream) {
  const LzLayout L = lz_layout(bt.nmax, bt.D, bt.r, g);
  if ((size_t)groups * L.total > scratch_bytes) return SLS_ERR_WORKSPACE;
  // barrier words and group sums of every group start at zero (one strided memset)
  SLS_CUDA_TRY(cudaMemset2DAsync((char*)scratch + L.bar, L.total, 0, L.zero_end - L.bar, groups,
                                 stream));
  const int C4 = bt.D / 4;
  const int P = (C4 >= LZ_CT) ? 1 : (LZ_CT / C4);
  const int gpt = gpt_of(bt.D);
  if (gpt == 0) return SLS_ERR_UNSUPPORTED;
  const int teams = lz_teams(gpt, P);
  // z' of the strip, rounded up to an even count so the arrays after it stay
  // 16-byte aligned
  const int rows_cap = (int)(((bt.nmax + g - 1) / g + 2) & ~(int64_t)1);
  const size_t limit = 227 * 1024 - 1024;  // leave room for static shared memory
  if (bt.phi_bf16 && (bt.D % 8)) return SLS_ERR_UNSUPPORTED;  // 16-byte rows for the copies
  const int esz = bt.phi_bf16 ? 2 : 4;
  // the stage count and the mbarriers that go with it: take the largest S
  // whose ring and other shared memory fit
  RingShape R = ring_shape(bt.D, q_ld(bt.r), 0, esz, teams);
  int stages = 0;
  for (int s = RING_MAX_STAGES; s >= 1; --s) {
    if ((size_t)s * R.stage + lz_smem_other(bt.D, bt.r, rows_cap, teams, s) <= limit) {
      stages = s;
      break;
    }
  }
  // Room for the pass ends' scratch in the ring, and at least 2 teams + 2
  // stages: a team refills the slots of its previous pair after the first
  // barrier of its current pair, so chunk c is issued after the first barrier
  // of the pair `teams` pairs after the one holding chunk c - S; with fewer
  // stages (or 2 teams + 1) a team would wait for a chunk that only its own
  // later refill issues.
  if (stages < 2 * teams + 2) return SLS_ERR_UNSUPPORTED;
  if ((size_t)stages * R.stage < lz_pass_end_bytes(gpt, bt.r, teams)) return SLS_ERR_UNSUPPORTED;
  const size_t smem = (size_t)stages * R.stage + lz_smem_other(bt.D, bt.r, rows_cap, teams, stages);
  const int kt = (bt.r <= 32) ? 1 : (bt.r <= 64) ? 2 : 4;  // 32-wide tiles of k < r
#define SLS_LZ_CALL(fn) \
  fn(bt, scratch, L.total, groups, g, rows_cap, stages, status, smem, stream, kt, teams)
  if (bt.phi_bf16) {
    switch (gpt) {
      case 1: return SLS_LZ_CALL(launch_lanczos_bf16_gpt1);
      case 2: return SLS_LZ_CALL(launch_lanczos_bf16_gpt2);
      case 4: return SLS_LZ_CALL(launch_lanczos_bf16_gpt4);
      case 8: return SLS_LZ_CALL(launch_lanczos_bf16_gpt8);
      default: break;
    }
  } else {
    switch (gpt) {
      case 1: return SLS_LZ_CALL(launch_lanczos_gpt1);
      case 2: return SLS_LZ_CALL(launch_lanczos_gpt2);
      case 4: return SLS_LZ_CALL(launch_lanczos_gpt4);
      case 8: return SLS_LZ_CALL(launch_lanczos_gpt8);
      default: break;
    }
  }
#undef SLS_LZ_CALL
  return SLS_ERR_UNSUPPORTED;
}

int launch_tridiag_eigen(const LanczosBatch& bt, cudaStream_t stream, bool values_done) {
  dim3 grid(bt.r, bt.nprob_max);
  if (!values_done) {
    if ((int64_t)bt.r * bt.nprob_max <= 1024) {
      tridiag_eigvals_cta_kernel<<<grid, EIG_THREADS, 0, stream>>>(bt);
    } else {
      dim3 vgrid((bt.r + EIG_WARPS - 1) / EIG_WARPS, bt.nprob_max);
      tridiag_eigvals_kernel<<<vgrid, EIG_WARPS * 32, 0, stream>>>(bt);
    }
    SLS_LAUNCH_CHECK();
  }
  if (bt.r <= EIGW_MAXR) {
    const int blocks = (bt.nprob_max + EIGW_WARPS - 1) / EIGW_WARPS;
    tridiag_eigvecs_warp_kernel<<<blocks, EIGW_WARPS * 32, 0, stream>>>(bt);
  } else {
    tridiag_eigvecs_kernel<<<grid, 32, 0, stream>>>(bt);
  }
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

int launch_ritz_vectors(const LanczosBatch& bt, float* U, cudaStream_t stream) {
  const int r = bt.r;
  const int TR = ritz_tile_rows(r);
  int64_t blocks = (bt.nmax + TR - 1) / TR;
  if (blocks > 4 * (int64_t)num_sms()) blocks = 4 * (int64_t)num_sms();
  if (blocks < 1) blocks = 1;
  const size_t smem = sizeof(float) * ((size_t)r * r + 2 * (size_t)TR * (r + 1));
  SLS_CUDA_TRY(cudaFuncSetAttribute(ritz_vectors_kernel,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  ritz_vectors_kernel<<<dim3((unsigned)blocks, bt.nprob_max), RITZ_THREADS, smem, stream>>>(bt, U);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

}  // namespace sls
