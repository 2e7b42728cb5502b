// Eigh(T) and Ritz vectors (Algorithm 1) after the implicit Lanczos of
// lanczos_kernel.cuh, plus the planning and launch of the Lanczos kernel.
//
// The r x r (r <= 128) tridiagonal T is solved on the device: Ritz values by
// Sturm-count multisection (one warp per eigenvalue, 32 shifts per round,
// float64), eigenvectors by inverse iteration with partial-pivoting LU, with
// modified Gram-Schmidt inside clusters of nearly equal eigenvalues.  Finally
// U = Q S.
#include "lanczos_kernel.cuh"

namespace sls {

namespace {

// ----------------------------------------------------------------------------
// Eigenvalues of T: multisection on Sturm counts (float64)
// ----------------------------------------------------------------------------

// Number of eigenvalues of the (scaled) tridiagonal below x, from the signs of
// the leading principal minors p_i(x) (three-term recurrence, Sturm sequence).
// Powers of two rescale the pair (p_{i-1}, p_i) to keep it in range; a zero
// minor takes the sign opposite to its predecessor.
SLS_DEV int sturm_count(const double* a, const double* b2, int n, double x) {
  double pm = 1.0, pc = a[0] - x;
  int sprev = 0;
  int s = (pc < 0.0) ? 1 : ((pc > 0.0) ? 0 : 1);
  int cnt = (s != sprev);
  sprev = s;
  for (int i = 1; i < n; ++i) {
    const double pn = fma(a[i] - x, pc, -b2[i - 1] * pm);
    pm = pc;
    pc = pn;
    const int ec = (__double2hiint(pc) >> 20) & 0x7ff;
    const int em = (__double2hiint(pm) >> 20) & 0x7ff;
    const int e = max(ec, em);
    if (e > 1023 + 400) {
      pc = pc * 0x1p-400;
      pm = pm * 0x1p-400;
    } else if (e < 1023 - 400) {
      pc = pc * 0x1p400;
      pm = pm * 0x1p400;
    }
    s = (pc < 0.0) ? 1 : ((pc > 0.0) ? 0 : 1 - sprev);
    cnt += (s != sprev);
    sprev = s;
  }
  return cnt;
}

__global__ void __launch_bounds__(32)
tridiag_eigvals_kernel(LanczosBatch bt) {
  __shared__ double sa[SLS_MAX_R], sb2[SLS_MAX_R];
  const int m = blockIdx.x, p = blockIdx.y, lane = threadIdx.x;
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  if (p >= nprob) return;
  const int r = bt.r;
  const int n = bt.r_eff[p];
  double* theta = bt.theta + (size_t)p * r;
  if (m >= n) {
    if (lane == 0) theta[m] = 0.0;
    return;
  }
  const double* a = bt.alpha + (size_t)p * r;
  const double* b = bt.beta + (size_t)p * r;
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
  const double big = fmax(fabs(glo), fabs(ghi));
  int ex = 0;
  frexp(big > 0.0 ? big : 1.0, &ex);
  const double sc = ldexp(1.0, -ex);  // power of two: exact scaling
  for (int i = lane; i < n; i += 32) {
    sa[i] = a[i] * sc;
    if (i < n - 1) {
      const double bs = b[i] * sc;
      sb2[i] = bs * bs;
    }
  }
  __syncwarp();
  double lo = glo * sc, hi = ghi * sc;
  const double pad = 4.0 * DBL_EPSILON * fmax(fabs(lo), fabs(hi)) + DBL_MIN;
  lo -= pad;
  hi += pad;
  const int k = n - 1 - m;  // ascending index of the wanted eigenvalue
  for (int round = 0; round < 64; ++round) {
    const double x = lo + (hi - lo) * ((double)(lane + 1) / 33.0);
    const int c = sturm_count(sa, sb2, n, x);
    const unsigned ball = __ballot_sync(0xffffffffu, c > k);
    if (ball == 0u) {
      lo = __shfl_sync(0xffffffffu, x, 31);
    } else {
      const int f = __ffs(ball) - 1;
      const double xf = __shfl_sync(0xffffffffu, x, f);
      const double xl = __shfl_sync(0xffffffffu, x, f > 0 ? f - 1 : 0);
      hi = xf;
      if (f > 0) lo = xl;
    }
    if (hi - lo <= 2.0 * DBL_EPSILON * fmax(fabs(lo), fabs(hi)) || hi - lo <= 2.0 * DBL_MIN)
      break;
  }
  if (lane == 0) theta[m] = (0.5 * (lo + hi)) / sc;
}

// ----------------------------------------------------------------------------
// Eigenvectors of T: inverse iteration (float64), MGS within clusters
// ----------------------------------------------------------------------------

__global__ void __launch_bounds__(32)
tridiag_eigvecs_kernel(LanczosBatch bt) {
  __shared__ double d[SLS_MAX_R], du[SLS_MAX_R], du2[SLS_MAX_R], dl[SLS_MAX_R];
  __shared__ double y[SLS_MAX_R];
  __shared__ unsigned char piv[SLS_MAX_R];
  const int m = blockIdx.x, p = blockIdx.y, lane = threadIdx.x;
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  if (p >= nprob) return;
  const int r = bt.r;
  const int n = bt.r_eff[p];
  double* S = bt.S + (size_t)p * r * r;
  if (m >= n) {
    for (int k = lane; k < r; k += 32) S[(size_t)k * r + m] = 0.0;
    return;
  }
  const double* th = bt.theta + (size_t)p * r;
  const double* a = bt.alpha + (size_t)p * r;
  const double* b = bt.beta + (size_t)p * r;
  const double tnorm = fmax(fabs(th[0]), fabs(th[n - 1])) + DBL_MIN;
  const double ctol = 1e-7 * tnorm;
  int first = m;
  while (first > 0 && th[first - 1] - th[first] <= ctol) --first;
  if (first != m) {
    // another CTA (the first member of this cluster) writes this column
    return;
  }
  int last = m;
  while (last + 1 < n && th[last] - th[last + 1] <= ctol) ++last;
  for (int k = lane + n; k < r; k += 32)
    for (int mm = first; mm <= last; ++mm) S[(size_t)k * r + mm] = 0.0;
  if (lane != 0) return;
  const double pert = DBL_EPSILON * tnorm;
  for (int mm = first; mm <= last; ++mm) {
    // distinct shifts inside a cluster
    const double shift = th[mm] - (double)(mm - first) * 4.0 * pert;
    for (int i = 0; i < n; ++i) {
      d[i] = a[i] - shift;
      if (i < n - 1) {
        du[i] = b[i];
        dl[i] = b[i];
      }
      du2[i] = 0.0;
    }
    if (n == 1) {
      y[0] = 1.0;
    } else {
      // LU with partial pivoting of T - shift I
      for (int i = 0; i < n - 1; ++i) {
        if (fabs(d[i]) >= fabs(dl[i])) {
          if (d[i] == 0.0) d[i] = pert;
          const double f = dl[i] / d[i];
          dl[i] = f;
          d[i + 1] -= f * du[i];
          piv[i] = 0;
        } else {
          const double f = d[i] / dl[i];
          d[i] = dl[i];
          dl[i] = f;
          const double tmp = du[i];
          du[i] = d[i + 1];
          d[i + 1] = tmp - f * d[i + 1];
          if (i < n - 2) {
            du2[i] = du[i + 1];
            du[i + 1] = -f * du[i + 1];
          }
          piv[i] = 1;
        }
      }
      if (d[n - 1] == 0.0) d[n - 1] = pert;
      // deterministic start vector
      for (int i = 0; i < n; ++i) {
        unsigned h = (unsigned)(i + 1) * 2654435761u ^ (unsigned)(mm + 7) * 40503u;
        h ^= h >> 13;
        h *= 0x5bd1e995u;
        h ^= h >> 15;
        y[i] = 0.5 + (double)(h & 0xffffu) / 65536.0;
      }
      for (int it = 0; it < 3; ++it) {
        for (int i = 0; i < n - 1; ++i) {
          if (!piv[i]) {
            y[i + 1] -= dl[i] * y[i];
          } else {
            const double t = y[i];
            y[i] = y[i + 1];
            y[i + 1] = t - dl[i] * y[i];
          }
        }
        y[n - 1] /= d[n - 1];
        y[n - 2] = (y[n - 2] - du[n - 2] * y[n - 1]) / d[n - 2];
        for (int i = n - 3; i >= 0; --i)
          y[i] = (y[i] - du[i] * y[i + 1] - du2[i] * y[i + 2]) / d[i];
        // orthogonalise against the cluster members found so far
        for (int pm = first; pm < mm; ++pm) {
          double dot = 0.0;
          for (int i = 0; i < n; ++i) dot += S[(size_t)i * r + pm] * y[i];
          for (int i = 0; i < n; ++i) y[i] -= dot * S[(size_t)i * r + pm];
        }
        double nr = 0.0;
        for (int i = 0; i < n; ++i) nr += y[i] * y[i];
        nr = sqrt(nr);
        if (!(nr > 0.0) || !isfinite(nr)) {
          for (int i = 0; i < n; ++i) y[i] = (i == mm) ? 1.0 : 0.0;
          nr = 1.0;
        }
        const double inv = 1.0 / nr;
        for (int i = 0; i < n; ++i) y[i] *= inv;
      }
    }
    const double sg = (y[0] < 0.0) ? -1.0 : 1.0;
    for (int i = 0; i < n; ++i) S[(size_t)i * r + mm] = sg * y[i];
    __threadfence_block();
  }
}

// ----------------------------------------------------------------------------
// Ritz vectors U = Q S (float32 output)
// ----------------------------------------------------------------------------

__global__ void __launch_bounds__(256)
ritz_vectors_kernel(LanczosBatch bt, float* __restrict__ U) {
  extern __shared__ float Ss[];  // r x r
  const int p = blockIdx.y;
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  if (p >= nprob) return;
  const int r = bt.r;
  const int kn = bt.r_eff[p];
  const int64_t row0 = bt.row0 ? bt.row0[p] : 0;
  const int64_t n = bt.n ? (int64_t)bt.n[p] : bt.n_single;
  const double* S = bt.S + (size_t)p * r * r;
  for (int e = threadIdx.x; e < r * r; e += blockDim.x) Ss[e] = (float)S[e];
  __syncthreads();
  const int rpb = blockDim.x / r;
  const int sub = threadIdx.x / r, m = threadIdx.x % r;
  if (sub >= rpb) return;
  for (int64_t i = (int64_t)blockIdx.x * rpb + sub; i < n; i += (int64_t)gridDim.x * rpb) {
    const float2* Qi = bt.Q + (row0 + i) * q_ld(r);
    float acc = 0.f;
    for (int k = 0; k < kn; ++k) {
      const float2 q = Qi[k];
      const float s = Ss[k * r + m];
      acc = fmaf(q.x, s, acc);
      acc = fmaf(q.y, s, acc);
    }
    U[(row0 + i) * r + m] = (m < kn) ? acc : 0.f;
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
    // a batch: enough CTAs per problem for ~256 rows each, as many groups as fit
    int64_t g = (nmax + 255) / 256;
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
  // barrier words start at zero
  for (int gi = 0; gi < groups; ++gi)
    SLS_CUDA_TRY(cudaMemsetAsync((char*)scratch + (size_t)gi * L.total + L.bar, 0, 256, stream));
  const int C4 = bt.D / 4;
  const int P = (C4 >= LZ_CT) ? 1 : (LZ_CT / C4);
  const int redn = (P > 1) ? P * bt.D : 0;
  const int rows_cap = (int)((bt.nmax + g - 1) / g) + 1;
  // shared memory besides the ring: w (hi, lo; only for D < 4 LZ_CT), phase
  // partials, z' of the strip, row-dot warp sums, coefficient partials and c,
  // barriers
  const size_t other = sizeof(float) * 2 * (size_t)(P > 1 ? bt.D : 0) +
                       sizeof(float2) * ((size_t)redn + (size_t)rows_cap + 16 * LZ_CW +
                                         (size_t)(LZ_CW + 1) * (bt.r + 1)) +
                       16 + 2 * RING_MAX_STAGES * 8;
  const size_t limit = 227 * 1024 - 1024;  // leave room for static shared memory
  if (other >= limit) return SLS_ERR_UNSUPPORTED;
  const RingShape R = ring_shape(bt.D, q_ld(bt.r), limit - other);
  if (R.S < 2) return SLS_ERR_UNSUPPORTED;
  const size_t smem = (size_t)R.S * R.stage + other;
  const int stages = R.S;
  const int kt = (bt.r <= 32) ? 1 : (bt.r <= 64) ? 2 : 4;  // 32-wide tiles of k < r
  switch (gpt_of(bt.D)) {
    case 1: return launch_lanczos_gpt1(bt, scratch, L.total, groups, g, rows_cap, stages, status, smem, stream, kt);
    case 2: return launch_lanczos_gpt2(bt, scratch, L.total, groups, g, rows_cap, stages, status, smem, stream, kt);
    case 4: return launch_lanczos_gpt4(bt, scratch, L.total, groups, g, rows_cap, stages, status, smem, stream, kt);
    case 8: return launch_lanczos_gpt8(bt, scratch, L.total, groups, g, rows_cap, stages, status, smem, stream, kt);
    default: break;
  }
  return SLS_ERR_UNSUPPORTED;
}

int launch_tridiag_eigen(const LanczosBatch& bt, cudaStream_t stream) {
  dim3 grid(bt.r, bt.nprob_max);
  tridiag_eigvals_kernel<<<grid, 32, 0, stream>>>(bt);
  SLS_LAUNCH_CHECK();
  tridiag_eigvecs_kernel<<<grid, 32, 0, stream>>>(bt);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

int launch_ritz_vectors(const LanczosBatch& bt, float* U, cudaStream_t stream) {
  const int r = bt.r;
  const int rpb = 256 / r;
  int64_t blocks = (bt.nmax + rpb - 1) / rpb;
  if (blocks > 1024) blocks = 1024;
  if (blocks < 1) blocks = 1;
  const size_t smem = sizeof(float) * r * r;
  SLS_CUDA_TRY(cudaFuncSetAttribute(ritz_vectors_kernel,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  ritz_vectors_kernel<<<dim3((unsigned)blocks, bt.nprob_max), 256, smem, stream>>>(bt, U);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

}  // namespace sls
