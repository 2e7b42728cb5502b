// Implicit Lanczos (Algorithm 2), Eigh(T) and Ritz vectors (Algorithm 1).
//
// Lanczos runs as one persistent cooperative kernel.  The grid is split into
// groups of CTAs; a group owns one problem at a time (one prompt, or one
// adaptive window) and its CTAs own contiguous row strips of that problem's
// feature matrix Phi (N x D, float32).  One step j costs two streaming sweeps
// over the strip and four group barriers:
//
//   A  u_j = z1 - Q c2 (second Gram-Schmidt correction of step j-1), stored
//      as column j of Q; w_part = Phi^T u_j and |u_j|^2 per CTA.
//      [barrier]  every CTA reduces a slice of the D columns
//      [barrier]  beta_{j-1} = |u_j|, w = Phi^T q_j = w_red / beta_{j-1},
//                 alpha_j = q_j^T A q_j = |w|^2, break test
//   B  z' = Phi w - alpha_j q_j - beta_{j-1} q_{j-1}   (the implicit matvec of
//      Eq. implicit_matvec and the three-term recurrence) and the first
//      Gram-Schmidt coefficients c = Q^T z' per CTA
//      [barrier]  c = sum of the CTA partials
//   D  z1 = z' - Q c and the second coefficients c2 = Q^T z1 per CTA
//      [barrier]  c2 = sum of the CTA partials
//
// Normalisation is deferred (q_j = u_j / |u_j| is applied in B), so |u_j|
// rides along with the first sweep.  All vectors are double-float (two
// float32) and every sum over N or D is Dot2-compensated; reductions use a
// fixed order, so results are bit-reproducible.  Barriers give up after a
// bounded number of polls and report SLS_ERR_TIMEOUT through the status word.
//
// The r x r (r <= 128) tridiagonal T is then solved on the device: Ritz values
// by Sturm-count multisection (one warp per eigenvalue, 32 shifts per round,
// float64), eigenvectors by inverse iteration with partial-pivoting LU, with
// modified Gram-Schmidt inside clusters of nearly equal eigenvalues.  Finally
// U = Q S.
#include <cfloat>

#include "common.cuh"
#include "kernels.cuh"

namespace sls {

namespace {

constexpr int LZ_THREADS = 256;
constexpr int LZ_WARPS = LZ_THREADS / 32;

// Per-group scratch layout (byte offsets), identical on host and device.
struct LzLayout {
  size_t z0, z1, wpart, wred, cpartB, cpartD, npart, bar, total;
};

__host__ __device__ inline size_t lz_al(size_t x) { return (x + 255) & ~(size_t)255; }

__host__ __device__ inline LzLayout lz_layout(int64_t nmax, int D, int r, int g) {
  LzLayout L;
  size_t o = 0;
  L.bar = o;    o += 256;
  L.z0 = o;     o += lz_al((size_t)nmax * sizeof(float2));
  L.z1 = o;     o += lz_al((size_t)nmax * sizeof(float2));
  L.wpart = o;  o += lz_al((size_t)g * D * sizeof(float2));
  L.wred = o;   o += lz_al((size_t)D * sizeof(float2));
  L.cpartB = o; o += lz_al((size_t)g * (r + 1) * sizeof(float2));
  L.cpartD = o; o += lz_al((size_t)g * (r + 1) * sizeof(float2));
  L.npart = o;  o += lz_al((size_t)g * sizeof(float2));
  L.total = o;
  return L;
}

SLS_DEV float2 f2(dfloat a) { return make_float2(a.hi, a.lo); }
SLS_DEV dfloat dfv(float2 a) { return df_make(a.x, a.y); }

SLS_DEV dfloat shfl_df(dfloat v, int src) {
  v.hi = __shfl_sync(0xffffffffu, v.hi, src);
  v.lo = __shfl_sync(0xffffffffu, v.lo, src);
  return v;
}

// Block-wide double-float sum; result valid in every thread.
SLS_DEV dfloat block_sum_df(dfloat v, float2* tmp /* LZ_WARPS */) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_sum_df(v);
  __syncthreads();
  if (lane == 0) tmp[warp] = f2(v);
  __syncthreads();
  dfloat s = df_make(0.f, 0.f);
#pragma unroll
  for (int w = 0; w < LZ_WARPS; ++w) s = df_add(s, dfv(tmp[w]));
  return s;
}

// Sweep A: w_part[c] = sum over the strip of Phi[i, c] * u_i (Dot2).
// GPT float4 column groups per thread; P row phases when D/4 < LZ_THREADS.
template <int GPT>
SLS_DEV void sweep_phi_t_u(const float* __restrict__ Phi, int D, int64_t rs, int64_t re,
                           const float2* __restrict__ us, float2* __restrict__ red,
                           float2* __restrict__ wpart_row) {
  const int tid = threadIdx.x;
  const int C4 = D >> 2;
  const int P = (C4 >= LZ_THREADS) ? 1 : (LZ_THREADS / C4);
  const int act = (P == 1) ? LZ_THREADS : P * C4;
  constexpr int UNR = (16 / GPT) < 2 ? 2 : (16 / GPT);
  if (tid < act) {
    const int ph = (P == 1) ? 0 : tid / C4;
    const int cb = (P == 1) ? tid : tid % C4;
    float ah[GPT][4], al[GPT][4];
#pragma unroll
    for (int q = 0; q < GPT; ++q)
#pragma unroll
      for (int c = 0; c < 4; ++c) ah[q][c] = al[q][c] = 0.f;
    const float4* base = reinterpret_cast<const float4*>(Phi);
    int64_t i = rs + ph;
    for (; i + (int64_t)(UNR - 1) * P < re; i += (int64_t)UNR * P) {
      float4 f[UNR][GPT];
      float2 uu[UNR];
#pragma unroll
      for (int t = 0; t < UNR; ++t) {
        const int64_t row = i + (int64_t)t * P;
        uu[t] = us[row - rs];
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          const int cg = cb + q * LZ_THREADS;
          f[t][q] = (cg < C4) ? __ldg(base + row * C4 + cg) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
#pragma unroll
      for (int t = 0; t < UNR; ++t)
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          dot2_acc(ah[q][0], al[q][0], f[t][q].x, uu[t].x, uu[t].y);
          dot2_acc(ah[q][1], al[q][1], f[t][q].y, uu[t].x, uu[t].y);
          dot2_acc(ah[q][2], al[q][2], f[t][q].z, uu[t].x, uu[t].y);
          dot2_acc(ah[q][3], al[q][3], f[t][q].w, uu[t].x, uu[t].y);
        }
    }
    for (; i < re; i += P) {
      const float2 u = us[i - rs];
#pragma unroll
      for (int q = 0; q < GPT; ++q) {
        const int cg = cb + q * LZ_THREADS;
        if (cg < C4) {
          const float4 f = __ldg(base + i * C4 + cg);
          dot2_acc(ah[q][0], al[q][0], f.x, u.x, u.y);
          dot2_acc(ah[q][1], al[q][1], f.y, u.x, u.y);
          dot2_acc(ah[q][2], al[q][2], f.z, u.x, u.y);
          dot2_acc(ah[q][3], al[q][3], f.w, u.x, u.y);
        }
      }
    }
    float2* dst = (P == 1) ? wpart_row : red + (size_t)ph * D;
#pragma unroll
    for (int q = 0; q < GPT; ++q) {
      const int cg = cb + q * LZ_THREADS;
      if (cg < C4) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          dfloat v = df_norm(ah[q][c], al[q][c]);
          dst[4 * cg + c] = f2(v);
        }
      }
    }
  }
  if (P > 1) {
    __syncthreads();
    for (int col = tid; col < D; col += LZ_THREADS) {
      dfloat s = df_make(0.f, 0.f);
      for (int ph = 0; ph < P; ++ph) s = df_add(s, dfv(red[(size_t)ph * D + col]));
      wpart_row[col] = f2(s);
    }
  }
}

// Row dot product s = Phi[i, :] . w with w in shared memory (double-float);
// one warp per row, every lane returns the sum.
SLS_DEV dfloat row_dot_w(const float* __restrict__ Phi, int D, int64_t i,
                         const float2* __restrict__ wsm) {
  const int lane = threadIdx.x & 31;
  const int C4 = D >> 2;
  const float4* rowp = reinterpret_cast<const float4*>(Phi) + i * C4;
  const float4* w4 = reinterpret_cast<const float4*>(wsm);  // (h0,l0,h1,l1),(h2,l2,h3,l3)
  float h[4] = {0.f, 0.f, 0.f, 0.f}, l[4] = {0.f, 0.f, 0.f, 0.f};
  constexpr int CH = 16;
  for (int q0 = 0; q0 < C4; q0 += CH * 32) {
    float4 f[CH];
#pragma unroll
    for (int t = 0; t < CH; ++t) {
      const int cg = q0 + lane + 32 * t;
      f[t] = (cg < C4) ? __ldg(rowp + cg) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int t = 0; t < CH; ++t) {
      const int cg = q0 + lane + 32 * t;
      if (cg < C4) {
        const float4 wa = w4[2 * cg], wb = w4[2 * cg + 1];
        dot2_acc(h[0], l[0], f[t].x, wa.x, wa.y);
        dot2_acc(h[1], l[1], f[t].y, wa.z, wa.w);
        dot2_acc(h[2], l[2], f[t].z, wb.x, wb.y);
        dot2_acc(h[3], l[3], f[t].w, wb.z, wb.w);
      }
    }
  }
  dfloat s = df_add(df_add(df_make(h[0], l[0]), df_make(h[1], l[1])),
                    df_add(df_make(h[2], l[2]), df_make(h[3], l[3])));
  return warp_sum_df(s);
}

template <int GPT>
__global__ void __launch_bounds__(LZ_THREADS, 1)
lanczos_kernel(LanczosBatch bt, char* scratch, size_t gstride, int g, int ngroups,
               int rows_cap, int* status) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ float2 tmpw[LZ_WARPS];
  __shared__ double shd[4];
  __shared__ int sflag, sbreak;

  const int D = bt.D, r = bt.r, C4 = D >> 2;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int gi = blockIdx.x / g, rank = blockIdx.x % g;
  const int P = (C4 >= LZ_THREADS) ? 1 : (LZ_THREADS / C4);
  const int redn = (P > 1) ? P * D : 0;

  float2* wsm = reinterpret_cast<float2*>(smem_raw);
  float2* red = wsm + D;
  float2* us = red + redn;
  float2* cw = us + rows_cap;                    // LZ_WARPS x (r+1)
  float2* cs = cw + (size_t)LZ_WARPS * (r + 1);  // r+1

  const LzLayout L = lz_layout(bt.nmax, D, r, g);
  char* gb = scratch + (size_t)gi * gstride;
  unsigned* barw = reinterpret_cast<unsigned*>(gb + L.bar);
  float2* z0 = reinterpret_cast<float2*>(gb + L.z0);
  float2* z1 = reinterpret_cast<float2*>(gb + L.z1);
  float2* wpart = reinterpret_cast<float2*>(gb + L.wpart);
  float2* wred = reinterpret_cast<float2*>(gb + L.wred);
  float2* cpartB = reinterpret_cast<float2*>(gb + L.cpartB);
  float2* cpartD = reinterpret_cast<float2*>(gb + L.cpartD);
  float2* npart = reinterpret_cast<float2*>(gb + L.npart);
  const GroupBarrier bar{barw, barw + 32, (unsigned)g};
  unsigned lgen = 0;

  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);

  for (int p = gi; p < nprob; p += ngroups) {
    const int64_t row0 = bt.row0 ? bt.row0[p] : 0;
    const int64_t n = bt.n ? (int64_t)bt.n[p] : bt.n_single;
    const int64_t q1o = bt.q1off ? bt.q1off[p] : row0;
    const float* Phi = bt.Phi + row0 * D;
    float2* Q = bt.Q + row0 * r;
    const double* q1 = bt.q1 + q1o;
    const int64_t rs = (int64_t)rank * n / g, re = (int64_t)(rank + 1) * n / g;
    double* alpha_out = bt.alpha + (size_t)p * r;
    double* beta_out = bt.beta + (size_t)p * r;
    const int cbeg = (int)((int64_t)rank * D / g), cend = (int)((int64_t)(rank + 1) * D / g);

    double scale = 0.0;
    double alpha_prev = 0.0;
    dfloat alpha_df = df_make(0.f, 0.f), beta_df = df_make(0.f, 0.f), invb_df;
    int reff = 0;

    for (int j = 0; j < r; ++j) {
      // ---------------- phase A: u_j, stored as column j of Q ----------------
      dfloat nacc = df_make(0.f, 0.f);
      for (int64_t i = rs + warp; i < re; i += LZ_WARPS) {
        dfloat u;
        if (j == 0) {
          u = df_make(0.f, 0.f);
          if (lane == 0) u = df_from_double(q1[i]);
          u = shfl_df(u, 0);
        } else {
          const float2* Qi = Q + i * r;
          float corr = 0.f;
          for (int k = lane; k < j; k += 32) {
            const float2 qk = Qi[k], ck = cs[k];
            corr = fmaf(qk.x, ck.x, fmaf(qk.x, ck.y, fmaf(qk.y, ck.x, corr)));
          }
          corr = warp_sum_f(corr);
          u = df_add(dfv(z1[i]), df_make(-corr, 0.f));
        }
        if (lane == 0) {
          Q[i * r + j] = f2(u);
          us[i - rs] = f2(u);
          dot2_acc_df(nacc.hi, nacc.lo, u, u);
        }
      }
      if (lane == 0) tmpw[warp] = f2(df_norm(nacc.hi, nacc.lo));
      __syncthreads();
      if (tid == 0) {
        dfloat s = df_make(0.f, 0.f);
        for (int w = 0; w < LZ_WARPS; ++w) s = df_add(s, dfv(tmpw[w]));
        npart[rank] = f2(s);
      }
      sweep_phi_t_u<GPT>(Phi, D, rs, re, us, red, wpart + (size_t)rank * D);
      if (!group_sync(bar, lgen, status, &sflag)) return;

      // slice reduction of w over the group's CTAs
      for (int c = cbeg + warp; c < cend; c += LZ_WARPS) {
        dfloat s = df_make(0.f, 0.f);
        for (int b = lane; b < g; b += 32) s = df_add(s, dfv(wpart[(size_t)b * D + c]));
        s = warp_sum_df(s);
        if (lane == 0) wred[c] = f2(s);
      }
      if (!group_sync(bar, lgen, status, &sflag)) return;

      // |u_j|^2, |w_red|^2, w into shared memory
      if (warp == 0) {
        dfloat s = df_make(0.f, 0.f);
        for (int b = lane; b < g; b += 32) s = df_add(s, dfv(npart[b]));
        s = warp_sum_df(s);
        if (lane == 0) shd[0] = df_to_double(s);
      }
      dfloat sq = df_make(0.f, 0.f);
      for (int c = tid; c < D; c += LZ_THREADS) {
        const float2 v = wred[c];
        wsm[c] = v;
        dot2_acc_df(sq.hi, sq.lo, dfv(v), dfv(v));
      }
      sq = block_sum_df(df_norm(sq.hi, sq.lo), tmpw);
      if (tid == 0) {
        const double nrm2 = shd[0];
        const double bnew = sqrt(nrm2);
        int brk = 0;
        if (j > 0) {
          scale = fmax(scale, fabs(alpha_prev) + bnew);
          if (!(bnew > bt.tol * scale)) brk = 1;
          else if (rank == 0) beta_out[j - 1] = bnew;
        } else if (!(bnew > 0.0)) {
          brk = 1;  // zero start vector: nothing to iterate
        }
        const double a = brk ? 0.0 : df_to_double(sq) / nrm2;
        if (!brk && rank == 0) alpha_out[j] = a;
        shd[1] = brk ? 0.0 : 1.0 / bnew;
        shd[2] = a;
        shd[3] = (j > 0) ? bnew : 0.0;
        sbreak = brk;
      }
      __syncthreads();
      if (sbreak) {
        reff = j;
        break;
      }
      invb_df = df_from_double(shd[1]);
      alpha_prev = shd[2];
      alpha_df = df_from_double(shd[2]);
      beta_df = df_from_double(shd[3]);
      for (int c = tid; c < D; c += LZ_THREADS) wsm[c] = f2(df_mul(dfv(wsm[c]), invb_df));
      __syncthreads();

      // ---------------- phase B: z' = A q_j - alpha q_j - beta q_{j-1} --------
      const bool last = (j == r - 1);
      dfloat cacc[(SLS_MAX_R + 1 + 31) / 32];
#pragma unroll
      for (int t = 0; t < (SLS_MAX_R + 1 + 31) / 32; ++t) cacc[t] = df_make(0.f, 0.f);
      for (int64_t i = rs + warp; i < re; i += LZ_WARPS) {
        const dfloat s = row_dot_w(Phi, D, i, wsm);
        const float2* Qi = Q + i * r;
        const dfloat qj = df_mul(dfv(Qi[j]), invb_df);
        dfloat zp = df_sub(s, df_mul(alpha_df, qj));
        if (j > 0) zp = df_sub(zp, df_mul(beta_df, dfv(Qi[j - 1])));
        __syncwarp();
        if (lane == 0) {
          Q[i * r + j] = f2(qj);
          z0[i] = f2(zp);
        }
        if (!last) {
#pragma unroll
          for (int t = 0; t < (SLS_MAX_R + 1 + 31) / 32; ++t) {
            const int k = lane + 32 * t;
            if (k <= j) {
              const dfloat qk = (k == j) ? qj : dfv(Qi[k]);
              dot2_acc_df(cacc[t].hi, cacc[t].lo, qk, zp);
            }
          }
        }
      }
      if (last) {
        reff = r;
        break;
      }
#pragma unroll
      for (int t = 0; t < (SLS_MAX_R + 1 + 31) / 32; ++t) {
        const int k = lane + 32 * t;
        if (k <= j) cw[(size_t)warp * (r + 1) + k] = f2(df_norm(cacc[t].hi, cacc[t].lo));
      }
      __syncthreads();
      for (int k = tid; k <= j; k += LZ_THREADS) {
        dfloat s = df_make(0.f, 0.f);
        for (int w = 0; w < LZ_WARPS; ++w) s = df_add(s, dfv(cw[(size_t)w * (r + 1) + k]));
        cpartB[(size_t)rank * (r + 1) + k] = f2(s);
      }
      if (!group_sync(bar, lgen, status, &sflag)) return;
      for (int k = warp; k <= j; k += LZ_WARPS) {
        dfloat s = df_make(0.f, 0.f);
        for (int b = lane; b < g; b += 32) s = df_add(s, dfv(cpartB[(size_t)b * (r + 1) + k]));
        s = warp_sum_df(s);
        if (lane == 0) cs[k] = f2(s);
      }
      __syncthreads();

      // ---------------- phase D: z1 = z' - Q c, c2 = Q^T z1 ----------------------
#pragma unroll
      for (int t = 0; t < (SLS_MAX_R + 1 + 31) / 32; ++t) cacc[t] = df_make(0.f, 0.f);
      for (int64_t i = rs + warp; i < re; i += LZ_WARPS) {
        const float2* Qi = Q + i * r;
        float corr = 0.f;
        for (int k = lane; k <= j; k += 32) {
          const float2 qk = Qi[k], ck = cs[k];
          corr = fmaf(qk.x, ck.x, fmaf(qk.x, ck.y, fmaf(qk.y, ck.x, corr)));
        }
        corr = warp_sum_f(corr);
        const dfloat zz = df_add(dfv(z0[i]), df_make(-corr, 0.f));
        if (lane == 0) z1[i] = f2(zz);
#pragma unroll
        for (int t = 0; t < (SLS_MAX_R + 1 + 31) / 32; ++t) {
          const int k = lane + 32 * t;
          if (k <= j) dot2_acc_df(cacc[t].hi, cacc[t].lo, dfv(Qi[k]), zz);
        }
      }
#pragma unroll
      for (int t = 0; t < (SLS_MAX_R + 1 + 31) / 32; ++t) {
        const int k = lane + 32 * t;
        if (k <= j) cw[(size_t)warp * (r + 1) + k] = f2(df_norm(cacc[t].hi, cacc[t].lo));
      }
      __syncthreads();
      for (int k = tid; k <= j; k += LZ_THREADS) {
        dfloat s = df_make(0.f, 0.f);
        for (int w = 0; w < LZ_WARPS; ++w) s = df_add(s, dfv(cw[(size_t)w * (r + 1) + k]));
        cpartD[(size_t)rank * (r + 1) + k] = f2(s);
      }
      if (!group_sync(bar, lgen, status, &sflag)) return;
      for (int k = warp; k <= j; k += LZ_WARPS) {
        dfloat s = df_make(0.f, 0.f);
        for (int b = lane; b < g; b += 32) s = df_add(s, dfv(cpartD[(size_t)b * (r + 1) + k]));
        s = warp_sum_df(s);
        if (lane == 0) cs[k] = f2(s);
      }
      __syncthreads();
    }
    if (rank == 0 && tid == 0) {
      bt.r_eff[p] = reff;
      for (int k = reff; k < r; ++k) alpha_out[k] = 0.0;
      for (int k = (reff > 0 ? reff - 1 : 0); k < r; ++k) beta_out[k] = 0.0;
    }
    // problems on the same group run back to back; keep them apart
    if (!group_sync(bar, lgen, status, &sflag)) return;
  }
}

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
    const float2* Qi = bt.Q + (row0 + i) * r;
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

template <int GPT>
int launch_lanczos_t(const LanczosBatch& bt, void* scratch, size_t gstride, int groups, int g,
                     int rows_cap, int* status, size_t smem, cudaStream_t stream) {
  auto fn = lanczos_kernel<GPT>;
  SLS_CUDA_TRY(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  char* sc = (char*)scratch;
  void* args[] = {(void*)&bt, (void*)&sc, (void*)&gstride, (void*)&g, (void*)&groups,
                  (void*)&rows_cap, (void*)&status};
  SLS_CUDA_TRY(cudaLaunchCooperativeKernel((const void*)fn, dim3(groups * g), dim3(LZ_THREADS),
                                           args, smem, stream));
  count_launch(1);
  return SLS_OK;
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
  const int P = (C4 >= LZ_THREADS) ? 1 : (LZ_THREADS / C4);
  const int redn = (P > 1) ? P * bt.D : 0;
  const int rows_cap = (int)((bt.nmax + g - 1) / g) + 1;
  const size_t smem = sizeof(float2) * ((size_t)bt.D + redn + rows_cap +
                                        (size_t)(LZ_WARPS + 1) * (bt.r + 1));
  if (smem > 200 * 1024) return SLS_ERR_UNSUPPORTED;
  const int gpt = (C4 + LZ_THREADS - 1) / LZ_THREADS;
  if (gpt <= 1) return launch_lanczos_t<1>(bt, scratch, L.total, groups, g, rows_cap, status, smem, stream);
  if (gpt <= 2) return launch_lanczos_t<2>(bt, scratch, L.total, groups, g, rows_cap, status, smem, stream);
  if (gpt <= 4) return launch_lanczos_t<4>(bt, scratch, L.total, groups, g, rows_cap, status, smem, stream);
  if (gpt <= 8) return launch_lanczos_t<8>(bt, scratch, L.total, groups, g, rows_cap, status, smem, stream);
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
