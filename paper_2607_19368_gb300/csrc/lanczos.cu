// Implicit Lanczos (Algorithm 2), Eigh(T) and Ritz vectors (Algorithm 1).
//
// Lanczos runs as one persistent cooperative kernel.  The grid is split into
// groups of CTAs; a group owns one problem at a time (one prompt, or one
// adaptive window) and every CTA owns a contiguous strip of the problem's rows
// of the feature matrix Phi (N x D, float32) and of the basis Q.  One copy warp
// per CTA streams the Phi strip through a shared-memory ring with
// one-dimensional bulk copies (cp.async.bulk + mbarrier), twice per step, and
// runs ahead of the eight compute warps by as many chunks as the ring holds.
// All work on basis rows happens in two dense row phases between the sweeps,
// with the strip's rows split over the compute warps (batches of 32 rows,
// lanes over the basis index, transposed butterflies for the row sums).
//
// Step j (0-based):
//
//   row phase A         z1 = z' - Q c (first Gram-Schmidt pass of step j-1, c
//                       from the previous barrier 3), c2 += Q^T z1, |z1|^2.
//   sweep A (forward)   Phi^T z1, column-parallel.
//                       [barrier 1]
//   slice phase         c2 = sum of the CTA partials (second Gram-Schmidt
//                       coefficients); each CTA finishes a slice of the D
//                       columns of Phi^T u_j = Phi^T z1 - sum_k c2_k w_k with
//                       w_k = Phi^T q_k kept from earlier steps.
//                       [barrier 2]
//                       beta_{j-1} = |u_j| = sqrt(|z1|^2 - |c2|^2), the break
//                       test, w_j = Phi^T q_j, alpha_j = |w_j|^2.
//   sweep B (backward)  s = Phi w_j, the implicit matvec (Eq. implicit_matvec):
//                       all compute threads share each chunk, w_j in registers.
//   row phase B         u = z1 - Q c2, q_j = u / beta_{j-1}, the three-term
//                       recurrence z' = s - alpha_j q_j - beta_{j-1} q_{j-1},
//                       and c += Q^T z'.
//                       [barrier 3]  c = sum of the CTA partials
//
// For j = 0, z1 is the start vector q1.  This is Algorithm 2 with two-pass
// classical Gram-Schmidt re-orthogonalisation, regrouped so that the two
// passes over Phi per step are pure streams; in exact arithmetic it equals the
// textbook order.  Sweep B runs backward so the rows sweep A touched last are
// still in L2.  Vectors are double-float (two float32), every sum over N or D
// is Dot2-compensated, reductions have a fixed order (bit-reproducible runs).
// Barriers and waits give up after a bounded number of polls and report
// SLS_ERR_TIMEOUT through the status word.
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

constexpr int LZ_CW = 8;                  // compute warps
constexpr int LZ_CT = LZ_CW * 32;         // compute threads
constexpr int LZ_THREADS = LZ_CT + 32;    // plus one copy warp
constexpr unsigned BAR_COMPUTE = 1;       // named barrier: the compute warps
constexpr int KT_MAX = (SLS_MAX_R + 31) / 32;  // basis columns k < r per lane

// leading dimension (float2) of the basis rows: even, so rows are 16-byte aligned
__host__ __device__ inline int q_ld(int r) { return (r + 1) & ~1; }

// Per-group scratch layout (byte offsets), identical on host and device.
struct LzLayout {
  size_t bar, wpart, wred, Wm, cpartA, cpartB, npart, sqpart, total;
};

__host__ __device__ inline size_t lz_al(size_t x) { return (x + 255) & ~(size_t)255; }

__host__ __device__ inline LzLayout lz_layout(int64_t nmax, int D, int r, int g) {
  (void)nmax;
  LzLayout L;
  size_t o = 0;
  L.bar = o;    o += 256;
  L.wpart = o;  o += lz_al((size_t)g * D * sizeof(float2));
  L.wred = o;   o += lz_al((size_t)D * sizeof(float2));
  L.Wm = o;     o += lz_al((size_t)D * r * sizeof(float2));
  L.cpartA = o; o += lz_al((size_t)g * (r + 1) * sizeof(float2));
  L.cpartB = o; o += lz_al((size_t)g * (r + 1) * sizeof(float2));
  L.npart = o;  o += lz_al((size_t)g * sizeof(float2));
  L.sqpart = o; o += lz_al((size_t)g * sizeof(float2));
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

// Ring stage: cr rows of Phi (cr * D floats).  For D >= 4 * LZ_CT (one
// column group per compute thread or more) a stage holds TEAM_ELEMS / D rows,
// so that sweep B can give every compute thread the same number of elements
// per chunk; smaller D takes as many rows as fit RING_STAGE bytes.
struct RingShape {
  int cr;          // rows per chunk
  int S;           // stages
  unsigned stage;  // bytes per stage
};

constexpr int RING_STAGE = 32 * 1024;
constexpr int RING_MAX_STAGES = 8;
constexpr int WB_ROWS = 64;  // rows per window of sweep-B warp partials

// float4 column groups per compute thread, rounded up to a power of two
// (1, 2, 4 or 8; 0 when D is too wide)
__host__ __device__ inline int gpt_of(int D) {
  const int need = (D / 4 + LZ_CT - 1) / LZ_CT;
  return need <= 1 ? 1 : need <= 2 ? 2 : need <= 4 ? 4 : need <= 8 ? 8 : 0;
}
// rows per chunk of the team sweep B: 8 / GPT (GPT * 4 * rows = 32 elements
// per thread per chunk)
__host__ __device__ constexpr int team_rows(int gpt) { return gpt >= 8 ? 1 : 8 / gpt; }

__host__ __device__ inline RingShape ring_shape(int D, size_t budget) {
  RingShape R;
  if (D / 4 >= LZ_CT) {
    R.cr = team_rows(gpt_of(D));
  } else {
    R.cr = RING_STAGE / (4 * D);
    if (R.cr < 1) R.cr = 1;
  }
  R.stage = (unsigned)R.cr * (unsigned)D * 4u;
  R.S = (int)(budget / R.stage);
  if (R.S > RING_MAX_STAGES) R.S = RING_MAX_STAGES;
  return R;
}

// Sweep A over one chunk: acc[c] += Phi[i, c] * z1_i for the chunk's rows,
// column-parallel (GPT float4 groups per thread, P row phases), Dot2.  With
// TRACK the thread also keeps the largest |Phi| it has seen in *mx.
template <int GPT, bool TRACK>
SLS_DEV void sweepA_chunk(const float* __restrict__ chunk, int nr, int D, int lb,
                          const float2* __restrict__ us, f32x2_t (&ah)[GPT][2],
                          f32x2_t (&al)[GPT][2], float* mx) {
  const int tid = threadIdx.x;
  const int C4 = D >> 2;
  const int P = (C4 >= LZ_CT) ? 1 : (LZ_CT / C4);
  if (P > 1 && tid >= P * C4) return;
  const int ph = (P == 1) ? 0 : tid / C4;
  const int cb = (P == 1) ? tid : tid % C4;
  const float4* c4 = reinterpret_cast<const float4*>(chunk);
  for (int i = ph; i < nr; i += P) {
    const float2 u = us[lb + i];
    const f32x2_t uh = pk2(u.x, u.x), nuh = pk2(-u.x, -u.x), ul = pk2(u.y, u.y);
#pragma unroll
    for (int q = 0; q < GPT; ++q) {
      const int cg = cb + q * LZ_CT;
      if (cg < C4) {
        const float4 f = c4[i * C4 + cg];
        dot2_acc2n(ah[q][0], al[q][0], pk2(f.x, f.y), uh, nuh, ul);
        dot2_acc2n(ah[q][1], al[q][1], pk2(f.z, f.w), uh, nuh, ul);
        if (TRACK)
          *mx = fmaxf(*mx, fmaxf(fmaxf(fabsf(f.x), fabsf(f.y)), fmaxf(fabsf(f.z), fabsf(f.w))));
      }
    }
  }
}

SLS_DEV dfloat shfl_xor_df(dfloat v, int m) {
  v.hi = __shfl_xor_sync(0xffffffffu, v.hi, m);
  v.lo = __shfl_xor_sync(0xffffffffu, v.lo, m);
  return v;
}

// Transposed butterfly over CR rows (CR a power of two <= 32): every lane
// holds one partial per row; afterwards lane L holds the warp sum of row
// L >> (5 - log2 CR).  CR - 1 + 5 - log2 CR shuffles instead of 5 per row.
template <int CR>
SLS_DEV float transpose_sum_f(float (&v)[CR]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int s = 0; s < 5; ++s) {
    const int h = 16 >> s;
    const int nv = (CR >> s) > 1 ? (CR >> s) : 1;
    if (nv > 1) {
      const bool up = (lane & h) != 0;
#pragma unroll
      for (int i = 0; i < nv / 2; ++i) {
        const float send = up ? v[i] : v[i + nv / 2];
        const float keep = up ? v[i + nv / 2] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, h);
      }
    } else {
      v[0] += __shfl_xor_sync(0xffffffffu, v[0], h);
    }
  }
  return v[0];
}

// Sweep A over two ring chunks at once (D >= 4 * LZ_CT; CR rows each, the
// second chunk may be absent: nr1 = 0) with offset accumulators: ah starts at
// the power-of-two offset of the column sums.  FULL: both chunks full and
// D = 4 * LZ_CT * GPT, so no guards.
template <int GPT, int CR, bool FULL>
SLS_DEV void sweepA_team_pair(const float* __restrict__ c0, int nr0, int lb0,
                              const float* __restrict__ c1, int nr1, int lb1, int C4,
                              const float2* __restrict__ us, f32x2_t (&ah)[GPT][2],
                              f32x2_t (&al)[GPT][2]) {
  const int tid = threadIdx.x;
#pragma unroll
  for (int i = 0; i < 2 * CR; ++i) {
    const bool first = i < CR;
    const int ii = first ? i : i - CR;
    if (FULL || ii < (first ? nr0 : nr1)) {
      const float4* c4 = reinterpret_cast<const float4*>(first ? c0 : c1);
      const float2 u = us[(first ? lb0 : lb1) + ii];
      const f32x2_t uh = pk2(u.x, u.x), nuh = pk2(-u.x, -u.x), ul = pk2(u.y, u.y);
#pragma unroll
      for (int q = 0; q < GPT; ++q) {
        const int cg = tid + q * LZ_CT;
        if (FULL || cg < C4) {
          const float4 f = c4[ii * C4 + cg];
          ofs_acc2n(ah[q][0], al[q][0], pk2(f.x, f.y), uh, nuh, ul);
          ofs_acc2n(ah[q][1], al[q][1], pk2(f.z, f.w), uh, nuh, ul);
        }
      }
    }
  }
}

// Double-float sum without the second renormalisation (11 operations): the
// error is a few units of the low part, enough for partial sums that are
// combined once.
SLS_DEV dfloat df_add_fast(dfloat a, dfloat b) {
  float s, e;
  two_sum(a.hi, b.hi, s, e);
  e = __fadd_rn(e, __fadd_rn(a.lo, b.lo));
  float h, l;
  fast_two_sum(s, e, h, l);
  return df_make(h, l);
}

// Transposed butterfly over CR rows (CR a power of two <= 32), double-float:
// every lane holds one partial per row; afterwards lane L holds the warp sum
// of row L >> (5 - log2 CR).  CR - 1 + 5 - log2 CR shuffles instead of 5 per
// row.
template <int CR>
SLS_DEV dfloat transpose_sum_df(dfloat (&v)[CR]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int s = 0; s < 5; ++s) {
    const int h = 16 >> s;
    const int nv = (CR >> s) > 1 ? (CR >> s) : 1;
    if (nv > 1) {
      const bool up = (lane & h) != 0;
#pragma unroll
      for (int i = 0; i < nv / 2; ++i) {
        const dfloat send = up ? v[i] : v[i + nv / 2];
        const dfloat keep = up ? v[i + nv / 2] : v[i];
        v[i] = df_add_fast(keep, shfl_xor_df(send, h));
      }
    } else {
      v[0] = df_add_fast(v[0], shfl_xor_df(v[0], h));
    }
  }
  return v[0];
}

// Sweep B over two ring chunks at once with all compute threads (D >= 4 *
// LZ_CT): thread t owns the float4 column groups t + LZ_CT q of every row, w
// for those columns sits in registers.  Each thread accumulates its part of
// a row against its own offset Ct (a power of two above twice max|Phi| times
// the l1 norm of its slice of w), so the FastTwoSum steps lose nothing to a
// loose global bound; the 2 CR per-row double-float partials are then summed
// over the warp by one transposed butterfly and the warp sums stored to
// bp0 / bp1 [i * LZ_CW + warp].
template <int GPT, int CR, bool FULL>
SLS_DEV void sweepB_team_pair(const float* __restrict__ c0, int nr0, const float* __restrict__ c1,
                              int nr1, int C4, const f32x2_t (&wh)[GPT][2],
                              const f32x2_t (&nwh)[GPT][2], const f32x2_t (&wl)[GPT][2],
                              float Ct, float2* __restrict__ bp0, float2* __restrict__ bp1) {
  constexpr int R2 = 2 * CR;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  dfloat v[R2];
#pragma unroll
  for (int i = 0; i < R2; ++i) {
    const bool first = i < CR;
    const int ii = first ? i : i - CR;
    f32x2_t s = pk2(Ct, Ct), lo = 0ull;
    if (FULL || ii < (first ? nr0 : nr1)) {
      const float4* c4 = reinterpret_cast<const float4*>(first ? c0 : c1);
#pragma unroll
      for (int q = 0; q < GPT; ++q) {
        const int cg = tid + q * LZ_CT;
        if (FULL || cg < C4) {
          const float4 f = c4[ii * C4 + cg];
          ofs_acc2n(s, lo, pk2(f.x, f.y), wh[q][0], nwh[q][0], wl[q][0]);
          ofs_acc2n(s, lo, pk2(f.z, f.w), wh[q][1], nwh[q][1], wl[q][1]);
        }
      }
    }
    float sx, sy, lx, ly;
    upk2(s, sx, sy);
    upk2(lo, lx, ly);
    const float x = sy - Ct;  // exact
    const float s1 = sx + x;
    v[i] = df_make(s1 - Ct, (lx + ly) + (x - (s1 - sx)));
  }
  const dfloat r = transpose_sum_df<R2>(v);
  constexpr int SH = (R2 >= 32) ? 0 : (R2 >= 16) ? 1 : (R2 >= 8) ? 2 : (R2 >= 4) ? 3 : 4;
  if ((lane & ((1 << SH) - 1)) == 0) {
    const int i = lane >> SH;
    if (i < CR) {
      if (i < nr0) bp0[i * LZ_CW + warp] = f2(r);
    } else if (i - CR < nr1) {
      bp1[(i - CR) * LZ_CW + warp] = f2(r);
    }
  }
}

// Row dot product with w from shared memory (separate hi / lo arrays); one
// warp per row, all lanes get the sum.  Used by sweep B when D < 4 * LZ_CT.
SLS_DEV dfloat row_dot_smem(const float* __restrict__ row, int D, const float* __restrict__ wsh,
                            const float* __restrict__ wsl) {
  const int lane = threadIdx.x & 31;
  const int C4 = D >> 2;
  const float4* r4 = reinterpret_cast<const float4*>(row);
  const float4* h4 = reinterpret_cast<const float4*>(wsh);
  const float4* l4 = reinterpret_cast<const float4*>(wsl);
  f32x2_t h01 = 0, l01 = 0, h23 = 0, l23 = 0;
  for (int cg = lane; cg < C4; cg += 32) {
    const float4 f = r4[cg];
    const float4 wh = h4[cg], wl = l4[cg];
    dot2_acc2(h01, l01, pk2(f.x, f.y), pk2(wh.x, wh.y), pk2(wl.x, wl.y));
    dot2_acc2(h23, l23, pk2(f.z, f.w), pk2(wh.z, wh.w), pk2(wl.z, wl.w));
  }
  float a0, a1, b0, b1, c0, c1, d0, d1;
  upk2(h01, a0, a1);
  upk2(l01, b0, b1);
  upk2(h23, c0, c1);
  upk2(l23, d0, d1);
  dfloat s = df_add(df_add(df_make(a0, b0), df_make(a1, b1)),
                    df_add(df_make(c0, d0), df_make(c1, d1)));
  return warp_sum_df(s);
}

// Position in the ring: chunks consumed, current slot and its phase parity.
struct RingCursor {
  unsigned cnt;
  int slot;
  unsigned par;
};

SLS_DEV void rc_next(RingCursor& c, int S) {
  ++c.cnt;
  if (++c.slot == S) {
    c.slot = 0;
    c.par ^= 1u;
  }
}

SLS_DEV int nprob_of(const LanczosBatch& bt) {
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  return nprob;
}

// Sum of the per-CTA partial coefficients part[b * (r+1) + k] over the g CTAs
// of a group, for k < K, into cs[k].  Every CTA does it redundantly; the loads
// are spread over all compute threads so they are in flight together.
SLS_DEV void reduce_coeffs(const float2* __restrict__ part, int g, int r, int K,
                           float2* __restrict__ cs, float2* __restrict__ tmp) {
  const int tid = threadIdx.x;
  if (K <= 0) return;
  int PH = LZ_CT / K;
  if (PH < 1) PH = 1;
  if (PH > 8) PH = 8;
  while (PH > 1 && PH * K > 4 * LZ_CT) --PH;
  for (int idx = tid; idx < K * PH; idx += LZ_CT) {
    const int k = idx % K, ph = idx / K;
    dfloat s = df_make(0.f, 0.f);
    int b = ph;
    for (; b + 7 * PH < g; b += 8 * PH) {
      float2 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = part[(size_t)(b + u * PH) * (r + 1) + k];
#pragma unroll
      for (int u = 0; u < 8; ++u) s = df_add(s, dfv(v[u]));
    }
    for (; b < g; b += PH) s = df_add(s, dfv(part[(size_t)b * (r + 1) + k]));
    tmp[ph * K + k] = f2(s);
  }
  named_sync(BAR_COMPUTE, LZ_CT);
  for (int k = tid; k < K; k += LZ_CT) {
    dfloat s = df_make(0.f, 0.f);
    for (int ph = 0; ph < PH; ++ph) s = df_add(s, dfv(tmp[ph * K + k]));
    cs[k] = f2(s);
  }
  named_sync(BAR_COMPUTE, LZ_CT);
}

// Per-warp partial coefficients (lanes over k < K) -> the CTA's partial row.
SLS_DEV void store_coeff_partials(dfloat (&cacc)[KT_MAX], int K, int r, float2* __restrict__ cw,
                                  float2* __restrict__ dst) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
#pragma unroll
  for (int t = 0; t < KT_MAX; ++t) {
    const int k = lane + 32 * t;
    if (k < K) cw[(size_t)warp * (r + 1) + k] = f2(df_norm(cacc[t].hi, cacc[t].lo));
  }
  named_sync(BAR_COMPUTE, LZ_CT);
  for (int k = tid; k < K; k += LZ_CT) {
    dfloat s = df_make(0.f, 0.f);
    for (int w = 0; w < LZ_CW; ++w) s = df_add(s, dfv(cw[(size_t)w * (r + 1) + k]));
    dst[k] = f2(s);
  }
}

constexpr int RG = 8;  // basis rows per register group in the row phases

// Basis rows 0 .. RG-1 of Qb (those < ng) at the columns k = lane + 32 kt < K,
// zero elsewhere; all loads of a group are in flight together.
SLS_DEV void load_qgroup(const float2* __restrict__ Qb, int ldq, int ng, int K,
                         float2 (&q)[RG][KT_MAX]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < RG; ++i) {
#pragma unroll
    for (int kt = 0; kt < KT_MAX; ++kt) {
      const int k = lane + 32 * kt;
      q[i][kt] = make_float2(0.f, 0.f);
      if (i < ng && 32 * kt < K && k < K) q[i][kt] = Qb[(size_t)i * ldq + k];
    }
  }
}

// sum_k q[i][k] c_k for the RG rows of a group (float32: the coefficients are
// at rounding level); lane L gets row L >> 2.
SLS_DEV float group_correction(const float2 (&q)[RG][KT_MAX], const float2 (&cv)[KT_MAX]) {
  float v[RG];
#pragma unroll
  for (int i = 0; i < RG; ++i) {
    float s = 0.f;
#pragma unroll
    for (int kt = 0; kt < KT_MAX; ++kt)
      s = fmaf(q[i][kt].x, cv[kt].x, fmaf(q[i][kt].x, cv[kt].y, fmaf(q[i][kt].y, cv[kt].x, s)));
    v[i] = s;
  }
  return transpose_sum_f<RG>(v);
}

// Row phase A of step j >= 1 for the warp's rows [wr0, wr1) of the strip, in
// groups of RG rows held in registers (lanes over the basis index k):
// z1 = z' - Q c (first pass), us = z1, |z1|^2, sum |z1|, c2 += Q^T z1.
SLS_DEV void row_phase_A(const float2* __restrict__ Qs, int ldq, int wr0, int wr1, int j,
                         const float2* __restrict__ cs, const float2* __restrict__ zps,
                         float2* __restrict__ us, dfloat& nacc, float& zl1,
                         dfloat (&c2acc)[KT_MAX]) {
  const int lane = threadIdx.x & 31;
  float2 cv[KT_MAX];
#pragma unroll
  for (int kt = 0; kt < KT_MAX; ++kt) {
    const int k = lane + 32 * kt;
    cv[kt] = (k < j) ? cs[k] : make_float2(0.f, 0.f);
  }
  for (int b = wr0; b < wr1; b += RG) {
    const int ng = min(RG, wr1 - b);
    const float2* Qb = Qs + (size_t)b * ldq;
    float2 q[RG][KT_MAX];
    load_qgroup(Qb, ldq, ng, j, q);
    const int i = lane >> 2;
    const float2 zin = (i < ng) ? zps[b + i] : make_float2(0.f, 0.f);
    const float corr = group_correction(q, cv);
    dfloat z = df_make(0.f, 0.f);
    if (i < ng) {
      z = df_add(dfv(zin), df_make(-corr, 0.f));
      if ((lane & 3) == 0) {
        us[b + i] = f2(z);
        dot2_acc_df(nacc.hi, nacc.lo, z, z);
        zl1 += fabsf(z.hi);
      }
    }
#pragma unroll
    for (int ii = 0; ii < RG; ++ii) {
      const dfloat zb = shfl_df(z, 4 * ii);
#pragma unroll
      for (int kt = 0; kt < KT_MAX; ++kt) {
        const int k = lane + 32 * kt;
        if (32 * kt < j && k < j) dot2_acc_df(c2acc[kt].hi, c2acc[kt].lo, dfv(q[ii][kt]), zb);
      }
    }
  }
}

// Row phase B of step j for the warp's rows: u = z1 - Q c2 (second pass),
// q_j = u / beta_{j-1}, z' = s - alpha_j q_j - beta_{j-1} q_{j-1} with
// s = (Phi w_j)_i from sweep B (held in zps on entry), Q[:, j] = q_j, and
// c += Q^T z' over k <= j unless this is the last step.
SLS_DEV void row_phase_B(float2* __restrict__ Qs, int ldq, int wr0, int wr1, int j, bool last,
                         const float2* __restrict__ c2s, const float2* __restrict__ us,
                         float2* __restrict__ zps, dfloat invb, dfloat alpha, dfloat beta,
                         dfloat (&cacc)[KT_MAX]) {
  const int lane = threadIdx.x & 31;
  float2 cv[KT_MAX];
#pragma unroll
  for (int kt = 0; kt < KT_MAX; ++kt) {
    const int k = lane + 32 * kt;
    cv[kt] = (k < j) ? c2s[k] : make_float2(0.f, 0.f);
  }
  for (int b = wr0; b < wr1; b += RG) {
    const int ng = min(RG, wr1 - b);
    float2* Qb = Qs + (size_t)b * ldq;
    float2 q[RG][KT_MAX];
    load_qgroup(Qb, ldq, ng, j, q);
    const int i = lane >> 2;
    float2 sin = make_float2(0.f, 0.f), uin = sin, qprev = sin;
    if (i < ng) {
      sin = zps[b + i];
      uin = us[b + i];
      if (j > 0) qprev = Qb[(size_t)i * ldq + j - 1];
    }
    const float corr = group_correction(q, cv);
    dfloat qj = df_make(0.f, 0.f), zp = df_make(0.f, 0.f);
    if (i < ng) {
      dfloat u = dfv(uin);
      if (j > 0) u = df_add(u, df_make(-corr, 0.f));
      qj = df_mul(u, invb);
      zp = df_sub(dfv(sin), df_mul(alpha, qj));
      if (j > 0) zp = df_sub(zp, df_mul(beta, dfv(qprev)));
      if ((lane & 3) == 0) {
        Qb[(size_t)i * ldq + j] = f2(qj);
        zps[b + i] = f2(zp);
      }
    }
    if (!last) {
#pragma unroll
      for (int ii = 0; ii < RG; ++ii) {
        const dfloat zb = shfl_df(zp, 4 * ii);
        const dfloat qb = shfl_df(qj, 4 * ii);
#pragma unroll
        for (int kt = 0; kt < KT_MAX; ++kt) {
          const int k = lane + 32 * kt;
          if (32 * kt <= j && k <= j) {
            const dfloat qk = (k == j) ? qb : dfv(q[ii][kt]);
            dot2_acc_df(cacc[kt].hi, cacc[kt].lo, qk, zb);
          }
        }
      }
    }
  }
}

template <int GPT>
__global__ void __launch_bounds__(LZ_THREADS, 1)
lanczos_kernel(LanczosBatch bt, char* scratch, size_t gstride, int g, int ngroups,
               int rows_cap, int ring_stages, int* status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ float2 tmpw[LZ_CW];
  __shared__ float s_red1[LZ_CW];  // per-warp max |Phi| and sum |z1| (offset bounds)
  __shared__ double shd[4];
  __shared__ int sflag, sbreak;
  // copy warp <-> compute warps handshake (no named barrier involves the copy
  // warp, so an early exit of either side can never leave the other blocked in
  // bar.sync; every wait on these flags is bounded)
  __shared__ volatile int s_halt;        // compute -> copy: stop issuing this problem
  __shared__ volatile int s_go;          // compute -> copy: may start problem s_go - 1
  __shared__ volatile int s_pdone;       // copy -> compute: finished problem s_pdone - 1
  __shared__ volatile unsigned s_issued;  // copy -> compute: chunks issued so far

  constexpr int TCR = team_rows(GPT);
  const int D = bt.D, r = bt.r, ldq = q_ld(bt.r);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int gi = blockIdx.x / g, rank = blockIdx.x % g;
  const int C4 = D >> 2;
  const int P = (C4 >= LZ_CT) ? 1 : (LZ_CT / C4);
  const int redn = (P > 1) ? P * D : 0;
  const bool fullD = (C4 == GPT * LZ_CT);  // no ragged column groups

  const RingShape shp0 = ring_shape(D, 0);
  const int S = ring_stages;
  const int cr = shp0.cr;
  const unsigned stage = shp0.stage;
  unsigned char* ring = smem_raw;
  unsigned char* after_ring = smem_raw + (size_t)S * stage;
  float* wsh = reinterpret_cast<float*>(after_ring);   // D
  float* wsl = wsh + D;                                // D
  float2* red = reinterpret_cast<float2*>(wsl + D);    // redn
  float2* us = red + redn;                             // rows_cap (z1 of the strip)
  float2* zps = us + rows_cap;                         // rows_cap (s, then z')
  float2* bpart = zps + rows_cap;                      // 2 x WB_ROWS x LZ_CW
  float2* cw = bpart + 2 * WB_ROWS * LZ_CW;            // LZ_CW x (r+1)
  float2* cs = cw + (size_t)LZ_CW * (r + 1);           // r+1 (c, first pass)
  float2* c2s = cs + (r + 1);                          // r+1 (c2, second pass)
  float2* red2 = c2s + (r + 1);                        // 4 * LZ_CT
  uint64_t* bars = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(red2 + 4 * LZ_CT) + 15) & ~(uintptr_t)15);
  uint64_t* fullb = bars;
  uint64_t* emptyb = bars + S;

  const LzLayout L = lz_layout(bt.nmax, D, r, g);
  char* gb = scratch + (size_t)gi * gstride;
  unsigned* barw = reinterpret_cast<unsigned*>(gb + L.bar);
  float2* wpart = reinterpret_cast<float2*>(gb + L.wpart);
  float2* wred = reinterpret_cast<float2*>(gb + L.wred);
  float2* Wm = reinterpret_cast<float2*>(gb + L.Wm);
  float2* cpartA = reinterpret_cast<float2*>(gb + L.cpartA);
  float2* cpartB = reinterpret_cast<float2*>(gb + L.cpartB);
  float2* npart = reinterpret_cast<float2*>(gb + L.npart);
  float2* sqpart = reinterpret_cast<float2*>(gb + L.sqpart);
  const GroupBarrier bar{barw, barw + 32, (unsigned)g};

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&fullb[s], 1);
      mbar_init(&emptyb[s], LZ_CW);
    }
    mbar_fence_init();
    s_halt = 0;
    s_go = 0;
    s_pdone = 0;
    s_issued = 0;
  }
  __syncthreads();

  const int nprob = nprob_of(bt);

  // ========================= copy warp ======================================
  // Phi is read-only, so the copy warp runs ahead of the compute warps by as
  // many chunks as the ring holds: sweep A forward, sweep B backward, per step.
  if (warp == LZ_CW) {
    if (lane != 0) return;
    const uint64_t pol = l2_policy_normal();
    unsigned cnt = 0;
    int pp = 0;
    for (int p = gi; p < nprob; p += ngroups, ++pp) {
      bool ok = false;
      for (unsigned it = 0; it < (1u << 26); ++it) {
        if (s_go == pp + 1) {
          ok = true;
          break;
        }
        __nanosleep(64);
      }
      if (!ok) {
        atomicExch(status, SLS_ERR_TIMEOUT);
        break;
      }
      const int64_t row0 = bt.row0 ? bt.row0[p] : 0;
      const int64_t n = bt.n ? (int64_t)bt.n[p] : bt.n_single;
      const int64_t rs = (int64_t)rank * n / g, re = (int64_t)(rank + 1) * n / g;
      const int nch = (int)((re - rs + cr - 1) / cr);
      const float* Phi = bt.Phi + (row0 + rs) * D;
      bool stop = false;
      for (int j = 0; j < r && !stop; ++j) {
        for (int sweep = 0; sweep < 2 && !stop; ++sweep) {
          for (int t = 0; t < nch; ++t) {
            if (s_halt) {
              stop = true;
              break;
            }
            const int k = (sweep == 0) ? t : nch - 1 - t;
            const int slot = (int)(cnt % (unsigned)S);
            const unsigned par = (cnt / (unsigned)S) & 1u;
            if (!mbar_wait(&emptyb[slot], par ^ 1u)) {
              atomicExch(status, SLS_ERR_TIMEOUT);
              stop = true;
              break;
            }
            const int64_t nr = min((int64_t)cr, (re - rs) - (int64_t)k * cr);
            const unsigned b1 = (unsigned)(nr * D * 4);
            unsigned char* dst = ring + (size_t)slot * stage;
            mbar_expect_tx(&fullb[slot], b1);
            bulk_g2s(dst, Phi + (int64_t)k * cr * D, b1, &fullb[slot], pol);
            ++cnt;
            __threadfence_block();
            s_issued = cnt;
          }
        }
      }
      __threadfence_block();
      s_pdone = pp + 1;
      if (*((volatile int*)status) == SLS_ERR_TIMEOUT) break;
    }
    // every copy issued has landed before the CTA may exit
    for (unsigned c = (cnt > (unsigned)S ? cnt - S : 0); c < cnt; ++c)
      mbar_wait(&fullb[c % S], (c / S) & 1u);
    return;
  }

  // ========================= compute warps ===================================
  unsigned lgen = 0;
  RingCursor rc{0u, 0, 0u};  // chunks consumed
  int pp = 0;
  for (int p = gi; p < nprob; p += ngroups, ++pp) {
    if (tid == 0) {
      s_halt = 0;
      __threadfence_block();
      s_go = pp + 1;
    }
    const int64_t row0 = bt.row0 ? bt.row0[p] : 0;
    const int64_t n = bt.n ? (int64_t)bt.n[p] : bt.n_single;
    const int64_t q1o = bt.q1off ? bt.q1off[p] : row0;
    const double* q1 = bt.q1 + q1o;
    const int64_t rs = (int64_t)rank * n / g, re = (int64_t)(rank + 1) * n / g;
    float2* Qs = bt.Q + (row0 + rs) * ldq;  // this CTA's rows of the basis
    const int nrows = (int)(re - rs);
    const int nch = (nrows + cr - 1) / cr;
    const int wr0 = warp * nrows / LZ_CW, wr1 = (warp + 1) * nrows / LZ_CW;
    double* alpha_out = bt.alpha + (size_t)p * r;
    double* beta_out = bt.beta + (size_t)p * r;
    const int cbeg = (int)((int64_t)rank * D / g), cend = (int)((int64_t)(rank + 1) * D / g);

    double scale = 0.0, alpha_prev = 0.0;
    float phimax = 0.f;  // max |Phi| over this CTA's strip (step 0, sweep A)
    dfloat alpha_df = df_make(0.f, 0.f), beta_df = df_make(0.f, 0.f), invb_df;
    int reff = 0;
    sbreak = 0;

    for (int j = 0; j < r; ++j) {
      // ---------------- row phase A and sweep A: z1, then Phi^T z1 -----------
      {
        dfloat c2acc[KT_MAX];
#pragma unroll
        for (int t = 0; t < KT_MAX; ++t) c2acc[t] = df_make(0.f, 0.f);
        dfloat nacc = df_make(0.f, 0.f);
        float zl1 = 0.f;
        if (j == 0) {
          for (int il = tid; il < nrows; il += LZ_CT) {
            const dfloat z = df_from_double(q1[rs + il]);
            us[il] = f2(z);
            dot2_acc_df(nacc.hi, nacc.lo, z, z);
          }
        } else {
          row_phase_A(Qs, ldq, wr0, wr1, j, cs, zps, us, nacc, zl1, c2acc);
        }
        zl1 = warp_sum_f(zl1);
        if (lane == 0) s_red1[warp] = zl1;
        named_sync(BAR_COMPUTE, LZ_CT);
        // offset for the column sums: all partial sums of Phi^T z1 over the
        // strip are bounded by max|Phi| * sum_i |z1_i|
        const bool ofsA = (P == 1) && (j > 0);
        float Ca = 0.f;
        if (ofsA) {
          float z1sum = 0.f;
#pragma unroll
          for (int w = 0; w < LZ_CW; ++w) z1sum += s_red1[w];
          Ca = ofs_pow2(phimax * z1sum);
        }

        f32x2_t ah[GPT][2], al[GPT][2];
        const f32x2_t a0 = pk2(Ca, Ca);
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          ah[q][0] = ah[q][1] = a0;
          al[q][0] = al[q][1] = 0ull;
        }
        float mx = 0.f;
        if (ofsA) {
          // two chunks per pass: more independent rows in flight per thread
          for (int t = 0; t < nch; t += 2) {
            const bool two = t + 1 < nch;
            const int s0 = rc.slot;
            if (!mbar_wait(&fullb[s0], rc.par)) atomicExch(status, SLS_ERR_TIMEOUT);
            rc_next(rc, S);
            int s1 = s0;
            if (two) {
              s1 = rc.slot;
              if (!mbar_wait(&fullb[s1], rc.par)) atomicExch(status, SLS_ERR_TIMEOUT);
              rc_next(rc, S);
            }
            const float* ch0 = reinterpret_cast<const float*>(ring + (size_t)s0 * stage);
            const float* ch1 = reinterpret_cast<const float*>(ring + (size_t)s1 * stage);
            const int nr0 = min(cr, nrows - t * cr);
            const int nr1 = two ? min(cr, nrows - (t + 1) * cr) : 0;
            if (fullD && nr0 == TCR && nr1 == TCR)
              sweepA_team_pair<GPT, TCR, true>(ch0, nr0, t * cr, ch1, nr1, (t + 1) * cr, C4, us, ah, al);
            else
              sweepA_team_pair<GPT, TCR, false>(ch0, nr0, t * cr, ch1, nr1, (t + 1) * cr, C4, us, ah, al);
            __syncwarp();
            if (lane == 0) {
              mbar_arrive(&emptyb[s0]);
              if (two) mbar_arrive(&emptyb[s1]);
            }
          }
        } else {
          for (int t = 0; t < nch; ++t) {
            const int slot = rc.slot;
            if (!mbar_wait(&fullb[slot], rc.par))
              atomicExch(status, SLS_ERR_TIMEOUT);  // leave at the next group barrier
            const float* chunk = reinterpret_cast<const float*>(ring + (size_t)slot * stage);
            const int nr = min(cr, nrows - t * cr);
            if (j == 0)
              sweepA_chunk<GPT, true>(chunk, nr, D, t * cr, us, ah, al, &mx);
            else
              sweepA_chunk<GPT, false>(chunk, nr, D, t * cr, us, ah, al, &mx);
            __syncwarp();
            if (lane == 0) mbar_arrive(&emptyb[slot]);
            rc_next(rc, S);
          }
        }
        if (j == 0) {
          for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
          named_sync(BAR_COMPUTE, LZ_CT);  // s_red1 (sum |z1|) has been read
          if (lane == 0) s_red1[warp] = mx;
        }
        // CTA partials: Phi^T z1, c2, |z1|^2
        const int ph = (P == 1) ? 0 : tid / C4;
        const int cb = (P == 1) ? tid : tid % C4;
        float2* dst = (P == 1) ? wpart + (size_t)rank * D : red + (size_t)ph * D;
        if (P == 1 || tid < P * C4) {
#pragma unroll
          for (int q = 0; q < GPT; ++q) {
            const int cg = cb + q * LZ_CT;
            if (cg < C4) {
              float h0, h1, l0, l1, h2, h3, l2, l3;
              upk2(ah[q][0], h0, h1);
              upk2(al[q][0], l0, l1);
              upk2(ah[q][1], h2, h3);
              upk2(al[q][1], l2, l3);
              dst[4 * cg + 0] = f2(df_norm(h0 - Ca, l0));
              dst[4 * cg + 1] = f2(df_norm(h1 - Ca, l1));
              dst[4 * cg + 2] = f2(df_norm(h2 - Ca, l2));
              dst[4 * cg + 3] = f2(df_norm(h3 - Ca, l3));
            }
          }
        }
        if (P > 1) {
          named_sync(BAR_COMPUTE, LZ_CT);
          for (int col = tid; col < D; col += LZ_CT) {
            dfloat s = df_make(0.f, 0.f);
            for (int q = 0; q < P; ++q) s = df_add(s, dfv(red[(size_t)q * D + col]));
            wpart[(size_t)rank * D + col] = f2(s);
          }
        }
        nacc = warp_sum_df(df_norm(nacc.hi, nacc.lo));
        if (lane == 0) tmpw[warp] = f2(nacc);
        store_coeff_partials(c2acc, j, r, cw, cpartA + (size_t)rank * (r + 1));
        if (tid == 0) {
          dfloat s = df_make(0.f, 0.f);
          for (int w = 0; w < LZ_CW; ++w) s = df_add(s, dfv(tmpw[w]));
          npart[rank] = f2(s);
        }
      }
      if (!group_sync_named(bar, lgen, status, &sflag, BAR_COMPUTE, LZ_CT)) return;

      // ---------------- slice phase: c2, Phi^T u_j for this CTA's columns --------
      reduce_coeffs(cpartA, g, r, j, c2s, red2);
      {
        dfloat sq = df_make(0.f, 0.f);
        for (int c = cbeg + warp; c < cend; c += LZ_CW) {
          dfloat s = df_make(0.f, 0.f);
          for (int b = lane; b < g; b += 32) s = df_add(s, dfv(wpart[(size_t)b * D + c]));
          s = warp_sum_df(s);
          // - sum_k c2_k w_k[c]
          dfloat cor = df_make(0.f, 0.f);
#pragma unroll
          for (int tt = 0; tt < KT_MAX; ++tt) {
            const int k = lane + 32 * tt;
            if (k < j) dot2_acc_df(cor.hi, cor.lo, dfv(Wm[(size_t)c * r + k]), dfv(c2s[k]));
          }
          cor = warp_sum_df(df_norm(cor.hi, cor.lo));
          s = df_sub(s, cor);
          if (lane == 0) {
            wred[c] = f2(s);
            dot2_acc_df(sq.hi, sq.lo, s, s);
          }
        }
        if (lane == 0) tmpw[warp] = f2(df_norm(sq.hi, sq.lo));
        named_sync(BAR_COMPUTE, LZ_CT);
        if (tid == 0) {
          dfloat s = df_make(0.f, 0.f);
          for (int w = 0; w < LZ_CW; ++w) s = df_add(s, dfv(tmpw[w]));
          sqpart[rank] = f2(s);
        }
      }
      if (!group_sync_named(bar, lgen, status, &sflag, BAR_COMPUTE, LZ_CT)) return;

      // ---------------- beta_{j-1}, alpha_j, break test -------------------------
      if (warp == 0) {
        dfloat s = df_make(0.f, 0.f), q = df_make(0.f, 0.f);
        for (int b = lane; b < g; b += 32) {
          s = df_add(s, dfv(npart[b]));
          q = df_add(q, dfv(sqpart[b]));
        }
        s = warp_sum_df(s);
        q = warp_sum_df(q);
        dfloat c2n = df_make(0.f, 0.f);
#pragma unroll
        for (int tt = 0; tt < KT_MAX; ++tt) {
          const int k = lane + 32 * tt;
          if (k < j) dot2_acc_df(c2n.hi, c2n.lo, dfv(c2s[k]), dfv(c2s[k]));
        }
        c2n = warp_sum_df(df_norm(c2n.hi, c2n.lo));
        if (lane == 0) {
          const double nrm2 = df_to_double(s) - df_to_double(c2n);  // |u_j|^2
          const double bnew = sqrt(fmax(nrm2, 0.0));
          int brk = 0;
          if (j > 0) {
            scale = fmax(scale, fabs(alpha_prev) + bnew);
            if (!(bnew > bt.tol * scale)) brk = 1;
            else if (rank == 0) beta_out[j - 1] = bnew;
          } else if (!(bnew > 0.0)) {
            brk = 1;
          }
          const double a = brk ? 0.0 : df_to_double(q) / (bnew * bnew);
          if (!brk && rank == 0) alpha_out[j] = a;
          shd[1] = brk ? 0.0 : 1.0 / bnew;
          shd[2] = a;
          shd[3] = (j > 0) ? bnew : 0.0;
          sbreak = brk;
          if (brk) s_halt = 1;
        }
      }
      named_sync(BAR_COMPUTE, LZ_CT);
      if (sbreak) {
        reff = j;
        break;
      }
      invb_df = df_from_double(shd[1]);
      alpha_prev = shd[2];
      alpha_df = df_from_double(shd[2]);
      beta_df = df_from_double(shd[3]);
      if (j == 0) {
#pragma unroll
        for (int w = 0; w < LZ_CW; ++w) phimax = fmaxf(phimax, s_red1[w]);
      }
      // w_j = (Phi^T u_j) / beta into shared memory; keep w_j (slice) for the
      // second Gram-Schmidt correction of later steps
      for (int c = tid; c < D; c += LZ_CT) {
        const dfloat a = df_mul(dfv(wred[c]), invb_df);
        wsh[c] = a.hi;
        wsl[c] = a.lo;
        if (c >= cbeg && c < cend) Wm[(size_t)c * r + j] = f2(a);
      }
      named_sync(BAR_COMPUTE, LZ_CT);

      // ---------------- sweep B (backward): s = Phi w_j per row -----------------
      if (P == 1) {
        f32x2_t wh[GPT][2], nwh[GPT][2], wl[GPT][2];
        float wt1 = 0.f;  // l1 norm of this thread's slice of w_j
        const float4* h4 = reinterpret_cast<const float4*>(wsh);
        const float4* l4 = reinterpret_cast<const float4*>(wsl);
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          const int cg = tid + q * LZ_CT;
          float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a;
          if (cg < C4) {
            a = h4[cg];
            b = l4[cg];
          }
          wh[q][0] = pk2(a.x, a.y);
          wh[q][1] = pk2(a.z, a.w);
          nwh[q][0] = pk2(-a.x, -a.y);
          nwh[q][1] = pk2(-a.z, -a.w);
          wl[q][0] = pk2(b.x, b.y);
          wl[q][1] = pk2(b.z, b.w);
          wt1 += (fabsf(a.x) + fabsf(a.y)) + (fabsf(a.z) + fabsf(a.w));
        }
        // offset of this thread's row partials: each is bounded by
        // max|Phi| * |w slice|_1
        const float Ct = ofs_pow2(phimax * wt1);
        constexpr int WCH = WB_ROWS / TCR;  // chunks per window (even)
        for (int t0p = 0; t0p < nch; t0p += 2) {
          const bool two = t0p + 1 < nch;
          const int kc0 = nch - 1 - t0p, kc1 = kc0 - 1;
          const int s0 = rc.slot;
          if (!mbar_wait(&fullb[s0], rc.par)) atomicExch(status, SLS_ERR_TIMEOUT);
          rc_next(rc, S);
          int s1 = s0;
          if (two) {
            s1 = rc.slot;
            if (!mbar_wait(&fullb[s1], rc.par)) atomicExch(status, SLS_ERR_TIMEOUT);
            rc_next(rc, S);
          }
          const float* ch0 = reinterpret_cast<const float*>(ring + (size_t)s0 * stage);
          const float* ch1 = reinterpret_cast<const float*>(ring + (size_t)s1 * stage);
          const int nr0 = min(cr, nrows - kc0 * cr);
          const int nr1 = two ? cr : 0;
          const int win = t0p / WCH, tw0 = t0p % WCH;
          float2* bp0 = bpart + (size_t)((win & 1) * WB_ROWS + tw0 * TCR) * LZ_CW;
          float2* bp1 = bp0 + (size_t)TCR * LZ_CW;
          if (fullD && nr0 == TCR && nr1 == TCR)
            sweepB_team_pair<GPT, TCR, true>(ch0, nr0, ch1, nr1, C4, wh, nwh, wl, Ct, bp0, bp1);
          else
            sweepB_team_pair<GPT, TCR, false>(ch0, nr0, ch1, nr1, C4, wh, nwh, wl, Ct, bp0, bp1);
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(&emptyb[s0]);
            if (two) mbar_arrive(&emptyb[s1]);
          }
          const int t = two ? t0p + 1 : t0p;  // last chunk of the pass
          const int tw = t % WCH;
          (void)kc1;
          if (tw == WCH - 1 || t == nch - 1) {
            // the window's warp partials are complete: one row per thread sums
            // them (the summing threads rotate from window to window)
            named_sync(BAR_COMPUTE, LZ_CT);
            const int t0 = t - tw;
            const int pidx = (tid - 64 * (win & 3) + LZ_CT) % LZ_CT;
            if (pidx < (tw + 1) * TCR) {
              const int il = (nch - 1 - (t0 + pidx / TCR)) * cr + pidx % TCR;
              if (il < nrows) {
                const float2* src = bpart + (size_t)((win & 1) * WB_ROWS + pidx) * LZ_CW;
                dfloat s = df_make(0.f, 0.f);
#pragma unroll
                for (int w = 0; w < LZ_CW; ++w) s = df_add(s, dfv(src[w]));
                zps[il] = f2(s);
              }
            }
          }
        }
      } else {
        for (int t = 0; t < nch; ++t) {
          const int kc = nch - 1 - t;
          const int slot = rc.slot;
          if (!mbar_wait(&fullb[slot], rc.par))
            atomicExch(status, SLS_ERR_TIMEOUT);  // leave at the next group barrier
          const float* chunk = reinterpret_cast<const float*>(ring + (size_t)slot * stage);
          const int nr = min(cr, nrows - kc * cr);
          for (int ii = warp; ii < nr; ii += LZ_CW) {
            const dfloat s = row_dot_smem(chunk + (size_t)ii * D, D, wsh, wsl);
            if (lane == 0) zps[kc * cr + ii] = f2(s);
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&emptyb[slot]);
          rc_next(rc, S);
        }
      }
      named_sync(BAR_COMPUTE, LZ_CT);

      // ---------------- row phase B: q_j, z', c ----------------------------------
      const bool last = (j == r - 1);
      dfloat cacc[KT_MAX];
#pragma unroll
      for (int t = 0; t < KT_MAX; ++t) cacc[t] = df_make(0.f, 0.f);
      row_phase_B(Qs, ldq, wr0, wr1, j, last, c2s, us, zps, invb_df, alpha_df, beta_df, cacc);
      if (last) {
        reff = r;
        break;
      }
      store_coeff_partials(cacc, j + 1, r, cw, cpartB + (size_t)rank * (r + 1));
      if (!group_sync_named(bar, lgen, status, &sflag, BAR_COMPUTE, LZ_CT)) return;
      reduce_coeffs(cpartB, g, r, j + 1, cs, red2);
    }
    // a break leaves chunks issued ahead of it: consume them until the copy
    // warp reports that it stopped
    if (sbreak) {
      for (unsigned it = 0; it < (1u << 26); ++it) {
        const unsigned iss = s_issued;
        if (rc.cnt < iss) {
          const int slot = rc.slot;
          if (!mbar_wait(&fullb[slot], rc.par)) {
            atomicExch(status, SLS_ERR_TIMEOUT);
            break;
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&emptyb[slot]);
          rc_next(rc, S);
        } else if (s_pdone == pp + 1) {
          if (s_issued == rc.cnt) break;
        } else {
          __nanosleep(64);
        }
      }
    }
    if (rank == 0 && tid == 0) {
      bt.r_eff[p] = reff;
      for (int k = reff; k < r; ++k) alpha_out[k] = 0.0;
      for (int k = (reff > 0 ? reff - 1 : 0); k < r; ++k) beta_out[k] = 0.0;
    }
    // problems on the same group run back to back; keep them apart
    if (!group_sync_named(bar, lgen, status, &sflag, BAR_COMPUTE, LZ_CT)) return;
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

template <int GPT>
int launch_lanczos_t(const LanczosBatch& bt, void* scratch, size_t gstride, int groups, int g,
                     int rows_cap, int stages, int* status, size_t smem, cudaStream_t stream) {
  auto fn = lanczos_kernel<GPT>;
  SLS_CUDA_TRY(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  char* sc = (char*)scratch;
  void* args[] = {(void*)&bt, (void*)&sc, (void*)&gstride, (void*)&g, (void*)&groups,
                  (void*)&rows_cap, (void*)&stages, (void*)&status};
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
  const int P = (C4 >= LZ_CT) ? 1 : (LZ_CT / C4);
  const int redn = (P > 1) ? P * bt.D : 0;
  const int rows_cap = (int)((bt.nmax + g - 1) / g) + 1;
  // shared memory besides the ring: w (hi, lo), phase partials, z1 and z' of
  // the strip, sweep-B warp partials, coefficient partials and vectors,
  // reduction scratch, barriers
  const size_t other = sizeof(float) * 2 * (size_t)bt.D +
                       sizeof(float2) * ((size_t)redn + 2 * (size_t)rows_cap +
                                         2 * WB_ROWS * LZ_CW +
                                         (size_t)(LZ_CW + 2) * (bt.r + 1) + 4 * LZ_CT) +
                       16 + 2 * RING_MAX_STAGES * 8;
  const size_t limit = 227 * 1024 - 1024;  // leave room for static shared memory
  if (other >= limit) return SLS_ERR_UNSUPPORTED;
  const RingShape R = ring_shape(bt.D, limit - other);
  if (R.S < 2) return SLS_ERR_UNSUPPORTED;
  const size_t smem = (size_t)R.S * R.stage + other;
  const int stages = R.S;
  switch (gpt_of(bt.D)) {
    case 1: return launch_lanczos_t<1>(bt, scratch, L.total, groups, g, rows_cap, stages, status, smem, stream);
    case 2: return launch_lanczos_t<2>(bt, scratch, L.total, groups, g, rows_cap, stages, status, smem, stream);
    case 4: return launch_lanczos_t<4>(bt, scratch, L.total, groups, g, rows_cap, stages, status, smem, stream);
    case 8: return launch_lanczos_t<8>(bt, scratch, L.total, groups, g, rows_cap, stages, status, smem, stream);
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
