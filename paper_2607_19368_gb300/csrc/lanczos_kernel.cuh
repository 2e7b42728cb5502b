// Implicit Lanczos (Algorithm 2): the persistent kernel.
//
// Lanczos runs as one persistent cooperative kernel.  The grid is split into
// groups of CTAs; a group owns one problem at a time (one prompt, or one
// adaptive window) and every CTA owns a contiguous strip of the problem's rows
// of the feature matrix Phi (N x D, float32) and of the basis Q.  One copy warp
// per CTA streams the strip through a shared-memory ring with one-dimensional
// bulk copies (cp.async.bulk + mbarrier): each stage holds a few rows of Phi
// and the same rows of Q.  Eight compute warps consume the ring.
//
// The whole run makes r passes over Phi: a prologue pass Phi^T q1, then one
// fused pass per step but the last.  Step j starts from z' (the new Lanczos
// direction before its re-orthogonalisation; z' = q1 for j = 0) and the CTA
// partials of Phi^T z', of c = Q^T z' (k < j) and of |z'|^2:
//
//   [barrier 1]
//   slice phase   c = sum of the CTA partials; each CTA finishes a slice of the
//                 D columns of Phi^T z1 = Phi^T z' - sum_k c_k w_k with
//                 z1 = z' - Q c and w_k = Phi^T q_k kept from earlier steps.
//   [barrier 2]
//                 beta_{j-1} = |z1| = sqrt(|z'|^2 - |c|^2), the break test,
//                 w_j = Phi^T q_j, alpha_j = |w_j|^2.
//   fused pass    per pair of ring chunks: z1 = z' - Q c and q_j = z1 / beta
//                 for its rows; the implicit matvec rows s = Phi w_j (Eq.
//                 implicit_matvec, all compute threads on each row, w_j in
//                 registers); the three-term recurrence z' = s - alpha_j q_j -
//                 beta_{j-1} q_{j-1} with its partials of c and |z'|^2; and
//                 the columns Phi^T z' of the next step, from the same rows
//                 while they are in shared memory.
//
// The last step only forms q_{r-1}.  This is Algorithm 2 with full
// re-orthogonalisation by one classical Gram-Schmidt pass per step, applied to
// Phi^T z' through the stored w_k so that one pass over Phi per step carries
// both halves of the matvec.  The projection c = Q^T z' of a fully
// re-orthogonalised Lanczos run stays at rounding level, so a second pass
// would change z1 only in the second order of the rounding unit.  Passes
// alternate direction so each starts on the rows the previous one left in
// L2.  Vectors are double-float (two float32), every sum over N or D is
// compensated, reductions have a fixed order (bit-reproducible runs).
// Barriers and waits poll without sleeping and give up after about a second
// of clock cycles, reporting SLS_ERR_TIMEOUT through the status word.
//
// The kernel is a template over GPT (float4 column groups of Phi per compute
// thread) and KT (32-wide tiles of the basis index k < r per lane); each
// lanczos_g<GPT>.cu instantiates one GPT for every KT.
#pragma once

#include <cfloat>

#include "common.cuh"
#include "kernels.cuh"

namespace sls {

namespace {

constexpr int LZ_CW = 8;                  // compute warps
constexpr int LZ_CT = LZ_CW * 32;         // compute threads
constexpr int LZ_THREADS = LZ_CT + 32;    // plus one copy warp
constexpr unsigned BAR_COMPUTE = 1;       // named barrier: the compute warps


// Per-group scratch layout (byte offsets), identical on host and device.
struct LzLayout {
  size_t bar, wpart, wred, Wm, cpart, npart, sqpart, total;
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
  L.cpart = o;  o += lz_al((size_t)g * (r + 1) * sizeof(float2));
  L.npart = o;  o += lz_al((size_t)2 * g * sizeof(float2));  // by step parity
  L.sqpart = o; o += lz_al((size_t)g * sizeof(float2));
  L.total = o;
  return L;
}


SLS_DEV dfloat shfl_df(dfloat v, int src) {
  v.hi = __shfl_sync(0xffffffffu, v.hi, src);
  v.lo = __shfl_sync(0xffffffffu, v.lo, src);
  return v;
}

// Ring stage: cr rows of Phi (cr * D elements of esz bytes: 4 for float32, 2
// for bfloat16) followed by the same cr rows of
// the basis Q (cr * ldq float2).  For D >= 4 * LZ_CT (one column group per
// compute thread or more) a stage holds team_rows(GPT) rows, so that the team
// row dots give every compute thread the same number of elements per chunk;
// smaller D takes as many rows as fit RING_STAGE bytes.
struct RingShape {
  int cr;          // rows per chunk
  int S;           // stages
  unsigned phib;   // bytes of Phi per full chunk
  unsigned stage;  // bytes per stage
};

constexpr int RING_STAGE = 32 * 1024;
constexpr int RING_MAX_STAGES = 8;
constexpr int SLICE_LOADS = 5;  // per-CTA values per lane in flight in warp sums (g <= 160)

// float4 column groups per compute thread, rounded up to a power of two
// (1, 2, 4 or 8; 0 when D is too wide)
__host__ __device__ inline int gpt_of(int D) {
  const int need = (D / 4 + LZ_CT - 1) / LZ_CT;
  return need <= 1 ? 1 : need <= 2 ? 2 : need <= 4 ? 4 : need <= 8 ? 8 : 0;
}
// rows per chunk of the team row dots: 8 / GPT (GPT * 4 * rows = 32 elements
// per thread per chunk)
__host__ __device__ constexpr int team_rows(int gpt) { return gpt >= 8 ? 1 : 8 / gpt; }

__host__ __device__ inline RingShape ring_shape(int D, int ldq, size_t budget, int esz) {
  RingShape R;
  if (D / 4 >= LZ_CT) {
    R.cr = team_rows(gpt_of(D));
  } else {
    R.cr = RING_STAGE / (esz * D + 8 * ldq);
    if (R.cr < 1) R.cr = 1;
  }
  R.phib = (unsigned)R.cr * (unsigned)D * (unsigned)esz;
  R.stage = R.phib + (unsigned)R.cr * (unsigned)ldq * 8u;
  R.S = (int)(budget / R.stage);
  if (R.S > RING_MAX_STAGES) R.S = RING_MAX_STAGES;
  return R;
}

// Sweep A over one chunk: acc[c] += Phi[i, c] * z1_i for the chunk's rows,
// column-parallel (GPT float4 groups per thread, P row phases), Dot2.  With
// TRACK the thread also keeps the largest |Phi| it has seen in *mx.
template <int GPT, bool TRACK, typename PT>
SLS_DEV void sweepA_chunk(const PT* __restrict__ chunk, int nr, int D, int lb,
                          const float2* __restrict__ us, f32x2_t (&ah)[GPT][2],
                          f32x2_t (&al)[GPT][2], float* mx) {
  const int tid = threadIdx.x;
  const int C4 = D >> 2;
  const int P = (C4 >= LZ_CT) ? 1 : (LZ_CT / C4);
  if (P > 1 && tid >= P * C4) return;
  const int ph = (P == 1) ? 0 : tid / C4;
  const int cb = (P == 1) ? tid : tid % C4;
  for (int i = ph; i < nr; i += P) {
    const float2 u = us[lb + i];
    const f32x2_t uh = pk2(u.x, u.x), nuh = pk2(-u.x, -u.x), ul = pk2(u.y, u.y);
#pragma unroll
    for (int q = 0; q < GPT; ++q) {
      const int cg = cb + q * LZ_CT;
      if (cg < C4) {
        const float4 f = phi_ld4(chunk, (size_t)i * C4 + cg);
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

// Column pass over two ring chunks at once (D >= 4 * LZ_CT; CR rows each, the
// second chunk may be absent: nr1 = 0): acc[c] += Phi[i, c] * z'_i.  The
// pair's rows are summed against a power-of-two offset C above twice max|Phi|
// times the l1 norm of their z' (offset accumulation, 5 operations per pair of
// elements), then (s - C) + lo, exact in its high part, joins the column sums
// (ah, al) by one TwoSum.  FULL: both chunks full and D = 4 LZ_CT GPT (the
// steady state), so the row and column guards vanish.
template <int GPT, int CR, bool FULL, typename PT>
SLS_DEV void sweepA_team_pair(const PT* __restrict__ c0, int nr0, int lb0,
                              const PT* __restrict__ c1, int nr1, int lb1, int C4,
                              const float2* __restrict__ us, float phimax,
                              f32x2_t (&ah)[GPT][2], f32x2_t (&al)[GPT][2]) {
  const int tid = threadIdx.x;
  float ut1 = 0.f;
#pragma unroll
  for (int i = 0; i < 2 * CR; ++i) {
    const bool first = i < CR;
    const int ii = first ? i : i - CR;
    if (FULL || ii < (first ? nr0 : nr1)) ut1 += fabsf(us[(first ? lb0 : lb1) + ii].x);
  }
  const float C = ofs_pow2(phimax * ut1);
  const f32x2_t Cp = pk2(C, C);
  f32x2_t s[GPT][2], lo[GPT][2];
#pragma unroll
  for (int q = 0; q < GPT; ++q) {
    s[q][0] = s[q][1] = Cp;
    lo[q][0] = lo[q][1] = 0ull;
  }
#pragma unroll
  for (int i = 0; i < 2 * CR; ++i) {
    const bool first = i < CR;
    const int ii = first ? i : i - CR;
    if (FULL || ii < (first ? nr0 : nr1)) {
      const PT* ch = first ? c0 : c1;
      const float2 u = us[(first ? lb0 : lb1) + ii];
      const f32x2_t uh = pk2(u.x, u.x), ul = pk2(u.y, u.y);
#pragma unroll
      for (int q = 0; q < GPT; ++q) {
        const int cg = tid + q * LZ_CT;
        if (FULL || cg < C4) {
          const float4 f = phi_ld4(ch, (size_t)ii * C4 + cg);
          ofs_fma_acc2(s[q][0], lo[q][0], pk2(f.x, f.y), uh, ul);
          ofs_fma_acc2(s[q][1], lo[q][1], pk2(f.z, f.w), uh, ul);
        }
      }
    }
  }
#pragma unroll
  for (int q = 0; q < GPT; ++q) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const f32x2_t x = sub2(s[q][h], Cp);  // exact (Sterbenz)
      const f32x2_t t = add2(ah[q][h], x);
      const f32x2_t bb = sub2(t, ah[q][h]);
      const f32x2_t e = add2(sub2(ah[q][h], sub2(t, bb)), sub2(x, bb));  // TwoSum error
      ah[q][h] = t;
      al[q][h] = add2(al[q][h], add2(e, lo[q][h]));
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

// Sweep B over two ring chunks at once with all compute threads (D >= 4 *
// LZ_CT): thread t owns the float4 column groups t + LZ_CT q of every row, w
// for those columns sits in registers.  Every thread of a warp accumulates
// its part of a row against the warp's offset Ct, a power of two above twice
// max|Phi| times the l1 norm of the warp's slice of w: each partial s - Ct is
// then exact, a multiple of ulp(Ct) / 2 below Ct / 2 in magnitude, and so is
// every sum of them over the warp, which makes the high parts of the
// transposed butterfly exact additions.  The rounding errors of the
// accumulation (each formed by an FMA at the scale of the low part) travel in
// the low parts; each warp sum is renormalised once by TwoSum and stored to bp0 / bp1
// [i * LZ_CW + warp].
template <int GPT, int CR, bool FULL, typename PT>
SLS_DEV void sweepB_team_pair(const PT* __restrict__ c0, int nr0, const PT* __restrict__ c1,
                              int nr1, int C4, const f32x2_t (&wh)[GPT][2],
                              const f32x2_t (&wl)[GPT][2], float Ct, float2* __restrict__ bp0, float2* __restrict__ bp1) {
  constexpr int R2 = 2 * CR;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float vh[R2], vl[R2];
#pragma unroll
  for (int i = 0; i < R2; ++i) {
    const bool first = i < CR;
    const int ii = first ? i : i - CR;
    f32x2_t s = pk2(Ct, Ct), lo = 0ull;
    if (FULL || ii < (first ? nr0 : nr1)) {
      const PT* ch = first ? c0 : c1;
#pragma unroll
      for (int q = 0; q < GPT; ++q) {
        const int cg = tid + q * LZ_CT;
        if (FULL || cg < C4) {
          const float4 f = phi_ld4(ch, (size_t)ii * C4 + cg);
          ofs_fma_acc2(s, lo, pk2(f.x, f.y), wh[q][0], wl[q][0]);
          ofs_fma_acc2(s, lo, pk2(f.z, f.w), wh[q][1], wl[q][1]);
        }
      }
    }
    float sx, sy, lx, ly;
    upk2(s, sx, sy);
    upk2(lo, lx, ly);
    vh[i] = (sx - Ct) + (sy - Ct);  // exact (one grid, below Ct / 2)
    vl[i] = lx + ly;
  }
  // the high parts add exactly; the low parts are orders of magnitude smaller
  const float th = transpose_sum_f<R2>(vh);
  const float tl = transpose_sum_f<R2>(vl);
  float rh, rl;
  two_sum(th, tl, rh, rl);
  const dfloat r = df_make(rh, rl);
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
template <typename PT>
SLS_DEV dfloat row_dot_smem(const PT* __restrict__ row, int D, const float* __restrict__ wsh,
                            const float* __restrict__ wsl) {
  const int lane = threadIdx.x & 31;
  const int C4 = D >> 2;
  const float4* h4 = reinterpret_cast<const float4*>(wsh);
  const float4* l4 = reinterpret_cast<const float4*>(wsl);
  f32x2_t h01 = 0, l01 = 0, h23 = 0, l23 = 0;
  for (int cg = lane; cg < C4; cg += 32) {
    const float4 f = phi_ld4(row, cg);
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

// A wait of this CTA gave up: report it and leave at the next group barrier.
SLS_DEV void lz_fail(int* status, volatile int* err) {
  atomicExch(status, SLS_ERR_TIMEOUT);
  *err = 1;
}

SLS_DEV int nprob_of(const LanczosBatch& bt) {
  int nprob = bt.nprob_max;
  if (bt.nprob_dev) nprob = min(nprob, *bt.nprob_dev);
  return nprob;
}

// Column sums over the CTAs of a group, eight items per warp: lane (bq, xx)
// = (lane >> 3, lane & 7) loads base[b * stride + x] for b = bq, bq + 4, ...
// (all loads of a batch in flight, 64 contiguous bytes per b), adds them as
// a pairwise tree and the four b-groups by two butterfly steps; every lane
// with lane & 7 == xx returns the sum for its item x.  One batch covers the
// partials of up to 160 CTAs, so a group's sums take one round of loads.
constexpr int CS_BATCH = 40;

__device__ __noinline__ dfloat warp_colsum8(const float2* __restrict__ base, size_t stride, int nb, int x,
                            bool valid) {
  const int lane = threadIdx.x & 31, bq = lane >> 3;
  dfloat acc = df_make(0.f, 0.f);
  for (int b0 = bq; b0 < nb; b0 += 4 * CS_BATCH) {
    dfloat v[CS_BATCH];
#pragma unroll
    for (int u = 0; u < CS_BATCH; ++u) {
      const int b = b0 + 4 * u;
      v[u] = (valid && b < nb) ? dfv(base[(size_t)b * stride + x]) : df_make(0.f, 0.f);
    }
#pragma unroll
    for (int w = 1; w < CS_BATCH; w *= 2) {
#pragma unroll
      for (int i = 0; i + w < CS_BATCH; i += 2 * w) v[i] = df_add_fast(v[i], v[i + w]);
    }
    acc = df_add_fast(acc, v[0]);
  }
  acc = df_add_fast(acc, shfl_xor_df(acc, 8));
  acc = df_add_fast(acc, shfl_xor_df(acc, 16));
  return acc;
}

// Sum of the per-CTA partial coefficients part[b * (r+1) + k] over the g CTAs
// of a group, for k < K, into cs[k].  Every CTA does it redundantly, warp w
// the coefficients 8 w .. 8 w + 7 (+ 8 LZ_CW m).
__device__ __noinline__ void reduce_coeffs(const float2* __restrict__ part, int g, int r, int K,
                           float2* __restrict__ cs) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int k0 = warp * 8; k0 < K; k0 += LZ_CW * 8) {
    const int k = k0 + (lane & 7);
    const dfloat v = warp_colsum8(part, (size_t)(r + 1), g, k, k < K);
    if (lane < 8 && k < K) cs[k] = f2(v);
  }
  named_sync(BAR_COMPUTE, LZ_CT);
}

// sum_{k < j} Wm[k * D + c] * c_k for the warp's eight columns, with the same
// lane layout as warp_colsum8 (lanes k-group bq = lane >> 3, Dot2).
__device__ __noinline__ dfloat warp_wcorr8(const float2* __restrict__ Wm, int D, int j, int c,
                                           bool valid, const float2* __restrict__ cs) {
  const int lane = threadIdx.x & 31, bq = lane >> 3;
  float sh = 0.f, sl = 0.f;
  for (int k0 = bq; k0 < j; k0 += 4 * 16) {
    float2 wv[16];
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      const int k = k0 + 4 * u;
      wv[u] = (valid && k < j) ? Wm[(size_t)k * D + c] : make_float2(0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      const int k = k0 + 4 * u;
      if (k < j) dot2_acc_df(sh, sl, dfv(wv[u]), dfv(cs[k]));
    }
  }
  dfloat acc = df_norm(sh, sl);
  acc = df_add_fast(acc, shfl_xor_df(acc, 8));
  acc = df_add_fast(acc, shfl_xor_df(acc, 16));
  return acc;
}

// Sums of a[0 .. n) and b[0 .. n) over the warp, both batches of loads in
// flight together; every lane gets both.
__device__ __noinline__ void warp_sum_vec2(const float2* __restrict__ a,
                                           const float2* __restrict__ b, int n, float2* out) {
  const int lane = threadIdx.x & 31;
  dfloat x[SLICE_LOADS], y[SLICE_LOADS];
#pragma unroll
  for (int m = 0; m < SLICE_LOADS; ++m) {
    const int i = lane + 32 * m;
    x[m] = (i < n) ? dfv(a[i]) : df_make(0.f, 0.f);
    y[m] = (i < n) ? dfv(b[i]) : df_make(0.f, 0.f);
  }
  dfloat s = x[0], t = y[0];
#pragma unroll
  for (int m = 1; m < SLICE_LOADS; ++m) {
    s = df_add_fast(s, x[m]);
    t = df_add_fast(t, y[m]);
  }
  for (int i = lane + 32 * SLICE_LOADS; i < n; i += 32) {
    s = df_add_fast(s, dfv(a[i]));
    t = df_add_fast(t, dfv(b[i]));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    s = df_add_fast(s, shfl_xor_df(s, o));
    t = df_add_fast(t, shfl_xor_df(t, o));
  }
  out[0] = f2(s);
  out[1] = f2(t);
}

// Per-warp partial coefficients (lanes over k < K) -> the CTA's partial row.
template <int KT>
SLS_DEV void store_coeff_partials(dfloat (&cacc)[KT], int K, int r, float2* __restrict__ cw,
                                  float2* __restrict__ dst) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
#pragma unroll
  for (int t = 0; t < KT; ++t) {
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

// Basis rows per register group in the row phases: RG * KT = 32 basis
// elements per lane in registers.
template <int KT>
struct RowGroup {
  static constexpr int RG = 32 / KT;                       // rows per group
  static constexpr int SH = (KT == 1) ? 0 : (KT == 2) ? 1 : 2;  // lane >> SH owns a row
};

// Basis rows 0 .. RG-1 of Qb (those < ng) at the columns k = lane + 32 kt < K,
// zero elsewhere; all loads of a group are in flight together.
template <int KT, int RG>
SLS_DEV void load_qgroup(const float2* __restrict__ Qb, int ldq, int ng, int K,
                         float2 (&q)[RG][KT]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < RG; ++i) {
#pragma unroll
    for (int kt = 0; kt < KT; ++kt) {
      const int k = lane + 32 * kt;
      q[i][kt] = make_float2(0.f, 0.f);
      if (i < ng && k < K) q[i][kt] = Qb[(size_t)i * ldq + k];
    }
  }
}

// sum_k q[i][k] c_k for the RG rows of a group (float32: the coefficients are
// at rounding level); lane L gets row L >> (5 - log2 RG).
template <int KT, int RG>
SLS_DEV float group_correction(const float2 (&q)[RG][KT], const float2 (&cv)[KT]) {
  float v[RG];
#pragma unroll
  for (int i = 0; i < RG; ++i) {
    float s = 0.f;
#pragma unroll
    for (int kt = 0; kt < KT; ++kt)
      s = fmaf(q[i][kt].x, cv[kt].x, fmaf(q[i][kt].x, cv[kt].y, fmaf(q[i][kt].y, cv[kt].x, s)));
    v[i] = s;
  }
  return transpose_sum_f<RG>(v);
}

// sum_{k < K} qrow[k] * c[k] over the warp (lanes over k), float32: the
// coefficients are at rounding level; every lane gets the result.
template <int KT>
SLS_DEV float row_corr(const float2* __restrict__ qrow, const float2* __restrict__ c, int K) {
  const int lane = threadIdx.x & 31;
  float s = 0.f;
#pragma unroll
  for (int kt = 0; kt < KT; ++kt) {
    const int k = lane + 32 * kt;
    if (k < K) {
      const float2 q = qrow[k], cc = c[k];
      s = fmaf(q.x, cc.x, fmaf(q.x, cc.y, fmaf(q.y, cc.x, s)));
    }
  }
  return warp_sum_f(s);
}

// Block sum of a double-float per-thread partial into *dst (tmpw: LZ_CW
// shared scratch).
SLS_DEV void store_cta_sum(dfloat acc, float2* tmpw, float2* __restrict__ dst) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  acc = df_norm(acc.hi, acc.lo);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc = df_add_fast(acc, shfl_xor_df(acc, o));
  if (lane == 0) tmpw[warp] = f2(acc);
  named_sync(BAR_COMPUTE, LZ_CT);
  if (tid == 0) {
    dfloat t = df_make(0.f, 0.f);
    for (int w = 0; w < LZ_CW; ++w) t = df_add(t, dfv(tmpw[w]));
    *dst = f2(t);
  }
  named_sync(BAR_COMPUTE, LZ_CT);
}

// The CTA's column partials of Phi^T z' (accumulators of the column pass, with
// offset C, zero for Dot2) to dst[0 .. D): directly for P = 1, through the P
// row-phase sums in red otherwise.
template <int GPT>
SLS_DEV void store_col_partials(const f32x2_t (&ah)[GPT][2], const f32x2_t (&al)[GPT][2],
                                float C, int P, int C4, int D, float2* __restrict__ dst,
                                float2* __restrict__ red) {
  const int tid = threadIdx.x;
  const int ph = (P == 1) ? 0 : tid / C4;
  const int cb = (P == 1) ? tid : tid % C4;
  float2* d = (P == 1) ? dst : red + (size_t)ph * D;
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
        d[4 * cg + 0] = f2(df_norm(h0 - C, l0));
        d[4 * cg + 1] = f2(df_norm(h1 - C, l1));
        d[4 * cg + 2] = f2(df_norm(h2 - C, l2));
        d[4 * cg + 3] = f2(df_norm(h3 - C, l3));
      }
    }
  }
  if (P > 1) {
    named_sync(BAR_COMPUTE, LZ_CT);
    for (int col = tid; col < D; col += LZ_CT) {
      dfloat s = df_make(0.f, 0.f);
      for (int q = 0; q < P; ++q) s = df_add(s, dfv(red[(size_t)q * D + col]));
      dst[col] = f2(s);
    }
  }
}

// Row phase of step j for the warp's rows [wr0, wr1) of the strip, in groups
// of RG rows held in registers (lanes over the basis index k):
//   z1 = z' - Q c                    (the re-orthogonalisation, c = Q^T z'
//                                     from the previous step, float32: the
//                                     coefficients are at rounding level)
//   q_j = z1 / beta_{j-1},  Q[:, j] = q_j
//   z' <- s - alpha_j q_j - beta_{j-1} q_{j-1}   (s = Phi w_j from sweep B)
// and, unless this is the last step, the partials of the next step:
// c += Q^T z' over k <= j, |z'|^2, sum |z'|.
template <int KT>
SLS_DEV void row_phase(float2* __restrict__ Qs, int ldq, int wr0, int wr1, int j, bool last,
                       const float2* __restrict__ cs, const float2* __restrict__ sv,
                       float2* __restrict__ zps, dfloat invb, dfloat alpha, dfloat beta,
                       dfloat (&cacc)[KT], dfloat& nacc, float& zl1) {
  constexpr int RG = RowGroup<KT>::RG, SH = RowGroup<KT>::SH;
  const int lane = threadIdx.x & 31;
  float2 cv[KT];
#pragma unroll
  for (int kt = 0; kt < KT; ++kt) {
    const int k = lane + 32 * kt;
    cv[kt] = (k < j) ? cs[k] : make_float2(0.f, 0.f);
  }
  for (int b = wr0; b < wr1; b += RG) {
    const int ng = min(RG, wr1 - b);
    float2* Qb = Qs + (size_t)b * ldq;
    float2 q[RG][KT];
    load_qgroup<KT, RG>(Qb, ldq, ng, j, q);
    const int i = lane >> SH;
    float2 sin = make_float2(0.f, 0.f), zin = sin, qprev = sin;
    if (i < ng) {
      sin = sv[b + i];
      zin = zps[b + i];
      if (j > 0) qprev = Qb[(size_t)i * ldq + j - 1];
    }
    const float corr = group_correction<KT, RG>(q, cv);
    dfloat qj = df_make(0.f, 0.f), zp = df_make(0.f, 0.f);
    if (i < ng) {
      dfloat z1 = dfv(zin);
      if (j > 0) z1 = df_add(z1, df_make(-corr, 0.f));
      qj = df_mul(z1, invb);
      zp = df_sub(dfv(sin), df_mul(alpha, qj));
      if (j > 0) zp = df_sub(zp, df_mul(beta, dfv(qprev)));
      if ((lane & ((1 << SH) - 1)) == 0) {
        Qb[(size_t)i * ldq + j] = f2(qj);
        zps[b + i] = f2(zp);
        if (!last) {
          dot2_acc_df(nacc.hi, nacc.lo, zp, zp);
          zl1 += fabsf(zp.hi);
        }
      }
    }
    if (!last) {
#pragma unroll
      for (int ii = 0; ii < RG; ++ii) {
        const dfloat zb = shfl_df(zp, ii << SH);
        const dfloat qb = shfl_df(qj, ii << SH);
#pragma unroll
        for (int kt = 0; kt < KT; ++kt) {
          const int k = lane + 32 * kt;
          if (k <= j) {
            const dfloat qk = (k == j) ? qb : dfv(q[ii][kt]);
            dot2_acc_df(cacc[kt].hi, cacc[kt].lo, qk, zb);
          }
        }
      }
    }
  }
}

template <int GPT, int KT, typename PT>
__global__ void __launch_bounds__(LZ_THREADS, 1)
lanczos_kernel(LanczosBatch bt, char* scratch, size_t gstride, int g, int ngroups,
               int rows_cap, int ring_stages, int* status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ float2 tmpw[LZ_CW];
  __shared__ float s_red1[LZ_CW];  // per-warp max |Phi| (offset bounds)
  __shared__ double shd[4];
  __shared__ int sflag, sbreak;
  // copy warp <-> compute warps handshake (no named barrier involves the copy
  // warp, so an early exit of either side can never leave the other blocked in
  // bar.sync; every wait on these flags is bounded)
  __shared__ volatile int s_halt;        // compute -> copy: stop issuing this problem
  __shared__ volatile int s_go;          // compute -> copy: may start problem s_go - 1
  __shared__ volatile int s_pass;        // compute -> copy: passes completed (+ 256 per problem)
  __shared__ volatile int s_pdone;       // copy -> compute: finished problem s_pdone - 1
  __shared__ volatile unsigned s_issued;  // copy -> compute: chunks issued so far
  __shared__ volatile int s_err;          // a wait of this CTA gave up

  constexpr int TCR = team_rows(GPT);
  constexpr int RPW = (2 * TCR + LZ_CW - 1) / LZ_CW;  // rows of a chunk pair per warp
  const int D = bt.D, r = bt.r, ldq = q_ld(bt.r);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int gi = blockIdx.x / g, rank = blockIdx.x % g;
  const int C4 = D >> 2;
  const int P = (C4 >= LZ_CT) ? 1 : (LZ_CT / C4);
  const int redn = (P > 1) ? P * D : 0;
  const bool fullD = (C4 == GPT * LZ_CT);  // no ragged column groups

  const RingShape shp0 = ring_shape(D, ldq, 0, (int)sizeof(PT));
  const int S = ring_stages;
  const int cr = shp0.cr;
  const unsigned stage = shp0.stage, phib = shp0.phib;
  unsigned char* ring = smem_raw;
  unsigned char* after_ring = smem_raw + (size_t)S * stage;
  const int wn = (P > 1) ? D : 0;                      // w_j staged for row_dot_smem
  float* wsh = reinterpret_cast<float*>(after_ring);   // wn
  float* wsl = wsh + wn;                               // wn
  float2* red = reinterpret_cast<float2*>(wsl + wn);   // redn
  float2* zps = red + redn;                            // rows_cap (z' of the strip)
  float2* bpart = zps + rows_cap;                      // 16 x LZ_CW (row-dot warp sums)
  float2* cw = bpart + 16 * LZ_CW;                     // LZ_CW x (r+1)
  float2* cs = cw + (size_t)LZ_CW * (r + 1);           // r+1 (c = Q^T z')
  uint64_t* bars = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(cs + (r + 1)) + 15) & ~(uintptr_t)15);
  uint64_t* fullb = bars;
  uint64_t* emptyb = bars + S;

  const LzLayout L = lz_layout(bt.nmax, D, r, g);
  char* gb = scratch + (size_t)gi * gstride;
  unsigned* barw = reinterpret_cast<unsigned*>(gb + L.bar);
  float2* wpart = reinterpret_cast<float2*>(gb + L.wpart);
  float2* wred = reinterpret_cast<float2*>(gb + L.wred);
  float2* Wm = reinterpret_cast<float2*>(gb + L.Wm);
  float2* cpart = reinterpret_cast<float2*>(gb + L.cpart);
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
    s_pass = 0;
    s_pdone = 0;
    s_issued = 0;
    s_err = 0;
  }
  __syncthreads();

  const int nprob = nprob_of(bt);

  // ========================= copy warp ======================================
  // Streams r passes over the strip per problem (the prologue pass and one
  // fused pass per step but the last), alternating direction so that each
  // pass starts on the rows the previous one left in L2.  Each ring stage
  // holds rows of Phi and the same rows of the basis Q; a pass is fetched only
  // once the previous pass has written its column of Q.
  if (warp == LZ_CW) {
    if (lane != 0) return;
    // Phi and Q stream through L2 once per pass: evict-first (measured faster
    // than evict-normal, and no slower than keeping the rows the next pass
    // reads first with evict-last)
    const uint64_t pol = l2_policy_evict_first();
    unsigned cnt = 0;
    int pp = 0;
    for (int p = gi; p < nprob; p += ngroups, ++pp) {
      bool ok = false;
      const long long t0 = clock64();
      for (unsigned it = 0;; ++it) {
        if (s_go == pp + 1) {
          ok = true;
          break;
        }
        if ((it & 63) == 63 && clock64() - t0 > SLS_WAIT_CYCLES) break;
      }
      if (!ok) {
        lz_fail(status, &s_err);
        break;
      }
      const int64_t row0 = bt.row0 ? bt.row0[p] : 0;
      const int64_t n = bt.n ? (int64_t)bt.n[p] : bt.n_single;
      const int64_t rs = (int64_t)rank * n / g, re = (int64_t)(rank + 1) * n / g;
      const int nch = (int)((re - rs + cr - 1) / cr);
      const PT* Phi = reinterpret_cast<const PT*>(bt.Phi) + (row0 + rs) * D;
      const float2* Qs = bt.Q + (row0 + rs) * ldq;
      bool stop = false;
      for (int pass = 0; pass < r && !stop; ++pass) {
        if (pass > 0) {
          const int need = pp * 256 + pass;
          // poll without sleeping: the ring refill of the next pass starts
          // as soon as the compute warps open it
          bool open = false;
          const long long t0 = clock64();
          for (unsigned it = 0;; ++it) {
            if (s_halt) break;
            if (s_pass >= need) {
              open = true;
              break;
            }
            if ((it & 63) == 63 && clock64() - t0 > SLS_WAIT_CYCLES) break;
          }
          if (!open) {
            if (!s_halt) lz_fail(status, &s_err);
            break;
          }
        }
        for (int t = 0; t < nch; ++t) {
          if (s_halt) {
            stop = true;
            break;
          }
          const int k = (pass & 1) ? nch - 1 - t : t;
          const int slot = (int)(cnt % (unsigned)S);
          const unsigned par = (cnt / (unsigned)S) & 1u;
          if (!mbar_wait(&emptyb[slot], par ^ 1u)) {
            lz_fail(status, &s_err);
            stop = true;
            break;
          }
          const int64_t nr = min((int64_t)cr, (re - rs) - (int64_t)k * cr);
          const unsigned b1 = (unsigned)(nr * D * (int64_t)sizeof(PT));
          const unsigned b2 = (unsigned)(nr * ldq * 8);
          unsigned char* dst = ring + (size_t)slot * stage;
          mbar_expect_tx(&fullb[slot], b1 + b2);
          bulk_g2s(dst, Phi + (int64_t)k * cr * D, b1, &fullb[slot], pol);
          bulk_g2s(dst + phib, Qs + (int64_t)k * cr * ldq, b2, &fullb[slot], pol);
          ++cnt;
          __threadfence_block();
          s_issued = cnt;
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
    dfloat alpha_df = df_make(0.f, 0.f), beta_df = df_make(0.f, 0.f), invb_df;
    float phimax = 0.f;  // max |Phi| over this CTA's strip (prologue pass)
    int reff = 0;
    sbreak = 0;

    // ---------------- prologue: z' = q1, |z'|^2 and Phi^T z' (pass 0) ------------
    {
      dfloat nacc = df_make(0.f, 0.f);
      for (int il = tid; il < nrows; il += LZ_CT) {
        const dfloat z = df_from_double(q1[rs + il]);
        zps[il] = f2(z);
        dot2_acc_df(nacc.hi, nacc.lo, z, z);
      }
      store_cta_sum(nacc, tmpw, npart + (size_t)rank);
      f32x2_t ah[GPT][2], al[GPT][2];
#pragma unroll
      for (int q = 0; q < GPT; ++q) ah[q][0] = ah[q][1] = al[q][0] = al[q][1] = 0ull;
      float mx = 0.f;
      for (int t = 0; t < nch; ++t) {
        const int slot = rc.slot;
        if (!mbar_wait(&fullb[slot], rc.par)) lz_fail(status, &s_err);
        const PT* chunk = reinterpret_cast<const PT*>(ring + (size_t)slot * stage);
        const int nr = min(cr, nrows - t * cr);
        sweepA_chunk<GPT, true>(chunk, nr, D, t * cr, zps, ah, al, &mx);
        __syncwarp();
        if (lane == 0) mbar_arrive(&emptyb[slot]);
        rc_next(rc, S);
      }
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      if (lane == 0) s_red1[warp] = mx;
      store_col_partials<GPT>(ah, al, 0.f, P, C4, D, wpart + (size_t)rank * D, red);
      named_sync(BAR_COMPUTE, LZ_CT);
      if (tid == 0) {
        __threadfence_block();
        s_pass = pp * 256 + 1;
      }
    }

    if (bt.inject_fail && rank == 0 && tid == 0) lz_fail(status, &s_err);
    for (int j = 0; j < r; ++j) {
      if (!group_sync_named(bar, lgen, status, &sflag, &s_err, BAR_COMPUTE, LZ_CT)) return;

      // ---------------- slice phase: c, Phi^T z1 for this CTA's columns ----------
      // c = Q^T z' (k < j) from the partials of the previous pass;
      // Phi^T z1 = Phi^T z' - sum_k c_k w_k with w_k = Phi^T q_k kept in Wm.
      reduce_coeffs(cpart, g, r, j, cs);
      {
        dfloat sq = df_make(0.f, 0.f);
        for (int c0 = cbeg + warp * 8; c0 < cend; c0 += LZ_CW * 8) {
          const int c = c0 + (lane & 7);
          const bool valid = c < cend;
          dfloat s = warp_colsum8(wpart, (size_t)D, g, c, valid);
          if (j > 0) s = df_sub(s, warp_wcorr8(Wm, D, j, c, valid, cs));
          if (lane < 8 && valid) {
            wred[c] = f2(s);
            dot2_acc_df(sq.hi, sq.lo, s, s);
          }
        }
        sq = df_norm(sq.hi, sq.lo);
#pragma unroll
        for (int o = 4; o > 0; o >>= 1) sq = df_add_fast(sq, shfl_xor_df(sq, o));
        if (lane == 0) tmpw[warp] = f2(sq);
        named_sync(BAR_COMPUTE, LZ_CT);
        if (tid == 0) {
          dfloat s = df_make(0.f, 0.f);
          for (int w = 0; w < LZ_CW; ++w) s = df_add(s, dfv(tmpw[w]));
          sqpart[rank] = f2(s);
        }
      }
      if (!group_sync_named(bar, lgen, status, &sflag, &s_err, BAR_COMPUTE, LZ_CT)) return;

      // ---------------- beta_{j-1}, alpha_j, break test -------------------------
      if (warp == 0) {
        // |z1|^2 = |z'|^2 - |c|^2 (Q orthonormal), |Phi^T z1|^2
        float2 sq2[2];
        warp_sum_vec2(npart + (size_t)(j & 1) * g, sqpart, g, sq2);
        const dfloat s = dfv(sq2[0]), q = dfv(sq2[1]);
        dfloat cn = df_make(0.f, 0.f);
#pragma unroll
        for (int tt = 0; tt < KT; ++tt) {
          const int k = lane + 32 * tt;
          if (k < j) dot2_acc_df(cn.hi, cn.lo, dfv(cs[k]), dfv(cs[k]));
        }
        cn = df_norm(cn.hi, cn.lo);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) cn = df_add_fast(cn, shfl_xor_df(cn, o));
        if (lane == 0) {
          const double nrm2 = df_to_double(s) - df_to_double(cn);  // |z1|^2
          // one reciprocal square root instead of a square root and two
          // divides (float64 runs at a fraction of the float32 rate here)
          const double inv = (nrm2 > 0.0) ? rsqrt(nrm2) : 0.0;    // 1 / beta
          const double bnew = (nrm2 > 0.0) ? nrm2 * inv : 0.0;
          int brk = 0;
          if (j > 0) {
            scale = fmax(scale, fabs(alpha_prev) + bnew);
            if (!(bnew > bt.tol * scale)) brk = 1;
            else if (rank == 0) beta_out[j - 1] = bnew;
          } else if (!(bnew > 0.0)) {
            brk = 1;
          }
          const double a = brk ? 0.0 : (df_to_double(q) * inv) * inv;
          if (!brk && rank == 0) alpha_out[j] = a;
          shd[1] = brk ? 0.0 : inv;
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

      if (j == r - 1) {
        // the last step needs no pass over Phi: q_{r-1} = z1 / beta_{r-2}
        dfloat cacc[KT];
#pragma unroll
        for (int t = 0; t < KT; ++t) cacc[t] = df_make(0.f, 0.f);
        dfloat nacc = df_make(0.f, 0.f);
        float zl1 = 0.f;
        row_phase<KT>(Qs, ldq, wr0, wr1, j, true, cs, zps, zps, invb_df, alpha_df, beta_df, cacc,
                      nacc, zl1);
        reff = r;
        break;
      }

      // w_j = (Phi^T z1) / beta: into shared memory for the row-per-warp row
      // dots (D < 4 LZ_CT; the team row dots take their columns straight into
      // registers below); keep w_j (slice) for the correction of later steps
      if (P > 1) {
        for (int c0 = tid; c0 < D; c0 += 8 * LZ_CT) {
          float2 wv[8];
#pragma unroll
          for (int m = 0; m < 8; ++m) {
            const int c = c0 + m * LZ_CT;
            wv[m] = (c < D) ? wred[c] : make_float2(0.f, 0.f);
          }
#pragma unroll
          for (int m = 0; m < 8; ++m) {
            const int c = c0 + m * LZ_CT;
            if (c < D) {
              const dfloat a = df_mul(dfv(wv[m]), invb_df);
              wsh[c] = a.hi;
              wsl[c] = a.lo;
              if (c >= cbeg && c < cend) Wm[(size_t)j * D + c] = f2(a);
            }
          }
        }
        named_sync(BAR_COMPUTE, LZ_CT);
      }

      // ---------------- fused pass j+1 over Phi ----------------------------------
      // per chunk (pair): z1 = z' - Q c, q_j = z1 / beta_{j-1} (row work);
      // s = Phi w_j (row dots); z' <- s - alpha_j q_j - beta_{j-1} q_{j-1} and
      // its partials of c = Q^T z' and |z'|^2 (row work); Phi^T z' (columns).
      const bool fwd = ((j + 1) & 1) == 0;
      f32x2_t ah[GPT][2], al[GPT][2];
#pragma unroll
      for (int q = 0; q < GPT; ++q) ah[q][0] = ah[q][1] = al[q][0] = al[q][1] = 0ull;
      dfloat cacc[KT];
#pragma unroll
      for (int t = 0; t < KT; ++t) cacc[t] = df_make(0.f, 0.f);
      dfloat nacc = df_make(0.f, 0.f);
      if (P == 1) {
        // this thread's columns of w_j, from the slices into registers
        f32x2_t wh[GPT][2], wl[GPT][2];
        float wt1 = 0.f;  // l1 norm of this thread's slice of w_j
        const float4* wr4 = reinterpret_cast<const float4*>(wred);
        float4 wv[GPT][2];
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          const int cg = tid + q * LZ_CT;
          wv[q][0] = wv[q][1] = make_float4(0.f, 0.f, 0.f, 0.f);
          if (cg < C4) {
            wv[q][0] = wr4[2 * cg];
            wv[q][1] = wr4[2 * cg + 1];
          }
        }
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          const int cg = tid + q * LZ_CT;
          float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a;
          if (cg < C4) {
            const dfloat w0 = df_mul(df_make(wv[q][0].x, wv[q][0].y), invb_df);
            const dfloat w1 = df_mul(df_make(wv[q][0].z, wv[q][0].w), invb_df);
            const dfloat w2 = df_mul(df_make(wv[q][1].x, wv[q][1].y), invb_df);
            const dfloat w3 = df_mul(df_make(wv[q][1].z, wv[q][1].w), invb_df);
            a = make_float4(w0.hi, w1.hi, w2.hi, w3.hi);
            b = make_float4(w0.lo, w1.lo, w2.lo, w3.lo);
            const int c = 4 * cg;
            if (c >= cbeg && c < cend) Wm[(size_t)j * D + c] = f2(w0);
            if (c + 1 >= cbeg && c + 1 < cend) Wm[(size_t)j * D + c + 1] = f2(w1);
            if (c + 2 >= cbeg && c + 2 < cend) Wm[(size_t)j * D + c + 2] = f2(w2);
            if (c + 3 >= cbeg && c + 3 < cend) Wm[(size_t)j * D + c + 3] = f2(w3);
          }
          wh[q][0] = pk2(a.x, a.y);
          wh[q][1] = pk2(a.z, a.w);
          wl[q][0] = pk2(b.x, b.y);
          wl[q][1] = pk2(b.z, b.w);
          wt1 += (fabsf(a.x) + fabsf(a.y)) + (fabsf(a.z) + fabsf(a.w));
        }
        // offset of the warp's row partials: every partial of a thread, and
        // their sum over the warp, is bounded by max|Phi| * |warp's w slice|_1
        float wtw = wt1;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) wtw += __shfl_xor_sync(0xffffffffu, wtw, o);
        const float Ct = ofs_pow2(phimax * wtw);
        for (int t0p = 0; t0p < nch; t0p += 2) {
          const bool two = t0p + 1 < nch;
          const int kc0 = fwd ? t0p : nch - 1 - t0p;
          const int kc1 = fwd ? t0p + 1 : nch - 2 - t0p;
          const int s0 = rc.slot;
          if (!mbar_wait(&fullb[s0], rc.par)) lz_fail(status, &s_err);
          rc_next(rc, S);
          int s1 = s0;
          if (two) {
            s1 = rc.slot;
            if (!mbar_wait(&fullb[s1], rc.par)) lz_fail(status, &s_err);
            rc_next(rc, S);
          }
          const PT* ch0 = reinterpret_cast<const PT*>(ring + (size_t)s0 * stage);
          const PT* ch1 = reinterpret_cast<const PT*>(ring + (size_t)s1 * stage);
          const float2* qb0 = reinterpret_cast<const float2*>(ring + (size_t)s0 * stage + phib);
          const float2* qb1 = reinterpret_cast<const float2*>(ring + (size_t)s1 * stage + phib);
          const int nr0 = min(cr, nrows - kc0 * cr);
          const int nr1 = two ? min(cr, nrows - kc1 * cr) : 0;
          // row work before the row dots: q_j of the warp's rows of the pair (it
          // feeds only the row work after them; with two or more column groups per
          // thread it runs after the row dots, measured faster there, with one
          // before them)
          dfloat qjv[RPW];
          float2 qpv[RPW];
          if constexpr (GPT == 1) {
#pragma unroll
            for (int m = 0; m < RPW; ++m) {
              const int ri = warp + m * LZ_CW;
              const bool first = ri < TCR;
              const int ii = first ? ri : ri - TCR;
              qjv[m] = df_make(0.f, 0.f);
              qpv[m] = make_float2(0.f, 0.f);
              if (ri < 2 * TCR && ii < (first ? nr0 : nr1)) {
                const int il = (first ? kc0 : kc1) * cr + ii;
                const float2* qrow = (first ? qb0 : qb1) + (size_t)ii * ldq;
                const float corr = row_corr<KT>(qrow, cs, j);
                dfloat z1 = dfv(zps[il]);
                if (j > 0) z1 = df_add(z1, df_make(-corr, 0.f));
                qjv[m] = df_mul(z1, invb_df);
                if (j > 0) qpv[m] = qrow[j - 1];
                if (lane == 0) Qs[(size_t)il * ldq + j] = f2(qjv[m]);
              }
            }
          }
          // row dots s = Phi w_j, warp sums into bpart[row * LZ_CW + warp]
          if (fullD && nr0 == TCR && nr1 == TCR)
            sweepB_team_pair<GPT, TCR, true>(ch0, nr0, ch1, nr1, C4, wh, wl, Ct, bpart,
                                             bpart + TCR * LZ_CW);
          else
            sweepB_team_pair<GPT, TCR, false>(ch0, nr0, ch1, nr1, C4, wh, wl, Ct, bpart,
                                              bpart + TCR * LZ_CW);
          if constexpr (GPT != 1) {
#pragma unroll
            for (int m = 0; m < RPW; ++m) {
              const int ri = warp + m * LZ_CW;
              const bool first = ri < TCR;
              const int ii = first ? ri : ri - TCR;
              qjv[m] = df_make(0.f, 0.f);
              qpv[m] = make_float2(0.f, 0.f);
              if (ri < 2 * TCR && ii < (first ? nr0 : nr1)) {
                const int il = (first ? kc0 : kc1) * cr + ii;
                const float2* qrow = (first ? qb0 : qb1) + (size_t)ii * ldq;
                const float corr = row_corr<KT>(qrow, cs, j);
                dfloat z1 = dfv(zps[il]);
                if (j > 0) z1 = df_add(z1, df_make(-corr, 0.f));
                qjv[m] = df_mul(z1, invb_df);
                if (j > 0) qpv[m] = qrow[j - 1];
                if (lane == 0) Qs[(size_t)il * ldq + j] = f2(qjv[m]);
              }
            }
          }
          named_sync(BAR_COMPUTE, LZ_CT);
          // row work after the row dots: z', its partials of c and |z'|^2
#pragma unroll
          for (int m = 0; m < RPW; ++m) {
            const int ri = warp + m * LZ_CW;
            const bool first = ri < TCR;
            const int ii = first ? ri : ri - TCR;
            if (ri < 2 * TCR && ii < (first ? nr0 : nr1)) {
              const int il = (first ? kc0 : kc1) * cr + ii;
              const float2* qrow = (first ? qb0 : qb1) + (size_t)ii * ldq;
              // the LZ_CW warp sums sit in lanes 0 .. LZ_CW - 1
              dfloat s = (lane < LZ_CW) ? dfv(bpart[ri * LZ_CW + lane]) : df_make(0.f, 0.f);
#pragma unroll
              for (int o = LZ_CW / 2; o > 0; o >>= 1) s = df_add_fast(s, shfl_xor_df(s, o));
              s = shfl_df(s, 0);
              dfloat zp = df_sub(s, df_mul(alpha_df, qjv[m]));
              if (j > 0) zp = df_sub(zp, df_mul(beta_df, dfv(qpv[m])));
              if (lane == 0) {
                zps[il] = f2(zp);
                dot2_acc_df(nacc.hi, nacc.lo, zp, zp);
              }
#pragma unroll
              for (int kt = 0; kt < KT; ++kt) {
                const int k = lane + 32 * kt;
                if (k <= j) {
                  const dfloat qk = (k == j) ? qjv[m] : dfv(qrow[k]);
                  dot2_acc_df(cacc[kt].hi, cacc[kt].lo, qk, zp);
                }
              }
            }
          }
          named_sync(BAR_COMPUTE, LZ_CT);
          // columns: Phi^T z' for the next step
          if (fullD && nr0 == TCR && nr1 == TCR)
            sweepA_team_pair<GPT, TCR, true>(ch0, nr0, kc0 * cr, ch1, nr1, kc1 * cr, C4, zps, phimax,
                                              ah, al);
          else
            sweepA_team_pair<GPT, TCR, false>(ch0, nr0, kc0 * cr, ch1, nr1, kc1 * cr, C4, zps, phimax,
                                               ah, al);
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(&emptyb[s0]);
            if (two) mbar_arrive(&emptyb[s1]);
          }
        }
      } else {
        float mx = 0.f;
        for (int t = 0; t < nch; ++t) {
          const int kc = fwd ? t : nch - 1 - t;
          const int slot = rc.slot;
          if (!mbar_wait(&fullb[slot], rc.par))
            lz_fail(status, &s_err);  // leave at the next group barrier
          const PT* chunk = reinterpret_cast<const PT*>(ring + (size_t)slot * stage);
          const float2* qblk = reinterpret_cast<const float2*>(ring + (size_t)slot * stage + phib);
          const int nr = min(cr, nrows - kc * cr);
          for (int ii = warp; ii < nr; ii += LZ_CW) {
            const int il = kc * cr + ii;
            const float2* qrow = qblk + (size_t)ii * ldq;
            const float corr = row_corr<KT>(qrow, cs, j);
            dfloat z1 = dfv(zps[il]);
            if (j > 0) z1 = df_add(z1, df_make(-corr, 0.f));
            const dfloat qj = df_mul(z1, invb_df);
            if (lane == 0) Qs[(size_t)il * ldq + j] = f2(qj);
            const dfloat s = row_dot_smem(chunk + (size_t)ii * D, D, wsh, wsl);
            dfloat zp = df_sub(s, df_mul(alpha_df, qj));
            if (j > 0) zp = df_sub(zp, df_mul(beta_df, dfv(qrow[j - 1])));
            if (lane == 0) {
              zps[il] = f2(zp);
              dot2_acc_df(nacc.hi, nacc.lo, zp, zp);
            }
#pragma unroll
            for (int kt = 0; kt < KT; ++kt) {
              const int k = lane + 32 * kt;
              if (k <= j) {
                const dfloat qk = (k == j) ? qj : dfv(qrow[k]);
                dot2_acc_df(cacc[kt].hi, cacc[kt].lo, qk, zp);
              }
            }
          }
          named_sync(BAR_COMPUTE, LZ_CT);
          sweepA_chunk<GPT, false>(chunk, nr, D, kc * cr, zps, ah, al, &mx);
          __syncwarp();
          if (lane == 0) mbar_arrive(&emptyb[slot]);
          rc_next(rc, S);
        }
      }
      // partials for step j+1 (read after its barrier 1): Phi^T z', c, |z'|^2
      store_col_partials<GPT>(ah, al, 0.f, P, C4, D, wpart + (size_t)rank * D, red);
      store_coeff_partials(cacc, j + 1, r, cw, cpart + (size_t)rank * (r + 1));
      store_cta_sum(nacc, tmpw, npart + (size_t)((j + 1) & 1) * g + rank);
      // the column j of Q written in this pass reaches the copy warp's bulk
      // reads of the next pass (async proxy)
      if (lane == 0) asm volatile("fence.proxy.async.global;" ::: "memory");
      named_sync(BAR_COMPUTE, LZ_CT);
      if (tid == 0) {
        __threadfence_block();
        s_pass = pp * 256 + j + 2;
      }
    }
    // a break leaves chunks issued ahead of it: consume them until the copy
    // warp reports that it stopped
    if (sbreak) {
      for (unsigned it = 0; it < (1u << 26); ++it) {
        const unsigned iss = s_issued;
        if (rc.cnt < iss) {
          const int slot = rc.slot;
          if (!mbar_wait(&fullb[slot], rc.par)) {
            lz_fail(status, &s_err);
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
    if (!group_sync_named(bar, lgen, status, &sflag, &s_err, BAR_COMPUTE, LZ_CT)) return;
  }
}

template <int GPT, int KT, typename PT>
int launch_lanczos_t(const LanczosBatch& bt, void* scratch, size_t gstride, int groups, int g,
                     int rows_cap, int stages, int* status, size_t smem, cudaStream_t stream) {
  auto fn = lanczos_kernel<GPT, KT, PT>;
  SLS_CUDA_TRY(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  char* sc = (char*)scratch;
  void* args[] = {(void*)&bt, (void*)&sc, (void*)&gstride, (void*)&g, (void*)&groups,
                  (void*)&rows_cap, (void*)&stages, (void*)&status};
  SLS_CUDA_TRY(cudaLaunchCooperativeKernel((const void*)fn, dim3(groups * g), dim3(LZ_THREADS),
                                           args, smem, stream));
  count_launch(1);
  return SLS_OK;
}

// KT = 1, 2 or 4 basis tiles for one GPT and element type
template <int GPT, typename PT>
int launch_lanczos_kt(const LanczosBatch& bt, void* scratch, size_t gstride, int groups, int g,
                      int rows_cap, int stages, int* status, size_t smem, cudaStream_t stream,
                      int kt) {
  switch (kt) {
    case 1:
      return launch_lanczos_t<GPT, 1, PT>(bt, scratch, gstride, groups, g, rows_cap, stages,
                                          status, smem, stream);
    case 2:
      return launch_lanczos_t<GPT, 2, PT>(bt, scratch, gstride, groups, g, rows_cap, stages,
                                          status, smem, stream);
    case 4:
      return launch_lanczos_t<GPT, 4, PT>(bt, scratch, gstride, groups, g, rows_cap, stages,
                                          status, smem, stream);
    default:
      return SLS_ERR_UNSUPPORTED;
  }
}

}  // namespace

// Launch the Lanczos kernel for GPT = 1, 2, 4 or 8 column groups per thread
// and KT = 1, 2 or 4 basis tiles, Phi in float32 (lanczos_g<GPT>.cu) or
// bfloat16 (lanczos_b<GPT>.cu).
#define SLS_LZ_LAUNCH_ARGS                                                                \
  const LanczosBatch &bt, void *scratch, size_t gstride, int groups, int g, int rows_cap, \
      int stages, int *status, size_t smem, cudaStream_t stream, int kt
int launch_lanczos_gpt1(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_gpt2(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_gpt4(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_gpt8(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_bf16_gpt1(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_bf16_gpt2(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_bf16_gpt4(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_bf16_gpt8(SLS_LZ_LAUNCH_ARGS);

}  // namespace sls
