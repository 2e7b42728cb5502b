// Implicit Lanczos (Algorithm 2): the persistent kernel.
//
// Lanczos runs as one persistent cooperative kernel.  The grid is split into
// groups of CTAs; a group owns one problem at a time (one prompt, or one
// adaptive window) and every CTA owns a contiguous strip of the problem's rows
// of the feature matrix Phi (N x D, float32) and of the basis Q.  The strip
// streams through a shared-memory ring with one-dimensional bulk copies
// (cp.async.bulk + mbarrier): each stage holds a few rows of Phi and the same
// rows of Q.  The warps of a CTA form teams of eight: with two teams, each
// takes every other pair of ring chunks, so that one team's latency-bound row
// work overlaps the other team's sweeps.  There is no copy warp: the first
// chunks of a pass are issued when the previous pass ends, and a team refills
// the slots of its previous pair as soon as its first barrier in the next
// pair shows that every warp of the team is done with them.
//
// The whole run makes r passes over Phi: a prologue pass Phi^T q1, then one
// fused pass per step but the last.  Step j starts from z' (the new Lanczos
// direction before its re-orthogonalisation; z' = q1 for j = 0), the CTA
// partials of Phi^T z' and the group sums of c = Q^T z' and of |z'|^2:
//
//   [barrier 1]
//   slice phase   c from the group sums; each CTA finishes a slice of the D
//                 columns of Phi^T z1 = Phi^T z' - sum_k c_k w_k with
//                 z1 = z' - Q c and w_k = Phi^T q_k kept from earlier steps.
//   [barrier 2]
//                 beta_{j-1} = |z1| = sqrt(|z'|^2 - |c|^2), the break test,
//                 w_j = Phi^T q_j, alpha_j = |w_j|^2.
//   fused pass    per pair of ring chunks: z1 = z' - Q c and q_j = z1 / beta
//                 for its rows; the implicit matvec rows s = Phi w_j (Eq.
//                 implicit_matvec, all threads of a team on each row, w_j in
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
// L2.  Vectors are double-float (two float32) and every sum over N or D is
// compensated.  The column sums of Phi^T z' are added over the CTAs in a fixed
// order; the group sums of the scalars (c, |z'|^2, |Phi^T z1|^2) are float64
// atomic additions, one per CTA, whose order may vary in the last float64 bit.
// Barriers and waits poll without sleeping and give up after about a second
// of clock cycles, reporting SLS_ERR_TIMEOUT through the status word.
//
// The kernel is a template over GPT (float4 column groups of Phi per compute
// thread), KT (32-wide tiles of the basis index k < r per lane), the element
// type of Phi and the number of compute teams; each lanczos_g<GPT>.cu /
// lanczos_b<GPT>.cu instantiates one GPT and element type.
#pragma once

#include <cfloat>

#include "common.cuh"
#include "kernels.cuh"

namespace sls {

namespace {

constexpr int LZ_CW = 8;                  // compute warps per team
constexpr int LZ_CT = LZ_CW * 32;         // compute threads per team
constexpr unsigned BAR_ALL = 1;           // named barrier: every compute warp
constexpr unsigned BAR_TEAM = 2;          // named barriers 2, 3: the warps of team 0, 1

// Teams of compute warps: two when each thread holds one float4 column group
// of a row (D = 4 LZ_CT = 1024), one otherwise.  Two teams give the scheduler
// another team's sweeps to issue while one team is in its latency-bound row
// work, at the price of chunk pairs half as long (more per-pair work per
// row); measured on both shapes (alternating builds on one GPU): at D = 1024
// two teams are faster (mistral7b 0.956 -> 0.858 ms, 76 adaptive windows
// 6.58 -> 5.97 ms), at D = 2048 one team (qwen7b 5.83 ms with two, 5.17 with
// one; the previous kernel with a copy warp 5.26).
__host__ __device__ constexpr int lz_teams(int gpt, int P) { return (P == 1 && gpt <= 1) ? 2 : 1; }
__host__ __device__ constexpr int lz_threads(int teams) { return teams * LZ_CT; }

// Per-group scratch layout (byte offsets), identical on host and device.
//   acc:   2 x (r + 4) float64 group sums by step parity: c_k (k <= r), |z'|^2
//          at r + 1, |Phi^T z1|^2 at r + 2 (float64 atomic additions)
//   wpart: g x D double-float CTA partials of Phi^T z'
//   wred:  D double-float: Phi^T z1, finished slice by slice
//   Wm:    r x D double-float: w_k = Phi^T q_k (each CTA writes its slice)
struct LzLayout {
  size_t bar, acc, zero_end, wpart, wred, Wm, total;
};

__host__ __device__ inline size_t lz_al(size_t x) { return (x + 255) & ~(size_t)255; }
__host__ __device__ inline int lz_acc_stride(int r) { return r + 4; }

__host__ __device__ inline LzLayout lz_layout(int64_t nmax, int D, int r, int g) {
  (void)nmax;
  LzLayout L;
  size_t o = 0;
  L.bar = o;    o += 256;
  L.acc = o;    o += lz_al((size_t)2 * lz_acc_stride(r) * sizeof(double));
  L.zero_end = o;  // [bar, zero_end) starts at zero before the launch
  L.wpart = o;  o += lz_al((size_t)g * D * sizeof(float2));
  L.wred = o;   o += lz_al((size_t)D * sizeof(float2));
  L.Wm = o;     o += lz_al((size_t)D * r * sizeof(float2));
  L.total = o;
  return L;
}

SLS_DEV dfloat shfl_df(dfloat v, int src) {
  v.hi = __shfl_sync(0xffffffffu, v.hi, src);
  v.lo = __shfl_sync(0xffffffffu, v.lo, src);
  return v;
}

SLS_DEV dfloat shfl_xor_df(dfloat v, int m) {
  v.hi = __shfl_xor_sync(0xffffffffu, v.hi, m);
  v.lo = __shfl_xor_sync(0xffffffffu, v.lo, m);
  return v;
}

// float64 atomic addition whose result is not used (a reduction operation)
SLS_DEV void red_add_f64(double* p, double v) { atomicAdd(p, v); }

// Ring stage: cr rows of Phi (cr * D elements of esz bytes: 4 for float32, 2
// for bfloat16) followed by the same cr rows of the basis Q (cr * ldq float2).
// For D >= 4 * LZ_CT (one column group per compute thread or more) a stage
// holds chunk_rows(GPT, teams) rows, so that the team row dots give every
// thread the same number of elements per chunk; smaller D takes as many rows
// as fit RING_STAGE bytes.
struct RingShape {
  int cr;          // rows per chunk
  int S;           // stages
  unsigned phib;   // bytes of Phi per full chunk
  unsigned stage;  // bytes per stage
};

constexpr int RING_STAGE = 32 * 1024;
constexpr int RING_MAX_STAGES = 16;

// float4 column groups per compute thread, rounded up to a power of two
// (1, 2, 4 or 8; 0 when D is too wide)
__host__ __device__ inline int gpt_of(int D) {
  const int need = (D / 4 + LZ_CT - 1) / LZ_CT;
  return need <= 1 ? 1 : need <= 2 ? 2 : need <= 4 ? 4 : need <= 8 ? 8 : 0;
}
// rows per ring chunk of the team row dots: GPT * 4 * rows = 32 elements per
// thread per chunk with one team, 16 with two (smaller stages keep the ring
// deep while two teams each hold a chunk pair)
__host__ __device__ constexpr int chunk_rows(int gpt, int teams) {
  return (teams == 2 ? 4 : 8) / gpt >= 1 ? (teams == 2 ? 4 : 8) / gpt : 1;
}

__host__ __device__ inline RingShape ring_shape(int D, int ldq, size_t budget, int esz,
                                                int teams) {
  RingShape R;
  if (D / 4 >= LZ_CT) {
    R.cr = chunk_rows(gpt_of(D), teams);
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

// Shared memory besides the ring (bytes), in the order the kernel carves it:
// w_j (hi, lo; only for D < 4 LZ_CT), the P row-phase partials, z' of the
// strip (rows_cap even), the row-dot warp sums of each team, c, then the
// mbarriers of the ring's stages (16-byte aligned).
__host__ __device__ inline size_t lz_smem_other(int D, int r, int rows_cap, int teams,
                                                int stages) {
  const int C4 = D / 4;
  const int P = (C4 >= LZ_CT) ? 1 : (LZ_CT / C4);
  const size_t wn = (P > 1) ? (size_t)D : 0;
  const size_t redn = (P > 1) ? (size_t)P * D : 0;
  size_t b = sizeof(float) * 2 * wn;
  b += sizeof(float2) * (redn + (size_t)rows_cap + (size_t)teams * 16 * LZ_CW + (size_t)(r + 1));
  b = (b + 15) & ~(size_t)15;
  b += (size_t)stages * 8;
  return b;
}

// Bytes of the ring the pass ends borrow: team 1's column sums (two teams)
// and the per-warp coefficient partials.
__host__ __device__ inline size_t lz_pass_end_bytes(int gpt, int r, int teams) {
  return sizeof(float2) * ((teams > 1 ? (size_t)4 * gpt * LZ_CT : 0) +
                           (size_t)teams * LZ_CW * (r + 1));
}

// Sweep A over one chunk: acc[c] += Phi[i, c] * z1_i for the chunk's rows,
// column-parallel (GPT float4 groups per thread, P row phases), Dot2.  With
// TRACK the thread also keeps the largest |Phi| it has seen in *mx.  tt: the
// thread's index in its team.
template <int GPT, bool TRACK, typename PT>
SLS_DEV void sweepA_chunk(const PT* __restrict__ chunk, int nr, int D, int lb, int tt,
                          const float2* __restrict__ us, f32x2_t (&ah)[GPT][2],
                          f32x2_t (&al)[GPT][2], float* mx) {
  const int C4 = D >> 2;
  const int P = (C4 >= LZ_CT) ? 1 : (LZ_CT / C4);
  if (P > 1 && tt >= P * C4) return;
  const int ph = (P == 1) ? 0 : tt / C4;
  const int cb = (P == 1) ? tt : tt % C4;
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
                              const PT* __restrict__ c1, int nr1, int lb1, int C4, int tt,
                              const float2* __restrict__ us, float phimax,
                              f32x2_t (&ah)[GPT][2], f32x2_t (&al)[GPT][2]) {
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
  if constexpr (GPT == 1) {
    // packed pairs
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
          const int cg = tt + q * LZ_CT;
          if (FULL || cg < C4) {
            const float4 f = phi_ld4(ch, (size_t)ii * C4 + cg);
            ofs_fma_acc2(s[q][0], lo[q][0], pk2(f.x, f.y), uh, ul);
            ofs_fma_acc2(s[q][1], lo[q][1], pk2(f.z, f.w), uh, ul);
          }
        }
      }
    }
  } else {
    // scalar steps for two or more column groups per thread: measured faster
    // there (qwen7b shape, alternating builds), and the instruction counters
    // show the packed form executing about 1.3 register moves per step, so
    // it saves fewer issue slots than its halved arithmetic count suggests
    float sc[GPT][4], lc[GPT][4];
#pragma unroll
    for (int q = 0; q < GPT; ++q)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        sc[q][e] = C;
        lc[q][e] = 0.f;
      }
#pragma unroll
    for (int i = 0; i < 2 * CR; ++i) {
      const bool first = i < CR;
      const int ii = first ? i : i - CR;
      if (FULL || ii < (first ? nr0 : nr1)) {
        const PT* ch = first ? c0 : c1;
        const float2 u = us[(first ? lb0 : lb1) + ii];
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          const int cg = tt + q * LZ_CT;
          if (FULL || cg < C4) {
            const float4 f = phi_ld4(ch, (size_t)ii * C4 + cg);
            ofs_fma_acc(sc[q][0], lc[q][0], f.x, u.x, u.y);
            ofs_fma_acc(sc[q][1], lc[q][1], f.y, u.x, u.y);
            ofs_fma_acc(sc[q][2], lc[q][2], f.z, u.x, u.y);
            ofs_fma_acc(sc[q][3], lc[q][3], f.w, u.x, u.y);
          }
        }
      }
    }
#pragma unroll
    for (int q = 0; q < GPT; ++q) {
      s[q][0] = pk2(sc[q][0], sc[q][1]);
      s[q][1] = pk2(sc[q][2], sc[q][3]);
      lo[q][0] = pk2(lc[q][0], lc[q][1]);
      lo[q][1] = pk2(lc[q][2], lc[q][3]);
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

// Sweep B over two ring chunks at once with the threads of one team (D >= 4 *
// LZ_CT): thread tt owns the float4 column groups tt + LZ_CT q of every row,
// w for those columns sits in registers.  Every thread of a warp accumulates
// its part of a row against the warp's offset Ct, a power of two above twice
// max|Phi| times the l1 norm of the warp's slice of w: each partial s - Ct is
// then exact, a multiple of ulp(Ct) / 2 below Ct / 2 in magnitude, and so is
// every sum of them over the warp, which makes the high parts of the
// transposed butterfly exact additions.  The rounding errors of the
// accumulation (each formed by an FMA at the scale of the low part) travel in
// the low parts; each warp sum is renormalised once by TwoSum and stored to
// bp0 / bp1 [i * LZ_CW + tw] (tw: the warp's index in its team).
template <int GPT, int CR, bool FULL, typename PT>
SLS_DEV void sweepB_team_pair(const PT* __restrict__ c0, int nr0, const PT* __restrict__ c1,
                              int nr1, int C4, int tt, const f32x2_t (&wh)[GPT][2],
                              const f32x2_t (&wl)[GPT][2], float Ct, float2* __restrict__ bp0,
                              float2* __restrict__ bp1) {
  constexpr int R2 = 2 * CR;
  const int lane = tt & 31, tw = tt >> 5;
  float vh[R2], vl[R2];
#pragma unroll
  for (int i = 0; i < R2; ++i) {
    const bool first = i < CR;
    const int ii = first ? i : i - CR;
    float sx, sy, lx, ly;
    if constexpr (GPT == 1) {
      f32x2_t s = pk2(Ct, Ct), lo = 0ull;
      if (FULL || ii < (first ? nr0 : nr1)) {
        const PT* ch = first ? c0 : c1;
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          const int cg = tt + q * LZ_CT;
          if (FULL || cg < C4) {
            const float4 f = phi_ld4(ch, (size_t)ii * C4 + cg);
            ofs_fma_acc2(s, lo, pk2(f.x, f.y), wh[q][0], wl[q][0]);
            ofs_fma_acc2(s, lo, pk2(f.z, f.w), wh[q][1], wl[q][1]);
          }
        }
      }
      upk2(s, sx, sy);
      upk2(lo, lx, ly);
    } else {
      // scalar steps (see sweepA_team_pair)
      sx = Ct;
      sy = Ct;
      lx = 0.f;
      ly = 0.f;
      if (FULL || ii < (first ? nr0 : nr1)) {
        const PT* ch = first ? c0 : c1;
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          const int cg = tt + q * LZ_CT;
          if (FULL || cg < C4) {
            const float4 f = phi_ld4(ch, (size_t)ii * C4 + cg);
            float a0, a1, b0, b1, c0_, c1_, d0, d1;
            upk2(wh[q][0], a0, a1);
            upk2(wl[q][0], b0, b1);
            upk2(wh[q][1], c0_, c1_);
            upk2(wl[q][1], d0, d1);
            ofs_fma_acc(sx, lx, f.x, a0, b0);
            ofs_fma_acc(sy, ly, f.y, a1, b1);
            ofs_fma_acc(sx, lx, f.z, c0_, d0);
            ofs_fma_acc(sy, ly, f.w, c1_, d1);
          }
        }
      }
    }
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
      if (i < nr0) bp0[i * LZ_CW + tw] = f2(r);
    } else if (i - CR < nr1) {
      bp1[(i - CR) * LZ_CW + tw] = f2(r);
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

// Basis rows per register group in the last step's row phase: RG * KT = 32
// basis elements per lane in registers.
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

// Row phase of the last step for the warp's rows [wr0, wr1) of the strip, in
// groups of RG rows held in registers (lanes over the basis index k):
//   z1 = z' - Q c  (the re-orthogonalisation with c = Q^T z' of the last
//                   pass, float32: the coefficients are at rounding level)
//   q_j = z1 / beta_{j-1},  Q[:, j] = q_j
template <int KT>
SLS_DEV void last_row_phase(float2* __restrict__ Qs, int ldq, int wr0, int wr1, int j,
                            const float2* __restrict__ cs, const float2* __restrict__ zps,
                            dfloat invb) {
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
    const float corr = group_correction<KT, RG>(q, cv);
    if (i < ng) {
      dfloat z1 = dfv(zps[b + i]);
      if (j > 0) z1 = df_add(z1, df_make(-corr, 0.f));
      const dfloat qj = df_mul(z1, invb);
      if ((lane & ((1 << SH) - 1)) == 0) Qb[(size_t)i * ldq + j] = f2(qj);
    }
  }
}

// Position in the ring of chunk number cnt (counted over the CTA's whole run):
// its slot and that slot's phase parity.  The divisions are taken once per
// pass; within a pass a RingPos advances by additions.
SLS_DEV int ring_slot(unsigned cnt, int S) { return (int)(cnt % (unsigned)S); }
SLS_DEV unsigned ring_par(unsigned cnt, int S) { return (cnt / (unsigned)S) & 1u; }

struct RingPos {
  int slot;
  unsigned par;
};

SLS_DEV RingPos ring_pos(unsigned cnt, int S) { return RingPos{ring_slot(cnt, S), ring_par(cnt, S)}; }

// the position k chunks further on (0 <= k <= S)
SLS_DEV RingPos ring_adv(RingPos q, int k, int S) {
  q.slot += k;
  if (q.slot >= S) {
    q.slot -= S;
    q.par ^= 1u;
  }
  return q;
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

// The CTA's column partials of Phi^T z' (double-float accumulators of the
// column pass) to dst[0 .. D): directly for P = 1, through the P row-phase
// sums in red otherwise (named barrier bar_id of nthr threads).
template <int GPT>
SLS_DEV void store_col_partials(const f32x2_t (&ah)[GPT][2], const f32x2_t (&al)[GPT][2],
                                int P, int C4, int D, int tt, float2* __restrict__ dst,
                                float2* __restrict__ red, unsigned bar_id, unsigned nthr) {
  const int ph = (P == 1) ? 0 : tt / C4;
  const int cb = (P == 1) ? tt : tt % C4;
  float2* d = (P == 1) ? dst : red + (size_t)ph * D;
  if (P == 1 || tt < P * C4) {
#pragma unroll
    for (int q = 0; q < GPT; ++q) {
      const int cg = cb + q * LZ_CT;
      if (cg < C4) {
        float h0, h1, l0, l1, h2, h3, l2, l3;
        upk2(ah[q][0], h0, h1);
        upk2(al[q][0], l0, l1);
        upk2(ah[q][1], h2, h3);
        upk2(al[q][1], l2, l3);
        const dfloat n0 = df_norm(h0, l0), n1 = df_norm(h1, l1);
        const dfloat n2 = df_norm(h2, l2), n3 = df_norm(h3, l3);
        float4* d4 = reinterpret_cast<float4*>(d + 4 * cg);
        d4[0] = make_float4(n0.hi, n0.lo, n1.hi, n1.lo);
        d4[1] = make_float4(n2.hi, n2.lo, n3.hi, n3.lo);
      }
    }
  }
  if (P > 1) {
    named_sync(bar_id, nthr);
    for (int col = tt; col < D; col += LZ_CT) {
      dfloat s = df_make(0.f, 0.f);
      for (int q = 0; q < P; ++q) s = df_add(s, dfv(red[(size_t)q * D + col]));
      dst[col] = f2(s);
    }
  }
}

// Slice phase of step j for the CTA's columns [cbeg, cend): the sum of the g
// CTA partials of Phi^T z' minus sum_{k < j} c_k w_k, into wred, and the
// CTA's part of |Phi^T z1|^2 (each thread returns its own columns' share).
// A column is summed by a segment of G lanes of one warp (G a power of two,
// as many as the compute threads allow), each lane over every G-th partial
// and every G-th basis index, then a butterfly within the segment.  The loads
// of the first column batch are issued before the named barrier after which
// c is ready (warp 0 fills it meanwhile); `synced` records that barrier.
// True when the last warp of the CTA sums no column in the slice phase (the
// column split of slice_columns below): it is free then for beta.
template <int NCW>
SLS_DEV bool slice_last_warp_idle(int ncol) {
  constexpr int NCT = NCW * 32;
  int G = 1;
  while (G < 32 && G * 2 * ncol <= NCT) G *= 2;
  return (NCW - 1) * (32 / G) >= ncol;
}

// c itself (cs[k] = the group sum accj[k], k < j) is loaded by warp cwarp:
// after it has issued its first batch when it sums columns, so that both
// round trips to L2 overlap, else before it reaches the named barrier.
template <int NCW>
SLS_DEV void load_c(float2* __restrict__ cs, const double* __restrict__ accj, int j) {
  const int lane = threadIdx.x & 31;
  for (int k = lane; k < j; k += 32) cs[k] = f2(df_from_double(accj[k]));
}

template <int NCW>
SLS_DEV dfloat slice_columns(const float2* __restrict__ wpart, const float2* __restrict__ Wm,
                             float2* __restrict__ wred, float2* __restrict__ cs,
                             const double* __restrict__ accj, int cwarp, int g, int D, int j,
                             int cbeg, int cend, bool& synced) {
  constexpr int NCT = NCW * 32;
  constexpr int BATCH = 8;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ncol = cend - cbeg;
  int G = 1;
  while (G < 32 && G * 2 * ncol <= NCT) G *= 2;
  const int cpw = 32 / G;
  const int sub = lane & (G - 1), slot = lane / G;
  dfloat sq = df_make(0.f, 0.f);
  for (int cb = warp * cpw; cb < ncol; cb += NCW * cpw) {
    const int cl = cb + slot;
    const bool valid = cl < ncol;
    const int c = cbeg + (valid ? cl : 0);
    // partials of Phi^T z' and basis columns: the first batches in flight together
    float2 pv[BATCH], wv[BATCH];
#pragma unroll
    for (int u = 0; u < BATCH; ++u) {
      const int b = sub + G * u;
      pv[u] = (valid && b < g) ? wpart[(size_t)b * D + c] : make_float2(0.f, 0.f);
      wv[u] = (valid && b < j) ? Wm[(size_t)b * D + c] : make_float2(0.f, 0.f);
    }
    if (!synced && warp == cwarp) load_c<NCW>(cs, accj, j);
    dfloat s = df_make(0.f, 0.f);
#pragma unroll
    for (int u = 0; u < BATCH; ++u) s = df_add_fast(s, dfv(pv[u]));
    for (int b0 = sub + G * BATCH; b0 < g; b0 += G * BATCH) {
#pragma unroll
      for (int u = 0; u < BATCH; ++u) {
        const int b = b0 + G * u;
        pv[u] = (valid && b < g) ? wpart[(size_t)b * D + c] : make_float2(0.f, 0.f);
      }
#pragma unroll
      for (int u = 0; u < BATCH; ++u) s = df_add_fast(s, dfv(pv[u]));
    }
    if (!synced) {
      named_sync(BAR_ALL, NCT);  // c is in shared memory
      synced = true;
    }
    // sum_k c_k w_k (Dot2), subtracted from the lane's part of the column sum
    float ch = 0.f, cl2 = 0.f;
#pragma unroll
    for (int u = 0; u < BATCH; ++u) {
      const int k = sub + G * u;
      if (k < j) dot2_acc_df(ch, cl2, dfv(wv[u]), dfv(cs[k]));
    }
    for (int k0 = sub + G * BATCH; k0 < j; k0 += G * BATCH) {
#pragma unroll
      for (int u = 0; u < BATCH; ++u) {
        const int k = k0 + G * u;
        wv[u] = (valid && k < j) ? Wm[(size_t)k * D + c] : make_float2(0.f, 0.f);
      }
#pragma unroll
      for (int u = 0; u < BATCH; ++u) {
        const int k = k0 + G * u;
        if (k < j) dot2_acc_df(ch, cl2, dfv(wv[u]), dfv(cs[k]));
      }
    }
    s = df_sub(s, df_norm(ch, cl2));
    for (int o = 1; o < G; o <<= 1) s = df_add_fast(s, shfl_xor_df(s, o));
    if (sub == 0 && valid) {
      wred[c] = f2(s);
      dot2_acc_df(sq.hi, sq.lo, s, s);
    }
  }
  if (!synced && warp == cwarp) load_c<NCW>(cs, accj, j);  // a warp without columns
  return sq;
}

// Ring chunks are numbered over the CTA's whole run; chunk cnt goes to slot
// cnt % S, whose mbarrier completes one phase per chunk.  slot_cnt[slot] holds
// the number of the last chunk issued to the slot (NO_CHUNK before the
// first): a chunk is issued only after the slot's previous chunk has been
// consumed, so once slot_cnt shows chunk cnt its phase parity is unambiguous.
constexpr unsigned NO_CHUNK = 0xffffffffu;

// Issue ring chunk number cnt: the rows of chunk k of the strip, Phi then the
// same rows of Q, one bulk copy each, completion counted on the slot's
// mbarrier.
template <typename PT>
SLS_DEV void issue_chunk(unsigned cnt, int slot, int k, int cr, int nrows, int D, int ldq,
                         unsigned stage, unsigned phib, unsigned char* ring, uint64_t* fullb,
                         volatile unsigned* slot_cnt, const PT* __restrict__ Phi,
                         const float2* __restrict__ Qs, uint64_t pol) {
  const int nr = min(cr, nrows - k * cr);
  const unsigned b1 = (unsigned)(nr * D * (int)sizeof(PT));
  const unsigned b2 = (unsigned)(nr * ldq * 8);
  unsigned char* dst = ring + (size_t)slot * stage;
  mbar_expect_tx(&fullb[slot], b1 + b2);
  bulk_g2s(dst, Phi + (int64_t)k * cr * D, b1, &fullb[slot], pol);
  bulk_g2s(dst + phib, Qs + (int64_t)k * cr * ldq, b2, &fullb[slot], pol);
  __threadfence_block();
  slot_cnt[slot] = cnt;
}

// Wait (bounded) until chunk cnt, at ring position q, has been issued and has
// landed; false if a wait gave up.  The chunk is normally issued long before
// its consumer arrives; otherwise the wait backs off instead of spinning.
SLS_DEV bool chunk_wait(unsigned cnt, RingPos q, uint64_t* fullb, volatile unsigned* slot_cnt) {
  if (slot_cnt[q.slot] != cnt) {
    const long long t0 = clock64();
    while (slot_cnt[q.slot] != cnt) {
      if (clock64() - t0 > SLS_WAIT_CYCLES) return false;
      __nanosleep(64);
    }
  }
  return mbar_wait(&fullb[q.slot], q.par);
}

template <int GPT, int KT, typename PT, int TEAMS>
__global__ void __launch_bounds__(TEAMS * LZ_CT, 1)
lanczos_kernel(LanczosBatch bt, char* scratch, size_t gstride, int g, int ngroups,
               int rows_cap, int ring_stages, int* status) {
  constexpr int NCW = TEAMS * LZ_CW;  // warps
  constexpr int NCT = NCW * 32;       // threads
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ float2 tmpw[NCW];
  __shared__ float s_red1[NCW];  // per-warp max |Phi| (offset bounds)
  __shared__ double shd[4];
  __shared__ float2 sdf[3];  // 1 / beta, alpha, beta of the step as double-float
  __shared__ int sflag, sbreak;
  __shared__ volatile unsigned slot_cnt[RING_MAX_STAGES];  // last chunk issued per slot
  __shared__ volatile int s_err;      // a wait of this CTA gave up

  constexpr int TCR = chunk_rows(GPT, TEAMS);
  constexpr int RPW = (2 * TCR + LZ_CW - 1) / LZ_CW;  // rows of a chunk pair per warp
  const int D = bt.D, r = bt.r, ldq = q_ld(bt.r);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int team = warp / LZ_CW, tw = warp % LZ_CW, tt = tid % LZ_CT;
  const int gi = blockIdx.x / g, rank = blockIdx.x % g;
  const int C4 = D >> 2;
  const int P = (C4 >= LZ_CT) ? 1 : (LZ_CT / C4);
  const int redn = (P > 1) ? P * D : 0;
  const bool fullD = (C4 == GPT * LZ_CT);  // no ragged column groups
  const unsigned bar_team = BAR_TEAM + (unsigned)team;

  const RingShape shp0 = ring_shape(D, ldq, 0, (int)sizeof(PT), TEAMS);
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
  float2* bpart = zps + rows_cap;                      // TEAMS x 16 x LZ_CW (row-dot warp sums)
  float2* cs = bpart + TEAMS * 16 * LZ_CW;             // r+1 (c = Q^T z')
  uint64_t* fullb = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(cs + (r + 1)) + 15) & ~(uintptr_t)15);  // S
  // scratch of the pass ends, in the ring (idle then: the next pass is
  // issued only once the pass has ended): team 1's column sums, then the
  // per-warp coefficient partials
  float2* tcol = reinterpret_cast<float2*>(ring);                   // 4 GPT x LZ_CT
  float2* cw = tcol + (TEAMS > 1 ? (size_t)4 * GPT * LZ_CT : 0);    // NCW x (r+1)

  const LzLayout L = lz_layout(bt.nmax, D, r, g);
  char* gb = scratch + (size_t)gi * gstride;
  unsigned* barw = reinterpret_cast<unsigned*>(gb + L.bar);
  double* acc = reinterpret_cast<double*>(gb + L.acc);
  float2* wpart = reinterpret_cast<float2*>(gb + L.wpart);
  float2* wred = reinterpret_cast<float2*>(gb + L.wred);
  float2* Wm = reinterpret_cast<float2*>(gb + L.Wm);
  const GroupBarrier bar{barw, barw + 32, (unsigned)g};
  const int accs = lz_acc_stride(r);
  // Phi and Q stream through L2 once per pass: evict-first (measured faster
  // than evict-normal, and no slower than keeping the rows the next pass
  // reads first with evict-last)
  const uint64_t pol = l2_policy_evict_first();

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&fullb[s], 1);
      slot_cnt[s] = NO_CHUNK;
    }
    mbar_fence_init();
    s_err = 0;
  }
  __syncthreads();

  // Before the CTA leaves: the last chunk issued to every slot has landed
  // (the slot's earlier chunks were consumed, so they landed before it).
  auto drain = [&]() {
    if (tid == 0) {
      for (int s = 0; s < S; ++s) {
        const unsigned c = slot_cnt[s];
        if (c != NO_CHUNK) mbar_wait(&fullb[s], ring_par(c, S));
      }
    }
  };

  const int nprob = nprob_of(bt);

  unsigned lgen = 0;
  unsigned base = 0;   // ring chunks consumed before the current pass
  unsigned gstep = 0;  // steps run by this group so far (parity of the group sums)
  for (int p = gi; p < nprob; p += ngroups) {
    const int64_t row0 = bt.row0 ? bt.row0[p] : 0;
    const int64_t n = bt.n ? (int64_t)bt.n[p] : bt.n_single;
    const int64_t q1o = bt.q1off ? bt.q1off[p] : row0;
    const double* q1 = bt.q1 + q1o;
    const int64_t rs = (int64_t)rank * n / g, re = (int64_t)(rank + 1) * n / g;
    const PT* Phis = reinterpret_cast<const PT*>(bt.Phi) + (row0 + rs) * D;  // this CTA's rows
    float2* Qs = bt.Q + (row0 + rs) * ldq;  // this CTA's rows of the basis
    const int nrows = (int)(re - rs);
    const int nch = (nrows + cr - 1) / cr;
    const int npairs = (nch + 1) / 2;
    double* alpha_out = bt.alpha + (size_t)p * r;
    double* beta_out = bt.beta + (size_t)p * r;
    const int cbeg = (int)((int64_t)rank * D / g), cend = (int)((int64_t)(rank + 1) * D / g);

    double scale = 0.0, alpha_prev = 0.0;
    // beta_{j-1} = 1 / e_inv and the break test of the step, in lane 0 of
    // warp bw: the last warp during the slice phase when that warp sums no
    // column there (measured 2% faster at the qwen7b shape), else warp 0
    // after group barrier 2
    double e_inv = 0.0, e_bnew = 0.0;
    int e_brk = 0;
    const bool beta_early = slice_last_warp_idle<NCW>(cend - cbeg);
    const int bw = beta_early ? NCW - 1 : 0;
    dfloat alpha_df = df_make(0.f, 0.f), beta_df = df_make(0.f, 0.f), invb_df;
    float phimax = 0.f;  // max |Phi| over this CTA's strip (prologue pass)
    int reff = 0;
    sbreak = 0;

    // The first min(S, nch) chunks of pass `pass` (0 = the prologue; passes
    // alternate direction), issued once the ring is idle, chunk t by lane 0
    // of warp t mod NCW: the thread that issues a bulk copy is held for a few
    // hundred cycles, so the copies are spread over warps.
    //
    // No chunk is issued once a wait of this CTA has given up (s_err, set
    // before the team or CTA barrier that precedes every issue): a slot then
    // never receives a chunk whose predecessor in the slot was not seen to
    // land, so the phase parity of each slot's mbarrier stays that of its
    // last chunk number and drain() waits for every copy still in flight.
    auto issue_pass_head = [&](int pass) {
      if (lane == 0 && !s_err) {
        const int m = min(S, nch);
        for (int t = warp; t < m; t += NCW)
          issue_chunk<PT>(base + (unsigned)t, ring_slot(base + (unsigned)t, S),
                          (pass & 1) ? nch - 1 - t : t, cr, nrows, D, ldq, stage, phib, ring,
                          fullb, slot_cnt, Phis, Qs, pol);
      }
    };
    // Refill of a team's previous pair in pass `pass`: chunk t0 + h + S of
    // the pass where it exists, into the slot of chunk t0 + h at ring
    // position q0 + h.  Called after a team barrier (no warp reads those
    // slots any more) by lane 0 of the team's last two warps, one chunk each
    // (measured 3.5% faster at the qwen7b shape than one thread issuing
    // both).
    auto refill_half = [&](int pass, int t0, RingPos q0) {
      const int h = tw - (LZ_CW - 2);
      if (t0 < 0 || lane != 0 || h < 0 || s_err) return;
      const int t = t0 + h + S;
      if (t >= nch) return;
      SLS_DBG_CHECK(status, t >= 0 && ring_adv(q0, h, S).slot < S);
      issue_chunk<PT>(base + (unsigned)t, ring_adv(q0, h, S).slot, (pass & 1) ? nch - 1 - t : t,
                      cr, nrows, D, ldq, stage, phib, ring, fullb, slot_cnt, Phis, Qs, pol);
    };

    // pass end: team 1's column sums join team 0's through the ring (idle
    // now), team 0 stores the CTA's partials of Phi^T z'; the per-warp
    // coefficient partials (k < K) and |z'|^2 join the group sums of parity
    // `par` (float64 atomics)
    auto pass_end = [&](f32x2_t (&ah)[GPT][2], f32x2_t (&al)[GPT][2], dfloat (&cacc)[KT], int K,
                        dfloat nacc, unsigned par) {
      named_sync(BAR_ALL, NCT);  // both teams are done with the ring
      if constexpr (TEAMS > 1) {
        if (team == 1) {
#pragma unroll
          for (int q = 0; q < GPT; ++q)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              float a0, a1, b0, b1;
              upk2(ah[q][h], a0, a1);
              upk2(al[q][h], b0, b1);
              tcol[(size_t)((q * 2 + h) * 2 + 0) * LZ_CT + tt] = make_float2(a0, b0);
              tcol[(size_t)((q * 2 + h) * 2 + 1) * LZ_CT + tt] = make_float2(a1, b1);
            }
        }
      }
#pragma unroll
      for (int t = 0; t < KT; ++t) {
        const int k = lane + 32 * t;
        if (k < K) cw[(size_t)warp * (r + 1) + k] = f2(df_norm(cacc[t].hi, cacc[t].lo));
      }
      {
        dfloat nv = df_norm(nacc.hi, nacc.lo);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) nv = df_add_fast(nv, shfl_xor_df(nv, o));
        if (lane == 0) tmpw[warp] = f2(nv);
      }
      named_sync(BAR_ALL, NCT);
      double* accn = acc + (size_t)(par & 1u) * accs;
      if (team == 0) {
        if constexpr (TEAMS > 1) {
#pragma unroll
          for (int q = 0; q < GPT; ++q)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              float a0, a1, b0, b1;
              upk2(ah[q][h], a0, a1);
              upk2(al[q][h], b0, b1);
              const dfloat x0 = df_add(df_make(a0, b0),
                                       dfv(tcol[(size_t)((q * 2 + h) * 2 + 0) * LZ_CT + tt]));
              const dfloat x1 = df_add(df_make(a1, b1),
                                       dfv(tcol[(size_t)((q * 2 + h) * 2 + 1) * LZ_CT + tt]));
              ah[q][h] = pk2(x0.hi, x1.hi);
              al[q][h] = pk2(x0.lo, x1.lo);
            }
        }
        store_col_partials<GPT>(ah, al, P, C4, D, tt, wpart + (size_t)rank * D, red, bar_team,
                                LZ_CT);
      }
      // coefficient k: the NCW warp partials summed by four lanes (each over
      // every fourth warp) and a butterfly over the four
      constexpr int LPK = 4;
      for (int k0 = 0; k0 < K; k0 += NCT / LPK) {
        const int k = k0 + tid / LPK, part = tid % LPK;
        dfloat s = df_make(0.f, 0.f);
        if (k < K)
          for (int w = part; w < NCW; w += LPK) s = df_add(s, dfv(cw[(size_t)w * (r + 1) + k]));
        s = df_add_fast(s, shfl_xor_df(s, 1));
        s = df_add_fast(s, shfl_xor_df(s, 2));
        if (part == 0 && k < K) red_add_f64(accn + k, df_to_double(s));
      }
      if (warp == NCW - 1) {
        dfloat t = (lane < NCW) ? dfv(tmpw[lane]) : df_make(0.f, 0.f);
#pragma unroll
        for (int o = 1; o < NCW; o <<= 1) t = df_add_fast(t, shfl_xor_df(t, o));
        if (lane == 0) red_add_f64(accn + r + 1, df_to_double(t));
      }
      // the column of Q written in this pass reaches the bulk reads of the
      // next pass (async proxy)
      if (lane == 0) asm volatile("fence.proxy.async.global;" ::: "memory");
      named_sync(BAR_ALL, NCT);
    };

    issue_pass_head(0);

    // ---------------- prologue: z' = q1, |z'|^2 and Phi^T z' (pass 0) ------------
    {
      dfloat nacc = df_make(0.f, 0.f);
      for (int il = tid; il < nrows; il += NCT) {
        const dfloat z = df_from_double(q1[rs + il]);
        SLS_DBG_GUARD(status, il < rows_cap) zps[il] = f2(z);
        dot2_acc_df(nacc.hi, nacc.lo, z, z);
      }
      f32x2_t ah[GPT][2], al[GPT][2];
#pragma unroll
      for (int q = 0; q < GPT; ++q) ah[q][0] = ah[q][1] = al[q][0] = al[q][1] = 0ull;
      float mx = 0.f;
      named_sync(BAR_ALL, NCT);  // z' of the strip is in shared memory
      int prev = -1;
      RingPos qprev{0, 0u};
      RingPos qc = ring_pos(base + 2u * (unsigned)team, S);  // the team's first pair
      for (int pi = team; pi < npairs; pi += TEAMS) {
        const int t0p = 2 * pi;
        const bool two = t0p + 1 < nch;
        const unsigned c0n = base + (unsigned)t0p;
        const RingPos q1p = ring_adv(qc, 1, S);
        if (!chunk_wait(c0n, qc, fullb, slot_cnt)) lz_fail(status, &s_err);
        if (two && !chunk_wait(c0n + 1, q1p, fullb, slot_cnt)) lz_fail(status, &s_err);
        named_sync(bar_team, LZ_CT);
        refill_half(0, prev, qprev);
        prev = t0p;
        qprev = qc;
        for (int h = 0; h < (two ? 2 : 1); ++h) {
          const int t = t0p + h;
          const PT* chunk =
              reinterpret_cast<const PT*>(ring + (size_t)(h ? q1p.slot : qc.slot) * stage);
          const int nr = min(cr, nrows - t * cr);
          sweepA_chunk<GPT, true>(chunk, nr, D, t * cr, tt, zps, ah, al, &mx);
        }
        qc = ring_adv(qc, 2 * TEAMS, S);
      }
      base += (unsigned)nch;
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      if (lane == 0) s_red1[warp] = mx;
      dfloat cacc0[KT];
#pragma unroll
      for (int t = 0; t < KT; ++t) cacc0[t] = df_make(0.f, 0.f);
      // |q1|^2 is the group sum of the first step
      pass_end(ah, al, cacc0, 0, nacc, gstep);
      if (r >= 2) issue_pass_head(1);
    }

    if (bt.inject_fail && rank == 0 && tid == 0) lz_fail(status, &s_err);
    for (int j = 0; j < r; ++j, ++gstep) {
      if (!group_sync_named(bar, lgen, status, &sflag, &s_err, BAR_ALL, NCT)) {
        drain();
        return;
      }
      const double* accj = acc + (size_t)(gstep & 1u) * accs;
      // |z1|^2 = |z'|^2 - |c|^2 (Q orthonormal): beta_{j-1} and the break
      // test (warp bw, once c is in shared memory)
      auto beta_phase = [&]() {
        const double zs = accj[r + 1];
        dfloat cn = df_make(0.f, 0.f);
#pragma unroll
        for (int t2 = 0; t2 < KT; ++t2) {
          const int k = lane + 32 * t2;
          if (k < j) dot2_acc_df(cn.hi, cn.lo, dfv(cs[k]), dfv(cs[k]));
        }
        cn = df_norm(cn.hi, cn.lo);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) cn = df_add_fast(cn, shfl_xor_df(cn, o));
        if (lane == 0) {
          const double nrm2 = zs - df_to_double(cn);  // |z1|^2
          // one reciprocal square root instead of a square root and two
          // divides (float64 runs at a fraction of the float32 rate here)
          e_inv = (nrm2 > 0.0) ? rsqrt(nrm2) : 0.0;  // 1 / beta
          e_bnew = (nrm2 > 0.0) ? nrm2 * e_inv : 0.0;
          e_brk = 0;
          if (j > 0) {
            scale = fmax(scale, fabs(alpha_prev) + e_bnew);
            if (!(e_bnew > bt.tol * scale)) e_brk = 1;
            else if (rank == 0) beta_out[j - 1] = e_bnew;
          } else if (!(e_bnew > 0.0)) {
            e_brk = 1;
          }
        }
      };

      // ---------------- slice phase: c, Phi^T z1 for this CTA's columns ----------
      // c = Q^T z' (k < j) from the group sums; Phi^T z1 = Phi^T z' - sum_k
      // c_k w_k with w_k = Phi^T q_k kept in Wm.  The group sums of the other
      // parity were read in the previous step by every CTA (all of them have
      // passed barrier 1 since): the first CTA clears them for the next step.
      if (rank == 0) {
        double* accz = acc + (size_t)((gstep + 1u) & 1u) * accs;
        for (int k = tid; k < accs; k += NCT) accz[k] = 0.0;
      }
      {
        // c is loaded by the last warp when it sums no column (it waits for
        // beta there anyway), else by warp 0
        bool synced = false;
        dfloat sq = slice_columns<NCW>(wpart, Wm, wred, cs, accj, beta_early ? NCW - 1 : 0, g, D,
                                       j, cbeg, cend, synced);
        if (!synced) named_sync(BAR_ALL, NCT);
        if (beta_early && warp == NCW - 1) beta_phase();
        sq = df_norm(sq.hi, sq.lo);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sq = df_add_fast(sq, shfl_xor_df(sq, o));
        if (lane == 0) tmpw[warp] = f2(sq);
        named_sync(BAR_ALL, NCT);
        if (warp == 0) {
          // the NCW warp sums by a butterfly over the first NCW lanes
          dfloat t = (lane < NCW) ? dfv(tmpw[lane]) : df_make(0.f, 0.f);
#pragma unroll
          for (int o = 1; o < NCW; o <<= 1) t = df_add_fast(t, shfl_xor_df(t, o));
          if (lane == 0) red_add_f64(const_cast<double*>(accj) + r + 2, df_to_double(t));
        }
      }
      if (!group_sync_named(bar, lgen, status, &sflag, &s_err, BAR_ALL, NCT)) {
        drain();
        return;
      }

      // ---------------- beta_{j-1}, alpha_j, break test; w_j gather ---------------
      // this thread's columns of Phi^T z1 (loads in flight while warp 0 works)
      float4 wv[GPT][2];
#pragma unroll
      for (int q = 0; q < GPT; ++q) wv[q][0] = wv[q][1] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (P == 1) {
        const float4* wr4 = reinterpret_cast<const float4*>(wred);
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          const int cg = tt + q * LZ_CT;
          if (cg < C4) {
            wv[q][0] = wr4[2 * cg];
            wv[q][1] = wr4[2 * cg + 1];
          }
        }
      }
      if (!beta_early && warp == 0) beta_phase();
      if (warp == bw && lane == 0) {
        const double q = accj[r + 2];  // |Phi^T z1|^2
        const double a = e_brk ? 0.0 : (q * e_inv) * e_inv;
        if (!e_brk && rank == 0) alpha_out[j] = a;
        shd[1] = e_brk ? 0.0 : e_inv;
        shd[2] = a;
        shd[3] = (j > 0) ? e_bnew : 0.0;
        // converted once here: float64 runs at a small fraction of the
        // float32 rate on this part, and every thread needs these
        sdf[0] = f2(df_from_double(shd[1]));
        sdf[1] = f2(df_from_double(a));
        sdf[2] = f2(df_from_double(shd[3]));
        sbreak = e_brk;
      }
      named_sync(BAR_ALL, NCT);
      if (sbreak) {
        reff = j;
        break;
      }
      invb_df = dfv(sdf[0]);
      alpha_prev = shd[2];
      alpha_df = dfv(sdf[1]);
      beta_df = dfv(sdf[2]);
      if (j == 0) {
#pragma unroll
        for (int w = 0; w < NCW; ++w) phimax = fmaxf(phimax, s_red1[w]);
      }

      if (j == r - 1) {
        // the last step needs no pass over Phi: q_{r-1} = z1 / beta_{r-2}
        const int wr0 = warp * nrows / NCW, wr1 = (warp + 1) * nrows / NCW;
        last_row_phase<KT>(Qs, ldq, wr0, wr1, j, cs, zps, invb_df);
        reff = r;
        break;
      }

      // w_j = (Phi^T z1) / beta: into shared memory for the row-per-warp row
      // dots (D < 4 LZ_CT; the team row dots take their columns straight into
      // registers below); keep w_j (slice) for the correction of later steps
      if (P > 1) {
        for (int c0 = tid; c0 < D; c0 += 8 * NCT) {
          float2 wv2[8];
#pragma unroll
          for (int m = 0; m < 8; ++m) {
            const int c = c0 + m * NCT;
            wv2[m] = (c < D) ? wred[c] : make_float2(0.f, 0.f);
          }
#pragma unroll
          for (int m = 0; m < 8; ++m) {
            const int c = c0 + m * NCT;
            if (c < D) {
              const dfloat a = df_mul(dfv(wv2[m]), invb_df);
              wsh[c] = a.hi;
              wsl[c] = a.lo;
              if (c >= cbeg && c < cend) Wm[(size_t)j * D + c] = f2(a);
            }
          }
        }
        named_sync(BAR_ALL, NCT);
      }

      // ---------------- fused pass j+1 over Phi ----------------------------------
      // per chunk (pair): z1 = z' - Q c, q_j = z1 / beta_{j-1} (row work);
      // s = Phi w_j (row dots); z' <- s - alpha_j q_j - beta_{j-1} q_{j-1} and
      // its partials of c = Q^T z' and |z'|^2 (row work); Phi^T z' (columns).
      const int pass = j + 1;
      const bool fwd = (pass & 1) == 0;
      f32x2_t ah[GPT][2], al[GPT][2];
#pragma unroll
      for (int q = 0; q < GPT; ++q) ah[q][0] = ah[q][1] = al[q][0] = al[q][1] = 0ull;
      dfloat cacc[KT];
#pragma unroll
      for (int t = 0; t < KT; ++t) cacc[t] = df_make(0.f, 0.f);
      dfloat nacc = df_make(0.f, 0.f);
      if (P == 1) {
        // this thread's columns of w_j into registers; team 0 keeps its slice
        f32x2_t wh[GPT][2], wl[GPT][2];
        float wt1 = 0.f;  // l1 norm of this thread's slice of w_j
#pragma unroll
        for (int q = 0; q < GPT; ++q) {
          const int cg = tt + q * LZ_CT;
          float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a;
          if (cg < C4) {
            const dfloat w0 = df_mul(df_make(wv[q][0].x, wv[q][0].y), invb_df);
            const dfloat w1 = df_mul(df_make(wv[q][0].z, wv[q][0].w), invb_df);
            const dfloat w2 = df_mul(df_make(wv[q][1].x, wv[q][1].y), invb_df);
            const dfloat w3 = df_mul(df_make(wv[q][1].z, wv[q][1].w), invb_df);
            a = make_float4(w0.hi, w1.hi, w2.hi, w3.hi);
            b = make_float4(w0.lo, w1.lo, w2.lo, w3.lo);
            const int c = 4 * cg;
            if (team == 0) {
              if (c >= cbeg && c < cend) Wm[(size_t)j * D + c] = f2(w0);
              if (c + 1 >= cbeg && c + 1 < cend) Wm[(size_t)j * D + c + 1] = f2(w1);
              if (c + 2 >= cbeg && c + 2 < cend) Wm[(size_t)j * D + c + 2] = f2(w2);
              if (c + 3 >= cbeg && c + 3 < cend) Wm[(size_t)j * D + c + 3] = f2(w3);
            }
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
        float2* bp = bpart + (size_t)team * 16 * LZ_CW;
        int prev = -1;
        RingPos qprev{0, 0u};
        RingPos qc = ring_pos(base + 2u * (unsigned)team, S);  // the team's first pair
        for (int pi = team; pi < npairs; pi += TEAMS) {
          const int t0p = 2 * pi;
          const bool two = t0p + 1 < nch;
          const int kc0 = fwd ? t0p : nch - 1 - t0p;
          const int kc1 = fwd ? t0p + 1 : nch - 2 - t0p;
          const unsigned c0n = base + (unsigned)t0p;
          const RingPos q1p = ring_adv(qc, 1, S);
          const int s0 = qc.slot;
          if (!chunk_wait(c0n, qc, fullb, slot_cnt)) lz_fail(status, &s_err);
          int s1 = s0;
          if (two) {
            s1 = q1p.slot;
            if (!chunk_wait(c0n + 1, q1p, fullb, slot_cnt)) lz_fail(status, &s_err);
          }
          const PT* ch0 = reinterpret_cast<const PT*>(ring + (size_t)s0 * stage);
          const PT* ch1 = reinterpret_cast<const PT*>(ring + (size_t)s1 * stage);
          const float2* qb0 = reinterpret_cast<const float2*>(ring + (size_t)s0 * stage + phib);
          const float2* qb1 = reinterpret_cast<const float2*>(ring + (size_t)s1 * stage + phib);
          const int nr0 = min(cr, nrows - kc0 * cr);
          const int nr1 = two ? min(cr, nrows - kc1 * cr) : 0;
          SLS_DBG_CHECK(status, kc0 >= 0 && kc0 < nch && nr0 >= 1 && (!two || (kc1 >= 0 && kc1 < nch && nr1 >= 1)));
          // row work before the row dots: q_j of the warp's rows of the pair
          // (it feeds only the row work after them)
          dfloat qjv[RPW];
          float2 qpv[RPW];
          if (fullD && nr0 == TCR && nr1 == TCR && 2 * TCR == LZ_CW) {
            // steady state, every warp owns one row of the pair: q_j of that
            // row and the row dots in one block, so that the warp reduction
            // of q_j interleaves with the sweep's arithmetic (measured 2.9%
            // faster at the qwen7b shape than q_j ahead of the sweep)
            const bool first = tw < TCR;
            const int ii = first ? tw : tw - TCR;
            const int il = (first ? kc0 : kc1) * cr + ii;
            const float2* qrow = (first ? qb0 : qb1) + (size_t)ii * ldq;
            const float corr = row_corr<KT>(qrow, cs, j);  // 0 at j = 0
            qjv[0] = df_mul(df_add(dfv(zps[il]), df_make(-corr, 0.f)), invb_df);
            qpv[0] = (j > 0) ? qrow[j > 0 ? j - 1 : 0] : make_float2(0.f, 0.f);
            sweepB_team_pair<GPT, TCR, true>(ch0, nr0, ch1, nr1, C4, tt, wh, wl, Ct, bp,
                                             bp + TCR * LZ_CW);
            if (lane == 0) SLS_DBG_GUARD(status, il < nrows) Qs[(size_t)il * ldq + j] = f2(qjv[0]);
          } else {
#pragma unroll
            for (int m = 0; m < RPW; ++m) {
              const int ri = tw + m * LZ_CW;
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
                if (lane == 0) SLS_DBG_GUARD(status, il < nrows) Qs[(size_t)il * ldq + j] = f2(qjv[m]);
              }
            }
            // row dots s = Phi w_j, warp sums into bp[row * LZ_CW + tw]
            if (fullD && nr0 == TCR && nr1 == TCR)
              sweepB_team_pair<GPT, TCR, true>(ch0, nr0, ch1, nr1, C4, tt, wh, wl, Ct, bp,
                                               bp + TCR * LZ_CW);
            else
              sweepB_team_pair<GPT, TCR, false>(ch0, nr0, ch1, nr1, C4, tt, wh, wl, Ct, bp,
                                                bp + TCR * LZ_CW);
          }
          named_sync(bar_team, LZ_CT);
          // every warp of the team is past its previous pair: refill those slots
          refill_half(pass, prev, qprev);
          prev = t0p;
          qprev = qc;
          qc = ring_adv(qc, 2 * TEAMS, S);
          // row work after the row dots: z', its partials of c and |z'|^2
#pragma unroll
          for (int m = 0; m < RPW; ++m) {
            const int ri = tw + m * LZ_CW;
            const bool first = ri < TCR;
            const int ii = first ? ri : ri - TCR;
            if (ri < 2 * TCR && ii < (first ? nr0 : nr1)) {
              const int il = (first ? kc0 : kc1) * cr + ii;
              const float2* qrow = (first ? qb0 : qb1) + (size_t)ii * ldq;
              // every lane adds the LZ_CW warp sums of the row (broadcast reads)
              const float4* b4 = reinterpret_cast<const float4*>(bp + ri * LZ_CW);
              dfloat v[LZ_CW];
#pragma unroll
              for (int u = 0; u < LZ_CW / 2; ++u) {
                const float4 x = b4[u];
                v[2 * u] = df_make(x.x, x.y);
                v[2 * u + 1] = df_make(x.z, x.w);
              }
#pragma unroll
              for (int wdt = 1; wdt < LZ_CW; wdt *= 2)
#pragma unroll
                for (int i = 0; i + wdt < LZ_CW; i += 2 * wdt) v[i] = df_add_fast(v[i], v[i + wdt]);
              dfloat zp = df_sub(v[0], df_mul(alpha_df, qjv[m]));
              if (j > 0) zp = df_sub(zp, df_mul(beta_df, dfv(qpv[m])));
              if (lane == 0) {
                SLS_DBG_GUARD(status, il < nrows) zps[il] = f2(zp);
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
          named_sync(bar_team, LZ_CT);
          // columns: Phi^T z' for the next step
          if (fullD && nr0 == TCR && nr1 == TCR)
            sweepA_team_pair<GPT, TCR, true>(ch0, nr0, kc0 * cr, ch1, nr1, kc1 * cr, C4, tt, zps,
                                              phimax, ah, al);
          else
            sweepA_team_pair<GPT, TCR, false>(ch0, nr0, kc0 * cr, ch1, nr1, kc1 * cr, C4, tt,
                                               zps, phimax, ah, al);
        }
      } else if constexpr (TEAMS == 1) {
        // D < 4 LZ_CT: one warp per row for the row dots (w_j in shared
        // memory), the column pass in P row phases
        float mx = 0.f;
        RingPos qc = ring_pos(base, S);
        for (int t = 0; t < nch; ++t, qc = ring_adv(qc, 1, S)) {
          const int kc = fwd ? t : nch - 1 - t;
          const unsigned cc = base + (unsigned)t;
          const int slot = qc.slot;
          if (!chunk_wait(cc, qc, fullb, slot_cnt))
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
            if (lane == 0) SLS_DBG_GUARD(status, il < nrows) Qs[(size_t)il * ldq + j] = f2(qj);
            const dfloat s = row_dot_smem(chunk + (size_t)ii * D, D, wsh, wsl);
            dfloat zp = df_sub(s, df_mul(alpha_df, qj));
            if (j > 0) zp = df_sub(zp, df_mul(beta_df, dfv(qrow[j - 1])));
            if (lane == 0) {
              SLS_DBG_GUARD(status, il < nrows) zps[il] = f2(zp);
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
          named_sync(BAR_ALL, NCT);
          sweepA_chunk<GPT, false>(chunk, nr, D, kc * cr, tt, zps, ah, al, &mx);
          // every warp is done with this chunk: refill its slot
          named_sync(BAR_ALL, NCT);
          if (tid == 0 && t + S < nch && !s_err)
            issue_chunk<PT>(base + (unsigned)(t + S), slot, fwd ? t + S : nch - 1 - (t + S), cr,
                            nrows, D, ldq, stage, phib, ring, fullb, slot_cnt, Phis, Qs, pol);
        }
      }
      base += (unsigned)nch;
      // partials for step j+1 (read after its barrier 1): Phi^T z', c, |z'|^2
      pass_end(ah, al, cacc, j + 1, nacc, gstep + 1u);
      if (pass + 1 <= r - 1) issue_pass_head(pass + 1);
    }
    // the loop always ends in a break (the break test, or the last step) with
    // gstep at that step; the slice phase of that step cleared the group sums
    // of the next parity, where the next problem's prologue starts
    ++gstep;
    // a break leaves the head of the next pass issued (chunks base ..): wait
    // for it to land and count it as consumed
    if (sbreak) {
      unsigned nb = base;
      for (int s2 = 0; s2 < S; ++s2) {
        const unsigned c = slot_cnt[s2];
        if (c != NO_CHUNK && c >= base) {
          if (tid == 0 && !mbar_wait(&fullb[s2], ring_par(c, S))) lz_fail(status, &s_err);
          nb = max(nb, c + 1u);
        }
      }
      named_sync(BAR_ALL, NCT);
      base = nb;
    }
    if (rank == 0 && tid == 0) {
      bt.r_eff[p] = reff;
      for (int k = reff; k < r; ++k) alpha_out[k] = 0.0;
      for (int k = (reff > 0 ? reff - 1 : 0); k < r; ++k) beta_out[k] = 0.0;
    }
    // problems on the same group run back to back; keep them apart
    if (!group_sync_named(bar, lgen, status, &sflag, &s_err, BAR_ALL, NCT)) {
      drain();
      return;
    }
  }
  drain();
}

template <int GPT, int KT, typename PT, int TEAMS>
int launch_lanczos_t(const LanczosBatch& bt, void* scratch, size_t gstride, int groups, int g,
                     int rows_cap, int stages, int* status, size_t smem, cudaStream_t stream) {
  auto fn = lanczos_kernel<GPT, KT, PT, TEAMS>;
  SLS_CUDA_TRY(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  char* sc = (char*)scratch;
  void* args[] = {(void*)&bt, (void*)&sc, (void*)&gstride, (void*)&g, (void*)&groups,
                  (void*)&rows_cap, (void*)&stages, (void*)&status};
  SLS_CUDA_TRY(cudaLaunchCooperativeKernel((const void*)fn, dim3(groups * g),
                                           dim3(lz_threads(TEAMS)), args, smem, stream));
  count_launch(1);
  return SLS_OK;
}

// KT = 1, 2 or 4 basis tiles for one GPT, element type and team count
template <int GPT, typename PT, int TEAMS>
int launch_lanczos_kt(const LanczosBatch& bt, void* scratch, size_t gstride, int groups, int g,
                      int rows_cap, int stages, int* status, size_t smem, cudaStream_t stream,
                      int kt) {
  switch (kt) {
    case 1:
      return launch_lanczos_t<GPT, 1, PT, TEAMS>(bt, scratch, gstride, groups, g, rows_cap,
                                                 stages, status, smem, stream);
    case 2:
      return launch_lanczos_t<GPT, 2, PT, TEAMS>(bt, scratch, gstride, groups, g, rows_cap,
                                                 stages, status, smem, stream);
    case 4:
      return launch_lanczos_t<GPT, 4, PT, TEAMS>(bt, scratch, gstride, groups, g, rows_cap,
                                                 stages, status, smem, stream);
    default:
      return SLS_ERR_UNSUPPORTED;
  }
}

}  // namespace

// Launch the Lanczos kernel for GPT = 1, 2, 4 or 8 column groups per thread
// and KT = 1, 2 or 4 basis tiles, Phi in float32 (lanczos_g<GPT>.cu) or
// bfloat16 (lanczos_b<GPT>.cu), with `teams` = lz_teams(GPT, P) compute teams.
#define SLS_LZ_LAUNCH_ARGS                                                                \
  const LanczosBatch &bt, void *scratch, size_t gstride, int groups, int g, int rows_cap, \
      int stages, int *status, size_t smem, cudaStream_t stream, int kt, int teams
int launch_lanczos_gpt1(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_gpt2(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_gpt4(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_gpt8(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_bf16_gpt1(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_bf16_gpt2(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_bf16_gpt4(SLS_LZ_LAUNCH_ARGS);
int launch_lanczos_bf16_gpt8(SLS_LZ_LAUNCH_ARGS);

}  // namespace sls
