// Double-float helpers for the symmetric tridiagonal T of Algorithm 1
// (Eigh(T)): division, power-of-two scaling and the Sturm count that
// bisection and multisection search on.
#pragma once

#include "common.cuh"

namespace sls {

SLS_DEV dfloat df_div(dfloat a, dfloat b) {
  const float q1 = __fdividef(a.hi, b.hi);
  float p, e;
  two_prod(q1, b.hi, p, e);
  const float rr = (((a.hi - p) - e) + a.lo) - q1 * b.lo;
  const float q2 = __fdividef(rr, b.hi);
  return df_norm(q1, q2);
}

SLS_DEV dfloat df_scale(dfloat a, float s) { return df_make(a.hi * s, a.lo * s); }

// Number of eigenvalues of the (scaled) tridiagonal below x, from the signs of
// the leading principal minors p_i(x) (three-term recurrence, Sturm sequence).
// Powers of two rescale the pair (p_{i-1}, p_i) to keep it in range; a zero
// minor takes the sign opposite to its predecessor.
SLS_DEV int sturm_count(const float2* __restrict__ a, const float2* __restrict__ b2, int n,
                        dfloat x) {
  dfloat pm = df_make(1.f, 0.f), pc = df_sub(dfv(a[0]), x);
  int sprev = 0;
  int s = (pc.hi < 0.f) ? 1 : ((pc.hi > 0.f) ? 0 : 1);
  int cnt = (s != sprev);
  sprev = s;
  for (int i = 1; i < n; ++i) {
    const dfloat d = df_sub(dfv(a[i]), x);
    const dfloat t = df_mul(dfv(b2[i - 1]), pm);
    const dfloat pn = df_sub(df_mul(d, pc), t);
    pm = pc;
    pc = pn;
    const float mg = fmaxf(fabsf(pc.hi), fabsf(pm.hi));
    if (mg > 0x1p60f) {
      pc = df_scale(pc, 0x1p-60f);
      pm = df_scale(pm, 0x1p-60f);
    } else if (mg < 0x1p-60f && mg > 0.f) {
      pc = df_scale(pc, 0x1p60f);
      pm = df_scale(pm, 0x1p60f);
    }
    s = (pc.hi < 0.f) ? 1 : ((pc.hi > 0.f) ? 0 : 1 - sprev);
    cnt += (s != sprev);
    sprev = s;
  }
  return cnt;
}

}  // namespace sls
