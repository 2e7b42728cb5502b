// Shared device helpers for the Spectral-LSH kernels (sm_103a).
//
//  * double-float ("df") arithmetic: a value is an unevaluated sum hi + lo of
//    two floats.  TwoSum (Knuth), Fast2Sum (Dekker) and TwoProduct through a
//    fused multiply-add give error-free transformations, and the compensated
//    dot product follows Ogita, Rump and Oishi, "Accurate Sum and Dot
//    Product", SIAM J. Sci. Comput. 26(6), 2005 (Dot2).  The GB300's fp64
//    rate is a small fraction of its fp32 rate, so every hot reduction runs
//    on the fp32 pipes in this form.
//  * a grid / CTA-group barrier with an iteration limit: a wait that gives up
//    records SLS_ERR_TIMEOUT in the workspace status word and the kernel
//    returns instead of hanging.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/sls.h"

#define SLS_DEV __device__ __forceinline__

// ---------------------------------------------------------------------------
// double-float arithmetic
// ---------------------------------------------------------------------------

struct dfloat {
  float hi, lo;
};

SLS_DEV void two_sum(float a, float b, float& s, float& e) {
  s = __fadd_rn(a, b);
  float bb = __fsub_rn(s, a);
  e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

// requires |a| >= |b| (or a == 0)
SLS_DEV void fast_two_sum(float a, float b, float& s, float& e) {
  s = __fadd_rn(a, b);
  e = __fsub_rn(b, __fsub_rn(s, a));
}

SLS_DEV void two_prod(float a, float b, float& p, float& e) {
  p = __fmul_rn(a, b);
  e = __fmaf_rn(a, b, -p);
}

SLS_DEV dfloat df_make(float hi, float lo) {
  dfloat r;
  r.hi = hi;
  r.lo = lo;
  return r;
}

SLS_DEV dfloat df_from_double(double x) {
  float hi = __double2float_rn(x);
  float lo = __double2float_rn(x - (double)hi);
  return df_make(hi, lo);
}

SLS_DEV double df_to_double(dfloat a) { return (double)a.hi + (double)a.lo; }

SLS_DEV dfloat df_norm(float s, float e) {
  float h, l;
  fast_two_sum(s, e, h, l);
  return df_make(h, l);
}

SLS_DEV dfloat df_add(dfloat a, dfloat b) {
  float s, e;
  two_sum(a.hi, b.hi, s, e);
  float t, f;
  two_sum(a.lo, b.lo, t, f);
  e = __fadd_rn(e, t);
  float h, l;
  fast_two_sum(s, e, h, l);
  l = __fadd_rn(l, f);
  fast_two_sum(h, l, s, e);
  return df_make(s, e);
}

SLS_DEV dfloat df_neg(dfloat a) { return df_make(-a.hi, -a.lo); }

SLS_DEV dfloat df_sub(dfloat a, dfloat b) { return df_add(a, df_neg(b)); }

SLS_DEV dfloat df_mul(dfloat a, dfloat b) {
  float p, e;
  two_prod(a.hi, b.hi, p, e);
  e = __fmaf_rn(a.hi, b.lo, e);
  e = __fmaf_rn(a.lo, b.hi, e);
  float h, l;
  fast_two_sum(p, e, h, l);
  return df_make(h, l);
}

SLS_DEV dfloat df_mul_f(dfloat a, float b) {
  float p, e;
  two_prod(a.hi, b, p, e);
  e = __fmaf_rn(a.lo, b, e);
  float h, l;
  fast_two_sum(p, e, h, l);
  return df_make(h, l);
}

// Compensated accumulation (Dot2 step): (sh, sl) += x * (yh + yl).
// The product x * yh is split exactly by TwoProduct; x * yl and the rounding
// errors are gathered in the low word.
SLS_DEV void dot2_acc(float& sh, float& sl, float x, float yh, float yl) {
  float p, pe;
  two_prod(x, yh, p, pe);
  pe = __fmaf_rn(x, yl, pe);
  float s, e;
  two_sum(sh, p, s, e);
  sh = s;
  sl = __fadd_rn(sl, __fadd_rn(e, pe));
}

// (sh, sl) += (xh + xl) * (yh + yl), both double-float.
SLS_DEV void dot2_acc_df(float& sh, float& sl, dfloat x, dfloat y) {
  float p, pe;
  two_prod(x.hi, y.hi, p, pe);
  pe = __fmaf_rn(x.hi, y.lo, pe);
  pe = __fmaf_rn(x.lo, y.hi, pe);
  float s, e;
  two_sum(sh, p, s, e);
  sh = s;
  sl = __fadd_rn(sl, __fadd_rn(e, pe));
}

// warp-wide sum of a double-float (butterfly; every lane gets the result)
SLS_DEV dfloat warp_sum_df(dfloat v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    dfloat w;
    w.hi = __shfl_xor_sync(0xffffffffu, v.hi, o);
    w.lo = __shfl_xor_sync(0xffffffffu, v.lo, o);
    v = df_add(v, w);
  }
  return v;
}

SLS_DEV float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// ---------------------------------------------------------------------------
// memory-model helpers
// ---------------------------------------------------------------------------

SLS_DEV unsigned ld_acquire_gpu(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

SLS_DEV void st_release_gpu(unsigned* p, unsigned v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

SLS_DEV unsigned atom_add_acq_rel_gpu(unsigned* p, unsigned v) {
  unsigned old;
  asm volatile("atom.add.acq_rel.gpu.global.u32 %0, [%1], %2;"
               : "=r"(old)
               : "l"(p), "r"(v)
               : "memory");
  return old;
}

// ---------------------------------------------------------------------------
// Barrier across a group of co-resident CTAs (all CTAs of a cooperative
// launch, or a subset).  `count` and `gen` live in global memory and start
// at 0.  Every CTA keeps its own copy of the generation in `local_gen`.
// Returns false (and sets *status = SLS_ERR_TIMEOUT) when the wait exceeded
// its iteration limit; the caller must then leave the kernel.
// ---------------------------------------------------------------------------

#ifndef SLS_SPIN_LIMIT
#define SLS_SPIN_LIMIT (1u << 21)  // ~2M polls of ~1 us each: a few seconds
#endif

struct GroupBarrier {
  unsigned* count;
  unsigned* gen;
  unsigned nblocks;
};

SLS_DEV bool group_sync(const GroupBarrier& bar, unsigned& local_gen, int* status,
                        int* smem_flag) {
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    unsigned g = local_gen;
    __threadfence();
    unsigned arrived = atom_add_acq_rel_gpu(bar.count, 1u);
    if (arrived == bar.nblocks - 1) {
      *bar.count = 0;
      __threadfence();
      st_release_gpu(bar.gen, g + 1);
    } else {
      unsigned it = 0;
      while (ld_acquire_gpu(bar.gen) == g) {
        if (++it > SLS_SPIN_LIMIT) {
          ok = 0;
          atomicExch(status, SLS_ERR_TIMEOUT);
          break;
        }
        __nanosleep(64);
      }
    }
    __threadfence();
    local_gen = g + 1;
    // a timeout anywhere (this CTA or another) stops every CTA at its next barrier
    if (ok && *((volatile int*)status) == SLS_ERR_TIMEOUT) ok = 0;
    *smem_flag = ok;
  }
  __syncthreads();
  return *((volatile int*)smem_flag) != 0;
}

// ---------------------------------------------------------------------------
// host-side helpers
// ---------------------------------------------------------------------------

static inline size_t sls_align256(size_t x) { return (x + 255) & ~(size_t)255; }

#define SLS_CUDA_TRY(expr)                          \
  do {                                              \
    cudaError_t e_ = (expr);                        \
    if (e_ != cudaSuccess) return SLS_ERR_CUDA;     \
  } while (0)

namespace sls {
void count_launch(int n);  // library-wide kernel launch counter (api.cu)
}

#define SLS_LAUNCH_CHECK()                                   \
  do {                                                       \
    cudaError_t e_ = cudaGetLastError();                     \
    if (e_ != cudaSuccess) return SLS_ERR_CUDA;              \
    sls::count_launch(1);                                    \
  } while (0)
