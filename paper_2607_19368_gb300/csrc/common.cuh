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
#include <cuda_bf16.h>
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

SLS_DEV float2 f2(dfloat a) { return make_float2(a.hi, a.lo); }

// Elements of the feature matrix as stored: float32, or raw bfloat16 bits
// (uint16), widened to float32 exactly.  phi_ld reads through the read-only
// cache (global memory); phi_ld4 reads the four elements 4 g .. 4 g + 3 of a
// row in shared or global memory (16-byte aligned for float32, 8 for bf16).
SLS_DEV float bf16_bits_to_float(uint32_t u) { return __uint_as_float(u << 16); }
SLS_DEV float phi_ld(const float* p, size_t i) { return __ldg(p + i); }
SLS_DEV float phi_ld(const uint16_t* p, size_t i) {
  return bf16_bits_to_float((uint32_t)__ldg(reinterpret_cast<const unsigned short*>(p) + i));
}
// Stores of a feature value: float32 as is, bfloat16 rounded to nearest even.
SLS_DEV void phi_st(float* p, float v) { *p = v; }
SLS_DEV void phi_st(uint16_t* p, float v) {
  *reinterpret_cast<unsigned short*>(p) = __bfloat16_as_ushort(__float2bfloat16_rn(v));
}
SLS_DEV float4 phi_ld4(const float* p, size_t g) { return reinterpret_cast<const float4*>(p)[g]; }
SLS_DEV float4 phi_ld4(const uint16_t* p, size_t g) {
  const uint2 u = reinterpret_cast<const uint2*>(p)[g];
  return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                     __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
}
SLS_DEV dfloat dfv(float2 a) { return df_make(a.x, a.y); }

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
// packed float32 pairs (sm_100-family f32x2 instructions): one instruction
// performs the same IEEE round-to-nearest operation on both halves.
// ---------------------------------------------------------------------------

typedef unsigned long long f32x2_t;

SLS_DEV f32x2_t pk2(float a, float b) {
  f32x2_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
SLS_DEV void upk2(f32x2_t v, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}
SLS_DEV f32x2_t add2(f32x2_t a, f32x2_t b) {
  f32x2_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
SLS_DEV f32x2_t sub2(f32x2_t a, f32x2_t b) {
  f32x2_t r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
SLS_DEV f32x2_t mul2(f32x2_t a, f32x2_t b) {
  f32x2_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
SLS_DEV f32x2_t fma2(f32x2_t a, f32x2_t b, f32x2_t c) {
  f32x2_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
SLS_DEV f32x2_t neg2(f32x2_t a) { return a ^ 0x8000000080000000ull; }

// Dot2 step on two lanes at once: (sh, sl) += x * (yh + yl), with the
// negated high part nyh = -yh supplied so that TwoProduct needs no sign flip.
SLS_DEV void dot2_acc2n(f32x2_t& sh, f32x2_t& sl, f32x2_t x, f32x2_t yh, f32x2_t nyh,
                        f32x2_t yl) {
  const f32x2_t np = mul2(x, nyh);      // -p, p = fl(x * yh)
  f32x2_t pe = fma2(x, yh, np);          // x * yh - p, exact
  pe = fma2(x, yl, pe);
  const f32x2_t s = sub2(sh, np);        // sh + p
  const f32x2_t bb = sub2(s, sh);
  const f32x2_t e = sub2(sub2(sh, sub2(s, bb)), add2(np, bb));  // TwoSum error
  sh = s;
  sl = add2(sl, add2(e, pe));
}

// Same step when only yh is at hand (the sign flip is an integer xor).
SLS_DEV void dot2_acc2(f32x2_t& sh, f32x2_t& sl, f32x2_t x, f32x2_t yh, f32x2_t yl) {
  const f32x2_t p = mul2(x, yh);
  const f32x2_t np = neg2(p);
  f32x2_t pe = fma2(x, yh, np);
  pe = fma2(x, yl, pe);
  const f32x2_t s = add2(sh, p);
  const f32x2_t bb = sub2(s, sh);
  const f32x2_t e = add2(sub2(sh, sub2(s, bb)), sub2(p, bb));
  sh = s;
  sl = add2(sl, add2(e, pe));
}

// Offset accumulation step on two lanes: (s, lo) += x * (yh + yl), 5
// operations.  s carries a power-of-two offset C and every partial sum it
// accumulates is at most C/2 in magnitude, so s and s1 = fl(s + x * yh) both
// lie in [C/2, 3C/2]: s1 - s is exact, and x * yh - (s1 - s) is the rounding
// error of the fused step, formed by a second FMA (rounded once, at the scale
// of the low part) before x * yl joins it in lo.  The value is (s - C) + lo,
// and s - C is exact (Sterbenz).
SLS_DEV void ofs_fma_acc2(f32x2_t& s, f32x2_t& lo, f32x2_t x, f32x2_t yh, f32x2_t yl) {
  const f32x2_t s1 = fma2(x, yh, s);
  f32x2_t e = fma2(x, yh, sub2(s, s1));  // x * yh - (s1 - s)
  e = fma2(x, yl, e);
  s = s1;
  lo = add2(lo, e);
}

// The same step on one lane.
SLS_DEV void ofs_fma_acc(float& s, float& lo, float x, float yh, float yl) {
  const float s1 = __fmaf_rn(x, yh, s);
  float e = __fmaf_rn(x, yh, __fsub_rn(s, s1));
  e = __fmaf_rn(x, yl, e);
  s = s1;
  lo = __fadd_rn(lo, e);
}

// The offset for a bound B on all partial sums: a power of two C > 2 B (with
// a little slack for the rounding of B itself), clamped to [2^-100, 2^126].
SLS_DEV float ofs_pow2(float bound) {
  const float x = 2.f * bound * 1.00390625f;
  if (!(x >= 0x1p-100f)) return 0x1p-100f;
  if (x >= 0x1p125f) return 0x1p126f;
  return __int_as_float((__float_as_int(x) & 0x7f800000) + 0x00800000);
}

// ---------------------------------------------------------------------------
// shared-memory barriers, bulk copies and named barriers
// ---------------------------------------------------------------------------

SLS_DEV uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

SLS_DEV void mbar_init(uint64_t* bar, unsigned count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

SLS_DEV void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

SLS_DEV void mbar_arrive(uint64_t* bar, unsigned count = 1) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(count)
               : "memory");
}

SLS_DEV void mbar_expect_tx(uint64_t* bar, unsigned bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(
                   smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

SLS_DEV bool mbar_try_wait(uint64_t* bar, unsigned parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Clock cycles after which a wait on a barrier gives up (about a second).
constexpr long long SLS_WAIT_CYCLES = 1ll << 31;

// Bounded wait for the phase with the given parity; false after about a
// second.  try_wait itself suspends the thread in hardware for a while, so
// the loop polls without sleeping (a sleep delays the waiter's wake-up and
// with it the stage hand-over of a copy ring).
SLS_DEV bool mbar_wait(uint64_t* bar, unsigned parity) {
  const long long t0 = clock64();
  for (unsigned it = 0;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 63) == 63 && clock64() - t0 > SLS_WAIT_CYCLES) return false;
  }
}

// One-dimensional bulk copy global -> shared, completion counted on `bar`.
SLS_DEV void bulk_g2s(void* dst, const void* src, unsigned bytes, uint64_t* bar,
                      uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
      "[%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

SLS_DEV uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

SLS_DEV uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

SLS_DEV uint64_t l2_policy_normal() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
  return p;
}

SLS_DEV void named_sync(unsigned id, unsigned nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}


// ---------------------------------------------------------------------------
// memory-model helpers
// ---------------------------------------------------------------------------

SLS_DEV unsigned ld_relaxed_gpu(const unsigned* p) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
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
// launch, or a subset).  `count` lives in global memory and starts at 0;
// `gen` is unused.  Every CTA counts the barriers it passed in `local_gen`.
// Returns false (and sets *status = SLS_ERR_TIMEOUT) when the wait exceeded
// about a second (SLS_WAIT_CYCLES) or another CTA gave up; the caller must
// then leave the kernel.
// ---------------------------------------------------------------------------

struct GroupBarrier {
  unsigned* count;
  unsigned* gen;
  unsigned nblocks;
};

// Bit of the arrival counter that releases every waiter with an error: a CTA
// that gives up sets it, so the other CTAs of the group stop at their next
// barrier instead of waiting out the time limit.
constexpr unsigned SLS_BAR_POISON = 0x80000000u;

SLS_DEV void fence_acq_rel_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }

// Same barrier for kernels where only `nthreads` threads (ids 0..nthreads-1,
// named barrier `bar_id`) take part, e.g. compute warps next to a copy warp.
// One monotonically increasing arrival counter: barrier number n (local_gen
// = n) is complete when the counter reaches (n + 1) * nblocks, so the last
// arrival's own atomic releases the group (one round trip to L2 less than a
// separate release word).  `local_err` is a shared-memory flag the CTA sets
// when one of its own waits gave up; such a CTA poisons the counter instead
// of arriving.
SLS_DEV bool group_sync_named(const GroupBarrier& bar, unsigned& local_gen, int* status,
                              int* smem_flag, volatile int* local_err, unsigned bar_id,
                              unsigned nthreads) {
  named_sync(bar_id, nthreads);
  if (threadIdx.x == 0) {
    int ok = (*local_err == 0);
    if (!ok) {
      atomicOr(bar.count, SLS_BAR_POISON);
    } else {
      const unsigned target = (local_gen + 1) * bar.nblocks;
      // the arrival is a release at GPU scope: it orders the CTA's writes,
      // which the named barrier above ordered before it; the polls are
      // relaxed and the fence after the last one is the acquire (measured
      // 0.6% faster on the Lanczos kernel than a fence before the arrival
      // and acquire polls)
      unsigned v = atom_add_acq_rel_gpu(bar.count, 1u) + 1u;
      const long long t0 = clock64();
      unsigned it = 0;
      while (v < target) {
        if ((++it & 63) == 0 && clock64() - t0 > SLS_WAIT_CYCLES) {
          ok = 0;
          atomicExch(status, SLS_ERR_TIMEOUT);
          atomicOr(bar.count, SLS_BAR_POISON);
          break;
        }
        v = ld_relaxed_gpu(bar.count);
      }
      if (v & SLS_BAR_POISON) ok = 0;
      fence_acq_rel_gpu();
    }
    local_gen += 1;
    *smem_flag = ok;
  }
  named_sync(bar_id, nthreads);
  return *((volatile int*)smem_flag) != 0;
}

// ---------------------------------------------------------------------------
// debug build (-DSLS_DEBUG): device-side bounds guards
// ---------------------------------------------------------------------------
// SLS_DBG_GUARD(status, cond) stmt;  runs stmt only when cond holds; in the
// debug build a false cond records SLS_ERR_BOUNDS in *status (when status is
// not NULL) and skips stmt instead of letting the access go out of bounds.
// In the ordinary build the check and the guard vanish: stmt always runs.
#ifdef SLS_DEBUG
#define SLS_DBG_GUARD(status, cond)                                 \
  if (!(cond)) {                                                    \
    if ((status) != nullptr) atomicExch((status), SLS_ERR_BOUNDS);  \
  } else
#define SLS_DBG_CHECK(status, cond)                                     \
  do {                                                                  \
    if (!(cond) && (status) != nullptr) atomicExch((status), SLS_ERR_BOUNDS); \
  } while (0)
#else
#define SLS_DBG_GUARD(status, cond)
#define SLS_DBG_CHECK(status, cond) \
  do {                              \
  } while (0)
#endif

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
