// SimHash (Sec. 3.3), clusters and the exact-length adjustment (Sec. 3.3),
// macro-token aggregation with positions (Sec. 3.4) and the window
// redundancy score of the adaptive router (Sec. 3.6, Eq. redundancy).
//
// Work is organised by "problems" (one token set compressed on its own; see
// segment.cuh).  The per-problem bookkeeping -- a stable radix sort of
// (code, token), cluster boundaries, the merge or D'Hondt split to exactly m
// groups, group positions and the ordering of groups by position -- runs in
// one 1024-thread CTA per problem and touches only integers.  Reading X and
// writing the macro-token embeddings is spread over the whole GPU.
#include <climits>

#include "common.cuh"
#include "kernels.cuh"
#include "segment.cuh"

namespace sls {

// ============================================================================
// SimHash: code[i] = sum_l [ fl32 dot(U[i,:k], R[l,:k]) > 0 ] << l
// ============================================================================

namespace {

// SimHash of rows 0 .. n-1 with one lane per hyperplane: a warp takes
// 32 / BP rows at a time (BP = bits rounded up to a power of two), lane
// slot * BP + l forms row slot's dot with hyperplane l by the fixed float32
// chain of the specification (acc = 0; for m = 0 .. k-1:
// acc = fl(acc + fl(U[i,m] * R[l,m])), multiply and add rounded separately),
// the row's elements read by every lane of its slot (the same addresses: one
// transaction), R from shared memory with the padded row stride rs (no bank
// conflicts between hyperplanes), and a ballot assembles the codes.  Warps
// w0, w0 + wstride, ... of the launch.
SLS_DEV void simhash_lanes(const float* __restrict__ U, int64_t n, int ldu, int kk,
                           const float* __restrict__ Rs, int rs, int bits,
                           uint32_t* __restrict__ codes, int64_t w0, int64_t wstride) {
  int BP = 1;
  while (BP < bits) BP <<= 1;
  const int lane = threadIdx.x & 31;
  const int slot = lane / BP, l = lane % BP, rpw = 32 / BP;
  const float* rl = Rs + (size_t)min(l, max(bits, 1) - 1) * rs;
  for (int64_t w = w0; w * rpw < n; w += wstride) {
    const int64_t i = w * rpw + slot;
    const bool live = i < n;
    float acc = 0.0f;
    if (live) {
      const float* u = U + i * ldu;
      for (int m = 0; m < kk; ++m) acc = __fadd_rn(acc, __fmul_rn(__ldg(u + m), rl[m]));
    }
    const unsigned ball = __ballot_sync(0xffffffffu, live && l < bits && acc > 0.0f);
    if (live && l == 0) {
      const unsigned mask = (BP == 32) ? 0xffffffffu : ((1u << BP) - 1u);
      codes[i] = (ball >> (slot * BP)) & mask;
    }
  }
}

// R (bits x kk) into shared memory with row stride kk + 1
SLS_DEV void simhash_stage_R(const float* __restrict__ R, int ldr, int bits, int kk, float* Rs) {
  for (int e = threadIdx.x; e < bits * kk; e += blockDim.x)
    Rs[(e / kk) * (kk + 1) + e % kk] = R[(e / kk) * ldr + e % kk];
}

__global__ void __launch_bounds__(256)
simhash_kernel(const float* __restrict__ U, int64_t N, int k, int ldu,
               const int32_t* __restrict__ k_dev, const float* __restrict__ R, int bits,
               int ldr, uint32_t* __restrict__ codes) {
  extern __shared__ float Rs[];
  int kk = k;
  if (k_dev) kk = min(kk, max(0, (int)*k_dev));
  simhash_stage_R(R, ldr, bits, kk, Rs);
  __syncthreads();
  const int64_t wpb = blockDim.x >> 5;
  simhash_lanes(U, N, ldu, kk, Rs, kk + 1, bits, codes,
                (int64_t)blockIdx.x * wpb + (threadIdx.x >> 5), (int64_t)gridDim.x * wpb);
}

// Batched over spectral problems: rows of problem p start at phi_row, k is
// the problem's r_eff, bits its own bit count; simhash_lanes per problem.
__global__ void __launch_bounds__(256)
simhash_batched_kernel(const ProbDesc* __restrict__ probs, const int* __restrict__ spec_list,
                       const int* __restrict__ nspec_dev, int nspec_max,
                       const int* __restrict__ r_eff, const float* __restrict__ U, int ldu,
                       const float* __restrict__ R, int ldr, uint32_t* __restrict__ codes) {
  extern __shared__ float Rs[];
  const int s = blockIdx.y;
  int nspec = nspec_max;
  if (nspec_dev) nspec = min(nspec, *nspec_dev);
  if (s >= nspec) return;
  const ProbDesc P = probs[spec_list ? spec_list[s] : s];
  const int kk = min(ldu, max(0, r_eff[s]));
  simhash_stage_R(R, ldr, P.bits, kk, Rs);
  __syncthreads();
  const int64_t wpb = blockDim.x >> 5;
  simhash_lanes(U + (int64_t)P.phi_row * ldu, P.n, ldu, kk, Rs, kk + 1, P.bits,
                codes + P.phi_row, (int64_t)blockIdx.x * wpb + (threadIdx.x >> 5),
                (int64_t)gridDim.x * wpb);
}

// Small problems (windows of at most SH_FLAT_MAX tokens): one thread per
// (problem, row) over all spectral problems, R read through the read-only
// cache (row l of R at R + l * ldr), the same float32 chain as simhash_lanes.
constexpr int SH_FLAT_MAX = 64;

__global__ void __launch_bounds__(256)
simhash_flat_kernel(const ProbDesc* __restrict__ probs, const int* __restrict__ spec_list,
                    const int* __restrict__ nspec_dev, int nspec_max, int nmax,
                    const int* __restrict__ r_eff, const float* __restrict__ U, int ldu,
                    const float* __restrict__ R, int ldr, uint32_t* __restrict__ codes) {
  int nspec = nspec_max;
  if (nspec_dev) nspec = min(nspec, *nspec_dev);
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int s = (int)(t / nmax), i = (int)(t % nmax);
  if (s >= nspec) return;
  const ProbDesc P = probs[spec_list ? spec_list[s] : s];
  if (i >= P.n) return;
  const int k = min(ldu, max(0, r_eff[s]));
  const float* __restrict__ u = U + (P.phi_row + i) * ldu;
  float acc[SLS_MAX_BITS];
#pragma unroll
  for (int l = 0; l < SLS_MAX_BITS; ++l) acc[l] = 0.0f;
  for (int m = 0; m < k; ++m) {
    const float um = __ldg(u + m);
#pragma unroll
    for (int l = 0; l < SLS_MAX_BITS; ++l)
      if (l < P.bits) acc[l] = __fadd_rn(acc[l], __fmul_rn(um, __ldg(R + (size_t)l * ldr + m)));
  }
  uint32_t code = 0;
#pragma unroll
  for (int l = 0; l < SLS_MAX_BITS; ++l)
    if (l < P.bits && acc[l] > 0.0f) code |= (1u << l);
  codes[P.phi_row + i] = code;
}

// ============================================================================
// block-level integer primitives (1024 threads)
// ============================================================================

constexpr int SEG_T = 1024;
constexpr int SEG_W = SEG_T / 32;

SLS_DEV unsigned lanemask_lt() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Exclusive scan of 1024 per-thread values; returns the exclusive prefix of
// the calling thread, *total receives the sum.  sh: SEG_W + 1 ints.
template <typename T>
SLS_DEV T block_excl_scan(T v, T* sh, T* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  T x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    T y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    T w = (lane < SEG_W) ? sh[lane] : (T)0;
    T z = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      T y = __shfl_up_sync(0xffffffffu, z, o);
      if (lane >= o) z += y;
    }
    if (lane < SEG_W) sh[lane] = z - w;
    if (lane == SEG_W - 1) sh[SEG_W] = z;
  }
  __syncthreads();
  const T res = sh[warp] + x - v;
  *total = sh[SEG_W];
  __syncthreads();
  return res;
}

// Exclusive scan of in[0..n) into out (may alias); returns the total.
// Each thread scans a contiguous chunk serially.
template <typename T>
SLS_DEV T block_scan_array(const T* in, T* out, int n, T* sh) {
  const int tid = threadIdx.x;
  const int chunk = (n + SEG_T - 1) / SEG_T;
  const int b = min(n, tid * chunk), e = min(n, b + chunk);
  T s = 0;
  for (int i = b; i < e; ++i) s += in[i];
  T total;
  T off = block_excl_scan<T>(s, sh, &total);
  for (int i = b; i < e; ++i) {
    const T v = in[i];
    out[i] = off;
    off += v;
  }
  __syncthreads();
  return total;
}

template <typename T>
SLS_DEV T block_sum(T v, T* sh) {
  T total;
  block_excl_scan<T>(v, sh, &total);
  return total;
}

// Stable LSD radix sort of (key, val) pairs on the low key_bits bits, one
// 8-bit digit per pass, ping-ponging between the (ka, va) and (kb, vb)
// buffers in global memory.  On return (ka, va) point at the sorted data.
// sh: 256 + 256 + SEG_W * 256 ints.
template <typename K>
SLS_DEV void block_radix_sort(K*& ka, int*& va, K*& kb, int*& vb, int n, int key_bits, int* sh) {
  int* base = sh;
  int* tot = sh + 256;
  int* wc = sh + 512;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int shift = 0; shift < key_bits; shift += 8) {
    if (tid < 256) base[tid] = 0;
    __syncthreads();
    for (int i = tid; i < n; i += SEG_T) atomicAdd(&base[(int)((ka[i] >> shift) & 255)], 1);
    __syncthreads();
    if (tid < 256) {
      // exclusive scan of 256 bins by the first 8 warps
      int v = base[tid];
      int x = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      if (lane == 31) tot[warp] = x;
      __syncwarp();
      x -= v;
      base[tid] = x;  // warp-local exclusive prefix
    }
    __syncthreads();
    if (tid < 256) {
      int add = 0;
      for (int w = 0; w < warp; ++w) add += tot[w];
      base[tid] += add;
    }
    __syncthreads();
    for (int t0 = 0; t0 < n; t0 += SEG_T) {
      for (int e = tid; e < SEG_W * 256; e += SEG_T) wc[e] = 0;
      __syncthreads();
      const int i = t0 + tid;
      const bool valid = i < n;
      K key = 0;
      int val = 0;
      unsigned dg = 256u + (unsigned)lane;
      if (valid) {
        key = ka[i];
        val = va[i];
        dg = (unsigned)((key >> shift) & 255);
      }
      const unsigned peers = __match_any_sync(0xffffffffu, dg);
      const int rank = __popc(peers & lanemask_lt());
      if (valid && rank == 0) wc[warp * 256 + dg] = __popc(peers);
      __syncthreads();
      if (tid < 256) {
        int run = 0;
        for (int w = 0; w < SEG_W; ++w) {
          const int c = wc[w * 256 + tid];
          wc[w * 256 + tid] = run;
          run += c;
        }
        tot[tid] = run;
      }
      __syncthreads();
      if (valid) {
        const int pos = base[dg] + wc[warp * 256 + dg] + rank;
        kb[pos] = key;
        vb[pos] = val;
      }
      __syncthreads();
      if (tid < 256) base[tid] += tot[tid];
      __syncthreads();
    }
    K* tk = ka;
    ka = kb;
    kb = tk;
    int* tv = va;
    va = vb;
    vb = tv;
  }
}

SLS_DEV int bit_length_u64(unsigned long long x) { return x ? 64 - __clzll((long long)x) : 0; }

// Per-problem scratch layout (ints unless noted), identical on host and device.
struct SegLayout {
  size_t ka, kb, va, vb, f, cst, grp, gst, gmax, gmin, gsum, ok_a, ok_b, ov_a, ov_b, oidx, rep,
      seat, gbar, ghist, gcsum, total;
};

__host__ __device__ inline size_t seg_al(size_t x) { return (x + 255) & ~(size_t)255; }

__host__ __device__ inline SegLayout seg_layout(int64_t nmax, int64_t mmax) {
  SegLayout L;
  size_t o = 0;
  const size_t n1 = (size_t)nmax + 1, m1 = (size_t)mmax + 1;
  L.ka = o;   o += seg_al(n1 * 8);   // keys (uint32 for codes, uint64 reused)
  L.kb = o;   o += seg_al(n1 * 8);
  L.va = o;   o += seg_al(n1 * 4);
  L.vb = o;   o += seg_al(n1 * 4);
  L.f = o;    o += seg_al(n1 * 4);
  L.cst = o;  o += seg_al(n1 * 4);
  L.grp = o;  o += seg_al(n1 * 4);
  L.gst = o;  o += seg_al(m1 * 4);
  L.gmax = o; o += seg_al(m1 * 4);
  L.gmin = o; o += seg_al(m1 * 4);
  L.gsum = o; o += seg_al(m1 * 8);
  L.ok_a = o; o += seg_al(m1 * 8);
  L.ok_b = o; o += seg_al(m1 * 8);
  L.ov_a = o; o += seg_al(m1 * 4);
  L.ov_b = o; o += seg_al(m1 * 4);
  L.oidx = o; o += seg_al(m1 * 4);
  L.rep = o;  o += seg_al(m1 * 4);
  L.seat = o; o += seg_al(n1 * 4);
  // grid version (one large problem): barrier words, digit counts per CTA,
  // CTA sums of the scans
  L.gbar = o;  o += 256;
  L.ghist = o; o += seg_al((size_t)256 * 256 * 4);
  L.gcsum = o; o += seg_al((size_t)256 * 4);
  L.total = o;
  return L;
}

// The segment kernel's sort buffers in shared memory (byte offsets): keys
// and values of the (code, token) sort and the 64-bit order keys with their
// values.
constexpr size_t SEG_SMEM_MAX = 180 * 1024;  // beside 35 KB of static shared memory

struct SegSmem {
  size_t ka, kb, va, vb, oka, okb, ova, ovb, total;
};

__host__ __device__ inline SegSmem seg_smem_layout(int64_t nmax, int64_t mmax) {
  SegSmem S;
  const size_t n1 = (size_t)nmax + 1, m1 = (size_t)mmax + 1;
  auto al = [](size_t x) { return (x + 15) & ~(size_t)15; };
  size_t o = 0;
  S.ka = o;  o += al(n1 * 4);
  S.kb = o;  o += al(n1 * 4);
  S.va = o;  o += al(n1 * 4);
  S.vb = o;  o += al(n1 * 4);
  S.oka = o; o += al(m1 * 8);
  S.okb = o; o += al(m1 * 8);
  S.ova = o; o += al(m1 * 4);
  S.ovb = o; o += al(m1 * 4);
  S.total = o;
  return S;
}

// Number of D'Hondt quotients n/m (2 <= m <= n) that are >= a / 2^40.
SLS_DEV long long dhondt_count_ge(long long n, long long a) {
  if (n < 2) return 0;
  long long k = (a == 0) ? n : min(n, (n << 40) / a);
  return k > 1 ? k - 1 : 0;
}

// ============================================================================
// segment kernel: one CTA per problem
// ============================================================================

__global__ void __launch_bounds__(SEG_T, 1)
segment_kernel(const ProbDesc* __restrict__ probs, int nprob, const uint32_t* __restrict__ codes,
               int pos_scheme, int pos_mode, char* scratch, size_t pstride, int64_t nmax,
               int64_t mmax, int* __restrict__ perm, int* __restrict__ mstart,
               int* __restrict__ mlen, int32_t* __restrict__ pos_out,
               int32_t* __restrict__ tok2macro, int chunk_done, int sort_in_smem) {
  __shared__ int sh_sort[512 + SEG_W * 256];
  __shared__ long long sh_ll[SEG_W + 1];
  __shared__ int sh_i[SEG_W + 1];
  extern __shared__ __align__(16) unsigned char seg_dyn[];
  const int tid = threadIdx.x;
  const SegLayout L = seg_layout(nmax, mmax);
  char* sb = scratch + (size_t)blockIdx.x * pstride;
  // the radix sorts' key and value buffers: in shared memory when the launch
  // gave room for them (seg_smem_layout), else in the problem's scratch
  const SegSmem SL = seg_smem_layout(nmax, mmax);
  char* sortb = sort_in_smem ? reinterpret_cast<char*>(seg_dyn) : nullptr;

  for (int p = blockIdx.x; p < nprob; p += gridDim.x) {
    const ProbDesc P = probs[p];
    const int n = P.n, M = P.m;
    if (n <= 0 || M <= 0) continue;
    if (chunk_done && !P.spectral) {
      // outputs already written by the score pass: nothing to aggregate
      for (int t = tid; t < M; t += SEG_T) mlen[P.out0 + t] = 0;
      continue;
    }
    int* va = reinterpret_cast<int*>(sortb ? sortb + SL.va : sb + L.va);
    int* vb = reinterpret_cast<int*>(sortb ? sortb + SL.vb : sb + L.vb);
    int* f = reinterpret_cast<int*>(sb + L.f);
    int* cst = reinterpret_cast<int*>(sb + L.cst);
    int* grp = reinterpret_cast<int*>(sb + L.grp);
    int* gst = reinterpret_cast<int*>(sb + L.gst);
    int* gmax = reinterpret_cast<int*>(sb + L.gmax);
    int* gmin = reinterpret_cast<int*>(sb + L.gmin);
    unsigned long long* gsum = reinterpret_cast<unsigned long long*>(sb + L.gsum);
    int* oidx = reinterpret_cast<int*>(sb + L.oidx);
    int* rep = reinterpret_cast<int*>(sb + L.rep);
    int* seat = reinterpret_cast<int*>(sb + L.seat);
    bool merged = false;

    if (P.spectral) {
      // ---- stable sort of (code, token) ----
      uint32_t* ka = reinterpret_cast<uint32_t*>(sortb ? sortb + SL.ka : sb + L.ka);
      uint32_t* kb = reinterpret_cast<uint32_t*>(sortb ? sortb + SL.kb : sb + L.kb);
      for (int i = tid; i < n; i += SEG_T) {
        ka[i] = codes[P.phi_row + i];
        va[i] = i;
      }
      __syncthreads();
      block_radix_sort<uint32_t>(ka, va, kb, vb, n, P.bits, sh_sort);
      // ---- clusters: runs of equal codes ----
      for (int s = tid; s < n; s += SEG_T) f[s] = (s == 0 || ka[s] != ka[s - 1]) ? 1 : 0;
      __syncthreads();
      const int C = block_scan_array<int>(f, grp, n, sh_i);  // grp[s] = clusters before s
      for (int s = tid; s < n; s += SEG_T)
        if (f[s]) cst[grp[s]] = s;
      if (tid == 0) cst[C] = n;
      __syncthreads();
      if (C >= M) {
        // merge: the cluster of rank t joins group floor(t M / C)
        merged = (C > M);
        for (int t = tid; t < C; t += SEG_T) {
          const int g = (int)(((long long)t * M) / C);
          const int gp = (t == 0) ? -1 : (int)(((long long)(t - 1) * M) / C);
          if (g != gp) gst[g] = cst[t];
        }
      } else {
        // split: D'Hondt seats, one guaranteed per cluster, ties to the lower code
        const long long K = (long long)(M - C);
        int maxn = 0;
        for (int t = tid; t < C; t += SEG_T) maxn = max(maxn, cst[t + 1] - cst[t]);
        // block max via the sum helper on a per-thread max is not valid; use atomics
        if (tid == 0) sh_i[0] = 0;
        __syncthreads();
        atomicMax(&sh_i[0], maxn);
        __syncthreads();
        maxn = sh_i[0];
        __syncthreads();
        long long lo = 0, hi = ((long long)maxn) << 40;
        while (hi - lo > 1) {
          const long long mid = lo + (hi - lo) / 2;
          long long c = 0;
          for (int t = tid; t < C; t += SEG_T) c += dhondt_count_ge(cst[t + 1] - cst[t], mid);
          c = block_sum<long long>(c, sh_ll);
          if (c >= K) lo = mid;
          else hi = mid;
        }
        // seats strictly above the K-th quotient, and ties at it (<= 1 per cluster)
        long long gt_sum = 0;
        for (int t = tid; t < C; t += SEG_T) {
          const long long nt = cst[t + 1] - cst[t];
          const long long ge = dhondt_count_ge(nt, lo);
          const long long gt = dhondt_count_ge(nt, lo + 1);
          seat[t] = (int)gt;
          f[t] = (int)(ge - gt);
          gt_sum += gt;
        }
        gt_sum = block_sum<long long>(gt_sum, sh_ll);
        const int R = (int)(K - gt_sum);
        __syncthreads();
        // exclusive scan of the tie flags in cluster order
        int* eqs = grp;  // reuse as scratch (size >= C)
        block_scan_array<int>(f, eqs, C, sh_i);
        for (int t = tid; t < C; t += SEG_T) {
          const int extra = (f[t] && eqs[t] < R) ? 1 : 0;
          seat[t] = 1 + seat[t] + extra;
        }
        __syncthreads();
        int* so = f;  // seat offsets
        block_scan_array<int>(seat, so, C, sh_i);
        for (int t = tid; t < C; t += SEG_T) {
          const int nt = cst[t + 1] - cst[t], pt = seat[t];
          const int q = nt / pt, rem = nt % pt;
          for (int k = 0; k < pt; ++k) {
            const int off = (k < rem) ? k * (q + 1) : rem * (q + 1) + (k - rem) * q;
            gst[so[t] + k] = cst[t] + off;
          }
        }
      }
      if (tid == 0) gst[M] = n;
      __syncthreads();
    } else {
      // chunk: contiguous groups (array_split into m, or runs of k)
      for (int i = tid; i < n; i += SEG_T) va[i] = i;
      for (int g = tid; g < M; g += SEG_T) {
        int off;
        if (P.chunk_k > 0) {
          off = min(n, g * P.chunk_k);
        } else {
          const int q = n / M, rem = n % M;
          off = (g < rem) ? g * (q + 1) : rem * (q + 1) + (g - rem) * q;
        }
        gst[g] = off;
      }
      if (tid == 0) gst[M] = n;
      __syncthreads();
    }
    const int* perm_l = va;  // sorted position -> local token
    // ---- group id of every sorted position ----
    for (int s = tid; s < n; s += SEG_T) f[s] = 0;
    __syncthreads();
    for (int g = tid; g < M; g += SEG_T) f[gst[g]] = 1;
    __syncthreads();
    block_scan_array<int>(f, grp, n, sh_i);
    for (int s = tid; s < n; s += SEG_T) grp[s] = grp[s] + f[s] - 1;
    for (int g = tid; g < M; g += SEG_T) {
      gmax[g] = -1;
      gmin[g] = INT_MAX;
      gsum[g] = 0ull;
    }
    __syncthreads();
    for (int s = tid; s < n; s += SEG_T) {
      const int g = grp[s], i = perm_l[s];
      atomicMax(&gmax[g], i);
      atomicMin(&gmin[g], i);
      if (pos_scheme == SLS_POS_MEAN) atomicAdd(&gsum[g], (unsigned long long)i);
    }
    __syncthreads();
    // ---- representative positions ----
    if (pos_scheme == SLS_POS_MEDIAN && merged) {
      // members of merged groups are not in token order: sort (group, token)
      uint32_t* ka = reinterpret_cast<uint32_t*>(sortb ? sortb + SL.ka : sb + L.ka);
      uint32_t* kb = reinterpret_cast<uint32_t*>(sortb ? sortb + SL.kb : sb + L.kb);
      int* xa = seat;
      int* xb = cst;
      for (int s = tid; s < n; s += SEG_T) ka[perm_l[s]] = (uint32_t)grp[s];
      for (int i = tid; i < n; i += SEG_T) xa[i] = i;
      __syncthreads();
      block_radix_sort<uint32_t>(ka, xa, kb, xb, n, bit_length_u64((unsigned long long)M), sh_sort);
      for (int g = tid; g < M; g += SEG_T) rep[g] = xa[gst[g] + (gst[g + 1] - gst[g] - 1) / 2];
    } else {
      for (int g = tid; g < M; g += SEG_T) {
        const int len = gst[g + 1] - gst[g];
        int rp;
        if (pos_scheme == SLS_POS_MAX) rp = gmax[g];
        else if (pos_scheme == SLS_POS_MEDIAN) rp = perm_l[gst[g] + (len - 1) / 2];
        else rp = (int)((2ull * gsum[g] + (unsigned long long)len) / (2ull * (unsigned long long)len));
        rep[g] = rp;
      }
    }
    __syncthreads();
    // ---- order groups by (position, first token) ----
    {
      unsigned long long* oka =
          reinterpret_cast<unsigned long long*>(sortb ? sortb + SL.oka : sb + L.ok_a);
      unsigned long long* okb =
          reinterpret_cast<unsigned long long*>(sortb ? sortb + SL.okb : sb + L.ok_b);
      int* ova = reinterpret_cast<int*>(sortb ? sortb + SL.ova : sb + L.ov_a);
      int* ovb = reinterpret_cast<int*>(sortb ? sortb + SL.ovb : sb + L.ov_b);
      for (int g = tid; g < M; g += SEG_T) {
        oka[g] = (unsigned long long)rep[g] * (unsigned long long)n + (unsigned long long)gmin[g];
        ova[g] = g;
      }
      __syncthreads();
      const int kbits = bit_length_u64((unsigned long long)n * (unsigned long long)n);
      block_radix_sort<unsigned long long>(oka, ova, okb, ovb, M, kbits, sh_sort);
      for (int t = tid; t < M; t += SEG_T) {
        const int g = ova[t];
        oidx[g] = t;
        const int64_t mrow = P.out0 + t;
        mstart[mrow] = (int)(P.tok_row + gst[g]);
        mlen[mrow] = gst[g + 1] - gst[g];
        pos_out[mrow] = (pos_mode == SLS_MODE_COMPACT) ? (P.out_local + t) : (P.pos0 + rep[g]);
      }
      __syncthreads();
      for (int s = tid; s < n; s += SEG_T) {
        const int i = perm_l[s];
        perm[P.tok_row + s] = (int)(P.tok_row + i);
        tok2macro[P.tok_row + i] = P.out_local + oidx[grp[s]];
      }
      __syncthreads();
    }
  }
}

// ============================================================================
// segment kernel for one large problem: the same computation spread over a
// cooperative grid (G CTAs of SEG_T threads), for the single-prompt pass
// ============================================================================

constexpr int SEGG_MAX = 256;           // CTAs of the grid segment kernel, at most
constexpr int64_t SEG_GRID_MIN_N = 8192;  // tokens from which one problem uses the grid kernel

struct GridSync {
  GroupBarrier bar;
  unsigned lgen;
  int* status;
  int* sflag;
  volatile int* serr;
};

SLS_DEV bool gsync(GridSync& gs) {
  return group_sync_named(gs.bar, gs.lgen, gs.status, gs.sflag, gs.serr, 1, SEG_T);
}

// Exclusive scan of in[0..n) into out over the grid; CTA b owns the slice
// [b n / G, (b+1) n / G).  On return this CTA's slice of out is final and the
// total is returned; other slices are final after the next gsync.  csum: G
// ints in global memory.
SLS_DEV bool grid_scan(const int* in, int* out, int n, int* csum, GridSync& gs, int* sh,
                       int* total) {
  const int G = gridDim.x, b = blockIdx.x, tid = threadIdx.x;
  const int c0 = (int)((int64_t)b * n / G), c1 = (int)((int64_t)(b + 1) * n / G);
  const int loc = block_scan_array<int>(in + c0, out + c0, c1 - c0, sh);
  if (tid == 0) csum[b] = loc;
  if (!gsync(gs)) return false;
  int pre = 0, tot = 0;
  for (int c = tid; c < G; c += SEG_T) {
    const int v = csum[c];
    tot += v;
    if (c < b) pre += v;
  }
  pre = block_sum<int>(pre, sh);
  tot = block_sum<int>(tot, sh);
  for (int i = c0 + tid; i < c1; i += SEG_T) out[i] += pre;
  *total = tot;
  __syncthreads();
  return true;
}

// One stable LSD pass (8 bits at `shift`) of (key, val) pairs over the grid:
// per-CTA digit counts, the prefix over (digit, CTA), then the CTA's slice is
// scattered in order (stable within the CTA as in block_radix_sort).
// hist: 256 x G ints in global memory.  sh: 256 + 256 + SEG_W * 256 ints.
template <typename K>
SLS_DEV bool grid_radix_pass(const K* ka, const int* va, K* kb, int* vb, int n, int shift,
                             int* hist, GridSync& gs, int* sh) {
  const int G = gridDim.x, b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int* base = sh;
  int* tot = sh + 256;
  int* wc = sh + 512;
  const int c0 = (int)((int64_t)b * n / G), c1 = (int)((int64_t)(b + 1) * n / G);
  if (tid < 256) base[tid] = 0;
  __syncthreads();
  for (int i = c0 + tid; i < c1; i += SEG_T) atomicAdd(&base[(int)((ka[i] >> shift) & 255)], 1);
  __syncthreads();
  if (tid < 256) hist[tid * G + b] = base[tid];
  if (!gsync(gs)) return false;
  if (tid < 256) {
    int all = 0, part = 0;
    for (int c = 0; c < G; ++c) {
      const int h = hist[tid * G + c];
      all += h;
      if (c < b) part += h;
    }
    // exclusive scan of the digit totals by the first 8 warps
    int x = all;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) tot[warp] = x;
    base[tid] = x - all + part;
  }
  __syncthreads();
  if (tid < 256) {
    int add = 0;
    for (int w = 0; w < warp; ++w) add += tot[w];
    base[tid] += add;
  }
  __syncthreads();
  for (int t0 = c0; t0 < c1; t0 += SEG_T) {
    for (int e = tid; e < SEG_W * 256; e += SEG_T) wc[e] = 0;
    __syncthreads();
    const int i = t0 + tid;
    const bool valid = i < c1;
    K key = 0;
    int val = 0;
    unsigned dg = 256u + (unsigned)lane;
    if (valid) {
      key = ka[i];
      val = va[i];
      dg = (unsigned)((key >> shift) & 255);
    }
    const unsigned peers = __match_any_sync(0xffffffffu, dg);
    const int rank = __popc(peers & lanemask_lt());
    if (valid && rank == 0) wc[warp * 256 + dg] = __popc(peers);
    __syncthreads();
    if (tid < 256) {
      int run = 0;
      for (int w = 0; w < SEG_W; ++w) {
        const int c = wc[w * 256 + tid];
        wc[w * 256 + tid] = run;
        run += c;
      }
      tot[tid] = run;
    }
    __syncthreads();
    if (valid) {
      const int pos = base[dg] + wc[warp * 256 + dg] + rank;
      kb[pos] = key;
      vb[pos] = val;
    }
    __syncthreads();
    if (tid < 256) base[tid] += tot[tid];
    __syncthreads();
  }
  return gsync(gs);
}

template <typename K>
SLS_DEV bool grid_radix_sort(K*& ka, int*& va, K*& kb, int*& vb, int n, int key_bits, int* hist,
                             GridSync& gs, int* sh) {
  for (int shift = 0; shift < key_bits; shift += 8) {
    if (!grid_radix_pass<K>(ka, va, kb, vb, n, shift, hist, gs, sh)) return false;
    K* tk = ka;
    ka = kb;
    kb = tk;
    int* tv = va;
    va = vb;
    vb = tv;
  }
  return true;
}

__global__ void __launch_bounds__(SEG_T, 1)
segment_grid_kernel(const ProbDesc* __restrict__ probs, const uint32_t* __restrict__ codes,
                    int pos_scheme, int pos_mode, char* sb, int64_t nmax, int64_t mmax,
                    int* __restrict__ perm, int* __restrict__ mstart, int* __restrict__ mlen,
                    int32_t* __restrict__ pos_out, int32_t* __restrict__ tok2macro,
                    int* status, int chunk_done) {
  __shared__ int sh_sort[512 + SEG_W * 256];
  __shared__ long long sh_ll[SEG_W + 1];
  __shared__ int sh_i[SEG_W + 1];
  __shared__ int sflag;
  __shared__ volatile int serr;
  const int tid = threadIdx.x, G = gridDim.x, b = blockIdx.x;
  const SegLayout L = seg_layout(nmax, mmax);
  if (tid == 0) serr = 0;
  __syncthreads();
  GridSync gs{GroupBarrier{reinterpret_cast<unsigned*>(sb + L.gbar),
                           reinterpret_cast<unsigned*>(sb + L.gbar) + 32, (unsigned)G},
              0u, status, &sflag, &serr};
  const ProbDesc P = probs[0];
  const int n = P.n, M = P.m;
  if (n <= 0 || M <= 0) return;
  if (chunk_done && !P.spectral) {  // the whole grid leaves before any grid barrier
    for (int t = b * SEG_T + tid; t < M; t += G * SEG_T) mlen[P.out0 + t] = 0;
    return;
  }
  uint32_t* ka = reinterpret_cast<uint32_t*>(sb + L.ka);
  uint32_t* kb = reinterpret_cast<uint32_t*>(sb + L.kb);
  int* va = reinterpret_cast<int*>(sb + L.va);
  int* vb = reinterpret_cast<int*>(sb + L.vb);
  int* f = reinterpret_cast<int*>(sb + L.f);
  int* cst = reinterpret_cast<int*>(sb + L.cst);
  int* grp = reinterpret_cast<int*>(sb + L.grp);
  int* gst = reinterpret_cast<int*>(sb + L.gst);
  int* gmax = reinterpret_cast<int*>(sb + L.gmax);
  int* gmin = reinterpret_cast<int*>(sb + L.gmin);
  unsigned long long* gsum = reinterpret_cast<unsigned long long*>(sb + L.gsum);
  int* oidx = reinterpret_cast<int*>(sb + L.oidx);
  int* rep = reinterpret_cast<int*>(sb + L.rep);
  int* seat = reinterpret_cast<int*>(sb + L.seat);
  int* hist = reinterpret_cast<int*>(sb + L.ghist);
  int* csum = reinterpret_cast<int*>(sb + L.gcsum);
  const int s0 = (int)((int64_t)b * n / G), s1 = (int)((int64_t)(b + 1) * n / G);
  const int m0 = (int)((int64_t)b * M / G), m1 = (int)((int64_t)(b + 1) * M / G);
  bool merged = false;

  if (P.spectral) {
    // ---- stable sort of (code, token) ----
    for (int i = s0 + tid; i < s1; i += SEG_T) {
      ka[i] = codes[P.phi_row + i];
      va[i] = i;
    }
    if (!gsync(gs)) return;
    if (!grid_radix_sort<uint32_t>(ka, va, kb, vb, n, P.bits, hist, gs, sh_sort)) return;
    // ---- clusters: runs of equal codes ----
    for (int s = s0 + tid; s < s1; s += SEG_T) f[s] = (s == 0 || ka[s] != ka[s - 1]) ? 1 : 0;
    __syncthreads();
    int C = 0;
    if (!grid_scan(f, grp, n, csum, gs, sh_i, &C)) return;  // grp[s] = clusters before s
    for (int s = s0 + tid; s < s1; s += SEG_T)
      if (f[s]) cst[grp[s]] = s;
    if (b == 0 && tid == 0) cst[C] = n;
    if (!gsync(gs)) return;
    if (C >= M) {
      // merge: the cluster of rank t joins group floor(t M / C)
      merged = (C > M);
      const int t0 = (int)((int64_t)b * C / G), t1 = (int)((int64_t)(b + 1) * C / G);
      for (int t = t0 + tid; t < t1; t += SEG_T) {
        const int g = (int)(((long long)t * M) / C);
        const int gp = (t == 0) ? -1 : (int)(((long long)(t - 1) * M) / C);
        if (g != gp) gst[g] = cst[t];
      }
    } else if (b == 0) {
      // split: D'Hondt seats, one guaranteed per cluster, ties to the lower
      // code (few clusters: one CTA)
      const long long K = (long long)(M - C);
      int maxn = 0;
      for (int t = tid; t < C; t += SEG_T) maxn = max(maxn, cst[t + 1] - cst[t]);
      if (tid == 0) sh_i[0] = 0;
      __syncthreads();
      atomicMax(&sh_i[0], maxn);
      __syncthreads();
      maxn = sh_i[0];
      __syncthreads();
      long long lo = 0, hi = ((long long)maxn) << 40;
      while (hi - lo > 1) {
        const long long mid = lo + (hi - lo) / 2;
        long long c = 0;
        for (int t = tid; t < C; t += SEG_T) c += dhondt_count_ge(cst[t + 1] - cst[t], mid);
        c = block_sum<long long>(c, sh_ll);
        if (c >= K) lo = mid;
        else hi = mid;
      }
      long long gt_sum = 0;
      for (int t = tid; t < C; t += SEG_T) {
        const long long nt = cst[t + 1] - cst[t];
        const long long ge = dhondt_count_ge(nt, lo);
        const long long gt = dhondt_count_ge(nt, lo + 1);
        seat[t] = (int)gt;
        f[t] = (int)(ge - gt);
        gt_sum += gt;
      }
      gt_sum = block_sum<long long>(gt_sum, sh_ll);
      const int R = (int)(K - gt_sum);
      __syncthreads();
      int* eqs = grp;  // scratch (size >= C)
      block_scan_array<int>(f, eqs, C, sh_i);
      for (int t = tid; t < C; t += SEG_T) {
        const int extra = (f[t] && eqs[t] < R) ? 1 : 0;
        seat[t] = 1 + seat[t] + extra;
      }
      __syncthreads();
      int* so = f;
      block_scan_array<int>(seat, so, C, sh_i);
      for (int t = tid; t < C; t += SEG_T) {
        const int nt = cst[t + 1] - cst[t], pt = seat[t];
        const int q = nt / pt, rem = nt % pt;
        for (int k = 0; k < pt; ++k) {
          const int off = (k < rem) ? k * (q + 1) : rem * (q + 1) + (k - rem) * q;
          gst[so[t] + k] = cst[t] + off;
        }
      }
    }
  } else {
    // chunk: contiguous groups (array_split into m, or runs of k)
    for (int i = s0 + tid; i < s1; i += SEG_T) va[i] = i;
    for (int g = m0 + tid; g < m1; g += SEG_T) {
      int off;
      if (P.chunk_k > 0) {
        off = min(n, g * P.chunk_k);
      } else {
        const int q = n / M, rem = n % M;
        off = (g < rem) ? g * (q + 1) : rem * (q + 1) + (g - rem) * q;
      }
      gst[g] = off;
    }
  }
  if (b == 0 && tid == 0) gst[M] = n;
  if (!gsync(gs)) return;
  const int* perm_l = va;  // sorted position -> local token
  // ---- group id of every sorted position ----
  for (int s = s0 + tid; s < s1; s += SEG_T) f[s] = 0;
  if (!gsync(gs)) return;
  for (int g = m0 + tid; g < m1; g += SEG_T) f[gst[g]] = 1;
  if (!gsync(gs)) return;
  int Mchk = 0;
  if (!grid_scan(f, grp, n, csum, gs, sh_i, &Mchk)) return;
  for (int s = s0 + tid; s < s1; s += SEG_T) grp[s] = grp[s] + f[s] - 1;
  for (int g = m0 + tid; g < m1; g += SEG_T) {
    gmax[g] = -1;
    gmin[g] = INT_MAX;
    gsum[g] = 0ull;
  }
  if (!gsync(gs)) return;
  for (int s = s0 + tid; s < s1; s += SEG_T) {
    const int g = grp[s], i = perm_l[s];
    atomicMax(&gmax[g], i);
    atomicMin(&gmin[g], i);
    if (pos_scheme == SLS_POS_MEAN) atomicAdd(&gsum[g], (unsigned long long)i);
  }
  if (!gsync(gs)) return;
  // ---- representative positions ----
  if (pos_scheme == SLS_POS_MEDIAN && merged) {
    // members of merged groups are not in token order: sort (group, token)
    int* xa = seat;
    int* xb = cst;
    uint32_t* ga = ka;
    uint32_t* gb2 = kb;
    for (int s = s0 + tid; s < s1; s += SEG_T) ga[perm_l[s]] = (uint32_t)grp[s];
    for (int i = s0 + tid; i < s1; i += SEG_T) xa[i] = i;
    if (!gsync(gs)) return;
    if (!grid_radix_sort<uint32_t>(ga, xa, gb2, xb, n, bit_length_u64((unsigned long long)M),
                                   hist, gs, sh_sort))
      return;
    for (int g = m0 + tid; g < m1; g += SEG_T) rep[g] = xa[gst[g] + (gst[g + 1] - gst[g] - 1) / 2];
  } else {
    for (int g = m0 + tid; g < m1; g += SEG_T) {
      const int len = gst[g + 1] - gst[g];
      int rp;
      if (pos_scheme == SLS_POS_MAX) rp = gmax[g];
      else if (pos_scheme == SLS_POS_MEDIAN) rp = perm_l[gst[g] + (len - 1) / 2];
      else rp = (int)((2ull * gsum[g] + (unsigned long long)len) / (2ull * (unsigned long long)len));
      rep[g] = rp;
    }
  }
  if (!gsync(gs)) return;
  // ---- order groups by (position, first token) ----
  if (pos_scheme != SLS_POS_MEAN) {
    // max and median positions are member tokens of disjoint groups, hence
    // distinct: the rank of a group is the number of marked positions below
    // its own (one scan over the token positions)
    for (int s = s0 + tid; s < s1; s += SEG_T) f[s] = 0;
    if (!gsync(gs)) return;
    for (int g = m0 + tid; g < m1; g += SEG_T) f[rep[g]] = 1;
    if (!gsync(gs)) return;
    int* rk = cst;  // rank of a marked position
    int tmk = 0;
    if (!grid_scan(f, rk, n, csum, gs, sh_i, &tmk)) return;
    if (!gsync(gs)) return;
    for (int g = m0 + tid; g < m1; g += SEG_T) oidx[g] = rk[rep[g]];
  } else {
    unsigned long long* oka = reinterpret_cast<unsigned long long*>(sb + L.ok_a);
    unsigned long long* okb = reinterpret_cast<unsigned long long*>(sb + L.ok_b);
    int* ova = reinterpret_cast<int*>(sb + L.ov_a);
    int* ovb = reinterpret_cast<int*>(sb + L.ov_b);
    for (int g = m0 + tid; g < m1; g += SEG_T) {
      oka[g] = (unsigned long long)rep[g] * (unsigned long long)n + (unsigned long long)gmin[g];
      ova[g] = g;
    }
    if (!gsync(gs)) return;
    const int kbits = bit_length_u64((unsigned long long)n * (unsigned long long)n);
    if (!grid_radix_sort<unsigned long long>(oka, ova, okb, ovb, M, kbits, hist, gs, sh_sort))
      return;
    for (int t = m0 + tid; t < m1; t += SEG_T) oidx[ova[t]] = t;
  }
  if (!gsync(gs)) return;
  // ---- outputs ----
  for (int g = m0 + tid; g < m1; g += SEG_T) {
    const int t = oidx[g];
    const int64_t mrow = P.out0 + t;
    mstart[mrow] = (int)(P.tok_row + gst[g]);
    mlen[mrow] = gst[g + 1] - gst[g];
    pos_out[mrow] = (pos_mode == SLS_MODE_COMPACT) ? (P.out_local + t) : (P.pos0 + rep[g]);
  }
  for (int s = s0 + tid; s < s1; s += SEG_T) {
    const int i = perm_l[s];
    perm[P.tok_row + s] = (int)(P.tok_row + i);
    tok2macro[P.tok_row + i] = P.out_local + oidx[grp[s]];
  }
}

// ============================================================================
// small problems (windows of at most 32 tokens): one warp per problem
// ============================================================================

// The same clusters, exact-length adjust, positions and causal order as
// segment_kernel for a problem of n <= 32 tokens, held in one warp: lane s
// holds the s-th token of the order the groups are cut from ((code, token)
// order for spectral windows, token order for chunk windows), so every group
// is a run of consecutive lanes.
constexpr int SEGW_WARPS = 8;

SLS_DEV unsigned long long shfl_u64(unsigned long long v, int src) {
  return ((unsigned long long)__shfl_sync(0xffffffffu, (unsigned)(v >> 32), src) << 32) |
         __shfl_sync(0xffffffffu, (unsigned)v, src);
}

__global__ void __launch_bounds__(SEGW_WARPS * 32)
segment_warp_kernel(const ProbDesc* __restrict__ probs, int nprob,
                    const uint32_t* __restrict__ codes, int pos_scheme, int pos_mode,
                    int* __restrict__ perm, int* __restrict__ mstart, int* __restrict__ mlen,
                    int32_t* __restrict__ pos_out, int32_t* __restrict__ tok2macro,
                    int chunk_done) {
  const unsigned FULL = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const int w0 = blockIdx.x * SEGW_WARPS + (threadIdx.x >> 5);
  const int nw = gridDim.x * SEGW_WARPS;
  for (int p = w0; p < nprob; p += nw) {
    const ProbDesc P = probs[p];
    const int n = P.n, M = P.m;
    if (n <= 0 || M <= 0) continue;
    if (chunk_done && !P.spectral) {
      for (int t = lane; t < M; t += 32) mlen[P.out0 + t] = 0;
      continue;
    }
    const bool valid = lane < n;
    // ---- order: (code, token) for spectral windows, token order otherwise ----
    unsigned long long key = ~0ull;
    if (valid)
      key = P.spectral ? (((unsigned long long)codes[P.phi_row + lane] << 5) | (unsigned)lane)
                       : (unsigned long long)lane;
    if (P.spectral) {
      // bitonic sort over the 32 lanes, ascending
#pragma unroll
      for (int k = 2; k <= 32; k <<= 1) {
#pragma unroll
        for (int j = k >> 1; j > 0; j >>= 1) {
          const unsigned long long o = shfl_u64(key, lane ^ j);
          const bool up = ((lane & k) == 0);
          const bool lower = (lane & j) == 0;
          // the lower lane of the pair keeps the smaller key when ascending
          const bool keep_min = (lower == up);
          key = keep_min ? (o < key ? o : key) : (o > key ? o : key);
        }
      }
    }
    const int tok = (int)(key & 31u);
    // ---- group of each position ----
    int g = 0;
    if (!P.spectral) {
      const int q = n / M, rem = n % M;
      g = (lane < (q + 1) * rem) ? lane / (q + 1) : rem + (lane - (q + 1) * rem) / max(q, 1);
    } else {
      const unsigned long long code = key >> 5;
      const unsigned long long prevc = shfl_u64(code, max(lane - 1, 0));
      const bool head = valid && (lane == 0 || code != prevc);
      const unsigned hm = __ballot_sync(FULL, head);
      const int C = __popc(hm);
      const int cl = __popc(hm & (0xffffffffu >> (31 - lane))) - 1;  // cluster of this position
      if (C >= M) {
        // merge: the cluster of rank t joins group floor(t M / C)
        g = (int)(((long long)cl * M) / C);
      } else {
        // split: D'Hondt seats, one guaranteed per cluster, ties to the lower
        // code; lane c holds cluster c
        const int cs = (lane < C) ? (int)__fns(hm, 0, lane + 1) : n;
        const int cn = (lane + 1 < C) ? (int)__fns(hm, 0, lane + 2) : n;
        const int size = (lane < C) ? cn - cs : 0;
        int seats = (lane < C) ? 1 : 0;
        for (int it = 0; it < M - C; ++it) {
          bool el = lane < C && seats < size;
          int num = size, den = seats + 1, idx = lane;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) {
            const bool el2 = __shfl_xor_sync(FULL, el ? 1 : 0, o) != 0;
            const int num2 = __shfl_xor_sync(FULL, num, o);
            const int den2 = __shfl_xor_sync(FULL, den, o);
            const int idx2 = __shfl_xor_sync(FULL, idx, o);
            const long long a = (long long)num2 * den, b = (long long)num * den2;
            const bool better = el2 && (!el || a > b || (a == b && idx2 < idx));
            if (better) {
              el = el2;
              num = num2;
              den = den2;
              idx = idx2;
            }
          }
          if (lane == idx) ++seats;
        }
        int gfirst = seats;  // exclusive prefix of seats: first group of each cluster
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(FULL, gfirst, o);
          if (lane >= o) gfirst += y;
        }
        gfirst -= seats;
        const int ccl = max(cl, 0);
        const int c_start = __shfl_sync(FULL, cs, ccl);
        const int c_size = __shfl_sync(FULL, size, ccl);
        const int c_seats = __shfl_sync(FULL, seats, ccl);
        const int c_g0 = __shfl_sync(FULL, gfirst, ccl);
        const int j = lane - c_start;
        const int q = c_size / max(c_seats, 1), rem = c_size % max(c_seats, 1);
        g = c_g0 + ((j < (q + 1) * rem) ? j / (q + 1) : rem + (j - (q + 1) * rem) / max(q, 1));
      }
    }
    if (!valid) g = M;  // past every group
    // ---- group runs: start, end, positions ----
    const int gp = __shfl_sync(FULL, g, max(lane - 1, 0));
    const bool ghead = valid && (lane == 0 || g != gp);
    const unsigned gm = __ballot_sync(FULL, ghead);
    const int gs = valid ? (int)__fns(gm, 0, g + 1) : 32;
    const int ge = (valid && g + 1 < M) ? (int)__fns(gm, 0, g + 2) : n;
    int vmax = valid ? tok : -1, vmin = valid ? tok : 1 << 30, vsum = valid ? tok : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int ymax = __shfl_down_sync(FULL, vmax, o);
      const int ymin = __shfl_down_sync(FULL, vmin, o);
      const int ysum = __shfl_down_sync(FULL, vsum, o);
      if (lane + o < ge) {
        vmax = max(vmax, ymax);
        vmin = min(vmin, ymin);
      }
      // a sum over [lane, ge) needs the partial of lane + o to cover
      // [lane + o, ge) exactly: doubling steps keep that true
      if (lane + o < ge) vsum += ysum;
    }
    // lower median: the member whose token has (len - 1) / 2 smaller members
    int rank = 0;
#pragma unroll
    for (int o = 0; o < 32; ++o) {
      const int t = __shfl_sync(FULL, tok, o);
      if (o >= gs && o < ge && t < tok) ++rank;
    }
    const int len = ge - gs;
    const bool ismed = valid && rank == (len - 1) / 2;
    const unsigned medm = __ballot_sync(FULL, ismed);
    // group g's summary moves to lane g
    const int src = (lane < M) ? (int)__fns(gm, 0, lane + 1) : 0;
    const int g_start = src;
    const int g_end = __shfl_sync(FULL, ge, src);
    const int g_len = g_end - g_start;
    const int g_max = __shfl_sync(FULL, vmax, src);
    const int g_min = __shfl_sync(FULL, vmin, src);
    const int g_sum = __shfl_sync(FULL, vsum, src);
    const unsigned g_end_mask = (g_end >= 32) ? 0xffffffffu : ((1u << g_end) - 1u);
    const unsigned g_mask = g_end_mask & ~((1u << g_start) - 1u);
    const int med_lane = (lane < M) ? (int)__fns(medm & g_mask, 0, 1) : 0;
    const int g_med = __shfl_sync(FULL, tok, med_lane);
    int rep = g_max;
    if (pos_scheme == SLS_POS_MEDIAN) rep = g_med;
    if (pos_scheme == SLS_POS_MEAN) rep = (2 * g_sum + g_len) / (2 * max(g_len, 1));
    // ---- causal order of the groups: by (position, first token) ----
    int orank = 0;
#pragma unroll
    for (int o = 0; o < 32; ++o) {
      const int r2 = __shfl_sync(FULL, rep, o), m2 = __shfl_sync(FULL, g_min, o);
      if (o < M && lane < M && (r2 < rep || (r2 == rep && m2 < g_min))) ++orank;
    }
    if (lane < M) {
      const int64_t mrow = P.out0 + orank;
      mstart[mrow] = (int)(P.tok_row + g_start);
      mlen[mrow] = g_len;
      pos_out[mrow] = (pos_mode == SLS_MODE_COMPACT) ? (P.out_local + orank) : (P.pos0 + rep);
    }
    const int my_rank = __shfl_sync(FULL, orank, min(g, 31));
    if (valid) {
      perm[P.tok_row + lane] = (int)(P.tok_row + tok);
      tok2macro[P.tok_row + tok] = P.out_local + my_rank;
    }
  }
}

// ============================================================================
// preserved tokens, identity
// ============================================================================

__global__ void preserved_kernel(int64_t B, int64_t N, int64_t M, int pf, int pl, int pos_mode,
                                 int* __restrict__ perm, int* __restrict__ mstart,
                                 int* __restrict__ mlen, int32_t* __restrict__ pos_out,
                                 int32_t* __restrict__ tok2macro) {
  const int per = pf + pl;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < B * per;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t b = e / per;
    const int k = (int)(e % per);
    int64_t tok, mac;
    if (k < pf) {
      tok = k;
      mac = k;
    } else {
      tok = N - pl + (k - pf);
      mac = M - pl + (k - pf);
    }
    const int64_t trow = b * N + tok, mrow = b * M + mac;
    perm[trow] = (int)trow;
    mstart[mrow] = (int)trow;
    mlen[mrow] = 1;
    pos_out[mrow] = (int32_t)((pos_mode == SLS_MODE_COMPACT) ? mac : tok);
    tok2macro[trow] = (int32_t)mac;
  }
}

template <typename T>
SLS_DEV float to_f32(T v);
template <>
SLS_DEV float to_f32<float>(float v) {
  return v;
}
template <>
SLS_DEV float to_f32<uint16_t>(uint16_t v) {
  return __uint_as_float(((unsigned)v) << 16);
}

template <typename T>
__global__ void identity_kernel(const T* __restrict__ X, int64_t B, int64_t N, int d, int64_t ldx,
                                float* __restrict__ Xt, int32_t* __restrict__ pos,
                                int32_t* __restrict__ tok2macro) {
  const int64_t total = B * N * d;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = e / d;
    const int c = (int)(e % d);
    Xt[e] = to_f32<T>(X[row * ldx + c]);
    if (c == 0) {
      pos[row] = (int32_t)(row % N);
      tok2macro[row] = (int32_t)(row % N);
    }
  }
}

// ============================================================================
// token norms and macro-token embeddings (Eq. macro_embed)
// ============================================================================

constexpr int AGG_T = 256;
constexpr int AGG_CH = 64;      // members per work item

// Work items: macro-token m is split into ceil(len / AGG_CH) items, listed in
// macro order.  Three grid-wide passes: per-block totals over the macro
// lengths; per macro its item offset, member-row offset, partial-sum slot and
// (for macros spanning several items) its place in a compact list; then one
// thread per item finds its macro by binary search over the increasing item
// offsets, writes the item and, for each of the G member-pass CTAs whose
// balanced row boundary falls inside the item, that CTA's first item.
constexpr int AI_BLOCK = SEG_T;           // macros per block (one per thread)
constexpr int AGG_MAX_GRID = 2048;        // member-pass CTAs at most

// Auxiliary integers of the aggregation: counts (16), block totals (4 per
// block), CTA range starts (AGG_MAX_GRID + 1), multi-item macro list, and per
// macro its first item and first member row.
struct AggAux {
  int* counts;  // [0] items, [1] partial slots, [2] multi-item macros, [3] member rows
  int4* btot;
  int* cta_first;
  int* multi;
  int* it_start;
  int* r_start;
};

__host__ __device__ inline int64_t agg_blocks(int64_t Mtot) { return (Mtot + AI_BLOCK - 1) / AI_BLOCK; }

__host__ __device__ inline AggAux agg_aux(int* base, int64_t Mtot, int64_t Ntot) {
  AggAux A;
  A.counts = base;
  A.btot = reinterpret_cast<int4*>(base + 16);
  A.cta_first = base + 16 + 4 * agg_blocks(Mtot);
  A.multi = A.cta_first + AGG_MAX_GRID + 1;
  A.it_start = A.multi + Ntot / AGG_CH + 2;
  A.r_start = A.it_start + Mtot;
  return A;
}

SLS_DEV int nchunks(int len) { return (len + AGG_CH - 1) / AGG_CH; }

__global__ void __launch_bounds__(SEG_T)
agg_count_kernel(const int* __restrict__ mlen, int64_t Mtot, int64_t Ntot, int* __restrict__ aux) {
  __shared__ int sh[SEG_W + 1];
  const AggAux A = agg_aux(aux, Mtot, Ntot);
  const int64_t m = (int64_t)blockIdx.x * AI_BLOCK + threadIdx.x;
  const int len = (m < Mtot) ? mlen[m] : 0, nch = nchunks(len);
  int t0, t1, t2, t3;
  block_excl_scan<int>(nch, sh, &t0);
  block_excl_scan<int>((nch > 1) ? nch : 0, sh, &t1);
  block_excl_scan<int>((nch > 1) ? 1 : 0, sh, &t2);
  block_excl_scan<int>(len, sh, &t3);
  if (threadIdx.x == 0) A.btot[blockIdx.x] = make_int4(t0, t1, t2, t3);
}

__global__ void __launch_bounds__(SEG_T)
agg_offsets_kernel(const int* __restrict__ mlen, int64_t Mtot, int64_t Ntot,
                   int* __restrict__ aux, int* __restrict__ pt_start) {
  __shared__ int sh[SEG_W + 1];
  const AggAux A = agg_aux(aux, Mtot, Ntot);
  const int nb = (int)agg_blocks(Mtot);
  // offsets of this block (sum over the blocks before it) and the totals
  int b0 = 0, b1 = 0, b2 = 0, b3 = 0, a0 = 0, a1 = 0, a2 = 0, a3 = 0;
  for (int k = threadIdx.x; k < nb; k += SEG_T) {
    const int4 v = A.btot[k];
    if (k < (int)blockIdx.x) {
      b0 += v.x;
      b1 += v.y;
      b2 += v.z;
      b3 += v.w;
    }
    a0 += v.x;
    a1 += v.y;
    a2 += v.z;
    a3 += v.w;
  }
  int o0, o1, o2, o3, n0, n1, n2, n3;
  block_excl_scan<int>(b0, sh, &o0);
  block_excl_scan<int>(b1, sh, &o1);
  block_excl_scan<int>(b2, sh, &o2);
  block_excl_scan<int>(b3, sh, &o3);
  block_excl_scan<int>(a0, sh, &n0);
  block_excl_scan<int>(a1, sh, &n1);
  block_excl_scan<int>(a2, sh, &n2);
  block_excl_scan<int>(a3, sh, &n3);
  const int64_t m = (int64_t)blockIdx.x * AI_BLOCK + threadIdx.x;
  const int len = (m < Mtot) ? mlen[m] : 0, nch = nchunks(len);
  int tt;
  const int ito = o0 + block_excl_scan<int>(nch, sh, &tt);
  const int pto = o1 + block_excl_scan<int>((nch > 1) ? nch : 0, sh, &tt);
  const int muo = o2 + block_excl_scan<int>((nch > 1) ? 1 : 0, sh, &tt);
  const int ro = o3 + block_excl_scan<int>(len, sh, &tt);
  if (m < Mtot) {
    A.it_start[m] = ito;
    A.r_start[m] = ro;
    pt_start[m] = (nch > 1) ? pto : -1;
    if (nch > 1) A.multi[muo] = (int)m;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    A.cta_first[0] = 0;
    A.counts[0] = n0;
    A.counts[1] = n1;
    A.counts[2] = n2;
    A.counts[3] = n3;
  }
}

__global__ void __launch_bounds__(256)
agg_fill_kernel(const int* __restrict__ mlen, int64_t Mtot, int64_t Ntot, int G,
                int* __restrict__ aux, int2* __restrict__ items) {
  const AggAux A = agg_aux(aux, Mtot, Ntot);
  const int nitems = A.counts[0];
  const int64_t rtot = A.counts[3];
  // no items (every macro-token already written elsewhere): every CTA range
  // is empty
  if (nitems == 0 && blockIdx.x == 0)
    for (int t = threadIdx.x; t <= G; t += blockDim.x) A.cta_first[t] = 0;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < nitems; i += gridDim.x * blockDim.x) {
    // the macro of item i: the last m with it_start[m] <= i
    int lo = 0, hi = (int)Mtot - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (A.it_start[mid] <= i)
        lo = mid;
      else
        hi = mid - 1;
    }
    const int m = lo, c = i - A.it_start[m], len = mlen[m];
    items[i] = make_int2(m, c);
    // CTA t starts at the first item whose first row is at or past
    // t * rtot / G: the item after the last one starting before it
    const int64_t rs = (int64_t)A.r_start[m] + (int64_t)c * AGG_CH;
    const int64_t re = (int64_t)A.r_start[m] + min((int64_t)len, (int64_t)(c + 1) * AGG_CH);
    const int64_t tlo = rs * G / rtot + 1, thi = re * G / rtot;
    for (int64_t t = tlo; t <= thi && t <= G; ++t) A.cta_first[t] = i + 1;
  }
}

template <typename T>
struct VecOf;
template <>
struct VecOf<float> {
  static constexpr int V = 4;
};
template <>
struct VecOf<uint16_t> {
  static constexpr int V = 8;
};

template <typename T>
SLS_DEV void load_vec(const T* p, float* out);
template <>
SLS_DEV void load_vec<float>(const float* p, float* out) {
  const float4 v = __ldg(reinterpret_cast<const float4*>(p));
  out[0] = v.x;
  out[1] = v.y;
  out[2] = v.z;
  out[3] = v.w;
}
template <>
SLS_DEV void load_vec<uint16_t>(const uint16_t* p, float* out) {
  const uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
  const unsigned w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    out[2 * k] = __uint_as_float(w[k] << 16);
    out[2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
  }
}

SLS_DEV float agg_block_sum(float v, float* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_sum_f(v);
  __syncthreads();
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  float s = 0.f;
#pragma unroll
  for (int w = 0; w < AGG_T / 32; ++w) s += sh[w];
  return s;
}

SLS_DEV void store_vec4(float* p, float a, float b, float c, float e) {
  *reinterpret_cast<float4*>(p) = make_float4(a, b, c, e);
}

// Thread `tid` owns the V-wide column groups c0 = (tid + q * AGG_T) * V, q < NV.
template <int V, int NV>
SLS_DEV void store_row(const float (&acc)[NV * V], float scale, int d, float* __restrict__ out) {
  const int tid = threadIdx.x;
#pragma unroll
  for (int q = 0; q < NV; ++q) {
    const int c0 = (tid + q * AGG_T) * V;
    if (c0 < d)
#pragma unroll
      for (int v = 0; v < V; v += 4)
        store_vec4(out + c0 + v, acc[q * V + v] * scale, acc[q * V + v + 1] * scale,
                   acc[q * V + v + 2] * scale, acc[q * V + v + 3] * scale);
  }
}

// Finalise one macro-token row from the member sum `acc` (per thread), the
// member count and the sum of member norms: mean, then rescale to the mean
// norm (Eq. macro_embed); a singleton is its token unchanged.
template <int V, int NV>
SLS_DEV void agg_finalize(float (&acc)[NV * V], int len, float eta_sum, int renorm, int d,
                          float* __restrict__ out, float* sh) {
  if (len == 1) {
    store_row<V, NV>(acc, 1.0f, d, out);
    return;
  }
  const int tid = threadIdx.x;
  const float inv = 1.0f / (float)len;
  float sq = 0.f;
#pragma unroll
  for (int q = 0; q < NV; ++q) {
    const int c0 = (tid + q * AGG_T) * V;
    if (c0 < d)
#pragma unroll
      for (int v = 0; v < V; ++v) {
        acc[q * V + v] *= inv;
        sq = fmaf(acc[q * V + v], acc[q * V + v], sq);
      }
  }
  float scale = 1.0f;
  if (renorm) {
    const float nrm = sqrtf(agg_block_sum(sq, sh));
    if (nrm >= 1e-30f) scale = (eta_sum * inv) / nrm;
  }
  store_row<V, NV>(acc, scale, d, out);
}

// Member rows loaded per batch, so that about eight 16-byte loads per thread
// are in flight.
template <int NV>
constexpr int agg_batch() {
  return NV >= 8 ? 1 : 8 / NV;
}

// The macro-tokens whose members span several items: sum their partial rows
// and finalise (one CTA per macro-token of the compact list).
template <int V, int NV>
__global__ void __launch_bounds__(AGG_T)
agg_final_kernel(int d, const int* __restrict__ mlen, const int* __restrict__ pt_start,
                 int64_t Mtot, int64_t Ntot, int renorm, const int* __restrict__ aux,
                 const float* __restrict__ part, const float* __restrict__ part_eta,
                 float* __restrict__ Xt) {
  __shared__ float sh[AGG_T / 32];
  const int tid = threadIdx.x;
  const AggAux A = agg_aux(const_cast<int*>(aux), Mtot, Ntot);
  const int nmulti = A.counts[2];
  for (int t = blockIdx.x; t < nmulti; t += gridDim.x) {
    const int64_t m = A.multi[t];
    const int ps = pt_start[m];
    const int len = mlen[m];
    const int nch = (len + AGG_CH - 1) / AGG_CH;
    float acc[NV * V];
#pragma unroll
    for (int k = 0; k < NV * V; ++k) acc[k] = 0.f;
    float eta = 0.f;
    // AF_B partial rows in flight per thread (the chunks are independent)
    constexpr int AF_B = (NV * V <= 16) ? 4 : 2;
    for (int cb = 0; cb < nch; cb += AF_B) {
      float4 buf[AF_B][NV * V / 4];
#pragma unroll
      for (int j = 0; j < AF_B; ++j) {
        const float* src = part + (int64_t)(ps + cb + j) * d;
#pragma unroll
        for (int q = 0; q < NV; ++q) {
          const int c0 = (tid + q * AGG_T) * V;
#pragma unroll
          for (int k = 0; k < V; k += 4) {
            float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
            if (cb + j < nch && c0 < d) f = *reinterpret_cast<const float4*>(src + c0 + k);
            buf[j][(q * V + k) / 4] = f;
          }
        }
      }
#pragma unroll
      for (int j = 0; j < AF_B; ++j) {
        if (cb + j < nch) eta += part_eta[ps + cb + j];
#pragma unroll
        for (int e = 0; e < NV * V / 4; ++e) {
          acc[4 * e] += buf[j][e].x;
          acc[4 * e + 1] += buf[j][e].y;
          acc[4 * e + 2] += buf[j][e].z;
          acc[4 * e + 3] += buf[j][e].w;
        }
      }
    }
    agg_finalize<V, NV>(acc, len, eta, renorm, d, Xt + m * d, sh);
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Member pass with a shared-memory row ring.  Warp 0 is the producer: it walks
// this CTA's contiguous range of work items (balanced by member rows), loads each
// item's descriptor and member ids one item ahead, and streams every member
// row into an S-stage ring with one bulk async copy per row (mbarrier
// complete_tx); the item descriptor travels with the item's first row.  Warps
// 1..8 consume the rows in the same order: each consumer thread owns the
// column groups c0 = (ct + q * 256) * V, sums them and the row's |x|^2, and
// releases the stage.  At the end of an item the consumers meet at a named
// barrier (which also ORs their failure flags), form the sum of member norms
// and finalise the macro-token (Eq. macro_embed) or store a partial sum.
// Every wait is bounded; a wait that gives up records SLS_ERR_TIMEOUT, the
// other roles stop at their next check, and in-flight copies are drained.
// ---------------------------------------------------------------------------

constexpr int AGR_CW = 8;                    // consumer warps
constexpr int AGR_CT = AGR_CW * 32;          // consumer threads
constexpr int AGR_THREADS = AGR_CT + 32;     // + producer warp
constexpr int AGR_MAX_STAGES = 16;
constexpr int AGR_BAR = 1;                   // named barrier of the consumers

struct AggDesc {
  int m, c, n, len, ps, pad0, pad1, pad2;
};

SLS_DEV bool named_sync_or(unsigned id, unsigned nthreads, bool pred) {
  unsigned r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n"
      " bar.red.or.pred q, %2, %3, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((unsigned)pred), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}

template <typename T>
SLS_DEV void load_vec_smem(const T* p, float* out);
template <>
SLS_DEV void load_vec_smem<float>(const float* p, float* out) {
  const float4 v = *reinterpret_cast<const float4*>(p);
  out[0] = v.x;
  out[1] = v.y;
  out[2] = v.z;
  out[3] = v.w;
}
template <>
SLS_DEV void load_vec_smem<uint16_t>(const uint16_t* p, float* out) {
  const uint4 v = *reinterpret_cast<const uint4*>(p);
  const unsigned w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    out[2 * k] = __uint_as_float(w[k] << 16);
    out[2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
  }
}

// Bounded wait (about a second of clock cycles) that also returns early once
// another role has aborted.  The producer polls without sleeping so that it
// refills a stage as soon as it is released; the eight consumer warps back
// off after a few polls so that their polling does not take the producer's
// issue slots.
template <bool BACKOFF>
SLS_DEV bool agr_wait(uint64_t* bar, unsigned parity, volatile int* abort_flag) {
  const long long t0 = clock64();
  for (unsigned it = 0;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 63) == 63 && (*abort_flag || clock64() - t0 > SLS_WAIT_CYCLES)) return false;
    if (BACKOFF && it > 64) __nanosleep(32);
  }
}

// Descriptor of the local item kidx of this CTA (item i0 + kidx of its
// contiguous range [i0, i1)), or an empty one past the end.
struct LaneDesc {
  int m, c, n, len, ps, off;
};

SLS_DEV LaneDesc agr_lane_desc(const int2* __restrict__ items, const int* __restrict__ mlen,
                               const int* __restrict__ mstart, const int* __restrict__ pt_start,
                               int i0, int i1, int kidx) {
  LaneDesc L{0, 0, 0, 0, -1, 0};
  const int it = i0 + kidx;
  if (it < i1) {
    const int2 item = items[it];
    L.m = item.x;
    L.c = item.y;
    L.len = mlen[L.m];
    L.n = min(L.len - L.c * AGG_CH, AGG_CH);
    L.ps = pt_start[L.m];
    L.off = mstart[L.m] + L.c * AGG_CH;
  }
  return L;
}

// Member row f (flattened over the 32 items of a batch whose inclusive row
// prefix is `pre`): its item j, index s inside the item and token row id.
SLS_DEV void agr_fetch_row(const int* __restrict__ perm, int pre, int nrows, int off, int f0,
                           int lane, int& rid, int& rj, int& rs) {
  const int f = f0 + lane;
  int j = 0;
#pragma unroll
  for (int step = 16; step >= 1; step >>= 1) {
    const int pv = __shfl_sync(0xffffffffu, pre, j + step - 1);
    if (pv <= f) j += step;
  }
  j = min(j, 31);
  const int base = __shfl_sync(0xffffffffu, pre, j > 0 ? j - 1 : 0);
  const int off_j = __shfl_sync(0xffffffffu, off, j);
  rs = f - (j > 0 ? base : 0);
  rj = j;
  rid = (f < nrows) ? perm[off_j + rs] : 0;
}

template <typename T, int NV>
__global__ void __launch_bounds__(AGR_THREADS, 2)
agg_ring_kernel(const T* __restrict__ X, int d, int64_t ldx, const int* __restrict__ perm,
                const int* __restrict__ mstart, const int* __restrict__ mlen,
                const int2* __restrict__ items, const int* __restrict__ cta_first,
                const int* __restrict__ pt_start, int renorm, float* __restrict__ Xt,
                float* __restrict__ part, float* __restrict__ part_eta, int S, int stage_bytes,
                int* status, int64_t ntot) {
  constexpr int V = VecOf<T>::V;
  extern __shared__ __align__(128) unsigned char agr_smem[];
  (void)ntot;  // bounds of the member rows (debug-build checks)
  __shared__ uint64_t fullb[AGR_MAX_STAGES], emptyb[AGR_MAX_STAGES];
  __shared__ AggDesc dring[AGR_MAX_STAGES + 2];
  __shared__ float shq[2][AGR_CW][AGG_CH];
  __shared__ float shm[2][AGR_CW];  // per-warp |member sum|^2 of the item
  __shared__ volatile int s_abort;
  const int DQ = S + 2;
  const int i0 = cta_first[blockIdx.x], i1 = cta_first[blockIdx.x + 1];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const unsigned row_bytes = (unsigned)d * sizeof(T);
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&fullb[s], 1);
      mbar_init(&emptyb[s], AGR_CW);
    }
    mbar_fence_init();
    s_abort = 0;
  }
  __syncthreads();

  if (warp == 0) {
    // ------------------------------ producer ------------------------------
    // Lane j holds the descriptor of local item kb + j; the member ids of the
    // batch are fetched 32 rows at a time, one chunk ahead of the copies.
    const uint64_t pol = l2_policy_evict_first();
    const int GP = S / 2 < 8 ? (S / 2 < 1 ? 1 : S / 2) : 8;  // rows issued together
    unsigned issued = 0;
    bool ok = true;
    int kb = 0;
    LaneDesc cd = agr_lane_desc(items, mlen, mstart, pt_start, i0, i1, kb + lane);
    while (ok) {
      int pre = cd.n;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, pre, o);
        if (lane >= o) pre += t;
      }
      const int nrows = __shfl_sync(0xffffffffu, pre, 31);
      if (nrows == 0) break;
      const LaneDesc nd = agr_lane_desc(items, mlen, mstart, pt_start, i0, i1, kb + 32 + lane);
      int rid, rj, rs;
      agr_fetch_row(perm, pre, nrows, cd.off, 0, lane, rid, rj, rs);
      for (int f0 = 0; f0 < nrows && ok; f0 += 32) {
        int nrid = 0, nrj = 0, nrs = 0;
        if (f0 + 32 < nrows) agr_fetch_row(perm, pre, nrows, cd.off, f0 + 32, lane, nrid, nrj, nrs);
        const int cnt = min(32, nrows - f0);
        // rows g0 .. g0 + GP - 1 of the batch go out together, one per lane:
        // each lane waits for its own ring stage, then issues its copy (a
        // thread issuing a bulk copy is held for a few hundred cycles, so
        // one lane issuing every row made the producer the bottleneck)
        for (int g0 = 0; g0 < cnt; g0 += GP) {
          const int gn = min(GP, cnt - g0);
          const bool act = lane < gn;
          const int row = __shfl_sync(0xffffffffu, rid, (g0 + lane) & 31);
          const int j = __shfl_sync(0xffffffffu, rj, (g0 + lane) & 31);
          const int s = __shfl_sync(0xffffffffu, rs, (g0 + lane) & 31);
          AggDesc D;
          D.m = __shfl_sync(0xffffffffu, cd.m, j);
          D.c = __shfl_sync(0xffffffffu, cd.c, j);
          D.n = __shfl_sync(0xffffffffu, cd.n, j);
          D.len = __shfl_sync(0xffffffffu, cd.len, j);
          D.ps = __shfl_sync(0xffffffffu, cd.ps, j);
          D.pad0 = D.pad1 = D.pad2 = 0;
          const unsigned mine = issued + (unsigned)lane;
          const int st = (int)(mine % (unsigned)S);
          const unsigned par = (mine / (unsigned)S) & 1u;
          bool w_ok = true;
          if (act) w_ok = agr_wait<false>(&emptyb[st], par ^ 1u, &s_abort);
          if (!__all_sync(0xffffffffu, w_ok)) {
            ok = false;
            if (lane == 0) {
              s_abort = 1;
              atomicExch(status, SLS_ERR_TIMEOUT);
            }
            break;
          }
          if (act) {
            if (s == 0) dring[(kb + j) % DQ] = D;
            unsigned char* dst = agr_smem + (size_t)st * stage_bytes;
            mbar_expect_tx(&fullb[st], row_bytes);
            int64_t src_row = row;
#ifdef SLS_DEBUG
            // a member row outside the token set is not fetched: the stage
            // gets row 0 instead and the status records SLS_ERR_BOUNDS
            if (!(row >= 0 && (int64_t)row < ntot)) {
              atomicExch(status, SLS_ERR_BOUNDS);
              src_row = 0;
            }
#endif
            bulk_g2s(dst, X + src_row * ldx, row_bytes, &fullb[st], pol);
          }
          issued += (unsigned)gn;
        }
        rid = nrid;
        rj = nrj;
        rs = nrs;
      }
      kb += 32;
      cd = nd;
    }
    // every issued copy has landed before the CTA may exit
    if (lane == 0) {
      const unsigned first = issued > (unsigned)S ? issued - (unsigned)S : 0u;
      for (unsigned c = first; c < issued; ++c) {
        for (unsigned w = 0; w < (1u << 25); ++w) {
          if (mbar_try_wait(&fullb[c % (unsigned)S], (c / (unsigned)S) & 1u)) break;
          __nanosleep(32);
        }
      }
    }
  } else {
    // ------------------------------ consumers -----------------------------
    const int cw = warp - 1, ct = threadIdx.x - 32;
    unsigned consumed = 0;
    bool ok = true;
    int k = 0;
    for (int it = i0; it < i1; ++it, ++k) {
      float acc[NV * V];
#pragma unroll
      for (int e = 0; e < NV * V; ++e) acc[e] = 0.f;
      AggDesc D{};
      D.n = 1;
      float* q = &shq[k & 1][cw][0];
      for (int s = 0; s < D.n && ok; ++s) {
        const int st = (int)(consumed % (unsigned)S);
        const unsigned par = (consumed / (unsigned)S) & 1u;
        if (!agr_wait<true>(&fullb[st], par, &s_abort)) {
          ok = false;
          if (lane == 0) {
            s_abort = 1;
            atomicExch(status, SLS_ERR_TIMEOUT);
          }
          break;
        }
        if (s == 0) D = dring[k % DQ];
        const T* rowp = reinterpret_cast<const T*>(agr_smem + (size_t)st * stage_bytes);
        float sq = 0.f;
#pragma unroll
        for (int qv = 0; qv < NV; ++qv) {
          const int c0 = (ct + qv * AGR_CT) * V;
          if (c0 < d) {
            float v[V];
            load_vec_smem<T>(rowp + c0, v);
#pragma unroll
            for (int e = 0; e < V; ++e) {
              acc[qv * V + e] += v[e];
              sq = fmaf(v[e], v[e], sq);
            }
          }
        }
        sq = warp_sum_f(sq);
        __syncwarp();
        if (lane == 0) {
          q[s] = sq;
          mbar_arrive(&emptyb[st]);
        }
        ++consumed;
      }
      // this warp's share of |sum of the members|^2, published with the
      // item-end barrier (the renorm needs no barrier of its own)
      {
        float msq = 0.f;
#pragma unroll
        for (int e = 0; e < NV * V; ++e) msq = fmaf(acc[e], acc[e], msq);
        msq = warp_sum_f(msq);
        if (lane == 0) shm[k & 1][cw] = msq;
      }
      if (named_sync_or(AGR_BAR, AGR_CT, !ok)) break;
      // sum of member norms (every warp forms the same total)
      float eta = 0.f;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int s = lane + 32 * h;
        if (s < D.n) {
          float t = 0.f;
#pragma unroll
          for (int w = 0; w < AGR_CW; ++w) t += shq[k & 1][w][s];
          eta += sqrtf(t);
        }
      }
      eta = warp_sum_f(eta);
      float scale = 1.0f;
      float* dst;
      if (D.ps < 0) {
        dst = Xt + (int64_t)D.m * d;
        if (D.len > 1) {
          // mean = sum / len, rescaled to the mean member norm
          const float inv = 1.0f / (float)D.len;
          scale = inv;
          if (renorm) {
            float tot = 0.f;
#pragma unroll
            for (int w = 0; w < AGR_CW; ++w) tot += shm[k & 1][w];
            const float nrm = sqrtf(tot) * inv;
            if (nrm >= 1e-30f) scale = inv * ((eta * inv) / nrm);
          }
        }
      } else {
        dst = part + (int64_t)(D.ps + D.c) * d;
        if (ct == 0) part_eta[D.ps + D.c] = eta;
      }
#pragma unroll
      for (int qv = 0; qv < NV; ++qv) {
        const int c0 = (ct + qv * AGR_CT) * V;
        if (c0 < d)
#pragma unroll
          for (int e = 0; e < V; e += 4)
            store_vec4(dst + c0 + e, acc[qv * V + e] * scale, acc[qv * V + e + 1] * scale,
                       acc[qv * V + e + 2] * scale, acc[qv * V + e + 3] * scale);
      }
    }
  }
}

// ============================================================================
// adaptive router: window redundancy score (Eq. redundancy)
// ============================================================================

// score = (1/L) sum_i cos(x_i, c) with c the window centroid; computed in one
// pass over X as (sum_i x_i/|x_i|) . (sum_i x_i) / (L |sum_i x_i|).  Zero rows
// add 0.  Every window is cut into parts of SCORE_PR rows (so that a batch of
// windows spreads evenly over the SMs); a CTA takes a part at a time, gathers
// its rows in batches of agg_batch<NV>(), reduces each row's |x|^2 from the
// same registers (per warp, then across warps through a double-buffered
// shared array, one barrier per batch) and writes the part's sums of x and of
// x/|x|; window_score_combine_kernel adds a window's parts and forms the
// score.
constexpr int SCORE_PR = 512;  // rows per part

__host__ __device__ inline int score_parts(int64_t nmax) {
  return (int)((nmax + SCORE_PR - 1) / SCORE_PR);
}

template <typename T, int NV>
__global__ void __launch_bounds__(AGG_T, 2)
window_score_kernel(const T* __restrict__ X, int d, int64_t ldx,
                    const ProbDesc* __restrict__ probs, int nprob, int KP,
                    float* __restrict__ part) {
  constexpr int V = VecOf<T>::V;
  constexpr int MB = agg_batch<NV>();
  constexpr int NW = AGG_T / 32;
  __shared__ float shq[2][MB][NW];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int units = nprob * KP;
  for (int u = blockIdx.x; u < units; u += gridDim.x) {
    const int p = u / KP, k = u % KP;
    const ProbDesc P = probs[p];
    const int r0 = min(P.n, k * SCORE_PR), r1 = min(P.n, r0 + SCORE_PR);
    if (r0 >= r1) continue;
    float cs[NV * V], ns[NV * V];
#pragma unroll
    for (int e = 0; e < NV * V; ++e) cs[e] = ns[e] = 0.f;
    int buf = 0;
    for (int s0 = r0; s0 < r1; s0 += MB, buf ^= 1) {
      float v[MB][NV * V];
#pragma unroll
      for (int j = 0; j < MB; ++j) {
        const bool live = s0 + j < r1;
        const T* x = X + (P.tok_row + s0 + j) * ldx;
#pragma unroll
        for (int q = 0; q < NV; ++q) {
          const int c0 = (tid + q * AGG_T) * V;
          if (live && c0 < d) {
            load_vec<T>(x + c0, &v[j][q * V]);
          } else {
#pragma unroll
            for (int e = 0; e < V; ++e) v[j][q * V + e] = 0.f;
          }
        }
      }
#pragma unroll
      for (int j = 0; j < MB; ++j) {
        float sq = 0.f;
#pragma unroll
        for (int e = 0; e < NV * V; ++e) sq = fmaf(v[j][e], v[j][e], sq);
        sq = warp_sum_f(sq);
        if (lane == 0) shq[buf][j][warp] = sq;
      }
      __syncthreads();
#pragma unroll
      for (int j = 0; j < MB; ++j) {
        float t = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) t += shq[buf][j][w];
        const float inv = (t > 0.f) ? 1.0f / sqrtf(t) : 0.f;
#pragma unroll
        for (int e = 0; e < NV * V; ++e) {
          cs[e] += v[j][e];
          ns[e] = fmaf(v[j][e], inv, ns[e]);
        }
      }
    }
    float* dst = part + (size_t)u * 2 * d;
#pragma unroll
    for (int q = 0; q < NV; ++q) {
      const int c0 = (tid + q * AGG_T) * V;
      if (c0 < d)
#pragma unroll
        for (int e = 0; e < V; e += 4) {
          store_vec4(dst + c0 + e, cs[q * V + e], cs[q * V + e + 1], cs[q * V + e + 2],
                     cs[q * V + e + 3]);
          store_vec4(dst + d + c0 + e, ns[q * V + e], ns[q * V + e + 1], ns[q * V + e + 2],
                     ns[q * V + e + 3]);
        }
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// The score pass with the chunk path folded in (adaptive backend below rho =
// 16, Sec. 3.6): the windows whose score falls below tau are averaged in
// consecutive groups (numpy array_split of the window's n tokens into its m
// macro-tokens), and those means need the same rows the score reads.  So the
// score pass computes, for every window, the chunk macro-tokens as if it were
// routed to the chunk path -- renormalised means (Eq. macro_embed), their
// positions and the token map -- and the segment and aggregation steps then
// handle the spectral windows only, whose outputs replace these.  Parts are
// cut on group boundaries (about SCORE_PR rows each), so no group spans two
// CTAs; a batch's shared-memory reduction carries, besides the row norms,
// the squared norms of the group means that end in the batch.
// ---------------------------------------------------------------------------

// first token of chunk group g (g <= m; group m starts at n)
__host__ __device__ inline int chunk_gstart(int n, int m, int g) {
  const int q = n / m, rem = n % m;
  return (g < rem) ? g * (q + 1) : rem * (q + 1) + (g - rem) * q;
}
// groups per part: about SCORE_PR rows, at least one group
__host__ __device__ inline int chunk_gpp(int n, int m) {
  const int gp = SCORE_PR / (n / m + 1);
  return gp < 1 ? 1 : gp;
}
__host__ __device__ inline int chunk_nparts(int n, int m) {
  const int gp = chunk_gpp(n, m);
  return (m + gp - 1) / gp;
}
// a bound on chunk_nparts over windows of at most nmax tokens: every part but
// the last holds at least SCORE_PR / 2 rows
__host__ __device__ inline int chunk_parts_max(int64_t nmax) {
  return (int)((nmax + SCORE_PR / 2 - 1) / (SCORE_PR / 2));
}

// Element e of a 16-byte word of X as loaded: four floats, or eight bf16
// values widened exactly.  Keeping the loaded rows as raw words halves their
// registers for bf16 inputs.
template <typename T>
SLS_DEV float raw_elem(const uint4& r, int e);
template <>
SLS_DEV float raw_elem<float>(const uint4& r, int e) {
  const unsigned w = (e == 0) ? r.x : (e == 1) ? r.y : (e == 2) ? r.z : r.w;
  return __uint_as_float(w);
}
template <>
SLS_DEV float raw_elem<uint16_t>(const uint4& r, int e) {
  const int k = e >> 1;
  const unsigned w = (k == 0) ? r.x : (k == 1) ? r.y : (k == 2) ? r.z : r.w;
  return (e & 1) ? __uint_as_float(w & 0xffff0000u) : __uint_as_float(w << 16);
}

// 16-byte asynchronous copy global -> shared (zero-filled when !live), and
// the wait for all but the newest `pending` groups of a thread's copies.
SLS_DEV void cp16_async(void* dst, const void* src, bool live) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src),
               "r"(live ? 16 : 0)
               : "memory");
}
SLS_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int PENDING>
SLS_DEV void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(PENDING) : "memory");
}

// Rows of a batch staged per thread: slot [buffer][row][column group][thread];
// two batches of MB * NV = 8 words, the next in flight while one is used (a
// third stage measured slower: its registers spill).
constexpr int CHK_RING_BYTES = 2 * 8 * AGG_T * 16;

template <typename T, int NV>
__global__ void __launch_bounds__(AGG_T, 2)
window_score_chunk_kernel(const T* __restrict__ X, int d, int64_t ldx,
                          const ProbDesc* __restrict__ probs, int nprob, int KP,
                          float* __restrict__ part, int pos_scheme, int pos_mode, int renorm,
                          float* __restrict__ Xt, int32_t* __restrict__ pos_out,
                          int32_t* __restrict__ tok2macro) {
  constexpr int V = VecOf<T>::V;
  constexpr int MB = agg_batch<NV>();
  constexpr int NW = AGG_T / 32;
  static_assert(MB * NV == 8, "staging ring sized for eight 16-byte words per thread");
  __shared__ float shq[2][MB][NW];  // row |x|^2 partials
  __shared__ float shg[2][MB][NW];  // |group mean|^2 partials, slot = the group's last row
  extern __shared__ uint4 chk_ring[];  // [2][MB][NV][AGG_T]: each thread reads only its own words
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int units = nprob * KP;
  for (int u = blockIdx.x; u < units; u += gridDim.x) {
    const int p = u / KP, k = u % KP;
    const ProbDesc P = probs[p];
    const int n = P.n, m = P.m;
    if (n <= 0 || m <= 0) continue;
    const int gp = chunk_gpp(n, m);
    if (k >= (m + gp - 1) / gp) continue;
    const int g0 = k * gp, g1 = min(m, g0 + gp);
    const int r0 = chunk_gstart(n, m, g0), r1 = chunk_gstart(n, m, g1);
    const int q = n / m, rem = n % m;
    // positions of the part's groups and the token map
    for (int g = g0 + tid; g < g1; g += AGG_T) {
      const int a = chunk_gstart(n, m, g), len = chunk_gstart(n, m, g + 1) - a;
      int rp;
      if (pos_scheme == SLS_POS_MAX) {
        rp = a + len - 1;
      } else if (pos_scheme == SLS_POS_MEDIAN) {
        rp = a + (len - 1) / 2;
      } else {
        const unsigned long long sum =
            (unsigned long long)len * a + (unsigned long long)len * (len - 1) / 2;
        rp = (int)((2ull * sum + (unsigned long long)len) / (2ull * (unsigned long long)len));
      }
      pos_out[P.out0 + g] = (pos_mode == SLS_MODE_COMPACT) ? (P.out_local + g) : (P.pos0 + rp);
    }
    for (int i = r0 + tid; i < r1; i += AGG_T) {
      const int g = (i < rem * (q + 1)) ? i / (q + 1) : rem + (i - rem * (q + 1)) / q;
      tok2macro[P.tok_row + i] = P.out_local + g;
    }
    float cs[NV * V], ns[NV * V], gs[NV * V];
#pragma unroll
    for (int e = 0; e < NV * V; ++e) cs[e] = ns[e] = gs[e] = 0.f;
    int gcur = g0, gend = chunk_gstart(n, m, g0 + 1), gcnt = 0;  // before the barrier
    int pcur = g0, pend = gend, pcnt = 0;                          // after it
    float geta = 0.f;
    // the copies of batch s0 go to ring slot b; the next batch is in flight
    // while this one is processed
    auto issue = [&](int s0, int b) {
#pragma unroll
      for (int j = 0; j < MB; ++j) {
        const bool rl = s0 + j < r1;
        const T* x = X + (P.tok_row + (rl ? s0 + j : r0)) * ldx;
#pragma unroll
        for (int qv = 0; qv < NV; ++qv) {
          const int c0 = (tid + qv * AGG_T) * V;
          const bool live = rl && c0 < d;
          cp16_async(&chk_ring[((b * MB + j) * NV + qv) * AGG_T + tid], live ? x + c0 : x, live);
        }
      }
      cp_async_commit();
    };
    issue(r0, 0);
    int buf = 0;
    for (int s0 = r0; s0 < r1; s0 += MB, buf ^= 1) {
      if (s0 + MB < r1) {
        issue(s0 + MB, buf ^ 1);
        cp_async_wait<1>();
      } else {
        cp_async_wait<0>();
      }
      uint4 raw[MB][NV];
#pragma unroll
      for (int j = 0; j < MB; ++j)
#pragma unroll
        for (int qv = 0; qv < NV; ++qv)
          raw[j][qv] = chk_ring[((buf * MB + j) * NV + qv) * AGG_T + tid];
      // before the barrier: row |x|^2 partials; the group sums, and for every
      // group that ends in this batch its mean (stored unscaled; a singleton is
      // its token) and the |mean|^2 partial
#pragma unroll
      for (int j = 0; j < MB; ++j) {
        float sq = 0.f;
#pragma unroll
        for (int e = 0; e < NV * V; ++e) {
          const float x = raw_elem<T>(raw[j][e / V], e % V);
          sq = fmaf(x, x, sq);
        }
        sq = warp_sum_f(sq);
        if (lane == 0) shq[buf][j][warp] = sq;
        if (s0 + j < r1) {
#pragma unroll
          for (int e = 0; e < NV * V; ++e) gs[e] += raw_elem<T>(raw[j][e / V], e % V);
          ++gcnt;
          if (s0 + j + 1 == gend) {
            const float ginv = (gcnt > 1) ? 1.0f / (float)gcnt : 1.0f;
            float gq = 0.f;
#pragma unroll
            for (int e = 0; e < NV * V; ++e) {
              if (gcnt > 1) gs[e] *= ginv;
              gq = fmaf(gs[e], gs[e], gq);
            }
            gq = warp_sum_f(gq);
            if (lane == 0) shg[buf][j][warp] = gq;
            store_row<V, NV>(gs, 1.0f, d, Xt + (P.out0 + gcur) * (int64_t)d);
#pragma unroll
            for (int e = 0; e < NV * V; ++e) gs[e] = 0.f;
            gcnt = 0;
            ++gcur;
            gend = chunk_gstart(n, m, gcur + 1);
          }
        }
      }
      __syncthreads();
      // after it: the score sums, and each finished group's mean rescaled in
      // place to the mean member norm (Eq. macro_embed)
#pragma unroll
      for (int j = 0; j < MB; ++j) {
        if (s0 + j >= r1) break;
        float tq = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) tq += shq[buf][j][w];
        const float nrm = sqrtf(tq);
        const float inv = (tq > 0.f) ? 1.0f / nrm : 0.f;
#pragma unroll
        for (int e = 0; e < NV * V; ++e) {
          const float x = raw_elem<T>(raw[j][e / V], e % V);
          cs[e] += x;
          ns[e] = fmaf(x, inv, ns[e]);
        }
        geta += nrm;
        ++pcnt;
        if (s0 + j + 1 == pend) {
          if (pcnt > 1 && renorm) {
            float gq = 0.f;
#pragma unroll
            for (int w = 0; w < NW; ++w) gq += shg[buf][j][w];
            const float gn = sqrtf(gq);
            if (gn >= 1e-30f) {
              const float scale = (geta * (1.0f / (float)pcnt)) / gn;
              float* out = Xt + (P.out0 + pcur) * (int64_t)d;
#pragma unroll
              for (int qv = 0; qv < NV; ++qv) {
                const int c0 = (tid + qv * AGG_T) * V;
                if (c0 < d)
#pragma unroll
                  for (int e = 0; e < V; e += 4) {
                    const float4 mv = *reinterpret_cast<const float4*>(out + c0 + e);
                    store_vec4(out + c0 + e, mv.x * scale, mv.y * scale, mv.z * scale,
                               mv.w * scale);
                  }
              }
            }
          }
          geta = 0.f;
          pcnt = 0;
          ++pcur;
          pend = chunk_gstart(n, m, pcur + 1);
        }
      }
    }
    float* dst = part + (size_t)u * 2 * d;
#pragma unroll
    for (int qv = 0; qv < NV; ++qv) {
      const int c0 = (tid + qv * AGG_T) * V;
      if (c0 < d)
#pragma unroll
        for (int e = 0; e < V; e += 4) {
          store_vec4(dst + c0 + e, cs[qv * V + e], cs[qv * V + e + 1], cs[qv * V + e + 2],
                     cs[qv * V + e + 3]);
          store_vec4(dst + d + c0 + e, ns[qv * V + e], ns[qv * V + e + 1], ns[qv * V + e + 2],
                     ns[qv * V + e + 3]);
        }
    }
    __syncthreads();
  }
}

// score[p] = (sum of the parts' x / |x|) . (sum of the parts' x) / (n |sum x|)
__global__ void __launch_bounds__(AGG_T)
window_score_combine_kernel(int d, const ProbDesc* __restrict__ probs, int nprob, int KP,
                            int chunked, const float* __restrict__ part,
                            float* __restrict__ score) {
  __shared__ float sh[AGG_T / 32];
  for (int p = blockIdx.x; p < nprob; p += gridDim.x) {
    const int n = probs[p].n;
    const int kp = chunked ? chunk_nparts(n, probs[p].m) : score_parts(n);
    float dot = 0.f, cc = 0.f;
    for (int c = threadIdx.x; c < d; c += AGG_T) {
      float cs = 0.f, ns = 0.f;
      for (int k = 0; k < kp; ++k) {
        const float* src = part + ((size_t)p * KP + k) * 2 * d;
        cs += src[c];
        ns += src[d + c];
      }
      dot = fmaf(ns, cs, dot);
      cc = fmaf(cs, cs, cc);
    }
    dot = agg_block_sum(dot, sh);
    cc = agg_block_sum(cc, sh);
    if (threadIdx.x == 0) score[p] = (cc > 0.f) ? dot / ((float)n * sqrtf(cc)) : 0.f;
    __syncthreads();
  }
}

}  // namespace

// ============================================================================
// launchers
// ============================================================================

int launch_simhash(const float* U, int64_t N, int k, int ldu, const int32_t* k_dev,
                   const float* R, int bits, int ldr, uint32_t* codes, cudaStream_t stream) {
  if (N == 0) return SLS_OK;
  const size_t smem = sizeof(float) * bits * (k + 1);
  int bp = 1;
  while (bp < bits) bp <<= 1;
  int64_t blocks = (N * bp + 255) / 256;  // 8 warps of 32 / bp rows
  if (blocks > 4096) blocks = 4096;
  if (smem > 48 * 1024)
    SLS_CUDA_TRY(cudaFuncSetAttribute(simhash_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)smem));
  simhash_kernel<<<(unsigned)blocks, 256, smem, stream>>>(U, N, k, ldu, k_dev, R, bits, ldr, codes);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

size_t segment_scratch_bytes(int64_t nmax, int64_t mmax, int slots) {
  return (size_t)slots * seg_layout(nmax, mmax).total;
}

int launch_simhash_problems(const ProbDesc* probs, const int* spec_list, const int* nspec_dev,
                            int nspec_max, int64_t nmax, const int* r_eff, const float* U, int ldu,
                            const float* R, int ldr, int bits_max, uint32_t* codes,
                            cudaStream_t stream) {
  if (nspec_max <= 0) return SLS_OK;
  if (nmax <= SH_FLAT_MAX) {
    const int64_t threads = (int64_t)nspec_max * nmax;
    const int64_t blocks = (threads + 255) / 256;
    if (blocks > 0x7fffffffLL) return SLS_ERR_UNSUPPORTED;
    simhash_flat_kernel<<<(unsigned)blocks, 256, 0, stream>>>(
        probs, spec_list, nspec_dev, nspec_max, (int)nmax, r_eff, U, ldu, R, ldr, codes);
    SLS_LAUNCH_CHECK();
    return SLS_OK;
  }
  const size_t smem = sizeof(float) * bits_max * (ldu + 1);
  // warps of 32 / BP rows (BP: bits rounded up to a power of two): enough
  // CTAs of 8 warps for the rows of the largest problem
  int bpmax = 1;
  while (bpmax < bits_max) bpmax <<= 1;
  int64_t bx = (nmax * bpmax + 255) / 256;
  if (bx > 1024) bx = 1024;
  // at most about 8192 CTAs in all (the CTAs loop over their problem's
  // rows): the launch is sized by the bound on the spectral problems, most
  // of which may be empty at run time
  const int64_t cap = 8192 / (nspec_max > 0 ? nspec_max : 1);
  if (bx > cap) bx = cap;
  if (bx < 1) bx = 1;
  if (smem > 48 * 1024)
    SLS_CUDA_TRY(cudaFuncSetAttribute(simhash_batched_kernel,
                                      cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  simhash_batched_kernel<<<dim3((unsigned)bx, nspec_max), 256, smem, stream>>>(
      probs, spec_list, nspec_dev, nspec_max, r_eff, U, ldu, R, ldr, codes);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

int launch_segment(const ProbDesc* probs, int nprob, const uint32_t* codes, int pos_scheme,
                   int pos_mode, void* scratch, int slots, int64_t nmax, int64_t mmax, int* perm,
                   int* mstart, int* mlen, int32_t* pos_out, int32_t* tok2macro, int* status,
                   cudaStream_t stream, int chunk_done) {
  if (nprob <= 0) return SLS_OK;
  const SegLayout L = seg_layout(nmax, mmax);
  const size_t stride = L.total;
  if (nmax <= 32) {
    // windows of at most 32 tokens: one warp per window
    int64_t blocks = ((int64_t)nprob + SEGW_WARPS - 1) / SEGW_WARPS;
    if (blocks > 65535) blocks = 65535;
    segment_warp_kernel<<<(unsigned)blocks, SEGW_WARPS * 32, 0, stream>>>(
        probs, nprob, codes, pos_scheme, pos_mode, perm, mstart, mlen, pos_out, tok2macro,
        chunk_done);
    SLS_LAUNCH_CHECK();
    return SLS_OK;
  }
  if (nprob == 1 && nmax >= SEG_GRID_MIN_N && status) {
    // one large problem: spread it over a cooperative grid
    int dev = 0, sms = 0;
    SLS_CUDA_TRY(cudaGetDevice(&dev));
    SLS_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    int G = sms < SEGG_MAX ? sms : SEGG_MAX;
    const int64_t want = (nmax + 255) / 256;
    if (want < G) G = (int)want;
    if (G < 1) G = 1;
    char* sb = (char*)scratch;
    SLS_CUDA_TRY(cudaMemsetAsync(sb + L.gbar, 0, 256, stream));
    int64_t nm = nmax, mm = mmax;
    void* args[] = {(void*)&probs, (void*)&codes, (void*)&pos_scheme, (void*)&pos_mode,
                    (void*)&sb, (void*)&nm, (void*)&mm, (void*)&perm, (void*)&mstart,
                    (void*)&mlen, (void*)&pos_out, (void*)&tok2macro, (void*)&status,
                    (void*)&chunk_done};
    SLS_CUDA_TRY(cudaLaunchCooperativeKernel((const void*)segment_grid_kernel, dim3(G), dim3(SEG_T),
                                             args, 0, stream));
    count_launch(1);
    return SLS_OK;
  }
  const int grid = nprob < slots ? nprob : slots;
  // the sort buffers in shared memory when they fit beside the static arrays
  // (the mistral7b prompt's segment step 85 -> 81 us)
  const size_t dyn = seg_smem_layout(nmax, mmax).total;
  const int in_smem = dyn <= SEG_SMEM_MAX ? 1 : 0;
  const size_t dyn_bytes = in_smem ? dyn : 0;
  if (in_smem)
    SLS_CUDA_TRY(cudaFuncSetAttribute(segment_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)dyn_bytes));
  segment_kernel<<<grid, SEG_T, dyn_bytes, stream>>>(probs, nprob, codes, pos_scheme, pos_mode,
                                                     (char*)scratch, stride, nmax, mmax, perm,
                                                     mstart, mlen, pos_out, tok2macro,
                                                     chunk_done, in_smem);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

int launch_preserved(int64_t B, int64_t N, int64_t M, int pf, int pl, int pos_mode, int* perm,
                     int* mstart, int* mlen, int32_t* pos_out, int32_t* tok2macro,
                     cudaStream_t stream) {
  if (pf + pl == 0 || B == 0) return SLS_OK;
  int64_t blocks = (B * (pf + pl) + 255) / 256;
  if (blocks > 1024) blocks = 1024;
  preserved_kernel<<<(unsigned)blocks, 256, 0, stream>>>(B, N, M, pf, pl, pos_mode, perm, mstart,
                                                         mlen, pos_out, tok2macro);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

int launch_identity(const void* X, int x_dtype, int64_t B, int64_t N, int d, int64_t ldx,
                    float* Xt, int32_t* pos, int32_t* tok2macro, cudaStream_t stream) {
  if (B * N == 0) return SLS_OK;
  int64_t blocks = (B * N * d + 255) / 256;
  if (blocks > 65536) blocks = 65536;
  if (x_dtype == SLS_F32)
    identity_kernel<float><<<(unsigned)blocks, 256, 0, stream>>>((const float*)X, B, N, d, ldx,
                                                                  Xt, pos, tok2macro);
  else
    identity_kernel<uint16_t><<<(unsigned)blocks, 256, 0, stream>>>((const uint16_t*)X, B, N, d,
                                                                     ldx, Xt, pos, tok2macro);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

size_t agg_item_capacity(int64_t Mtot, int64_t Ntot) { return (size_t)(Mtot + Ntot / AGG_CH + 2); }
size_t agg_aux_ints(int64_t Mtot, int64_t Ntot) {
  return (size_t)(16 + 4 * agg_blocks(Mtot) + (AGG_MAX_GRID + 1) + Ntot / AGG_CH + 2 + 2 * Mtot);
}
size_t agg_part_capacity(int64_t Ntot) { return (size_t)(2 * (Ntot / AGG_CH) + 2); }

namespace {
template <typename T, int NV>
int launch_agg_t(const void* X, int d, int64_t ldx, const int* perm, const int* mstart,
                 const int* mlen, int64_t Mtot, int64_t Ntot, int64_t fblocks, int renorm,
                 float* Xt,
                 int* pt_start, int2* items, int* aux, float* part, float* part_eta,
                 int* status, cudaStream_t stream) {
  constexpr int V = VecOf<T>::V;
  const int stage = (int)(((size_t)d * sizeof(T) + 127) & ~(size_t)127);
  // two CTAs per SM when each still gets at least 6 ring stages in ~100 KB
  int per_sm = 2;
  int S = (100 * 1024) / stage;
  if (S < 6) {
    per_sm = 1;
    S = (200 * 1024) / stage;
  }
  if (S > AGR_MAX_STAGES) S = AGR_MAX_STAGES;
  if (S < 2) return SLS_ERR_UNSUPPORTED;
  const size_t smem = (size_t)S * stage;
  SLS_CUDA_TRY(cudaFuncSetAttribute(agg_ring_kernel<T, NV>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  int occ = 0;
  SLS_CUDA_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, agg_ring_kernel<T, NV>,
                                                             AGR_THREADS, smem));
  if (occ < 1) return SLS_ERR_UNSUPPORTED;
  if (occ < per_sm) per_sm = occ;
  int dev = 0, sms = 0;
  SLS_CUDA_TRY(cudaGetDevice(&dev));
  SLS_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  int grid = sms * per_sm;
  if (grid > AGG_MAX_GRID) grid = AGG_MAX_GRID;
  // work items, partial slots and the balanced CTA ranges
  const unsigned nb = (unsigned)agg_blocks(Mtot);
  agg_count_kernel<<<nb, SEG_T, 0, stream>>>(mlen, Mtot, Ntot, aux);
  SLS_LAUNCH_CHECK();
  agg_offsets_kernel<<<nb, SEG_T, 0, stream>>>(mlen, Mtot, Ntot, aux, pt_start);
  SLS_LAUNCH_CHECK();
  int64_t fill = (Mtot + Ntot / AGG_CH + 255) / 256;
  if (fill > 8 * (int64_t)sms) fill = 8 * (int64_t)sms;
  agg_fill_kernel<<<(unsigned)fill, 256, 0, stream>>>(mlen, Mtot, Ntot, grid, aux, items);
  SLS_LAUNCH_CHECK();
  const AggAux A = agg_aux(aux, Mtot, Ntot);
  agg_ring_kernel<T, NV><<<grid, AGR_THREADS, smem, stream>>>(
      (const T*)X, d, ldx, perm, mstart, mlen, items, A.cta_first, pt_start, renorm, Xt, part,
      part_eta, S, stage, status, Ntot);
  SLS_LAUNCH_CHECK();
  agg_final_kernel<V, NV><<<(unsigned)fblocks, AGG_T, 0, stream>>>(
      d, mlen, pt_start, Mtot, Ntot, renorm, aux, part, part_eta, Xt);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

template <typename T>
int launch_agg_dtype(const void* X, int d, int64_t ldx, const int* perm, const int* mstart,
                     const int* mlen, int64_t Mtot, int64_t Ntot, int64_t fblocks, int renorm,
                     float* Xt,
                     int* pt_start, int2* items, int* aux, float* part, float* part_eta,
                     int* status, cudaStream_t stream) {
  constexpr int V = VecOf<T>::V;
  const int nv = (d / V + AGR_CT - 1) / AGR_CT;
#define SLS_AGG_NV(N)                                                                       \
  return launch_agg_t<T, N>(X, d, ldx, perm, mstart, mlen, Mtot, Ntot, fblocks, renorm, Xt, \
                            pt_start, items, aux, part, part_eta, status, stream)
  if (nv <= 1) SLS_AGG_NV(1);
  if (nv <= 2) SLS_AGG_NV(2);
  if (nv <= 4) SLS_AGG_NV(4);
  if (nv <= 8) SLS_AGG_NV(8);
#undef SLS_AGG_NV
  return SLS_ERR_UNSUPPORTED;
}
}  // namespace

int launch_aggregate(const void* X, int x_dtype, int d, int64_t ldx, const int* perm,
                     const int* mstart, const int* mlen, int64_t Mtot, int64_t Ntot, int renorm,
                     float* Xt, int* pt_start, int2* items, int* aux, float* part,
                     float* part_eta, int* status, cudaStream_t stream) {
  if (Mtot == 0) return SLS_OK;
  int64_t fblocks = Ntot / AGG_CH + 1;
  if (fblocks > 1024) fblocks = 1024;
  if (x_dtype == SLS_F32)
    return launch_agg_dtype<float>(X, d, ldx, perm, mstart, mlen, Mtot, Ntot, fblocks, renorm,
                                   Xt, pt_start, items, aux, part, part_eta, status, stream);
  return launch_agg_dtype<uint16_t>(X, d, ldx, perm, mstart, mlen, Mtot, Ntot, fblocks, renorm,
                                    Xt, pt_start, items, aux, part, part_eta, status, stream);
}

namespace {
template <typename T>
int launch_score_dtype(const void* X, int d, int64_t ldx, const ProbDesc* probs, int nprob,
                       int64_t nmax, float* part, float* score, cudaStream_t stream) {
  constexpr int V = VecOf<T>::V;
  const int nv = (d / V + AGG_T - 1) / AGG_T;
  const int KP = score_parts(nmax);
  const int64_t units = (int64_t)nprob * KP;
  const int blocks = (int)(units < 65535 ? units : 65535);
#define SLS_SCORE_NV(N)                                                                    \
  window_score_kernel<T, N><<<blocks, AGG_T, 0, stream>>>((const T*)X, d, ldx, probs, nprob, \
                                                          KP, part)
  if (nv <= 1)
    SLS_SCORE_NV(1);
  else if (nv <= 2)
    SLS_SCORE_NV(2);
  else if (nv <= 4)
    SLS_SCORE_NV(4);
  else if (nv <= 8)
    SLS_SCORE_NV(8);
  else
    return SLS_ERR_UNSUPPORTED;
#undef SLS_SCORE_NV
  SLS_LAUNCH_CHECK();
  const int cb = nprob < 4096 ? nprob : 4096;
  window_score_combine_kernel<<<cb, AGG_T, 0, stream>>>(d, probs, nprob, KP, 0, part, score);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}
}  // namespace

namespace {
template <typename T>
int launch_score_chunk_dtype(const void* X, int d, int64_t ldx, const ProbDesc* probs, int nprob,
                             int64_t nmax, float* part, float* score, int pos_scheme,
                             int pos_mode, int renorm, float* Xt, int32_t* pos,
                             int32_t* tok2macro, cudaStream_t stream) {
  constexpr int V = VecOf<T>::V;
  const int nv = (d / V + AGG_T - 1) / AGG_T;
  const int KP = chunk_parts_max(nmax);
  const int64_t units = (int64_t)nprob * KP;
  const int blocks = (int)(units < 65535 ? units : 65535);
#define SLS_SCORE_NV(N)                                                                   \
  do {                                                                                     \
    SLS_CUDA_TRY(cudaFuncSetAttribute(window_score_chunk_kernel<T, N>,                      \
                                      cudaFuncAttributeMaxDynamicSharedMemorySize,          \
                                      CHK_RING_BYTES));                                     \
    window_score_chunk_kernel<T, N><<<blocks, AGG_T, CHK_RING_BYTES, stream>>>(             \
        (const T*)X, d, ldx, probs, nprob, KP, part, pos_scheme, pos_mode, renorm, Xt, pos, \
        tok2macro);                                                                        \
  } while (0)
  if (nv <= 1)
    SLS_SCORE_NV(1);
  else if (nv <= 2)
    SLS_SCORE_NV(2);
  else if (nv <= 4)
    SLS_SCORE_NV(4);
  else if (nv <= 8)
    SLS_SCORE_NV(8);
  else
    return SLS_ERR_UNSUPPORTED;
#undef SLS_SCORE_NV
  SLS_LAUNCH_CHECK();
  const int cb = nprob < 4096 ? nprob : 4096;
  window_score_combine_kernel<<<cb, AGG_T, 0, stream>>>(d, probs, nprob, KP, 1, part, score);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}
}  // namespace

size_t score_part_floats(int64_t nprob, int64_t nmax, int d) {
  const int64_t kp = chunk_parts_max(nmax) > score_parts(nmax) ? chunk_parts_max(nmax)
                                                                 : score_parts(nmax);
  return (size_t)nprob * (size_t)kp * 2 * (size_t)d;
}

int launch_window_score_chunk(const void* X, int x_dtype, int d, int64_t ldx,
                              const ProbDesc* probs, int nprob, int64_t nmax, float* part,
                              float* score, int pos_scheme, int pos_mode, int renorm, float* Xt,
                              int32_t* pos, int32_t* tok2macro, cudaStream_t stream) {
  if (nprob <= 0) return SLS_OK;
  if (x_dtype == SLS_F32)
    return launch_score_chunk_dtype<float>(X, d, ldx, probs, nprob, nmax, part, score,
                                           pos_scheme, pos_mode, renorm, Xt, pos, tok2macro,
                                           stream);
  return launch_score_chunk_dtype<uint16_t>(X, d, ldx, probs, nprob, nmax, part, score,
                                            pos_scheme, pos_mode, renorm, Xt, pos, tok2macro,
                                            stream);
}

int launch_window_score(const void* X, int x_dtype, int d, int64_t ldx, const ProbDesc* probs,
                        int nprob, int64_t nmax, float* part, float* score, cudaStream_t stream) {
  if (nprob <= 0) return SLS_OK;
  if (x_dtype == SLS_F32)
    return launch_score_dtype<float>(X, d, ldx, probs, nprob, nmax, part, score, stream);
  return launch_score_dtype<uint16_t>(X, d, ldx, probs, nprob, nmax, part, score, stream);
}

}  // namespace sls
