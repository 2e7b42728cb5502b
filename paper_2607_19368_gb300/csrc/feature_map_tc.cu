// Random Fourier feature map on the 5th-generation tensor cores (sm_103a):
//   Phi = sqrt(2/D) * cos(X W^T + b)      (Sec. 3.2, Eq. rff_map)
// X (N x d) and W = Omega^T (D x d) are bf16, K-major (row-major, K = d
// contiguous); the contraction accumulates in fp32 in tensor memory; the
// epilogue adds b, takes the cosine, scales and stores Phi once (float32, or
// bfloat16 rounded to nearest even when the caller asks for bf16 storage).
//
// One persistent CTA per SM, 128 x 256 output tiles (tile index -> prompt,
// then m-block, then n-block innermost, so the D/256 tiles that share an X
// block run at the same time and X is read from HBM once).  One launch covers
// a batch of prompts (equal row counts, a fixed row stride in X); with a
// per-window route table, the row tiles whose windows all went to the chunk
// path (Sec. 3.6) are skipped by every role alike.  Warp roles:
//   warp 0  TMA producer: 128B-swizzled 128x64 (X) and 256x64 (W) bf16 tiles
//           into a 4-stage shared-memory ring (mbarrier complete_tx);
//   warp 1  MMA issuer: one elected thread issues tcgen05.mma (M=128, N=256,
//           K=16 per instruction, kind::f16 with bf16 inputs) into one of two
//           256-column fp32 accumulators in tensor memory; tcgen05.commit
//           releases ring stages and hands finished accumulators over;
//   warps 2-5 epilogue: tcgen05.ld 32x32b (one TMEM lane = one output row
//           per thread), cos epilogue; float32 features go through a
//           128B-swizzled 32 x 32 staging block per warp (two per warp, in
//           turn) and leave by TMA tensor stores, bfloat16 ones by direct
//           stores; then release the accumulator, so the next tile's MMAs
//           overlap this epilogue.
// Every wait is bounded; a wait that gives up records SLS_ERR_TIMEOUT, the
// other roles stop at their next wait, in-flight copies and MMAs are drained
// and the tensor memory is freed before the CTA exits.
#include <cuda.h>

#include <cstring>

#include "common.cuh"
#include "kernels.cuh"

namespace sls {

namespace {

constexpr int TC_BM = 128;
constexpr int TC_BN = 256;
constexpr int TC_BK = 64;  // one 128-byte swizzle atom of bf16
constexpr int TC_STAGES = 4;
constexpr int TC_A_BYTES = TC_BM * TC_BK * 2;
constexpr int TC_B_BYTES = TC_BN * TC_BK * 2;
constexpr int TC_STAGE_BYTES = TC_A_BYTES + TC_B_BYTES;
constexpr int TC_THREADS = 192;
constexpr int TC_TMEM_COLS = 2 * TC_BN;
constexpr int TC_EPI_WARPS = 4;
constexpr int TC_OUT_BYTES = 32 * 32 * 4;  // one 32 x 32 float32 staging block
constexpr size_t TC_SMEM =
    (size_t)TC_STAGES * TC_STAGE_BYTES + (size_t)TC_EPI_WARPS * 2 * TC_OUT_BYTES + 1024 + 256;

__device__ int g_fm_status;  // timeouts when the caller passes no status word

// K-major, 128-byte swizzle shared-memory matrix descriptor (tcgen05 format):
// start address >> 4, leading byte offset 16 B (unused for this layout),
// stride byte offset 1024 B (eight 128-byte rows), descriptor version 1,
// swizzle mode 2 (128B).
SLS_DEV uint64_t sw128_desc(uint32_t smem_addr) {
  uint64_t d = 0;
  d |= (uint64_t)((smem_addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)(16u >> 4) << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, M = 128, N = 256.
constexpr uint32_t TC_IDESC = (1u << 4) | (1u << 7) | (1u << 10) |
                              ((uint32_t)(TC_BN >> 3) << 17) | ((uint32_t)(TC_BM >> 4) << 24);

SLS_DEV void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

SLS_DEV void tc_mma(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(TC_IDESC), "r"(accumulate)
      : "memory");
}

SLS_DEV void tc_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

SLS_DEV void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
SLS_DEV void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

SLS_DEV void tc_ld32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
        "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
        "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Bounded wait that also gives up as soon as another role aborted.
SLS_DEV bool tc_wait(uint64_t* bar, unsigned parity, volatile int* abort_flag) {
  for (unsigned it = 0; it < (1u << 25); ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255) == 255 && *abort_flag) return false;
    if (it > 64) __nanosleep(20);
  }
  return false;
}

// cos(x) for the epilogue, branch-free for |x| <= 8192: Cody and Waite's
// reduction (W. J. Cody and W. Waite, "Software Manual for the Elementary
// Functions", 1980) by k = rint(x 2/pi) against pi/2 split into three
// float32 parts (P1 + P2 + P3, each the float32 rounding of what the
// previous parts leave of pi/2; with fused multiply-adds the first step is
// exact for |k| < 2^13), then the Taylor series of cos and sin on the
// reduced |r| <= pi/4 (truncation below 2e-9) in Horner form, and the
// quadrant k mod 4 picks cos r, -sin r, -cos r or sin r.  Larger or
// non-finite arguments take the library cosine (rff_cos_wide).
constexpr float RFF_COS_FAST_MAX = 8192.f;

__device__ __noinline__ float rff_cos_wide(float x) { return cosf(x); }

SLS_DEV float rff_cos_fast(float x) {
  const float k = rintf(x * 0x1.45f306p-1f);  // x * (2/pi)
  float r = __fmaf_rn(-k, 0x1.921fb6p+0f, x);
  r = __fmaf_rn(-k, -0x1.777a5cp-25f, r);
  r = __fmaf_rn(-k, -0x1.ee59dap-50f, r);
  const float z = r * r;
  // cos r = 1 - z/2! + z^2/4! - z^3/6! + z^4/8! - z^5/10!
  float c = __fmaf_rn(z, -1.f / 3628800.f, 1.f / 40320.f);
  c = __fmaf_rn(z, c, -1.f / 720.f);
  c = __fmaf_rn(z, c, 1.f / 24.f);
  c = __fmaf_rn(z, c, -0.5f);
  c = __fmaf_rn(z, c, 1.f);
  // sin r = r (1 - z/3! + z^2/5! - z^3/7! + z^4/9!)
  float s = __fmaf_rn(z, 1.f / 362880.f, -1.f / 5040.f);
  s = __fmaf_rn(z, s, 1.f / 120.f);
  s = __fmaf_rn(z, s, -1.f / 6.f);
  s = __fmaf_rn(r * z, s, r);
  const int q = (int)k;
  const float v = (q & 1) ? s : c;
  // quadrants 1 and 2 are negative
  return __uint_as_float(__float_as_uint(v) ^ ((unsigned)((q + 1) & 2) << 30));
}

// TMA tensor store of a 32 x 32 float32 block (3-d map: feature, row, prompt)
// from shared memory, tracked as a bulk async group of the issuing thread.
SLS_DEV void tma_store_3d(const CUtensorMap* map, uint32_t src, int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(src), "r"(x), "r"(y), "r"(z)
      : "memory");
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// at most one bulk group of this thread still reading shared memory
SLS_DEV void bulk_wait_read_le1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
SLS_DEV void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
SLS_DEV void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Rows of one launch: nb prompts of `rows` rows each, prompt b starting at
// X row b * x_stride (of the tensor map) and Phi row b * rows.  live, when
// set, holds one flag per window of `win` rows (nwin per prompt,
// prompt-major); a row tile is computed only if a window it touches is live.
struct FmJob {
  int nb;
  int rows;
  int x_stride;
  const int* live;
  int nwin;
  int win;
};

SLS_DEV bool fm_tile_live(const FmJob& J, int b, int mb) {
  if (!J.live) return true;
  const int r0 = mb * 128;
  const int r1 = min(J.rows, r0 + 128) - 1;
  for (int k = r0 / J.win; k <= r1 / J.win && k < J.nwin; ++k)
    if (J.live[(int64_t)b * J.nwin + k]) return true;
  return false;
}

// Four consecutive bfloat16 features, rounded to nearest even: one 8-byte
// store.
SLS_DEV void store4(uint16_t* p, float4 o) {
  const __nv_bfloat162 a = __floats2bfloat162_rn(o.x, o.y), b = __floats2bfloat162_rn(o.z, o.w);
  uint2 u;
  u.x = *reinterpret_cast<const unsigned*>(&a);
  u.y = *reinterpret_cast<const unsigned*>(&b);
  *reinterpret_cast<uint2*>(p) = u;
}

// OT: element type of Phi (float, or uint16_t for bfloat16 storage).
template <typename OT>
__global__ void __launch_bounds__(TC_THREADS, 1)
feature_map_tc_kernel(const __grid_constant__ CUtensorMap tmX,
                      const __grid_constant__ CUtensorMap tmW,
                      const __grid_constant__ CUtensorMap tmPhi, const float* __restrict__ bvec,
                      OT* __restrict__ Phi, FmJob J, int D, int K, float scale, int* status) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ uint64_t full_bar[TC_STAGES], empty_bar[TC_STAGES], tfull[2], tempty[2], done_bar;
  __shared__ uint32_t tmem_holder;
  __shared__ volatile int s_abort;

  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  const uint32_t smem_base = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m_tiles = (J.rows + TC_BM - 1) / TC_BM;
  const int n_tiles = D / TC_BN;
  const int per_prompt = m_tiles * n_tiles;
  const int num_tiles = J.nb * per_prompt;
  const int k_blocks = (K + TC_BK - 1) / TC_BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < TC_STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 4);
    }
    mbar_init(&done_bar, 1);
    mbar_fence_init();
    s_abort = 0;
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&tmem_holder)),
                 "r"(TC_TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tmem_holder;

  auto fail = [&]() {
    s_abort = 1;
    atomicExch(status, SLS_ERR_TIMEOUT);
  };

  if (warp == 0) {
    // ------------------------------ TMA producer ------------------------------
    if (lane == 0) {
      unsigned it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        const int pb = tile / per_prompt, rem = tile % per_prompt;
        const int mb = rem / n_tiles, nb = rem % n_tiles;
        if (!fm_tile_live(J, pb, mb)) continue;
        const int y = pb * J.x_stride + mb * TC_BM;
        for (int kb = 0; kb < k_blocks; ++kb, ++it) {
          const int s = it % TC_STAGES;
          const unsigned par = (it / TC_STAGES) & 1u;
          if (!tc_wait(&empty_bar[s], par ^ 1u, &s_abort)) {
            fail();
            ok = false;
            break;
          }
          const uint32_t a_dst = smem_base + s * TC_STAGE_BYTES;
          const uint32_t b_dst = a_dst + TC_A_BYTES;
          mbar_expect_tx(&full_bar[s], TC_STAGE_BYTES);
          tma_load_2d(a_dst, &tmX, kb * TC_BK, y, smem_u32(&full_bar[s]));
          tma_load_2d(b_dst, &tmW, kb * TC_BK, nb * TC_BN, smem_u32(&full_bar[s]));
        }
      }
      // drain: every issued stage has landed before the CTA may exit
      const unsigned first = it > TC_STAGES ? it - TC_STAGES : 0;
      for (unsigned c = first; c < it; ++c) {
        for (unsigned w = 0; w < (1u << 25); ++w) {
          if (mbar_try_wait(&full_bar[c % TC_STAGES], (c / TC_STAGES) & 1u)) break;
          __nanosleep(20);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer --------------------------------
    if (lane == 0) {
      unsigned it = 0, acc_it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        if (!fm_tile_live(J, tile / per_prompt, (tile % per_prompt) / n_tiles)) continue;
        const int acc = acc_it & 1;
        const unsigned apar = (acc_it >> 1) & 1u;
        if (!tc_wait(&tempty[acc], apar ^ 1u, &s_abort)) {
          fail();
          break;
        }
        tc_fence_after();
        const uint32_t tmem_d = tmem_base + (uint32_t)(acc * TC_BN);
        for (int kb = 0; kb < k_blocks; ++kb, ++it) {
          const int s = it % TC_STAGES;
          const unsigned par = (it / TC_STAGES) & 1u;
          if (!tc_wait(&full_bar[s], par, &s_abort)) {
            fail();
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_addr = smem_base + s * TC_STAGE_BYTES;
          const uint32_t b_addr = a_addr + TC_A_BYTES;
#pragma unroll
          for (int kk = 0; kk < TC_BK / 16; ++kk) {
            tc_mma(tmem_d, sw128_desc(a_addr + kk * 32), sw128_desc(b_addr + kk * 32),
                   (kb > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(smem_u32(&empty_bar[s]));
        }
        if (ok) tc_commit(smem_u32(&tfull[acc]));
        ++acc_it;
      }
      // all MMAs issued by this thread have completed before TMEM is freed
      tc_commit(smem_u32(&done_bar));
      for (unsigned w = 0; w < (1u << 25); ++w) {
        if (mbar_try_wait(&done_bar, 0)) break;
        __nanosleep(20);
      }
    }
  } else {
    // ------------------------------ epilogue ----------------------------------
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    // two 32 x 32 float32 staging blocks of this warp, 1024-byte aligned (the
    // 128-byte swizzle repeats every eight rows of 128 bytes)
    const uint32_t stg0 = smem_base + (uint32_t)(TC_STAGES * TC_STAGE_BYTES) +
                          (uint32_t)((warp - 2) * 2 * TC_OUT_BYTES);
    unsigned char* stg0p = smem + TC_STAGES * TC_STAGE_BYTES + (warp - 2) * 2 * TC_OUT_BYTES;
    unsigned acc_it = 0, blk = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
      const int pb = tile / per_prompt, rem = tile % per_prompt;
      const int mb = rem / n_tiles, nb = rem % n_tiles;
      if (!fm_tile_live(J, pb, mb)) continue;
      const int acc = acc_it & 1;
      const unsigned apar = (acc_it >> 1) & 1u;
      if (!tc_wait(&tfull[acc], apar, &s_abort)) {
        if (lane == 0) fail();
        break;
      }
      tc_fence_after();
      const int row = mb * TC_BM + q * 32 + lane;
      const float* bb = bvec + (size_t)nb * TC_BN;
      for (int c0 = 0; c0 < TC_BN; c0 += 32, ++blk) {
        uint32_t v[32];
        tc_ld32(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * TC_BN + c0), v);
        float th[32];
        float amax = 0.f;
#pragma unroll
        for (int e = 0; e < 32; e += 4) {
          const float4 bq = __ldg(reinterpret_cast<const float4*>(bb + c0 + e));
          th[e + 0] = __uint_as_float(v[e + 0]) + bq.x;
          th[e + 1] = __uint_as_float(v[e + 1]) + bq.y;
          th[e + 2] = __uint_as_float(v[e + 2]) + bq.z;
          th[e + 3] = __uint_as_float(v[e + 3]) + bq.w;
          amax = fmaxf(amax, fmaxf(fmaxf(fabsf(th[e]), fabsf(th[e + 1])),
                                   fmaxf(fabsf(th[e + 2]), fabsf(th[e + 3]))));
        }
        if (__all_sync(0xffffffffu, amax <= RFF_COS_FAST_MAX)) {
#pragma unroll
          for (int e = 0; e < 32; ++e) th[e] = scale * rff_cos_fast(th[e]);
        } else {
          for (int e = 0; e < 32; ++e) th[e] = scale * rff_cos_wide(th[e]);
        }
        if constexpr (sizeof(OT) == 4) {
          // row `lane` of the block: its eight 16-byte pieces at the swizzled
          // positions (piece c of row l goes to c ^ (l mod 8))
          const uint32_t sb = (blk & 1u) ? TC_OUT_BYTES : 0u;
          if (lane == 0) bulk_wait_read_le1();  // the block's previous store has read it
          __syncwarp();
          unsigned char* rowp = stg0p + sb + lane * 128;
#pragma unroll
          for (int c = 0; c < 8; ++c)
            *reinterpret_cast<float4*>(rowp + ((c ^ (lane & 7)) << 4)) =
                make_float4(th[4 * c], th[4 * c + 1], th[4 * c + 2], th[4 * c + 3]);
          fence_async_smem();
          __syncwarp();
          // a block wholly past the prompt's last row is not stored at all
          if (lane == 0 && mb * TC_BM + q * 32 < J.rows)
            tma_store_3d(&tmPhi, stg0 + sb, nb * TC_BN + c0, mb * TC_BM + q * 32, pb);
        } else {
          if (row < J.rows) {
            OT* out = Phi + ((int64_t)pb * J.rows + row) * D + (int64_t)nb * TC_BN + c0;
#pragma unroll
            for (int e = 0; e < 32; e += 4)
              store4(out + e, make_float4(th[e], th[e + 1], th[e + 2], th[e + 3]));
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
      ++acc_it;
    }
    // every tensor store of this warp has completed before the CTA exits
    if (lane == 0) bulk_wait_all();
    __syncwarp();
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(TC_TMEM_COLS)
                 : "memory");
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

bool make_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t ld,
              uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {ld * 2};
  const cuuint32_t box[2] = {(cuuint32_t)TC_BK, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// float32 output map: dims (D, rows, nb), 32 x 32 x 1 boxes, 128-byte
// swizzle (one box row is 128 bytes)
bool make_out_map(CUtensorMap* map, void* base, uint64_t D, uint64_t rows, uint64_t nb) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[3] = {D, rows, nb};
  const cuuint64_t strides[2] = {D * 4, rows * D * 4};
  const cuuint32_t box[3] = {32, 32, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && v > 0)
      sms = v;
    else
      return 1;
  }
  return sms;
}

}  // namespace

int launch_feature_map_tc_batched(const void* X, int64_t nb, int64_t rows, int64_t x_stride,
                                  int d, int64_t ldx, const void* W, const float* b, int D,
                                  void* Phi, const int* live, int nwin, int win,
                                  cudaStream_t stream, int* status, int phi_bf16) {
  // shapes the kernel covers; anything else takes the SIMT path
  if (nb <= 0 || rows <= 0 || x_stride < rows || D % TC_BN != 0 || d % 8 != 0 || ldx % 8 != 0)
    return SLS_ERR_UNSUPPORTED;
  const int64_t map_rows = (nb - 1) * x_stride + rows;
  const int64_t m_tiles = (rows + TC_BM - 1) / TC_BM;
  if (map_rows > (int64_t)INT32_MAX - TC_BM || nb * m_tiles * (D / TC_BN) > (int64_t)INT32_MAX)
    return SLS_ERR_UNSUPPORTED;
  if (live && (nwin < 1 || win < 1)) return SLS_ERR_INVALID_ARG;
  if (((uintptr_t)X & 15) || ((uintptr_t)W & 15) || ((uintptr_t)b & 15) || ((uintptr_t)Phi & 15))
    return SLS_ERR_UNSUPPORTED;
  CUtensorMap mx, mw, mp;
  if (!make_map(&mx, X, (uint64_t)map_rows, (uint64_t)d, (uint64_t)ldx, TC_BM))
    return SLS_ERR_UNSUPPORTED;
  if (!make_map(&mw, W, (uint64_t)D, (uint64_t)d, (uint64_t)d, TC_BN)) return SLS_ERR_UNSUPPORTED;
  // float32 Phi as (feature, row, prompt): a block's rows past the prompt's
  // last row fall outside the map and are not written
  if (phi_bf16) {
    memset(&mp, 0, sizeof(mp));
  } else if (!make_out_map(&mp, Phi, (uint64_t)D, (uint64_t)rows, (uint64_t)nb)) {
    return SLS_ERR_UNSUPPORTED;
  }
  int* st = status;
  if (!st) SLS_CUDA_TRY(cudaGetSymbolAddress((void**)&st, g_fm_status));
  SLS_CUDA_TRY(cudaFuncSetAttribute(feature_map_tc_kernel<float>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)TC_SMEM));
  SLS_CUDA_TRY(cudaFuncSetAttribute(feature_map_tc_kernel<uint16_t>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)TC_SMEM));
  const int64_t tiles = nb * m_tiles * (D / TC_BN);
  const int grid = tiles < sm_count() ? (int)tiles : sm_count();
  const float scale = (float)sqrt(2.0 / (double)D);
  FmJob J{(int)nb, (int)rows, (int)x_stride, live, nwin, win};
  if (phi_bf16)
    feature_map_tc_kernel<uint16_t><<<grid, TC_THREADS, TC_SMEM, stream>>>(
        mx, mw, mp, b, (uint16_t*)Phi, J, D, d, scale, st);
  else
    feature_map_tc_kernel<float><<<grid, TC_THREADS, TC_SMEM, stream>>>(mx, mw, mp, b, (float*)Phi,
                                                                      J, D, d, scale, st);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

int launch_feature_map_tc(const void* X, int64_t N, int d, int64_t ldx, const void* W,
                          const float* b, int D, void* Phi, cudaStream_t stream,
                          int* status, int phi_bf16) {
  return launch_feature_map_tc_batched(X, 1, N, N, d, ldx, W, b, D, Phi, nullptr, 0, 0, stream,
                                       status, phi_bf16);
}

}  // namespace sls
