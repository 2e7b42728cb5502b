// C ABI of the Spectral-LSH compression pass (include/sls.h).
//
// Host code here only validates arguments, carves caller-provided workspaces
// and enqueues kernels on the caller's stream; it never synchronises, never
// allocates and never computes any part of the method itself.
#include <cmath>
#include <cstring>

#include "common.cuh"
#include "kernels.cuh"
#include "segment.cuh"

#include <atomic>

using namespace sls;

namespace sls {
static std::atomic<long long> g_launches{0};
void count_launch(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
}  // namespace sls

namespace {

void* g_phase_events[2 * SLS_NUM_PHASES];
bool g_phase_on = false;

inline void phase_mark(int phase, int end, cudaStream_t s) {
  if (g_phase_on) cudaEventRecord((cudaEvent_t)g_phase_events[2 * phase + end], s);
}

// ---------------------------------------------------------------------------
// workspace carving
// ---------------------------------------------------------------------------

// In the debug build (-DSLS_DEBUG) every carved region is followed by a
// guard band of kGuardBytes filled with kGuardByte when a call starts and
// checked when it ends (guard_check_kernel): a write past the end of a
// region shows up as SLS_ERR_BOUNDS in the workspace status word.  The
// ordinary build carves no guards.
#ifdef SLS_DEBUG
constexpr size_t kGuardBytes = 256;
constexpr int kMaxGuards = 48;
#else
constexpr size_t kGuardBytes = 0;
constexpr int kMaxGuards = 1;
#endif
constexpr unsigned char kGuardByte = 0xA5;

struct GuardList {
  int n;
  size_t off[kMaxGuards];
};

struct Carver {
  char* base;
  size_t off = 0;
  GuardList guards{};
  explicit Carver(void* b) : base((char*)b) {}
  template <typename T>
  T* take(size_t count) {
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += sls_align256(count * sizeof(T));
    if (kGuardBytes) {
      if (guards.n < kMaxGuards) guards.off[guards.n++] = off;
      off += kGuardBytes;
    }
    return p;
  }
};

__global__ void guard_fill_kernel(unsigned char* base, GuardList g) {
  if ((int)blockIdx.x >= g.n) return;
  unsigned char* p = base + g.off[blockIdx.x];
  for (int b = threadIdx.x; b < (int)kGuardBytes; b += blockDim.x) p[b] = kGuardByte;
}

__global__ void guard_check_kernel(const unsigned char* base, GuardList g, int* status) {
  if ((int)blockIdx.x >= g.n) return;
  const unsigned char* p = base + g.off[blockIdx.x];
  for (int b = threadIdx.x; b < (int)kGuardBytes; b += blockDim.x)
    if (p[b] != kGuardByte) atomicExch(status, SLS_ERR_BOUNDS);
}

// Debug-build self-test: which = 0 writes one element past the end of a
// carved region of n ints (into its guard band: still inside the caller's
// workspace); which = 1 makes a guarded write at index n, which the guard
// skips.  Either must end in SLS_ERR_BOUNDS.
__global__ void debug_selftest_kernel(int* region, int n, int which, int* status) {
  if (threadIdx.x != 0) return;
  if (which == 0) {
    reinterpret_cast<unsigned char*>(region + n)[0] = (unsigned char)(kGuardByte ^ 0xFF);
  } else {
    const int idx = n;
    SLS_DBG_GUARD(status, idx < n) region[idx] = 1;
  }
}

// Debug build: fill the guard bands of a carved workspace (no-op otherwise).
int guards_arm(const Carver& cv, cudaStream_t s) {
  if (kGuardBytes == 0 || cv.base == nullptr || cv.guards.n == 0) return SLS_OK;
  guard_fill_kernel<<<cv.guards.n, 256, 0, s>>>((unsigned char*)cv.base, cv.guards);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

// Debug build: check the guard bands, SLS_ERR_BOUNDS into *status if one
// was written (no-op otherwise).
int guards_check(const Carver& cv, int* status, cudaStream_t s) {
  if (kGuardBytes == 0 || cv.base == nullptr || cv.guards.n == 0) return SLS_OK;
  guard_check_kernel<<<cv.guards.n, 256, 0, s>>>((const unsigned char*)cv.base, cv.guards,
                                                 status);
  SLS_LAUNCH_CHECK();
  return SLS_OK;
}

// host-side configuration arithmetic (Sec. 3.3, 3.5, 3.6)
struct Region {
  int64_t pf, pl, Nc;
};

Region region_of(const sls_config_t* c, int64_t N) {
  Region R;
  R.pf = c->preserve_first < 0 ? 0 : (c->preserve_first > N ? N : c->preserve_first);
  int64_t pl = c->preserve_last < 0 ? 0 : c->preserve_last;
  if (pl > N - R.pf) pl = N - R.pf;
  R.pl = pl;
  R.Nc = N - R.pf - R.pl;
  return R;
}

bool is_identity(const sls_config_t* c, int64_t N) {
  return !(c->rho > 1.0) || region_of(c, N).Nc <= 0;
}

int64_t target_count(int64_t n, double rho) { return (int64_t)std::ceil((double)n / rho); }

int auto_bits(int64_t n, double rho) {
  int b = 1;
  while (b < 32 && std::ldexp(1.0, b) * rho < (double)n) ++b;
  return b;
}

int64_t chunk_k(double rho) {
  const double k = std::rint(rho);
  return k < 1.0 ? 1 : (int64_t)k;
}

// Per-window budgets of the adaptive backend: one seat per window, the rest
// by largest remainder over quotas E (L_w - 1) / (N_c - W), ties to the lower
// window index.  All windows but the last have the same length, so the result
// is described by: full windows get m_full (+1 for the first left_full of
// them), the last window gets m_last.
struct Budgets {
  int64_t W, L_full, L_last, m_full, m_last, left_full;
};

bool adaptive_budgets(int64_t Nc, int64_t window, int64_t Mstar, Budgets* B) {
  const int64_t W = (Nc + window - 1) / window;
  if (W < 1 || Mstar < W || Mstar > Nc) return false;
  const int64_t L_last = Nc - (W - 1) * window;
  const bool partial = L_last != window;
  const int64_t W_full = partial ? W - 1 : W;
  const int64_t E = Mstar - W, den = Nc - W;
  B->W = W;
  B->L_full = window;
  B->L_last = L_last;
  if (E == 0 || den == 0) {
    B->m_full = 1;
    B->m_last = 1;
    B->left_full = 0;
    return true;
  }
  const int64_t base_f = E * (window - 1) / den, rem_f = E * (window - 1) % den;
  const int64_t base_l = E * (L_last - 1) / den, rem_l = E * (L_last - 1) % den;
  int64_t left = E - (W_full * base_f + (partial ? base_l : 0));
  int64_t left_full = 0, last_extra = 0;
  if (!partial) {
    left_full = left;
  } else if (rem_l > rem_f) {
    last_extra = left > 0 ? 1 : 0;
    left_full = left - last_extra;
  } else {
    left_full = left < W_full ? left : W_full;
    last_extra = left - left_full;
  }
  B->m_full = 1 + base_f;
  B->m_last = 1 + (partial ? base_l + last_extra : base_f);
  B->left_full = left_full;
  if (!partial) B->m_last = B->m_full + ((W - 1) < left_full ? 1 : 0);
  return true;
}

// ---------------------------------------------------------------------------
// device-side table construction (no host-to-device copies)
// ---------------------------------------------------------------------------

__global__ void plan_kernel(ProbDesc* __restrict__ probs, int64_t B, int64_t N, int64_t M,
                            int64_t pf, int64_t Nc, int64_t W, int64_t window, int64_t m_full,
                            int64_t m_last, int64_t left_full, int64_t L_last, double rho,
                            int cfg_bits, int spectral, int64_t k_chunk, int64_t q1_stride) {
  const int64_t total = B * W;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t b = e / W, w = e % W;
    const int64_t start = w * window;
    const int64_t n = (w == W - 1) ? L_last : window;
    int64_t m, prefix;
    if (w < W - 1 || W == 1) {
      m = (W == 1) ? m_last : m_full + (w < left_full ? 1 : 0);
      prefix = w * m_full + (w < left_full ? w : left_full);
    } else {
      m = m_last;
      prefix = w * m_full + (w < left_full ? w : left_full);
    }
    int bits = cfg_bits;
    if (bits <= 0) {
      bits = 1;
      while (bits < 32 && ldexp(1.0, bits) * rho < (double)n) ++bits;
    }
    ProbDesc P;
    P.tok_row = b * N + pf + start;
    P.q1off = b * q1_stride + start;
    P.out0 = b * M + pf + prefix;
    P.phi_row = b * Nc + start;
    P.pos0 = (int)(pf + start);
    P.n = (int)n;
    P.m = (int)m;
    P.bits = bits;
    P.spectral = spectral;
    P.chunk_k = (int)k_chunk;
    P.spec_idx = -1;
    P.out_local = (int)(pf + prefix);
    probs[e] = P;
  }
}

// Routing (Sec. 3.6) and compaction of the spectral problems, one CTA.
// mode: 0 = all spectral, 1 = none, 2 = adaptive router with `score`.
__global__ void __launch_bounds__(1024)
route_compact_kernel(ProbDesc* __restrict__ probs, int nprob, int mode,
                     const float* __restrict__ score, double rho, double tau,
                     int* __restrict__ spec_list, int64_t* __restrict__ lz_row0,
                     int* __restrict__ lz_n, int64_t* __restrict__ lz_q1off,
                     int* __restrict__ nspec, int32_t* __restrict__ route_out,
                     int* __restrict__ lz_reff) {
  __shared__ int sh[33];
  const int tid = threadIdx.x;
  const int chunk = (nprob + 1023) / 1024;
  const int b = min(nprob, tid * chunk), e = min(nprob, b + chunk);
  auto decide = [&](int p) -> int {
    if (mode == 0) return 1;
    if (mode == 1) return 0;
    if (rho >= 16.0) return 1;
    if (probs[p].n <= 4) return 0;
    return ((double)score[p] >= tau) ? 1 : 0;
  };
  int cnt = 0;
  for (int p = b; p < e; ++p) cnt += decide(p);
  // block exclusive scan
  const int lane = tid & 31, warp = tid >> 5;
  int x = cnt;
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = sh[lane];
    int z = w;
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, z, o);
      if (lane >= o) z += y;
    }
    sh[lane] = z - w;
    if (lane == 31) sh[32] = z;
  }
  __syncthreads();
  int off = sh[warp] + x - cnt;
  for (int p = b; p < e; ++p) {
    const int s = decide(p);
    probs[p].spectral = s;
    probs[p].spec_idx = s ? off : -1;
    if (route_out) route_out[p] = s;
    if (s) {
      spec_list[off] = p;
      lz_row0[off] = probs[p].phi_row;
      lz_n[off] = probs[p].n;
      lz_q1off[off] = probs[p].q1off;
      // -1 until the Lanczos kernel finishes; stays -1 if one of its waits
      // gave up, and the eigen and Ritz kernels then treat the problem as empty
      lz_reff[off] = -1;
      ++off;
    }
  }
  if (tid == 0) *nspec = sh[32];
}

__global__ void finish_reff_kernel(const ProbDesc* __restrict__ probs, int nprob,
                                   const int* __restrict__ r_eff_spec, int32_t* __restrict__ out) {
  for (int p = blockIdx.x * blockDim.x + threadIdx.x; p < nprob; p += gridDim.x * blockDim.x) {
    const int s = probs[p].spec_idx;
    out[p] = (s >= 0) ? r_eff_spec[s] : 0;
  }
}

__global__ void single_prob_kernel(ProbDesc* P, int64_t n, int64_t m, int bits) {
  ProbDesc d;
  d.tok_row = 0;
  d.q1off = 0;
  d.out0 = 0;
  d.phi_row = 0;
  d.pos0 = 0;
  d.n = (int)n;
  d.m = (int)m;
  d.bits = bits;
  d.spectral = 1;
  d.chunk_k = 0;
  d.spec_idx = 0;
  d.out_local = 0;
  *P = d;
}

// ---------------------------------------------------------------------------
// the compress pipeline's workspace
// ---------------------------------------------------------------------------

struct CompressPlan {
  int backend;
  int64_t B, N, M, pf, pl, Nc, Mstar;
  Budgets bud;
  int64_t nprob;     // problems (B * W)
  int64_t nmax, mmax;
  int D, r;
  int bits_max;
  int lz_groups, lz_g;
  int seg_slots;
  int64_t k_chunk;
  int normalize;
  int phi_bf16;
};

struct CompressWs {
  int* status;
  ProbDesc* probs;
  int* spec_list;
  int64_t* lz_row0;
  int* lz_n;
  int64_t* lz_q1off;
  int* nspec;
  float* score;
  float* score_part;  // window-score partial sums (adaptive backend)
  float2* norm_scratch;  // row-normalised operator: column sums
  int32_t* route;  // spectral flag per problem
  void* Phi;  // float32, or bfloat16 bits when the plan stores Phi as bf16
  float2* Q;
  double *alpha, *beta, *theta, *S;
  int* r_eff;
  float* U;
  uint32_t* codes;
  void* lz_scratch;
  size_t lz_bytes;
  void* seg_scratch;
  int *perm, *mstart, *mlen;
  int* pt_start;
  int2* items;
  int* counts;
  float *part, *part_eta;
  size_t total;
  Carver cv{nullptr};    // the head of the workspace (guards in the debug build)
  Carver tail{nullptr};  // the tail (aggregation partials, router partials)
};

int num_sms_host() {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        sms <= 0)
      sms = 152;
  }
  return sms;
}

int make_plan(const sls_config_t* c, int64_t B, int64_t N, CompressPlan* P,
              bool launch = true) {
  const Region R = region_of(c, N);
  P->backend = c->backend;
  P->B = B;
  P->N = N;
  P->pf = R.pf;
  P->pl = R.pl;
  P->Nc = R.Nc;
  P->D = c->D;
  P->r = c->r;
  P->k_chunk = chunk_k(c->rho);
  P->normalize = c->normalize ? 1 : 0;
  P->phi_bf16 = (c->phi_dtype == SLS_BF16) ? 1 : 0;
  if (c->backend == SLS_BACKEND_CHUNK) {
    P->Mstar = (R.Nc + P->k_chunk - 1) / P->k_chunk;
    P->bud = Budgets{1, R.Nc, R.Nc, P->Mstar, P->Mstar, 0};
  } else if (c->backend == SLS_BACKEND_GLOBAL) {
    P->Mstar = target_count(R.Nc, c->rho);
    P->bud = Budgets{1, R.Nc, R.Nc, P->Mstar, P->Mstar, 0};
  } else {
    P->Mstar = target_count(R.Nc, c->rho);
    if (c->window < 1) return SLS_ERR_INVALID_ARG;
    if (!adaptive_budgets(R.Nc, c->window, P->Mstar, &P->bud)) return SLS_ERR_INVALID_ARG;
  }
  P->M = R.pf + P->Mstar + R.pl;
  P->nprob = B * P->bud.W;
  P->nmax = P->bud.L_full > P->bud.L_last ? P->bud.L_full : P->bud.L_last;
  P->mmax = P->bud.m_full + 1 > P->bud.m_last ? P->bud.m_full + 1 : P->bud.m_last;
  if (P->mmax > P->nmax) P->mmax = P->nmax;
  if (c->bits > 0) {
    P->bits_max = c->bits;
  } else {
    P->bits_max = auto_bits(P->nmax, c->rho);
  }
  if (c->backend == SLS_BACKEND_CHUNK || !launch) {
    P->lz_groups = 0;
    P->lz_g = 0;
  } else {
    int st = lanczos_plan(P->nmax, c->D, c->r, (int)P->nprob, &P->lz_groups, &P->lz_g);
    if (st != SLS_OK) return st;
  }
  const int64_t slots = 2 * (int64_t)num_sms_host();
  P->seg_slots = (int)(P->nprob < slots ? P->nprob : slots);
  return SLS_OK;
}

void carve(const CompressPlan& P, void* ws, CompressWs* W) {
  Carver cv(ws);
  const int64_t np = P.nprob;
  const int64_t rows = P.B * P.Nc;  // compressible rows (Phi / Q / U)
  const int64_t toks = P.B * P.N, macs = P.B * P.M;
  const bool spectral = P.backend != SLS_BACKEND_CHUNK;
  W->status = cv.take<int>(64);
  W->probs = cv.take<ProbDesc>(np);
  W->spec_list = cv.take<int>(np);
  W->lz_row0 = cv.take<int64_t>(np);
  W->lz_n = cv.take<int>(np);
  W->lz_q1off = cv.take<int64_t>(np);
  W->nspec = cv.take<int>(1);
  W->score = cv.take<float>(np);
  W->route = cv.take<int>(np);
  W->Phi = cv.take<char>(spectral ? (size_t)rows * P.D * (P.phi_bf16 ? 2 : 4) : 0);
  W->norm_scratch = cv.take<float2>(
      (spectral && P.normalize)
          ? feature_normalize_scratch_bytes(P.nmax, P.D, (int)P.nprob) / sizeof(float2)
          : 0);
  W->Q = cv.take<float2>(spectral ? (size_t)rows * ((P.r + 1) & ~1) : 0);
  W->alpha = cv.take<double>(spectral ? (size_t)np * P.r : 0);
  W->beta = cv.take<double>(spectral ? (size_t)np * P.r : 0);
  W->theta = cv.take<double>(spectral ? (size_t)np * P.r : 0);
  W->S = cv.take<double>(spectral ? (size_t)np * P.r * P.r : 0);
  W->r_eff = cv.take<int>(np);
  W->U = cv.take<float>(spectral ? (size_t)rows * P.r : 0);
  W->codes = cv.take<uint32_t>(spectral ? (size_t)rows : 0);
  W->lz_bytes = spectral ? lanczos_scratch_bytes(P.nmax, P.D, P.r, P.lz_groups, P.lz_g) : 0;
  W->lz_scratch = cv.take<char>(W->lz_bytes);
  W->seg_scratch = cv.take<char>(segment_scratch_bytes(P.nmax, P.mmax, P.seg_slots));
  W->perm = cv.take<int>(toks);
  W->mstart = cv.take<int>(macs);
  W->mlen = cv.take<int>(macs);
  W->pt_start = cv.take<int>(macs);
  W->items = cv.take<int2>(agg_item_capacity(macs, toks));
  W->counts = cv.take<int>(agg_aux_ints(macs, toks));
  W->part = nullptr;  // carved from the tail (depends on d)
  W->part_eta = nullptr;
  W->total = cv.off;
  W->cv = cv;
}

bool ptr_ok(const void* p) { return p != nullptr && ((uintptr_t)p & 15u) == 0; }

int validate_config(const sls_config_t* c) {
  if (!c) return SLS_ERR_INVALID_ARG;
  if (c->backend < 0 || c->backend > 3) return SLS_ERR_INVALID_ARG;
  if (!(c->rho == c->rho)) return SLS_ERR_INVALID_ARG;
  if (c->rho > 1.0 && c->backend != SLS_BACKEND_CHUNK) {
    if (c->D < 4 || c->D > SLS_MAX_D || (c->D & 3)) return SLS_ERR_INVALID_ARG;
    if (c->r < 1 || c->r > SLS_MAX_R) return SLS_ERR_INVALID_ARG;
    if (c->bits < 0 || c->bits > SLS_MAX_BITS) return SLS_ERR_INVALID_ARG;
  }
  if (c->pos_scheme < 0 || c->pos_scheme > 2) return SLS_ERR_INVALID_ARG;
  if (c->pos_mode < 0 || c->pos_mode > 1) return SLS_ERR_INVALID_ARG;
  if (c->preserve_first < 0 || c->preserve_last < 0) return SLS_ERR_INVALID_ARG;
  if (c->phi_dtype != SLS_F32 && c->phi_dtype != SLS_BF16) return SLS_ERR_INVALID_ARG;
  // bf16 storage: 16-byte rows for the bulk copies; the normalised operator
  // scales float32 rows in place
  if (c->phi_dtype == SLS_BF16 && c->rho > 1.0 && c->backend != SLS_BACKEND_CHUNK &&
      ((c->D & 7) || c->normalize))
    return SLS_ERR_UNSUPPORTED;
  return SLS_OK;
}

// Bytes of the workspace tail: the aggregation partials (and the router's
// window partials for the adaptive backend), carved in this order.
size_t tail_bytes(const CompressPlan& P, int64_t toks, int d, int backend) {
  Carver cv(nullptr);
  cv.take<float>(agg_part_capacity(toks) * (size_t)d);
  cv.take<float>(agg_part_capacity(toks));
  if (backend == SLS_BACKEND_ADAPTIVE) cv.take<float>(score_part_floats(P.nprob, P.nmax, d));
  return cv.off;
}

// One Lanczos problem (sls_lanczos_topr_ex); inject_fail = 1 runs the
// failure self-test (the kernel's give-up path, see LanczosBatch).
int lanczos_single(const void* Phi, int phi_dtype, int64_t N, int D, int r, const double* q1,
                   double tol, double* theta, float* U, int32_t* r_eff, double* alpha,
                   double* beta, void* workspace, size_t workspace_bytes, void* stream,
                   int inject_fail) {
  if (N < 1 || D < 4 || D > SLS_MAX_D || r < 1 || r > SLS_MAX_R || !(tol >= 0.0))
    return SLS_ERR_INVALID_ARG;
  if (phi_dtype != SLS_F32 && phi_dtype != SLS_BF16) return SLS_ERR_INVALID_ARG;
  if ((D & 3) != 0 || (phi_dtype == SLS_BF16 && (D & 7) != 0)) return SLS_ERR_UNSUPPORTED;
  if (!ptr_ok(Phi) || !q1 || !theta || !U || !r_eff) return SLS_ERR_INVALID_ARG;
  const size_t need = sls_lanczos_workspace_size(N, D, r);
  if (need == 0) return SLS_ERR_UNSUPPORTED;
  if (!workspace || workspace_bytes < need) return SLS_ERR_WORKSPACE;
  int groups = 0, g = 0;
  int st = lanczos_plan(N, D, r, 1, &groups, &g);
  if (st != SLS_OK) return st;
  cudaStream_t s = (cudaStream_t)stream;
  Carver cv(workspace);
  int* status = cv.take<int>(64);
  float2* Q = cv.take<float2>((size_t)N * ((r + 1) & ~1));
  double* al = cv.take<double>(r);
  double* be = cv.take<double>(r);
  double* S = cv.take<double>((size_t)r * r);
  const size_t lzb = lanczos_scratch_bytes(N, D, r, groups, g);
  void* lz = cv.take<char>(lzb);
  SLS_CUDA_TRY(cudaMemsetAsync(status, 0, 256, s));
  if ((st = guards_arm(cv, s)) != SLS_OK) return st;
  // -1 until the Lanczos kernel finishes; stays -1 if one of its waits gave
  // up, and the eigen and Ritz kernels then treat the problem as empty
  SLS_CUDA_TRY(cudaMemsetAsync(r_eff, 0xff, sizeof(int32_t), s));
  LanczosBatch bt{};
  bt.Phi = Phi;
  bt.phi_bf16 = (phi_dtype == SLS_BF16) ? 1 : 0;
  bt.D = D;
  bt.r = r;
  bt.tol = tol;
  bt.q1 = q1;
  bt.n_single = N;
  bt.nprob_max = 1;
  bt.Q = Q;
  bt.alpha = al;
  bt.beta = be;
  bt.theta = theta;
  bt.S = S;
  bt.r_eff = r_eff;
  bt.nmax = N;
  bt.inject_fail = inject_fail;
  const bool small = lanczos_window_fits(N, D, r);
  if (small) {
    if ((st = launch_lanczos_window(bt, s)) != SLS_OK) return st;
  } else if ((st = launch_lanczos(bt, lz, lzb, status, groups, g, s)) != SLS_OK) {
    return st;
  }
  if ((st = launch_tridiag_eigen(bt, s, small)) != SLS_OK) return st;
  if ((st = launch_ritz_vectors(bt, U, s)) != SLS_OK) return st;
  if (alpha) SLS_CUDA_TRY(cudaMemcpyAsync(alpha, al, sizeof(double) * r, cudaMemcpyDeviceToDevice, s));
  if (beta) SLS_CUDA_TRY(cudaMemcpyAsync(beta, be, sizeof(double) * r, cudaMemcpyDeviceToDevice, s));
  return guards_check(cv, status, s);
}

}  // namespace

// ===========================================================================
// exported entry points
// ===========================================================================

extern "C" {

const char* sls_status_string(int status) {
  switch (status) {
    case SLS_OK: return "ok";
    case SLS_ERR_INVALID_ARG: return "invalid argument";
    case SLS_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case SLS_ERR_WORKSPACE: return "workspace missing or too small";
    case SLS_ERR_CUDA: return "CUDA launch or copy failed";
    case SLS_ERR_TIMEOUT: return "device wait reached its iteration limit";
    case SLS_ERR_BOUNDS: return "debug build: an access outside its range was caught and skipped";
    default: return "unknown status";
  }
}

int sls_version(void) { return 100; }

int sls_feature_map(const void* X, int x_dtype, int64_t N, int d, int64_t ldx, const void* W,
                    const float* b, int D, float* Phi, void* stream) {
  if (N < 0 || d < 1 || D < 4 || D > SLS_MAX_D || (D & 3) || ldx < d) return SLS_ERR_INVALID_ARG;
  if (x_dtype != SLS_F32 && x_dtype != SLS_BF16) return SLS_ERR_INVALID_ARG;
  if (N == 0) return SLS_OK;
  if (!X || !W || !b || !Phi) return SLS_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  if (x_dtype == SLS_BF16) {
    const int st = launch_feature_map_tc(X, N, d, ldx, W, b, D, Phi, s);
    if (st != SLS_ERR_UNSUPPORTED) return st;
  }
  return launch_feature_map_simt(X, x_dtype, N, d, ldx, W, b, D, Phi, s);
}

int sls_feature_map_ex(const void* X, int x_dtype, int64_t N, int d, int64_t ldx, const void* W,
                       const float* b, int D, void* Phi, int phi_dtype, void* stream) {
  if (phi_dtype == SLS_F32)
    return sls_feature_map(X, x_dtype, N, d, ldx, W, b, D, (float*)Phi, stream);
  if (phi_dtype != SLS_BF16) return SLS_ERR_INVALID_ARG;
  if (N < 0 || d < 1 || D < 4 || D > SLS_MAX_D || (D & 3) || ldx < d) return SLS_ERR_INVALID_ARG;
  if (x_dtype != SLS_F32 && x_dtype != SLS_BF16) return SLS_ERR_INVALID_ARG;
  if (N == 0) return SLS_OK;
  if (!X || !W || !b || !Phi) return SLS_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  if (x_dtype == SLS_BF16) {
    const int st = launch_feature_map_tc(X, N, d, ldx, W, b, D, Phi, s, nullptr, 1);
    if (st != SLS_ERR_UNSUPPORTED) return st;
  }
  return launch_feature_map_simt(X, x_dtype, N, d, ldx, W, b, D, Phi, s, 1);
}

int sls_feature_map_batched(const void* X, int64_t nb, int64_t rows, int64_t x_stride, int d,
                            int64_t ldx, const void* W, const float* b, int D, float* Phi,
                            const int32_t* live, int nwin, int win, void* stream) {
  if (nb < 0 || rows < 0 || x_stride < rows || d < 1 || ldx < d || D < 4 || D > SLS_MAX_D)
    return SLS_ERR_INVALID_ARG;
  if (live && (nwin < 1 || win < 1 || (int64_t)nwin * win < rows)) return SLS_ERR_INVALID_ARG;
  if (nb == 0 || rows == 0) return SLS_OK;
  if (!X || !W || !b || !Phi) return SLS_ERR_INVALID_ARG;
  return launch_feature_map_tc_batched(X, nb, rows, x_stride, d, ldx, W, b, D, Phi, live, nwin,
                                       win, (cudaStream_t)stream, nullptr);
}

size_t sls_feature_normalize_workspace_size(int64_t N, int D) {
  if (N < 1 || D < 1) return 0;
  return feature_normalize_scratch_bytes(N, D, 1);
}

int sls_feature_normalize(float* Phi, int64_t N, int D, double* s_hat, void* workspace,
                          size_t workspace_bytes, void* stream) {
  if (N < 0 || D < 1) return SLS_ERR_INVALID_ARG;
  if (N == 0) return SLS_OK;
  if (!ptr_ok(Phi)) return SLS_ERR_INVALID_ARG;
  const size_t need = sls_feature_normalize_workspace_size(N, D);
  if (!workspace || workspace_bytes < need) return SLS_ERR_WORKSPACE;
  return launch_feature_normalize(Phi, D, nullptr, nullptr, 1, nullptr, N, N,
                                  (float2*)workspace, s_hat, (cudaStream_t)stream);
}

size_t sls_lanczos_workspace_size(int64_t N, int D, int r) {
  if (N < 1 || D < 4 || r < 1 || r > SLS_MAX_R) return 0;
  int groups = 0, g = 0;
  if (lanczos_plan(N, D, r, 1, &groups, &g) != SLS_OK) return 0;
  Carver cv(nullptr);
  cv.take<int>(64);
  cv.take<float2>((size_t)N * ((r + 1) & ~1));
  cv.take<double>(r);
  cv.take<double>(r);
  cv.take<double>((size_t)r * r);
  cv.take<char>(lanczos_scratch_bytes(N, D, r, groups, g));
  return cv.off;
}

int sls_lanczos_topr(const float* Phi, int64_t N, int D, int r, const double* q1, double tol,
                     double* theta, float* U, int32_t* r_eff, double* alpha, double* beta,
                     void* workspace, size_t workspace_bytes, void* stream) {
  return sls_lanczos_topr_ex(Phi, SLS_F32, N, D, r, q1, tol, theta, U, r_eff, alpha, beta,
                             workspace, workspace_bytes, stream);
}

int sls_lanczos_topr_ex(const void* Phi, int phi_dtype, int64_t N, int D, int r, const double* q1,
                        double tol, double* theta, float* U, int32_t* r_eff, double* alpha,
                        double* beta, void* workspace, size_t workspace_bytes, void* stream) {
  return lanczos_single(Phi, phi_dtype, N, D, r, q1, tol, theta, U, r_eff, alpha, beta, workspace,
                        workspace_bytes, stream, 0);
}

int sls_selftest_lanczos_giveup(const float* Phi, int64_t N, int D, int r, const double* q1,
                                double* theta, float* U, int32_t* r_eff, void* workspace,
                                size_t workspace_bytes, void* stream) {
  if (lanczos_window_fits(N, D, r)) return SLS_ERR_UNSUPPORTED;  // no group barrier there
  return lanczos_single(Phi, SLS_F32, N, D, r, q1, 1e-10, theta, U, r_eff, nullptr, nullptr,
                        workspace, workspace_bytes, stream, 1);
}

size_t sls_lanczos_batched_workspace_size(int64_t rows, int64_t nmax, int D, int r, int nprob) {
  if (rows < 1 || nmax < 1 || D < 4 || r < 1 || r > SLS_MAX_R || nprob < 1) return 0;
  int groups = 0, g = 0;
  if (lanczos_plan(nmax, D, r, nprob, &groups, &g) != SLS_OK) return 0;
  Carver cv(nullptr);
  cv.take<int>(64);
  cv.take<float2>((size_t)rows * ((r + 1) & ~1));
  cv.take<double>((size_t)nprob * r);
  cv.take<double>((size_t)nprob * r);
  cv.take<double>((size_t)nprob * r * r);
  cv.take<char>(lanczos_scratch_bytes(nmax, D, r, groups, g));
  return cv.off;
}

int sls_lanczos_topr_batched(const void* Phi, int phi_dtype, int D, int r, int nprob,
                             const int64_t* row0, const int32_t* n, const int64_t* q1off,
                             int64_t nmax, int64_t rows, const double* q1, double tol,
                             double* theta, float* U, int32_t* r_eff, double* alpha,
                             double* beta, void* workspace, size_t workspace_bytes,
                             void* stream) {
  if (nprob < 1 || nmax < 1 || rows < 1 || D < 4 || D > SLS_MAX_D || r < 1 || r > SLS_MAX_R ||
      !(tol >= 0.0))
    return SLS_ERR_INVALID_ARG;
  if (phi_dtype != SLS_F32 && phi_dtype != SLS_BF16) return SLS_ERR_INVALID_ARG;
  if ((D & 3) != 0 || (phi_dtype == SLS_BF16 && (D & 7) != 0)) return SLS_ERR_UNSUPPORTED;
  if (!ptr_ok(Phi) || !row0 || !n || !q1 || !theta || !U || !r_eff) return SLS_ERR_INVALID_ARG;
  const size_t need = sls_lanczos_batched_workspace_size(rows, nmax, D, r, nprob);
  if (need == 0) return SLS_ERR_UNSUPPORTED;
  if (!workspace || workspace_bytes < need) return SLS_ERR_WORKSPACE;
  int groups = 0, g = 0;
  int st = lanczos_plan(nmax, D, r, nprob, &groups, &g);
  if (st != SLS_OK) return st;
  cudaStream_t s = (cudaStream_t)stream;
  Carver cv(workspace);
  int* status = cv.take<int>(64);
  float2* Q = cv.take<float2>((size_t)rows * ((r + 1) & ~1));
  double* al = cv.take<double>((size_t)nprob * r);
  double* be = cv.take<double>((size_t)nprob * r);
  double* S = cv.take<double>((size_t)nprob * r * r);
  const size_t lzb = lanczos_scratch_bytes(nmax, D, r, groups, g);
  void* lz = cv.take<char>(lzb);
  SLS_CUDA_TRY(cudaMemsetAsync(status, 0, 256, s));
  if ((st = guards_arm(cv, s)) != SLS_OK) return st;
  SLS_CUDA_TRY(cudaMemsetAsync(r_eff, 0xff, sizeof(int32_t) * (size_t)nprob, s));
  LanczosBatch bt{};
  bt.Phi = Phi;
  bt.phi_bf16 = (phi_dtype == SLS_BF16) ? 1 : 0;
  bt.D = D;
  bt.r = r;
  bt.tol = tol;
  bt.q1 = q1;
  bt.n_single = 0;
  bt.nprob_max = nprob;
  bt.nprob_dev = nullptr;
  bt.row0 = row0;
  bt.n = n;
  bt.q1off = q1off;
  bt.Q = Q;
  bt.alpha = al;
  bt.beta = be;
  bt.theta = theta;
  bt.S = S;
  bt.r_eff = r_eff;
  bt.nmax = nmax;
  const bool small = lanczos_window_fits(nmax, D, r);
  if (small) {
    if ((st = launch_lanczos_window(bt, s)) != SLS_OK) return st;
  } else if ((st = launch_lanczos(bt, lz, lzb, status, groups, g, s)) != SLS_OK) {
    return st;
  }
  if ((st = launch_tridiag_eigen(bt, s, small)) != SLS_OK) return st;
  if ((st = launch_ritz_vectors(bt, U, s)) != SLS_OK) return st;
  if (alpha)
    SLS_CUDA_TRY(cudaMemcpyAsync(alpha, al, sizeof(double) * r * (size_t)nprob,
                                 cudaMemcpyDeviceToDevice, s));
  if (beta)
    SLS_CUDA_TRY(cudaMemcpyAsync(beta, be, sizeof(double) * r * (size_t)nprob,
                                 cudaMemcpyDeviceToDevice, s));
  return guards_check(cv, status, s);
}

int sls_simhash(const float* U, int64_t N, int k, int ldu, const int32_t* k_dev, const float* R,
                int bits, int ldr, uint32_t* codes, void* stream) {
  if (N < 0 || k < 1 || k > SLS_MAX_R || ldu < k || bits < 1 || bits > SLS_MAX_BITS || ldr < k)
    return SLS_ERR_INVALID_ARG;
  if (N == 0) return SLS_OK;
  if (!U || !R || !codes) return SLS_ERR_INVALID_ARG;
  return launch_simhash(U, N, k, ldu, k_dev, R, bits, ldr, codes, (cudaStream_t)stream);
}

size_t sls_aggregate_workspace_size(int64_t N, int d, int64_t M_target) {
  if (N < 1 || d < 1 || M_target < 1 || M_target > N) return 0;
  Carver cv(nullptr);
  cv.take<int>(64);
  cv.take<ProbDesc>(1);
  cv.take<char>(segment_scratch_bytes(N, M_target, 1));
  cv.take<int>(N);
  cv.take<int>(M_target);
  cv.take<int>(M_target);
  cv.take<int>(M_target);
  cv.take<int2>(agg_item_capacity(M_target, N));
  cv.take<int>(agg_aux_ints(M_target, N));
  cv.take<float>(agg_part_capacity(N) * (size_t)d);
  cv.take<float>(agg_part_capacity(N));
  return cv.off;
}

int sls_aggregate(const void* X, int x_dtype, int64_t N, int d, int64_t ldx,
                  const uint32_t* codes, int64_t M_target, int pos_scheme, int renorm, float* Xt,
                  int32_t* pos, int32_t* tok2macro, void* workspace, size_t workspace_bytes,
                  void* stream) {
  if (N < 1 || d < 1 || ldx < d || M_target < 1 || M_target > N || N > (1 << 30))
    return SLS_ERR_INVALID_ARG;
  if (x_dtype != SLS_F32 && x_dtype != SLS_BF16) return SLS_ERR_INVALID_ARG;
  if (pos_scheme < 0 || pos_scheme > 2) return SLS_ERR_INVALID_ARG;
  if (!ptr_ok(X) || !codes || !Xt || !pos || !tok2macro) return SLS_ERR_INVALID_ARG;
  const int vec = (x_dtype == SLS_BF16) ? 8 : 4;
  if (d % vec || ldx % vec || d > SLS_MAX_D) return SLS_ERR_UNSUPPORTED;
  const size_t need = sls_aggregate_workspace_size(N, d, M_target);
  if (!workspace || workspace_bytes < need) return SLS_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  Carver cv(workspace);
  int* status = cv.take<int>(64);
  ProbDesc* prob = cv.take<ProbDesc>(1);
  void* seg = cv.take<char>(segment_scratch_bytes(N, M_target, 1));
  int* perm = cv.take<int>(N);
  int* mstart = cv.take<int>(M_target);
  int* mlen = cv.take<int>(M_target);
  int* pt_start = cv.take<int>(M_target);
  int2* items = cv.take<int2>(agg_item_capacity(M_target, N));
  int* counts = cv.take<int>(agg_aux_ints(M_target, N));
  float* part = cv.take<float>(agg_part_capacity(N) * (size_t)d);
  float* part_eta = cv.take<float>(agg_part_capacity(N));
  SLS_CUDA_TRY(cudaMemsetAsync(status, 0, 256, s));
  int st;
  if ((st = guards_arm(cv, s)) != SLS_OK) return st;
  single_prob_kernel<<<1, 1, 0, s>>>(prob, N, M_target, 32);
  SLS_LAUNCH_CHECK();
  if ((st = launch_segment(prob, 1, codes, pos_scheme, SLS_MODE_REPRESENTATIVE, seg, 1, N,
                           M_target, perm, mstart, mlen, pos, tok2macro, status, s)) != SLS_OK)
    return st;
  if ((st = launch_aggregate(X, x_dtype, d, ldx, perm, mstart, mlen, M_target, N, renorm, Xt,
                             pt_start, items, counts, part, part_eta, status, s)) != SLS_OK)
    return st;
  return guards_check(cv, status, s);
}

int64_t sls_output_count(const sls_config_t* cfg, int64_t N) {
  if (validate_config(cfg) != SLS_OK || N < 0) return -1;
  if (is_identity(cfg, N)) return N;
  CompressPlan P;
  if (make_plan(cfg, 1, N, &P, false) != SLS_OK) return -1;
  return P.M;
}

size_t sls_compress_workspace_size(const sls_config_t* cfg, int64_t B, int64_t N, int d) {
  if (validate_config(cfg) != SLS_OK || B < 1 || N < 1 || d < 1) return 0;
  if (is_identity(cfg, N)) return 256;
  CompressPlan P;
  if (make_plan(cfg, B, N, &P) != SLS_OK) return 0;
  CompressWs W;
  carve(P, nullptr, &W);
  return W.total + tail_bytes(P, B * N, d, cfg->backend);
}

int sls_compress(const sls_config_t* cfg, const void* X, int x_dtype, int64_t B, int64_t N, int d,
                 int64_t ldx, const sls_params_t* params, float* Xt, int32_t* pos,
                 int32_t* tok2macro, int32_t* r_eff, int32_t* route, void* workspace,
                 size_t workspace_bytes, void* stream) {
  int st = validate_config(cfg);
  if (st != SLS_OK) return st;
  if (B < 1 || N < 1 || d < 1 || ldx < d || B * N > (1LL << 30)) return SLS_ERR_INVALID_ARG;
  if (x_dtype != SLS_F32 && x_dtype != SLS_BF16) return SLS_ERR_INVALID_ARG;
  if (!ptr_ok(X) || !Xt || !pos || !tok2macro) return SLS_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  if (is_identity(cfg, N)) {
    // the workspace (if any) holds only the status word
    if (workspace && workspace_bytes >= 256) SLS_CUDA_TRY(cudaMemsetAsync(workspace, 0, 256, s));
    return launch_identity(X, x_dtype, B, N, d, ldx, Xt, pos, tok2macro, s);
  }
  const int vec = (x_dtype == SLS_BF16) ? 8 : 4;
  if (d % vec || ldx % vec || d > SLS_MAX_D) return SLS_ERR_UNSUPPORTED;
  CompressPlan P;
  if ((st = make_plan(cfg, B, N, &P)) != SLS_OK) return st;
  const bool spectral = cfg->backend != SLS_BACKEND_CHUNK;
  if (spectral) {
    if (!params || !params->W || !params->b || !params->R || !params->q1)
      return SLS_ERR_INVALID_ARG;
    if (params->R_ld < cfg->r || params->R_rows < P.bits_max) return SLS_ERR_INVALID_ARG;
    if (B > 1 && params->q1_stride < P.Nc) return SLS_ERR_INVALID_ARG;
  }
  CompressWs W;
  carve(P, workspace, &W);
  const size_t need = W.total + tail_bytes(P, B * N, d, cfg->backend);
  if (!workspace || workspace_bytes < need) return SLS_ERR_WORKSPACE;
  {
    Carver tail((char*)workspace + W.total);
    W.part = tail.take<float>(agg_part_capacity(B * N) * (size_t)d);
    W.part_eta = tail.take<float>(agg_part_capacity(B * N));
    W.score_part = (cfg->backend == SLS_BACKEND_ADAPTIVE)
                       ? tail.take<float>(score_part_floats(P.nprob, P.nmax, d))
                       : nullptr;
    W.tail = tail;
  }
  SLS_CUDA_TRY(cudaMemsetAsync(W.status, 0, 256, s));
  if ((st = guards_arm(W.cv, s)) != SLS_OK) return st;
  if ((st = guards_arm(W.tail, s)) != SLS_OK) return st;
  const int nprob = (int)P.nprob;
  phase_mark(0, 0, s);
  // problem table
  {
    int64_t blocks = (P.nprob + 255) / 256;
    plan_kernel<<<(unsigned)blocks, 256, 0, s>>>(
        W.probs, B, N, P.M, P.pf, P.Nc, P.bud.W, P.bud.L_full, P.bud.m_full, P.bud.m_last,
        P.bud.left_full, P.bud.L_last, cfg->rho, cfg->bits, spectral ? 1 : 0,
        cfg->backend == SLS_BACKEND_CHUNK ? P.k_chunk : 0, spectral ? params->q1_stride : 0);
    SLS_LAUNCH_CHECK();
  }
  // routing; at rho >= 16 every window is spectral and no score is needed
  int mode = spectral ? 0 : 1;
  if (cfg->backend == SLS_BACKEND_ADAPTIVE) {
    mode = 2;
    // below rho = 16 the score pass also writes every window's chunk-path
    // output, so the segment and aggregation steps only see spectral windows
    if (cfg->rho < 16.0 &&
        (st = launch_window_score_chunk(X, x_dtype, d, ldx, W.probs, nprob, P.nmax,
                                        W.score_part, W.score, cfg->pos_scheme, cfg->pos_mode,
                                        cfg->renorm, Xt, pos, tok2macro, s)) != SLS_OK)
      return st;
  }
  double tau = cfg->tau;
  if (cfg->tau_schedule) {
    tau = 0.75 - 0.05 * std::log2(cfg->rho);
    if (tau > 0.70) tau = 0.70;
    if (tau < 0.55) tau = 0.55;
  }
  int32_t* rflags = route ? route : W.route;
  route_compact_kernel<<<1, 1024, 0, s>>>(W.probs, nprob, mode, W.score, cfg->rho, tau,
                                          W.spec_list, W.lz_row0, W.lz_n, W.lz_q1off, W.nspec,
                                          rflags, W.r_eff);
  SLS_LAUNCH_CHECK();
  phase_mark(0, 1, s);
  phase_mark(1, 0, s);
  if (spectral) {
    // features of the compressible rows of every prompt, in one launch on the
    // tensor cores (bf16); windows routed to the chunk path are skipped
    st = SLS_ERR_UNSUPPORTED;
    if (x_dtype == SLS_BF16)
      st = launch_feature_map_tc_batched(
          (const char*)X + (size_t)P.pf * ldx * 2, B, P.Nc, N, d, ldx, params->W, params->b,
          cfg->D, W.Phi, mode == 2 ? rflags : nullptr, (int)P.bud.W, (int)P.bud.L_full, s,
          W.status, P.phi_bf16);
    if (st == SLS_ERR_UNSUPPORTED) {
      const size_t esz = P.phi_bf16 ? 2 : 4;
      for (int64_t b = 0; b < B; ++b) {
        const char* xb = (const char*)X +
                         (size_t)(b * N + P.pf) * ldx * (x_dtype == SLS_BF16 ? 2 : 4);
        st = sls_feature_map_ex(xb, x_dtype, P.Nc, d, ldx, params->W, params->b, cfg->D,
                                (char*)W.Phi + (size_t)b * P.Nc * cfg->D * esz,
                                P.phi_bf16 ? SLS_BF16 : SLS_F32, stream);
        if (st != SLS_OK) return st;
      }
    }
    if (st != SLS_OK) return st;
    // the row-normalised operator: each spectral problem's rows scaled by
    // 1 / sqrt of its estimated row sums (Sec. 3.2)
    if (cfg->normalize &&
        (st = launch_feature_normalize((float*)W.Phi, cfg->D, W.lz_row0, W.lz_n, nprob, W.nspec, 0,
                                       P.nmax, W.norm_scratch, nullptr, s)) != SLS_OK)
      return st;
    phase_mark(1, 1, s);
    phase_mark(2, 0, s);
    LanczosBatch bt{};
    bt.Phi = W.Phi;
    bt.phi_bf16 = P.phi_bf16;
    bt.D = cfg->D;
    bt.r = cfg->r;
    bt.tol = cfg->lanczos_tol;
    bt.q1 = params->q1;
    bt.n_single = 0;
    bt.nprob_max = nprob;
    bt.nprob_dev = W.nspec;
    bt.row0 = W.lz_row0;
    bt.n = W.lz_n;
    bt.q1off = W.lz_q1off;
    bt.Q = W.Q;
    bt.alpha = W.alpha;
    bt.beta = W.beta;
    bt.theta = W.theta;
    bt.S = W.S;
    bt.r_eff = W.r_eff;
    bt.nmax = P.nmax;
    // windows of at most 32 tokens: one warp per window (values of T included)
    const bool small = lanczos_window_fits(P.nmax, cfg->D, cfg->r);
    if (small) {
      if ((st = launch_lanczos_window(bt, s)) != SLS_OK) return st;
    } else if ((st = launch_lanczos(bt, W.lz_scratch, W.lz_bytes, W.status, P.lz_groups,
                                    P.lz_g, s)) != SLS_OK) {
      return st;
    }
    phase_mark(2, 1, s);
    phase_mark(3, 0, s);
    if ((st = launch_tridiag_eigen(bt, s, small)) != SLS_OK) return st;
    if ((st = launch_ritz_vectors(bt, W.U, s)) != SLS_OK) return st;
    phase_mark(3, 1, s);
    phase_mark(4, 0, s);
    if ((st = launch_simhash_problems(W.probs, W.spec_list, W.nspec, nprob, P.nmax, W.r_eff, W.U,
                                      cfg->r, params->R, params->R_ld, P.bits_max, W.codes, s)) !=
        SLS_OK)
      return st;
    if (r_eff) {
      finish_reff_kernel<<<(nprob + 255) / 256, 256, 0, s>>>(W.probs, nprob, W.r_eff, r_eff);
      SLS_LAUNCH_CHECK();
    }
    phase_mark(4, 1, s);
  } else {
    for (int ph = 1; ph <= 4; ++ph) {
      if (ph > 1) phase_mark(ph, 0, s);
      phase_mark(ph, 1, s);
    }
  }
  phase_mark(5, 0, s);
  const int chunk_done = (cfg->backend == SLS_BACKEND_ADAPTIVE && cfg->rho < 16.0) ? 1 : 0;
  if ((st = launch_segment(W.probs, nprob, W.codes, cfg->pos_scheme, cfg->pos_mode, W.seg_scratch,
                           P.seg_slots, P.nmax, P.mmax, W.perm, W.mstart, W.mlen, pos, tok2macro,
                           W.status, s, chunk_done)) != SLS_OK)
    return st;
  if ((st = launch_preserved(B, N, P.M, (int)P.pf, (int)P.pl, cfg->pos_mode, W.perm, W.mstart,
                             W.mlen, pos, tok2macro, s)) != SLS_OK)
    return st;
  phase_mark(5, 1, s);
  phase_mark(6, 0, s);
  st = launch_aggregate(X, x_dtype, d, ldx, W.perm, W.mstart, W.mlen, B * P.M, B * N,
                        cfg->renorm, Xt, W.pt_start, W.items, W.counts, W.part, W.part_eta,
                        W.status, s);
  phase_mark(6, 1, s);
  if (st != SLS_OK) return st;
  if ((st = guards_check(W.cv, W.status, s)) != SLS_OK) return st;
  return guards_check(W.tail, W.status, s);
}

int sls_embed_gather(const void* table, int x_dtype, int64_t V, int d, int64_t ld_table,
                     const int32_t* ids, int64_t N, void* X, int64_t ldx, int32_t* bad,
                     void* stream) {
  if (N < 0 || V < 1 || d < 1 || ld_table < d || ldx < d) return SLS_ERR_INVALID_ARG;
  if (x_dtype != SLS_F32 && x_dtype != SLS_BF16) return SLS_ERR_INVALID_ARG;
  if (N > 0 && (!table || !ids || !X)) return SLS_ERR_INVALID_ARG;
  return launch_embed_gather(table, x_dtype, V, d, ld_table, ids, N, X, ldx, bad,
                             (cudaStream_t)stream);
}

size_t sls_compress_tokens_workspace_size(const sls_config_t* cfg, int x_dtype, int64_t B,
                                          int64_t N, int d) {
  if (x_dtype != SLS_F32 && x_dtype != SLS_BF16) return 0;
  const size_t inner = sls_compress_workspace_size(cfg, B, N, d);
  if (inner == 0) return 0;
  const size_t elt = (x_dtype == SLS_BF16) ? 2 : 4;
  return sls_align256((size_t)B * (size_t)N * (size_t)d * elt) + inner;
}

int sls_compress_tokens(const sls_config_t* cfg, const void* table, int x_dtype, int64_t V, int d,
                        int64_t ld_table, const int32_t* ids, int64_t B, int64_t N,
                        const sls_params_t* params, float* Xt, int32_t* pos, int32_t* tok2macro,
                        int32_t* r_eff, int32_t* route, int32_t* bad_ids, void* workspace,
                        size_t workspace_bytes, void* stream) {
  const int vst = validate_config(cfg);
  if (vst != SLS_OK) return vst;
  if (B < 1 || N < 1 || V < 1 || d < 1 || ld_table < d) return SLS_ERR_INVALID_ARG;
  if (x_dtype != SLS_F32 && x_dtype != SLS_BF16) return SLS_ERR_INVALID_ARG;
  if (!table || !ids) return SLS_ERR_INVALID_ARG;
  const size_t need = sls_compress_tokens_workspace_size(cfg, x_dtype, B, N, d);
  if (need == 0) return SLS_ERR_INVALID_ARG;
  if (!ptr_ok(workspace) || workspace_bytes < need) return SLS_ERR_WORKSPACE;
  const size_t elt = (x_dtype == SLS_BF16) ? 2 : 4;
  const size_t xb = sls_align256((size_t)B * (size_t)N * (size_t)d * elt);
  void* X = workspace;
  int st = launch_embed_gather(table, x_dtype, V, d, ld_table, ids, B * N, X, d, bad_ids,
                               (cudaStream_t)stream);
  if (st != SLS_OK) return st;
  return sls_compress(cfg, X, x_dtype, B, N, d, d, params, Xt, pos, tok2macro, r_eff, route,
                      (char*)workspace + xb, workspace_bytes - xb, stream);
}

int sls_set_phase_events(void* const* events, int count) {
  if (count == 0 || events == nullptr) {
    g_phase_on = false;
    return SLS_OK;
  }
  if (count != 2 * SLS_NUM_PHASES) return SLS_ERR_INVALID_ARG;
  for (int i = 0; i < count; ++i) {
    if (!events[i]) return SLS_ERR_INVALID_ARG;
    g_phase_events[i] = events[i];
  }
  g_phase_on = true;
  return SLS_OK;
}

int64_t sls_launch_count(void) { return (int64_t)g_launches.load(); }

int sls_selftest_wait_limit(int which, void* workspace, size_t workspace_bytes, void* stream) {
  if (which != 0 && which != 1) return SLS_ERR_INVALID_ARG;
  if (!ptr_ok(workspace) || workspace_bytes < 512) return SLS_ERR_WORKSPACE;
  return launch_selftest_wait_limit(which, (int*)workspace,
                                    (unsigned*)((char*)workspace + 256), (cudaStream_t)stream);
}

int sls_debug_selftest(int which, void* workspace, size_t workspace_bytes, void* stream) {
  if (which != 0 && which != 1) return SLS_ERR_INVALID_ARG;
  if (kGuardBytes == 0) return SLS_ERR_UNSUPPORTED;  // the ordinary build has no checks
  if (!ptr_ok(workspace)) return SLS_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  Carver cv(workspace);
  int* status = cv.take<int>(64);
  int* region = cv.take<int>(64);
  if (workspace_bytes < cv.off) return SLS_ERR_WORKSPACE;
  SLS_CUDA_TRY(cudaMemsetAsync(status, 0, 256, s));
  int st;
  if ((st = guards_arm(cv, s)) != SLS_OK) return st;
  debug_selftest_kernel<<<1, 32, 0, s>>>(region, 64, which, status);
  SLS_LAUNCH_CHECK();
  return guards_check(cv, status, s);
}

int sls_workspace_status(void* workspace, void* stream) {
  if (!workspace) return SLS_ERR_INVALID_ARG;
  int h = 0;
  cudaStream_t s = (cudaStream_t)stream;
  SLS_CUDA_TRY(cudaMemcpyAsync(&h, workspace, sizeof(int), cudaMemcpyDeviceToHost, s));
  SLS_CUDA_TRY(cudaStreamSynchronize(s));
  SLS_CUDA_TRY(cudaMemsetAsync(workspace, 0, sizeof(int), s));
  return h == 0 ? SLS_OK : h;
}

}  // extern "C"
