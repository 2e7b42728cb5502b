/*
 * sls.h -- C ABI of the GB300 (sm_103a) Spectral-LSH compression pass.
 *
 * Spectral-LSH (arXiv 2607.19368) compresses a prompt's N x d input
 * embeddings X into M << N macro-tokens before prefill:
 *   1. random Fourier features Phi = sqrt(2/D) cos(X Omega + b)  (Sec. 3.2, Eq. rff_map)
 *   2. r steps of Lanczos on the implicit operator A(v) = Phi (Phi^T v),
 *      never forming the N x N kernel                            (Algorithm 2, Eq. implicit_matvec)
 *   3. Eigh of the tridiagonal T and the Ritz vectors U = Q V      (Algorithm 1)
 *   4. SimHash of the rows of U into b-bit codes                  (Sec. 3.3, Eq. simhash)
 *   5. clusters of equal codes, adjusted to exactly M* groups      (Sec. 3.3)
 *   6. macro-tokens: renormalised means with causal positions      (Sec. 3.4, Eq. macro_embed)
 *   7. optionally, the adaptive per-window router                 (Sec. 3.6, Eq. redundancy)
 *
 * Conventions for every entry point:
 *   - All array pointers are DEVICE pointers owned by the caller, unless a
 *     parameter says "host".  The library allocates no memory: calls that
 *     need scratch take a caller-provided device workspace sized by the
 *     matching *_workspace_size() function (256-byte aligned).
 *   - Matrices are row-major and contiguous unless a leading dimension is
 *     given.  X and W share one dtype: SLS_F32 (float) or SLS_BF16 (raw
 *     bfloat16 bit patterns, uint16).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Work is enqueued asynchronously; no call synchronises the
 *     host with the device.
 *   - Return value: SLS_OK or an SLS_ERR_* code.  Argument errors are
 *     detected on the host before anything is enqueued.  Errors raised by a
 *     running kernel (a device wait that gave up) are written to a status
 *     word in the workspace and read back with sls_workspace_status().
 *   - Random draws of the method (Omega, b, the hyperplanes R and the Lanczos
 *     start vector q1) are inputs, so any caller can reproduce a run.
 *   - Every pointer must be 16-byte aligned; D must be a multiple of 4.
 */
#ifndef SLS_H_
#define SLS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
#define SLS_OK 0
#define SLS_ERR_INVALID_ARG 1  /* a size, pointer or option is out of range      */
#define SLS_ERR_UNSUPPORTED 2  /* a valid but unsupported shape or dtype         */
#define SLS_ERR_WORKSPACE 3    /* workspace missing or smaller than required     */
#define SLS_ERR_CUDA 4         /* a CUDA launch or copy failed                   */
#define SLS_ERR_TIMEOUT 5      /* a device-side wait reached its iteration limit */
#define SLS_ERR_BOUNDS 6       /* debug build only: a device-side bounds check or a
                                  workspace guard band caught an access outside its
                                  range (the access was skipped)                  */

/* Embedding dtypes. */
#define SLS_F32 0
#define SLS_BF16 1

/* Position aggregation schemes (Sec. 3.4). */
#define SLS_POS_MAX 0     /* max of member positions (default, causal)        */
#define SLS_POS_MEDIAN 1  /* lower median of member positions                 */
#define SLS_POS_MEAN 2    /* floor(mean + 1/2) of member positions            */

/* Compressed position modes (Sec. 5.6, App. B.3). */
#define SLS_MODE_REPRESENTATIVE 0  /* keep aggregated original positions */
#define SLS_MODE_COMPACT 1         /* renumber 0..M-1                     */

/* Backends (Sec. 3.5 and 3.6). */
#define SLS_BACKEND_GLOBAL 0    /* Spectral-LSH over the whole compressible region */
#define SLS_BACKEND_ADAPTIVE 1  /* per-window router: chunk or Spectral-LSH         */
#define SLS_BACKEND_CHUNK 2     /* consecutive groups of max(1, round(rho)) tokens  */
#define SLS_BACKEND_LOCAL 3     /* Spectral-LSH inside every window (no routing)    */

/* Limits of this implementation. */
#define SLS_MAX_R 128      /* Krylov rank r                 */
#define SLS_MAX_BITS 32    /* SimHash bits b                */
#define SLS_MAX_D 8192     /* RFF features D (multiple of 4) */

/*
 * Compression configuration: the fields of the paper's CompressionConfig
 * (App. B.3, B.8) that the pass uses.
 */
typedef struct sls_config {
  int backend;          /* SLS_BACKEND_*                                        */
  double rho;           /* target compression; rho <= 1 is the exact identity  */
  int D;                /* RFF features                                        */
  int r;                /* Lanczos steps / Krylov rank, 1..SLS_MAX_R           */
  int bits;             /* SimHash bits; 0 = ceil(log2(n / rho)) (Sec. 3.3)     */
  int preserve_first;   /* leading tokens kept uncompressed (default 0)        */
  int preserve_last;    /* trailing tokens kept uncompressed (default 12)      */
  int pos_scheme;       /* SLS_POS_*                                           */
  int pos_mode;         /* SLS_MODE_*                                          */
  int renorm;           /* 1: rescale each mean to its mean member norm        */
  double lanczos_tol;   /* break when beta_j <= tol * max_i(|alpha_i|+beta_i)  */
  int window;           /* adaptive / local backend window length              */
  double tau;           /* fixed redundancy threshold (used if !tau_schedule)  */
  int tau_schedule;     /* 1: tau(rho) = clamp(0.75 - 0.05 log2 rho, .55, .70)  */
  int normalize;        /* 1: row-normalised operator (Sec. 3.2), see
                           sls_feature_normalize                               */
  int phi_dtype;        /* storage of the feature matrix Phi: SLS_F32 (default)
                           or SLS_BF16 (half the bytes; Lanczos then runs on
                           the bf16-rounded features, see sls_lanczos_topr_ex;
                           needs D % 8 == 0 and normalize = 0)                 */
} sls_config_t;

/*
 * Random parameters (device pointers).  W = Omega^T is D x d in the dtype of
 * X; b has D floats; R holds R_rows x R_ld float hyperplanes (row l is
 * hyperplane l, at least `bits` rows and r columns used); q1 holds the
 * Lanczos start vector (float64), one entry per compressible token (global
 * backend: N_c entries; adaptive: window w of prompt p reads q1 at offset
 * p * q1_stride + window start).
 */
typedef struct sls_params {
  const void* W;
  const float* b;
  const float* R;
  int R_rows;
  int R_ld;
  const double* q1;
  int64_t q1_stride;
} sls_params_t;

/* Human-readable name of a status code (static string). */
const char* sls_status_string(int status);

/* Library version, major * 10000 + minor * 100 + patch. */
int sls_version(void);

/*
 * Random Fourier features, Sec. 3.2 Eq. rff_map:
 *   Phi[i, c] = sqrt(2/D) * cos( sum_k X[i, k] * W[c, k] + b[c] ).
 * X: N x d (row stride ldx elements), W: D x d, both of dtype x_dtype;
 * b: D floats; Phi: N x D floats (output, row stride D).
 * bf16 inputs use the tcgen05 tensor cores (fp32 accumulation); fp32 inputs
 * use an fp32 SIMT path.  N may be 0.  Errors: INVALID_ARG for negative or
 * zero sizes, NULL pointers, D % 4 != 0 or D > SLS_MAX_D.
 */
int sls_feature_map(const void* X, int x_dtype, int64_t N, int d, int64_t ldx,
                    const void* W, const float* b, int D, float* Phi,
                    void* stream);

/*
 * sls_feature_map with a choice of storage for Phi: phi_dtype SLS_F32 (as
 * sls_feature_map) or SLS_BF16 (Phi: N x D raw bfloat16 values, uint16, each
 * the float32 feature rounded to nearest even).  Errors: those of
 * sls_feature_map, INVALID_ARG for another phi_dtype.
 */
int sls_feature_map_ex(const void* X, int x_dtype, int64_t N, int d, int64_t ldx,
                       const void* W, const float* b, int D, void* Phi,
                       int phi_dtype, void* stream);

/*
 * The same features for a batch of nb equal-length prompts in one launch
 * (Sec. 3.2 Eq. rff_map, per token), optionally only for the windows the
 * adaptive router sent to the spectral chain (Sec. 3.6):
 *   prompt k, row i < rows:  X row k * x_stride + i  ->  Phi row k * rows + i.
 * X rows have stride ldx elements; W: D x d; b: D floats; Phi: nb * rows x D.
 * live (may be NULL = every row): device int32, nwin flags per prompt
 * (prompt-major); flag w covers rows [w * win, (w + 1) * win) of its prompt.
 * Phi rows are written for every 128-row tile that touches a window with a
 * nonzero flag and may be left unwritten elsewhere.  bf16 only, on the
 * tensor cores; requires D % 256 == 0, d % 8 == 0, ldx % 8 == 0 and 16-byte
 * aligned pointers.  Errors: INVALID_ARG for bad sizes or NULL pointers,
 * UNSUPPORTED outside the shapes above.
 */
int sls_feature_map_batched(const void* X, int64_t nb, int64_t rows,
                            int64_t x_stride, int d, int64_t ldx,
                            const void* W, const float* b, int D, float* Phi,
                            const int32_t* live, int nwin, int win,
                            void* stream);

/*
 * The row-normalised operator of Sec. 3.2, diag(s)^-1 Phi (Phi^T v) with the
 * estimated row sums s = Phi (Phi^T 1), in the symmetric form Lanczos needs:
 * D^{-1/2} Phi Phi^T D^{-1/2} (D = diag(s); same eigenvalues, eigenvectors
 * D^{1/2}-scaled, which leaves every SimHash code unchanged) -- i.e. the rows
 * of Phi scaled in place by 1 / sqrt(s_i) (by 0 where s_i <= 0).
 *   Phi: N x D floats (device, in place); s_hat (may be NULL): N doubles
 *   (device, output); workspace: sls_feature_normalize_workspace_size(N, D)
 *   device bytes.  Column sums and row dots are compensated (double-float);
 *   each scaled element is x / sqrt(s_i) to within one float32 rounding.
 * Errors: INVALID_ARG for bad sizes or NULL pointers, WORKSPACE if the
 * workspace is too small.
 */
size_t sls_feature_normalize_workspace_size(int64_t N, int D);
int sls_feature_normalize(float* Phi, int64_t N, int D, double* s_hat,
                          void* workspace, size_t workspace_bytes, void* stream);

/* Device workspace bytes needed by sls_lanczos_topr for one problem. */
size_t sls_lanczos_workspace_size(int64_t N, int D, int r);

/*
 * Implicit Lanczos and Ritz pairs: Algorithm 2 with A(v) = Phi (Phi^T v)
 * (Eq. implicit_matvec) followed by Eigh(T) and U = Q V (Algorithm 1).
 *   Phi: N x D floats.  q1: N doubles (normalised by the callee).
 *   Full re-orthogonalisation is two classical Gram-Schmidt passes; the loop
 *   stops early (Lanczos breakdown, not an error) when
 *   beta_j <= tol * max_{i<=j}(|alpha_i| + beta_i); r_eff <= r steps are kept.
 * Outputs: theta[r] doubles, Ritz values in descending order (entries past
 * r_eff are 0); U: N x r floats, column m the Ritz vector of theta[m], signed
 * so that the first component of the eigenvector of T is positive (columns
 * past r_eff are 0); r_eff: one int32 (device), set to -1 when the call is
 * enqueued and left at -1 if a device-side wait of the Lanczos kernel gave up
 * (sls_workspace_status then reports SLS_ERR_TIMEOUT; theta and U are then
 * zero).  Optional (may be NULL):
 * alpha[r], beta[r] doubles receive the diagonal and off-diagonal of T.
 * Vectors are kept in double-float (two fp32) precision; Phi is read as
 * stored.  Errors: INVALID_ARG (sizes, NULL, r > SLS_MAX_R), WORKSPACE,
 * UNSUPPORTED (D % 4 != 0), CUDA.
 */
int sls_lanczos_topr(const float* Phi, int64_t N, int D, int r,
                     const double* q1, double tol, double* theta, float* U,
                     int32_t* r_eff, double* alpha, double* beta,
                     void* workspace, size_t workspace_bytes, void* stream);

/*
 * sls_lanczos_topr on a feature matrix stored as phi_dtype: SLS_F32 (exactly
 * sls_lanczos_topr) or SLS_BF16 (Phi: N x D raw bfloat16 values, uint16;
 * requires D % 8 == 0).  bf16 elements are widened exactly to float32, so the
 * run is Algorithm 2 on the operator of the stored (rounded) features, with
 * the same arithmetic as the float32 case; only the bytes read differ.
 * Errors: those of sls_lanczos_topr, INVALID_ARG for another phi_dtype,
 * UNSUPPORTED for bf16 with D % 8 != 0.
 */
int sls_lanczos_topr_ex(const void* Phi, int phi_dtype, int64_t N, int D, int r,
                        const double* q1, double tol, double* theta, float* U,
                        int32_t* r_eff, double* alpha, double* beta,
                        void* workspace, size_t workspace_bytes, void* stream);

/* Device workspace bytes needed by sls_lanczos_topr_batched. */
size_t sls_lanczos_batched_workspace_size(int64_t rows, int64_t nmax, int D, int r,
                                          int nprob);

/*
 * sls_lanczos_topr for nprob independent problems in one launch, with the
 * launch plan sls_compress uses for the windows of its adaptive and local
 * backends (Algorithm 2 per window, Sec. 3.5-3.6): the persistent kernel's
 * CTAs form groups and each group runs one problem at a time, each CTA of a
 * group a strip of the problem's rows; problems of at most 32 rows (r <= 32)
 * run one warp per problem instead.
 *   Phi: rows x D of phi_dtype (SLS_F32 or SLS_BF16, as sls_lanczos_topr_ex).
 *   row0, n, q1off: device arrays of nprob entries; problem p owns the rows
 *   [row0[p], row0[p] + n[p]) of Phi and of U, with 1 <= n[p] <= nmax and
 *   row0[p] + n[p] <= rows, and its start vector is q1[q1off[p] ..
 *   q1off[p] + n[p]) (q1off may be NULL: q1off = row0), normalised by the
 *   callee.
 *   Outputs: theta: nprob x r doubles (problem p at p * r, descending);
 *   U: rows x r floats (problem p's Ritz vectors in its rows); r_eff: nprob
 *   int32, -1 until the kernel finishes and left at -1 if a device-side wait
 *   gave up; alpha, beta (may be NULL): nprob x r doubles.
 * The problem table is read on the device only, so the host needs no copy of
 * it; nmax is a host upper bound on n[p] that sizes the plan.  Errors:
 * INVALID_ARG (sizes, NULL, misaligned Phi), UNSUPPORTED, WORKSPACE, CUDA.
 */
int sls_lanczos_topr_batched(const void* Phi, int phi_dtype, int D, int r, int nprob,
                             const int64_t* row0, const int32_t* n, const int64_t* q1off,
                             int64_t nmax, int64_t rows, const double* q1, double tol,
                             double* theta, float* U, int32_t* r_eff, double* alpha,
                             double* beta, void* workspace, size_t workspace_bytes,
                             void* stream);

/*
 * SimHash in the spectral subspace, Sec. 3.3 Eq. simhash:
 *   code[i] = sum_l [ dot(U[i, :k], R[l, :k]) > 0 ] << l,  l < bits.
 * The dot product is a fixed float32 chain (acc = 0; for m in 0..k-1:
 * acc = fl(acc + fl(U[i,m] * R[l,m])), no fused multiply-add), so codes are
 * reproducible bit for bit; a +-0 or NaN dot gives bit 0.  k = *k_dev if
 * k_dev is not NULL (device int32, e.g. r_eff), else k.  U: N rows with row
 * stride ldu floats; R: bits x ldr floats.  Errors: INVALID_ARG (bits outside
 * 1..32, k < 1 or > ldu, NULL pointers).
 */
int sls_simhash(const float* U, int64_t N, int k, int ldu, const int32_t* k_dev,
                const float* R, int bits, int ldr, uint32_t* codes,
                void* stream);

/* Device workspace bytes needed by sls_aggregate. */
size_t sls_aggregate_workspace_size(int64_t N, int d, int64_t M_target);

/*
 * Clusters, exact-length adjustment and macro-tokens (Sec. 3.3, Sec. 3.4,
 * Eq. macro_embed) for one token set of N tokens with codes[N]:
 *   - tokens with equal codes form clusters, in ascending code order;
 *   - adjusted to exactly M_target groups: if C > M_target the cluster of
 *     rank t joins group floor(t * M_target / C); if C < M_target clusters
 *     receive D'Hondt seats (one guaranteed each, ties to the lower code) and
 *     are cut into that many contiguous pieces in position order;
 *   - each group's embedding is the mean of its members rescaled to their
 *     mean norm (renorm = 1; a singleton is copied exactly; a mean of norm
 *     < 1e-30 is not rescaled); its position follows pos_scheme;
 *   - groups are output in increasing (position, first member) order.
 * Positions are token indices within the set (0..N-1).
 * Outputs: Xt: M_target x d floats; pos: M_target int32; tok2macro: N int32
 * (index of the macro-token holding each token).  1 <= M_target <= N.
 * Errors: INVALID_ARG, WORKSPACE, CUDA.
 */
int sls_aggregate(const void* X, int x_dtype, int64_t N, int d, int64_t ldx,
                  const uint32_t* codes, int64_t M_target, int pos_scheme,
                  int renorm, float* Xt, int32_t* pos, int32_t* tok2macro,
                  void* workspace, size_t workspace_bytes, void* stream);

/*
 * Number of output macro-tokens per prompt for a configuration (host
 * arithmetic only): N if rho <= 1 or no token is compressible, else
 * preserve_first + ceil(N_c / rho) + preserve_last with N_c the compressible
 * count (chunk backend: ceil(N_c / max(1, round(rho))) groups).  Returns -1
 * for an invalid configuration.
 */
int64_t sls_output_count(const sls_config_t* cfg, int64_t N);

/* Device workspace bytes needed by sls_compress for B prompts of N x d. */
size_t sls_compress_workspace_size(const sls_config_t* cfg, int64_t B,
                                   int64_t N, int d);

/*
 * The whole compression pass (Algorithm 1 and the backends of Sec. 3.5-3.6)
 * for B independent prompts of N tokens each (B = 1 for a single prompt).
 *   X: B x N x d embeddings (prompt stride N * ldx elements, row stride ldx);
 *   params: the random draws (see sls_params_t);
 *   Xt: B x M x d floats; pos: B x M int32; tok2macro: B x N int32,
 *   with M = sls_output_count(cfg, N).
 *   r_eff (may be NULL): device int32 per prompt (global backend) or per
 *   window (adaptive and local backends), the Lanczos steps kept (0 for chunk
 *   windows; -1 for a spectral problem whose Lanczos kernel gave up a
 *   device-side wait, see sls_workspace_status).
 *   route (may be NULL): device int32 per window, 1 = spectral, 0 = chunk
 *   (adaptive backend; all 1 for the local backend).
 * The windowed backends (adaptive, local) cut the compressible region into
 * windows of cfg->window tokens (the last one shorter) and give every window
 * an exact budget summing to ceil(N_c / rho) (App. B.8); INVALID_ARG if that
 * leaves a window without a macro-token (ceil(N_c / rho) < window count).
 * Preserved first/last tokens become singleton macro-tokens at their own
 * positions; rho <= 1 (or nothing compressible) returns the identity: Xt = X,
 * pos = 0..N-1, tok2macro = 0..N-1 (Sec. 5.6, App. B.6).
 * Errors: INVALID_ARG, UNSUPPORTED, WORKSPACE, CUDA.
 */
int sls_compress(const sls_config_t* cfg, const void* X, int x_dtype, int64_t B,
                 int64_t N, int d, int64_t ldx, const sls_params_t* params,
                 float* Xt, int32_t* pos, int32_t* tok2macro, int32_t* r_eff,
                 int32_t* route, void* workspace, size_t workspace_bytes,
                 void* stream);

/*
 * The step before the pass: a prompt's input embeddings, one row of the
 * model's input embedding table per token (Sec. 3.1: X is the output of the
 * LLM's input embedding layer; Fig. 1: prompt tokens -> input embeddings):
 *   X[i, :] = table[ids[i], :]   for i < N.
 * table: V x d of x_dtype (row stride ld_table elements); ids: N int32;
 * X: N x d of x_dtype (output, row stride ldx).  An id outside [0, V) gives a
 * zero row of X; bad (may be NULL): one device int32, set to the number of
 * such ids.  Rows move as 16-byte vectors when the table and X bases, their
 * row strides and d * element size are all multiples of 16 bytes, else by
 * element.  N may be 0.  Errors: INVALID_ARG for bad sizes, dtype or NULL
 * pointers.
 */
int sls_embed_gather(const void* table, int x_dtype, int64_t V, int d,
                     int64_t ld_table, const int32_t* ids, int64_t N, void* X,
                     int64_t ldx, int32_t* bad, void* stream);

/* Device workspace bytes needed by sls_compress_tokens. */
size_t sls_compress_tokens_workspace_size(const sls_config_t* cfg, int x_dtype,
                                          int64_t B, int64_t N, int d);

/*
 * sls_compress from token ids: B prompts of N ids each (ids: B x N int32,
 * prompt-major) are looked up in the embedding table (see sls_embed_gather)
 * into a B x N x d buffer at the start of the workspace, which sls_compress
 * then compresses; every other argument and output is that of sls_compress.
 * The macro-token embeddings Xt are what the frozen model's prefill takes
 * through its inputs_embeds interface (Sec. 3.4).  bad_ids (may be NULL):
 * one device int32, the number of ids outside [0, V) (their rows are zero).
 * workspace: sls_compress_tokens_workspace_size(cfg, x_dtype, B, N, d)
 * bytes, 16-byte aligned.  Errors: those of sls_compress.
 */
int sls_compress_tokens(const sls_config_t* cfg, const void* table, int x_dtype,
                        int64_t V, int d, int64_t ld_table, const int32_t* ids,
                        int64_t B, int64_t N, const sls_params_t* params,
                        float* Xt, int32_t* pos, int32_t* tok2macro,
                        int32_t* r_eff, int32_t* route, int32_t* bad_ids,
                        void* workspace, size_t workspace_bytes, void* stream);

/*
 * sls_lanczos_topr without a caller workspace.  The paper has no counterpart
 * to this entry point: it exists for callers that may not allocate device
 * memory themselves -- for example a plugin inside a host application whose
 * memory manager owns every device allocation, or a serving path that forbids
 * allocation after start-up -- and therefore cannot provide the workspace
 * that sls_lanczos_topr takes.  Arguments and results are those of
 * sls_lanczos_topr (the caller still passes Phi, q1 and the output arrays).
 *
 * Scratch lives in one statically sized device array of
 * SLS_NOALLOC_MAX_BYTES inside the library; every GPU that loads the library
 * holds it until the process exits.  No cudaMalloc, cudaFree or allocating
 * library routine is called.  The first call on a device (with that device
 * current) looks up the array's device address once; make that first call
 * before any stream capture.  All calls share the array and it keeps the
 * previous call's contents (what must start at zero is cleared by each
 * call), so calls that overlap on the GPU -- on different streams, or from
 * different host threads -- race and must be serialised by the caller.
 * The looked-up address is cached for the life of the process: after a
 * cudaDeviceReset() on a device (which destroys the array with the context)
 * this entry point must not be called on that device again in the same
 * process.  *r_eff is set to -1 when the call is enqueued and stays -1 if a
 * device-side wait gave up.  Errors: those of sls_lanczos_topr (arguments are
 * checked before anything is enqueued), and SLS_ERR_WORKSPACE, with nothing
 * enqueued, when sls_lanczos_workspace_size(N, D, r) exceeds
 * SLS_NOALLOC_MAX_BYTES.
 */
#define SLS_NOALLOC_MAX_BYTES (32u << 20)
int sls_lanczos_topr_noalloc(const float* Phi, int64_t N, int D, int r,
                             const double* q1, double tol, double* theta,
                             float* U, int32_t* r_eff, double* alpha,
                             double* beta, void* stream);

/*
 * Optional per-phase timing of sls_compress.  `events` is a host array of
 * 2 * SLS_NUM_PHASES cudaEvent_t handles (passed as void*) owned by the
 * caller; while set, every sls_compress call records events[2p] on its
 * stream before phase p and events[2p+1] after it.  Phases, in launch order:
 * 0 setup (problem table; token norms and router when adaptive), 1 feature
 * map, 2 Lanczos, 3 Eigh(T) and Ritz vectors, 4 SimHash, 5 clusters/adjust/
 * order, 6 macro-token aggregation.  count = 0 (or events = NULL) switches timing
 * off.  Process-wide setting, not thread-safe.  Errors: INVALID_ARG if
 * count is neither 0 nor 2 * SLS_NUM_PHASES.
 */
#define SLS_NUM_PHASES 7
int sls_set_phase_events(void* const* events, int count);

/* Total number of kernels this library has launched in the process. */
int64_t sls_launch_count(void);

/*
 * Self-test of the device-side wait limits that end a stuck kernel: every
 * wait of the library's kernels (on an mbarrier, a ring slot or a group
 * barrier) gives up after about a second of clock cycles, records
 * SLS_ERR_TIMEOUT in the workspace status word and returns, leaving the
 * context usable.  This call launches a kernel whose wait can never be
 * satisfied -- which = 0: an mbarrier that nothing arrives at; which = 1: a
 * group barrier of two CTAs that one CTA never reaches -- so that the limit
 * runs out (about one second).  workspace: at least 512 device bytes (status
 * word, then barrier words); read the outcome with sls_workspace_status().
 * Errors: INVALID_ARG (which), WORKSPACE, CUDA.
 */
int sls_selftest_wait_limit(int which, void* workspace, size_t workspace_bytes,
                            void* stream);

/*
 * Self-test of the Lanczos kernel's failure path (the paper has no
 * counterpart): sls_lanczos_topr (float32 Phi, tol = 1e-10, same arguments
 * and workspace) with its first CTA reporting, at its first barrier, a wait
 * that gave up.  The kernel then takes the path of a real give-up: the other
 * CTAs are released at once, the copy warps stop after their own bounded
 * wait (about a second), the status word reads SLS_ERR_TIMEOUT, *r_eff stays
 * -1, theta and U are zero, and the context stays usable.  No fault, trap or
 * hang is involved.  Errors: those of sls_lanczos_topr; UNSUPPORTED when the
 * problem runs on the one-warp small-window kernel (N <= 32), which has no
 * barrier to fail.
 */
int sls_selftest_lanczos_giveup(const float* Phi, int64_t N, int D, int r, const double* q1,
                                double* theta, float* U, int32_t* r_eff, void* workspace,
                                size_t workspace_bytes, void* stream);

/*
 * Self-test of the debug build's checks (a library built with -DSLS_DEBUG,
 * libsls_debug.so; the paper has no counterpart).  That build surrounds
 * every region it carves from a workspace with a guard band, filled when a
 * call starts and checked when it ends, and guards selected device-side
 * accesses (row indices of the Lanczos kernel, member rows of the
 * aggregation) so that an out-of-range access is skipped and reported as
 * SLS_ERR_BOUNDS in the workspace status word instead of faulting.
 * which = 0 writes into a guard band (inside the caller's workspace);
 * which = 1 makes a guarded out-of-range write.  Either leaves
 * SLS_ERR_BOUNDS in the status word (read it with sls_workspace_status).
 * workspace: at least 1024 device bytes.  Errors: INVALID_ARG (which),
 * WORKSPACE, UNSUPPORTED in the ordinary build (which has no checks).
 */
int sls_debug_selftest(int which, void* workspace, size_t workspace_bytes, void* stream);

/*
 * Reads (synchronously, on `stream`) the device status word of a workspace
 * used by sls_lanczos_topr or sls_compress: SLS_OK, or SLS_ERR_TIMEOUT when
 * a device-side wait gave up.  Clears the word.
 */
int sls_workspace_status(void* workspace, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SLS_H_ */
