// Internal launcher declarations shared by the library's translation units.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace sls {

// ---- feature map (Sec. 3.2) ----------------------------------------------
// Phi is written as float32, or as bfloat16 (round to nearest even from the
// float32 value) when phi_bf16 is set.
int launch_feature_map_simt(const void* X, int x_dtype, int64_t N, int d, int64_t ldx,
                            const void* W, const float* b, int D, void* Phi,
                            cudaStream_t stream, int phi_bf16 = 0);
// tcgen05 / TMA path for bf16 inputs; returns SLS_ERR_UNSUPPORTED when the
// shape is outside what the kernel handles (the caller then uses the SIMT path).
int launch_feature_map_tc(const void* X, int64_t N, int d, int64_t ldx, const void* W,
                          const float* b, int D, void* Phi, cudaStream_t stream,
                          int* status = nullptr, int phi_bf16 = 0);
// The same over nb prompts in one launch: prompt k has `rows` rows starting at
// X row k * x_stride and writes Phi rows [k * rows, (k + 1) * rows).  With
// `live` set (one flag per window of `win` rows, nwin per prompt,
// prompt-major), row tiles whose windows are all 0 are not computed.
int launch_feature_map_tc_batched(const void* X, int64_t nb, int64_t rows, int64_t x_stride,
                                  int d, int64_t ldx, const void* W, const float* b, int D,
                                  void* Phi, const int* live, int nwin, int win,
                                  cudaStream_t stream, int* status, int phi_bf16 = 0);

// ---- self-test of the device-side wait limits ---------------------------------
// which = 0: an mbarrier wait nothing completes; 1: a two-CTA group barrier
// one CTA never reaches.  The wait gives up and writes SLS_ERR_TIMEOUT to
// *status; barw: 256 bytes of barrier words.
int launch_selftest_wait_limit(int which, int* status, unsigned* barw, cudaStream_t stream);

// ---- input embeddings: X = E[ids] (Sec. 3.1) ---------------------------------
// Rows of a V x d table (row stride ld_table elements) gathered into X (row
// stride ldx); an id outside [0, V) gives a zero row and is counted in *bad
// (zeroed first; may be NULL).
int launch_embed_gather(const void* table, int x_dtype, int64_t V, int d, int64_t ld_table,
                        const int32_t* ids, int64_t N, void* X, int64_t ldx, int* bad,
                        cudaStream_t stream);

// ---- row-normalised operator (Sec. 3.2 variant) ------------------------------
// Rows of every problem (rows [row0[p], row0[p] + n[p]) of Phi, or one problem
// of n_single rows when row0 is NULL) scaled in place by 1 / sqrt(s_i) with
// s = Phi (Phi^T 1) of the problem; s_out (may be NULL) receives s per row.
size_t feature_normalize_scratch_bytes(int64_t nmax, int D, int nprob);
int launch_feature_normalize(float* Phi, int D, const int64_t* row0, const int* n,
                             int nprob_max, const int* nprob_dev, int64_t n_single, int64_t nmax,
                             float2* scratch, double* s_out, cudaStream_t stream);

// ---- Lanczos (Algorithm 2) --------------------------------------------------
// Row stride (in float2) of the double-float basis Q: r rounded up to even,
// so every basis row starts on a 16-byte boundary.
__host__ __device__ inline int q_ld(int r) { return (r + 1) & ~1; }

// A batch of independent problems, problem p owning rows
// [row0[p], row0[p] + n[p]) of Phi, Q and U and start vector q1 + q1off[p].
struct LanczosBatch {
  const void* Phi;      // rows x D: float32, or raw bfloat16 bits when phi_bf16
  int D;
  int r;
  double tol;
  const double* q1;
  // problem table: either a single problem (table pointers NULL, n_single
  // rows from row 0) or device arrays read by the kernels
  int64_t n_single;
  int nprob_max;            // host upper bound on the number of problems
  const int* nprob_dev;     // device count (may be NULL: nprob_max problems)
  const int64_t* row0;      // device, per problem
  const int* n;             // device, per problem
  const int64_t* q1off;     // device, per problem (NULL: = row0)
  // outputs, per problem p: Q rows as above (ld r); alpha/beta/theta at p*r;
  // S at p*r*r; r_eff at p
  float2* Q;
  double* alpha;
  double* beta;
  double* theta;
  double* S;
  int* r_eff;
  int64_t nmax;             // max rows of any problem
  int phi_bf16;             // Phi stored as bfloat16 (D % 8 == 0)
  // self-test of the failure path (0 in every ordinary call): the first CTA
  // reports a failed wait at its first group barrier, as a wait that gave up
  // would, so the kernel's give-up and clean-exit path runs without a fault
  int inject_fail;
};

size_t lanczos_scratch_bytes(int64_t nmax, int D, int r, int groups, int ctas_per_group);
int lanczos_plan(int64_t nmax, int D, int r, int nprob, int* groups, int* ctas_per_group);
int launch_lanczos(const LanczosBatch& bt, void* scratch, size_t scratch_bytes, int* status,
                   int groups, int ctas_per_group, cudaStream_t stream);
int launch_tridiag_eigen(const LanczosBatch& bt, cudaStream_t stream, bool values_done = false);
// Small problems (every window at most 32 rows, r <= 32): one warp per
// problem runs Algorithm 2 exactly (two Gram-Schmidt passes, beta = |z|) and
// the Ritz values; launch_tridiag_eigen(values_done = true) then adds S.
bool lanczos_window_fits(int64_t nmax, int D, int r);
int launch_lanczos_window(const LanczosBatch& bt, cudaStream_t stream);
int launch_ritz_vectors(const LanczosBatch& bt, float* U, cudaStream_t stream);

// ---- SimHash (Sec. 3.3) -----------------------------------------------------
int launch_simhash(const float* U, int64_t N, int k, int ldu, const int32_t* k_dev,
                   const float* R, int bits, int ldr, uint32_t* codes, cudaStream_t stream);

}  // namespace sls

// ---- segment / aggregation (hash_aggregate.cu) -------------------------------
namespace sls {
struct ProbDesc;
size_t segment_scratch_bytes(int64_t nmax, int64_t mmax, int slots);
int launch_simhash_problems(const ProbDesc* probs, const int* spec_list, const int* nspec_dev,
                            int nspec_max, int64_t nmax, const int* r_eff, const float* U, int ldu,
                            const float* R, int ldr, int bits_max, uint32_t* codes,
                            cudaStream_t stream);
// chunk_done: the chunk windows' outputs were written by the score pass
// (launch_window_score_chunk); they are skipped here, their macro lengths set
// to 0 so that the aggregation skips them too.
int launch_segment(const ProbDesc* probs, int nprob, const uint32_t* codes, int pos_scheme,
                   int pos_mode, void* scratch, int slots, int64_t nmax, int64_t mmax, int* perm,
                   int* mstart, int* mlen, int32_t* pos_out, int32_t* tok2macro, int* status,
                   cudaStream_t stream, int chunk_done = 0);
int launch_preserved(int64_t B, int64_t N, int64_t M, int pf, int pl, int pos_mode, int* perm,
                     int* mstart, int* mlen, int32_t* pos_out, int32_t* tok2macro,
                     cudaStream_t stream);
int launch_identity(const void* X, int x_dtype, int64_t B, int64_t N, int d, int64_t ldx,
                    float* Xt, int32_t* pos, int32_t* tok2macro, cudaStream_t stream);
size_t agg_item_capacity(int64_t Mtot, int64_t Ntot);
size_t agg_part_capacity(int64_t Ntot);
// Integers of the aggregation's auxiliary area (counts, block totals, CTA
// ranges, list of macro-tokens spanning several work items).
size_t agg_aux_ints(int64_t Mtot, int64_t Ntot);
int launch_aggregate(const void* X, int x_dtype, int d, int64_t ldx, const int* perm,
                     const int* mstart, const int* mlen, int64_t Mtot, int64_t Ntot, int renorm,
                     float* Xt, int* pt_start, int2* items, int* aux, float* part,
                     float* part_eta, int* status, cudaStream_t stream);
// Redundancy score of every window (Sec. 3.6, Eq. redundancy); part holds
// score_part_floats(nprob, nmax, d) floats of scratch.
size_t score_part_floats(int64_t nprob, int64_t nmax, int d);
int launch_window_score(const void* X, int x_dtype, int d, int64_t ldx, const ProbDesc* probs,
                        int nprob, int64_t nmax, float* part, float* score, cudaStream_t stream);
// The same score pass, which also writes every window's chunk-path output
// (array_split groups of its m macro-tokens: renormalised means into Xt,
// positions, token map) -- final for the windows the router sends to the
// chunk path, replaced by the spectral path for the others.
int launch_window_score_chunk(const void* X, int x_dtype, int d, int64_t ldx,
                              const ProbDesc* probs, int nprob, int64_t nmax, float* part,
                              float* score, int pos_scheme, int pos_mode, int renorm, float* Xt,
                              int32_t* pos, int32_t* tok2macro, cudaStream_t stream);
}  // namespace sls
