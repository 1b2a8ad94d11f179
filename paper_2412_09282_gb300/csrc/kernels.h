// Internal launchers of libcrvq (host side). Each enqueues on `stream` and returns a status.
#pragma once

#include "common.cuh"

namespace crvq {

constexpr int kD = 8;  // vector length supported by the kernels

// A vector set: M x (G_sub * d) block of a row-major matrix (leading dimension ldT) whose
// group g uses the Hessian block Hb[g].
struct SetView {
  const float* T;
  int64_t ldT;
  int64_t M;
  int64_t G_sub;
  const float* Hb;
};

crvq_status launch_hessian(const float* X, int64_t n, int64_t N, int d, float damp_rel,
                           float* H, float* xsq, float* H_blocks, float* delta,
                           cudaStream_t stream);
crvq_status launch_extract_blocks(const float* H, int64_t N, int d, const int32_t* perm,
                                  float* H_blocks, cudaStream_t stream);

// Tensor-core (tcgen05, 3xTF32) products.
// S = X^T X / n for X n x N row-major (S N x N, both triangles).
crvq_status launch_tc_syrk(const float* X, int64_t n, int64_t N, float* S, cudaStream_t stream);
// Xt = X^T (N x ldt, columns [n, ldt) zero) for X n x N row-major.
crvq_status launch_transpose(const float* X, int64_t n, int64_t N, float* Xt, int64_t ldt,
                             cudaStream_t stream);
// The 8 x 8 diagonal blocks of X^T X / n + delta I only, in the channel order perm (NULL: the
// stored order), bit-identical to the blocks of launch_hessian's dense H. delta_known: the
// damping is read from delta64; otherwise (stored order only) xsq, delta and delta64 are
// written.
crvq_status launch_tc_hessian_blocks(const float* Xt, int64_t ldt, int64_t n, int64_t N,
                                     const int32_t* perm, bool delta_known, float damp_rel,
                                     float* xsq, float* delta, double* delta64, float* Hb,
                                     cudaStream_t stream);
// dst[i][p] = src[i][idx[p]] for every row (M x N row-major; idx a permutation of 0..N-1,
// entries outside [0, N) reported and read as 0).
crvq_status launch_gather_cols(const float* src, int64_t M, int64_t N, const int32_t* idx,
                               float* dst, cudaStream_t stream);
// Partial sums of ||(A - A_sub) B'^T||_F^2 into part[0 .. *nparts): A, A_sub (optional) M x K,
// B Nb x K row-major, B' = B with its columns taken in the order B_cols (optional).
crvq_status launch_tc_sumsq(const float* A, const float* A_sub, int64_t M, const float* B,
                            const int32_t* B_cols, int64_t Nb, int64_t K, double* part,
                            int64_t part_cap, int64_t* nparts, cudaStream_t stream);

// C = A B^T on the tensor cores (3xTF32; K in chunks of 1024 added in order): A M x K
// (leading dimension lda), B Nb x K (ldb), C M x Nb (ldc); all row-major, 16-byte aligned rows.
crvq_status launch_tc_gemm_nt(const float* A, int64_t lda, int64_t M, const float* B,
                              int64_t ldb, int64_t Nb, int64_t K, float* C, int64_t ldc,
                              cudaStream_t stream);

// hinv[i] = [H^-1]_ii (fp64) of a symmetric positive definite H (N x N fp32): blocked fp64
// Cholesky, the inverse factor by blocked forward substitution, squared column norms.
crvq_status launch_hinv_diag(const float* H, int64_t N, double* hinv, cudaStream_t stream);

crvq_status launch_select_reorder(const float* W, int64_t M, int64_t N, int d,
                                  const float* W_pre, const float* xsq, const float* H,
                                  int mode, uint64_t seed, int32_t* perm, float* importance,
                                  float* W_sorted, float* H_blocks, cudaStream_t stream);

crvq_status launch_kmeans_init(const SetView& set, const CbList& fixed, int K, uint64_t seed,
                               float* C_out, cudaStream_t stream);

struct StatsView;

// Optional extras of an encode launch.
struct EncodeExtras {
  double* scores = nullptr;                // host: += (hypothesis, codeword) pairs scored
  const StatsView* stats = nullptr;        // accumulate LS statistics of the written codes
  unsigned long long* flag_total = nullptr;  // device: += vectors sent to the fp64 fallback
  // Scratch of the arg-min pass provided by the caller (e.g. once for a whole Lloyd loop, so
  // that its iterations allocate nothing); used when at least argmin_scratch_bytes long.
  char* work = nullptr;
  size_t work_bytes = 0;
  // Per-vector A-row terms of the arg-min pass for every group of the set (launch_row_terms),
  // valid while the target, the H blocks and the fixed codebooks stay put; null: computed in
  // the pass.
  const float4* rowterms = nullptr;
};

// The arg-min pass's per-vector terms for all M x G_sub vectors of the set (3 M G_sub float4).
crvq_status launch_row_terms(const SetView& set, const CbList& cbs, int n_fixed, float4* rt,
                             cudaStream_t stream);

// Scratch of one arg-min pass over a set of M rows and G_range groups with a K-entry codebook
// (B images, codeword terms, codebook maxima, flag list).
size_t argmin_scratch_bytes(int64_t M, int64_t G_range, int K);

// Encode / beam (see crvq_encode_beam).
crvq_status launch_encode_beam(const SetView& set, const CbList& cbs, int n_fixed, int B,
                               bool keep_if_better, float* vec_err, const EncodeExtras& ex,
                               cudaStream_t stream);

crvq_status launch_update_codebook(const SetView& set, const CbList& cbs, int which,
                                   float* C_out, int32_t* counts, cudaStream_t stream);

// Decode + block losses (+ optional W_hat in original order, + optional full loss).
// losses_dev: 3 doubles on the device [block, crit, full].
// delta_dev (device, 1 float) overrides damp_delta when not null.
crvq_status launch_reconstruct_error(const float* W_sorted, int64_t M, int64_t N,
                                     const float* Hb, const int32_t* perm, const CbList& cbs,
                                     int64_t n_crit_groups, const float* X, int64_t n_tok,
                                     double damp_delta, const float* delta_dev, float* W_hat,
                                     double* losses_dev, cudaStream_t stream);

// Gauss-Seidel sweeps of codebook `which` under the full loss (see crvq_coupled_sweep); W and
// H (N x N) in the sorted channel order; loss_dev: sweeps + 1 doubles on the device or null.
crvq_status launch_coupled_sweep(const float* W, int64_t M, int64_t N, const float* H,
                                 const CbList& cbs, int which, int sweeps, double* loss_dev,
                                 cudaStream_t stream);

// Y = X_in W_hat^T from the codes (see crvq_lut_matvec); b inputs of N channels (row stride
// ldx), M output rows (Y row stride ldy).
crvq_status launch_lut_matvec(const float* X, int64_t ldx, int64_t N, int b,
                              const int32_t* perm, const CbList& cbs, int64_t M, float* Y,
                              int64_t ldy, cudaStream_t stream);

}  // namespace crvq
