/*
 * crvq.h - C ABI of the GB300 (sm_103a) CRVQ code-search library (libcrvq.so).
 *
 * CRVQ (Channel-Relaxed Vector Quantization, arXiv 2412.09282) quantizes a weight matrix W
 * (M x N) by vector quantization of its length-d row segments, with one base codebook over
 * all vectors and extra "extended" codebooks fitted additively on the vectors of a small set
 * of reordered critical channels (Sec. 4, Alg. 1). This library runs the data-parallel hot
 * path of that procedure on one GPU: the Hessian proxy, channel scoring and reordering, the
 * vector x codeword score contraction with top-B (beam) selection, the codebook
 * least-squares update and the error evaluation.
 *
 * Conventions (every call):
 *  - Arrays are device pointers owned by the caller unless a parameter says "host". The
 *    library keeps no pointer after the call returns. Row-major; fp32 unless stated. The
 *    step calls (crvq_hessian ... crvq_reconstruct_error, crvq_update_codebook_noalloc)
 *    check that each device array is device or managed memory and return
 *    CRVQ_ERR_INVALID_ARG for a host pointer; crvq_quantize_layer accepts either.
 *  - Calls enqueue work on `stream` and return without waiting, except calls that return a
 *    value in host memory (their documentation says so): those synchronize `stream`.
 *  - Scratch memory is taken with stream-ordered cudaMallocAsync/cudaFreeAsync on `stream`.
 *  - Arguments are validated before any launch: a bad argument returns
 *    CRVQ_ERR_INVALID_ARG, an unsupported size CRVQ_ERR_UNSUPPORTED, and nothing is
 *    enqueued. crvq_last_error() then describes the problem (per host thread).
 *  - Faults found on the device (an index out of range, a non-SPD normal matrix, a bounded
 *    wait that ran out) set a per-device error word instead of trapping; crvq_sync() reports
 *    and clears it.
 *  - d (vector length) must be 8 in this version; larger d returns CRVQ_ERR_UNSUPPORTED.
 *
 * Vector sets. The encode/update/init calls work on a vector set: an M x (G_sub*d) block
 * T of a row-major matrix with leading dimension ldT (floats). Vector (i, g), 0 <= i < M,
 * 0 <= g < G_sub, is T[i*ldT + g*d .. + d) (the partition S of Sec. 3.1), and is scored with
 * the d x d Hessian block H_blocks[g] (pass H_blocks already offset to the set's first group).
 *
 * Codebooks. A codebook of a vector set covers the groups g < G_cov (a prefix of the set):
 * the base codebook covers every group, an extended codebook only the first G_c groups,
 * where the reordered critical channels sit (Sec. 4.3, Fig. 2). The reconstruction of vector
 * (i, g) is the sum, over the codebooks that cover g, of C[code(i, g)] (additive VQ).
 *
 * Score. Vector t against reconstruction r: err = (t - r)^T H_g (t - r), the block-diagonal
 * part of the Alg. 1 loss ||W X - W_enc X||^2 written with H = X^T X / n + delta I. With
 * H_g = c I it is the squared L2 distance of Sec. 3.1 Eq. (2)-(3). Code indices are decided
 * exactly: scores are computed in fp32 (on the tensor cores for one searched codebook) with
 * a rigorous error bound, and any decision closer than that bound is re-taken exactly (errs
 * as unevaluated fp32 pairs, about 2^-44 relative, or in fp64), so codes equal those of an
 * fp64 evaluation except for ties at rounding level (ties go to the smaller index / earlier
 * tuple).
 */
#ifndef CRVQ_H
#define CRVQ_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* crvq_stream_t; /* a cudaStream_t; NULL = the legacy default stream */
typedef int32_t crvq_status;

enum {
  CRVQ_OK = 0,
  CRVQ_ERR_INVALID_ARG = -1, /* a pointer, size or option is out of its documented range */
  CRVQ_ERR_UNSUPPORTED = -2, /* a valid request the library does not implement (e.g. d != 8) */
  CRVQ_ERR_CUDA = -3,        /* a CUDA runtime call failed */
  CRVQ_ERR_NOMEM = -4,       /* device memory allocation failed */
  CRVQ_ERR_TIMEOUT = -5,     /* a bounded device-side wait ran out */
  CRVQ_ERR_NUMERIC = -6,     /* non-finite input or a normal matrix that is not SPD */
  CRVQ_ERR_DEVICE = -7       /* a device-side index check failed (access skipped) */
};

/* Importance modes (Sec. 4.1; Table 2 "Reorder Strategy"). WA is the App. A.2 form (the
 * diagonal of X^T X); WA_INV is Eq. (wa) as printed, with the inverse-Hessian diagonal. */
enum {
  CRVQ_IMPORTANCE_WA = 0,
  CRVQ_IMPORTANCE_W_ONLY = 1,
  CRVQ_IMPORTANCE_RANDOM = 2,
  CRVQ_IMPORTANCE_WA_INV = 3
};

/* One codebook of a vector set (see "Codebooks" above). */
typedef struct crvq_codebook {
  const float* C; /* K x d codewords (device) */
  int32_t K;      /* number of codewords, 1 <= K <= 65536 */
  int32_t _pad;
  int32_t* codes; /* device; code of vector (i, g) is codes[i * ld + g] for g < G_cov */
  int64_t ld;     /* leading dimension of codes, ld >= G_cov */
  int64_t G_cov;  /* the codebook covers groups 0 <= g < G_cov of the set, G_cov <= G_sub */
} crvq_codebook;

/* Message describing the last failure on the calling host thread ("" when none). */
const char* crvq_last_error(void);

/* Waits for `stream`, then returns and clears the device error words of the current device
 * (the library's, and that of crvq_update_codebook_noalloc): CRVQ_OK, CRVQ_ERR_DEVICE,
 * CRVQ_ERR_NUMERIC or CRVQ_ERR_TIMEOUT (or CRVQ_ERR_CUDA). */
crvq_status crvq_sync(crvq_stream_t stream);

/* Library build string (compiler, architecture). Host memory, static. */
const char* crvq_version(void);

/* Self-test of the failure path of every bounded device wait: one thread waits on an
 * mbarrier that nothing ever arrives on, with the same bounded wait the tensor-core kernels
 * use (2 s of %globaltimer); it gives up, records the timeout in the device error word and
 * exits, so the context stays usable. The next crvq_sync on the device returns
 * CRVQ_ERR_TIMEOUT (and clears it). Enqueues on `stream`; no trap, no fault, no unbounded
 * spin. */
crvq_status crvq_selftest_bounded_wait(crvq_stream_t stream);

/* Per-kernel timing. Between crvq_profile_begin() and crvq_profile_end(), every kernel the
 * library launches is bracketed by CUDA events recorded on the stream it is launched on.
 * crvq_profile_end() waits for them and writes one entry per kernel name (host memory,
 * at most `cap` entries, *n_stats set to the number written). `units` is the algorithmic
 * work the launches were given (scores for the encode kernels, vectors for the update,
 * multiply-adds for the GEMMs, bytes for the streaming kernels). */
typedef struct crvq_kernel_stat {
  char name[64];
  int64_t launches;
  double ms;     /* summed event time */
  double units;  /* summed algorithmic work */
} crvq_kernel_stat;

crvq_status crvq_profile_begin(void);
crvq_status crvq_profile_end(crvq_kernel_stat* stats, int32_t cap, int32_t* n_stats);

/* Restricts the next profiling sessions to kernel names starting with `prefix` (host string,
 * copied; at most 63 characters); NULL or "" profiles every kernel again. Recording events
 * costs host time per launch, so a narrow filter keeps a timed region close to unprofiled.
 * Returns CRVQ_ERR_INVALID_ARG while a session is running or for a longer prefix. */
crvq_status crvq_profile_filter(const char* prefix);

/* Number of kernels this library has launched in this process (all devices). */
int64_t crvq_launch_count(void);

/*
 * S1. Hessian proxy (Alg. 1 "Require: XX^T"; App. A.2, where X is N x O and the proxy XX^T).
 * Here X is n_tok x N (row = token) and H = X^T X / n_tok + delta I with
 * delta = damp_rel * mean_i (X^T X / n_tok)_ii (damping is not in the paper; it keeps the
 * least-squares codebook solves well posed).
 *   X        [n_tok x N] calibration activations.
 *   H        [N x N] out, symmetric.
 *   xsq      [N] out, undamped diagonal (X^T X / n_tok)_ii, used by the W-A importance.
 *   H_blocks [(N/d) x d x d] out or NULL: diagonal blocks of H in the original channel order.
 *   delta    [1] out or NULL: the damping added to the diagonal.
 * Requires n_tok >= 1, N >= 1, N % d == 0, damp_rel >= 0 and finite.
 */
crvq_status crvq_hessian(const float* X, int64_t n_tok, int64_t N, int32_t d, float damp_rel,
                         float* H, float* xsq, float* H_blocks, float* delta,
                         crvq_stream_t stream);

/*
 * S1 / S3 without the dense H: the diagonal d x d blocks of H = X^T X / n_tok + delta I (as
 * crvq_hessian defines it) for the channel order `perm`:
 *   H_blocks[g][a][b] = H[perm[g*d + a]][perm[g*d + b]]   (perm NULL: the stored order).
 * The method reads H only through these blocks (the vector scores of Sec. 3.1 under the
 * block-diagonal reading of the Alg. 1 loss) and its diagonal (App. A.2 importance), so a
 * layer needs N * n_tok floats of scratch here instead of the N x N matrix. The values equal
 * crvq_hessian's dense H entries bit for bit (same tensor-core products, same split-K order).
 *   X        [n_tok x N] device, 16-byte aligned.
 *   perm     [N] device int32 channel order, or NULL. Entries outside [0, N) are reported as
 *            CRVQ_ERR_DEVICE by crvq_sync (the affected block rows are left unwritten).
 *   xsq      [N] out or NULL: the undamped diagonal, stored order.
 *   delta    [1] out or NULL.
 *   H_blocks [(N/d) x d x d] out.
 * Requires n_tok >= 1, N >= 1, N % d == 0, damp_rel >= 0 and finite; d = 8.
 */
crvq_status crvq_hessian_blocks(const float* X, int64_t n_tok, int64_t N, int32_t d,
                                float damp_rel, const int32_t* perm, float* xsq, float* delta,
                                float* H_blocks, crvq_stream_t stream);

/*
 * The diagonal of the inverse of a symmetric positive definite H (the denominator of Sec. 4.1
 * Eq. (wa)): hinv[i] = [H^-1]_ii in fp64, from a blocked fp64 Cholesky factor H = L L^T as the
 * squared column norms of L^-1 (about 2 N^3 / 3 fp64 flops; fp64 because the channel order
 * it decides must match an fp64 evaluation while cond(H) reaches 1e4 and more).
 *   H     [N x N] device, symmetric (the lower triangle is read), e.g. crvq_hessian's H.
 *   hinv  [N] device out (fp64).
 * A non-positive pivot (H not SPD) is reported as CRVQ_ERR_NUMERIC by crvq_sync.
 * Requires 1 <= N <= 49152. Scratch: two (N rounded up to 64)^2 fp64 matrices.
 */
crvq_status crvq_hessian_inverse_diag(const float* H, int64_t N, double* hinv,
                                      crvq_stream_t stream);

/*
 * S3. Channel importance and reordering (Alg. 1 ComputeImportance, ReorderChannels;
 * Sec. 4.1-4.2; App. A.2).
 *   mode W-A:    I_i = 1/2 * xsq_i * max_j (W_ji - W_pre_ji)^2 (App. A.2 form; W_pre is the
 *                prequantized W, original order).
 *   mode W-A inverse: I_i = max_j (W_ji - W_pre_ji)^2 / (2 [H^-1]_ii) (Eq. (wa) as printed;
 *                diag(H^-1) as crvq_hessian_inverse_diag computes it from H; xsq may be NULL).
 *   mode W-only: I_i = max_j W_ji^2 (Sec. 4.1). W_pre and xsq may be NULL.
 *   mode random: I_i = (SplitMix64(seed, i) >> 40) * 2^-24 (Table 2 "Random").
 * perm sorts channels by I descending, ties by original index (perm[new] = old).
 *   perm        [N] int32 out.      importance [N] out or NULL.
 *   W_sorted    [M x N] out, W_sorted[:, p] = W[:, perm[p]].
 *   H_blocks    [(N/d) x d x d] out, H_blocks[g][a][b] = H[perm[g d + a]][perm[g d + b]].
 *   n_crit_groups  host out: G_c = min(N/d, ceil(crit_frac * N / d)) (Sec. 4.3 ratio lambda,
 *               rounded up to whole groups of d channels).
 * Requires 0 <= crit_frac <= 1, N % d == 0, N <= 49152.
 */
crvq_status crvq_select_reorder_channels(const float* W, int64_t M, int64_t N, int32_t d,
                                         const float* W_pre, const float* xsq, const float* H,
                                         float crit_frac, int32_t mode, uint64_t seed,
                                         int32_t* perm, float* importance, float* W_sorted,
                                         float* H_blocks, int64_t* n_crit_groups,
                                         crvq_stream_t stream);

/*
 * k-means initial codebook (Eq. kmeans in Sec. 3.1; Alg. 1 KMeansCodebook). Draws one vector
 * from each of K equal strata of the vector index range v = i * G_sub + g:
 * v_k = floor(k n / K) + SplitMix64(seed, k) mod (floor((k+1) n / K) - floor(k n / K)),
 * n = M * G_sub; codeword k is that vector minus the reconstruction of the `fixed`
 * codebooks (residual, for extended codebooks), evaluated in fp64 and rounded once.
 *   fixed  host array of n_fixed codebooks (may be NULL when n_fixed == 0).
 *   C_out  [K x d] out.     Requires 1 <= K <= min(n, 65536).
 */
crvq_status crvq_kmeans_init(const float* T, int64_t ldT, int64_t M, int64_t G_sub, int32_t d,
                             const crvq_codebook* fixed, int32_t n_fixed, int32_t K,
                             uint64_t seed, float* C_out, crvq_stream_t stream);

/*
 * Encode / beam search (Sec. 3.1 Eq. (2)-(3); Alg. 1 VectorQuant, BeamSearchOptimize).
 * Codebooks 0..n_fixed-1 are fixed (their codes are read); codebooks n_fixed..n_cb-1 are
 * searched and their codes written. For each vector the target is t minus the fixed
 * reconstruction; the searched codebooks that cover the vector are taken in order as beam
 * stages: every kept partial tuple is extended by every codeword and the B best are kept,
 * ordered by (err, parent rank, codeword index). The best tuple of the last stage is written.
 * With one searched stage this is the arg-min assignment step of k-means.
 *   keep_if_better  nonzero: the searched codes hold a tuple on entry, which is kept when
 *                   its err is strictly smaller than the beam's best.
 *   vec_err         [M x G_sub] out or NULL: err of the written tuple (fp64, rounded).
 * Requires 1 <= B <= 16, 0 <= n_fixed < n_cb <= 8. Sets of more than 65535 groups return
 * CRVQ_ERR_UNSUPPORTED (a beam stage launches one grid row per group).
 * Beam stages over codebooks of at most 256 codewords with B <= 8 score on the tensor cores and
 * keep exactly the lists of the SIMT stages; CRVQ_BEAM_TC=0 in the environment (read at every
 * call) keeps every stage on the SIMT kernels. The results are identical either way.
 */
crvq_status crvq_encode_beam(const float* T, int64_t ldT, int64_t M, int64_t G_sub, int32_t d,
                             const float* H_blocks, const crvq_codebook* cbs, int32_t n_cb,
                             int32_t n_fixed, int32_t B, int32_t keep_if_better,
                             float* vec_err, crvq_stream_t stream);

/*
 * Least-squares codebook update (k-means update step; Alg. 1 FineTuneCodebook read as the
 * closed-form minimiser). Codebook `which` is refitted with all others fixed: the members v
 * of cluster k (vectors with code k, g < G_cov) have targets tau_v = t_v - sum over the other
 * covering codebooks of C[code]; c_k solves (sum_v H_{g_v}) c = sum_v H_{g_v} tau_v
 * (right side in 64-bit fixed point, normal matrix as fp32 pairs, both summed in a fixed order;
 * Cholesky with refinement in fp32 pairs, so results are reproducible bit for bit). Empty
 * clusters keep their codeword.   C_out [K x d] out (may alias cbs[which].C).
 *   counts [K] int32 out or NULL: cluster sizes.
 */
crvq_status crvq_update_codebook(const float* T, int64_t ldT, int64_t M, int64_t G_sub,
                                 int32_t d, const float* H_blocks, const crvq_codebook* cbs,
                                 int32_t n_cb, int32_t which, float* C_out, int32_t* counts,
                                 crvq_stream_t stream);

/*
 * crvq_update_codebook without device memory allocation. The paper has no counterpart: this
 * entry point exists for callers that cannot call cudaMalloc or cudaFree, such as runtimes
 * that hand out a fixed memory arena and forbid allocation after start-up, plugins whose host
 * owns every device allocation, and latency-critical callers that must not synchronise
 * (cudaFree synchronises the device). Arguments, validation (host pointers are refused with
 * CRVQ_ERR_INVALID_ARG), results and rounding are those of crvq_update_codebook; the caller
 * still passes the inputs and outputs. Its scratch is one file-scope device array of 4 MiB,
 * held by every GPU that loads the library until the process exits:
 *  - sizes whose statistics exceed it (G_cov * K * 4 + K * 64 + 256 + K * 296 bytes, each
 *    part rounded up to 256 bytes, above 4 MiB; e.g. K = 256 with more than ~3900 covered
 *    groups) return CRVQ_ERR_UNSUPPORTED before anything is enqueued;
 *  - every call shares the array and it keeps the last call's contents: each call clears
 *    what must start at zero, and calls that overlap on the GPU (on different streams, or
 *    host threads enqueueing on one device without ordering) race;
 *  - the first call on a device looks up the array's device address (cudaGetSymbolAddress)
 *    with that device current; make that first call before any stream capture;
 *  - what the kernels find on the device (codes outside [0, K), which are skipped; a
 *    non-finite input; a normal matrix without a Cholesky factor, whose codeword keeps its
 *    old value) is recorded in a second file-scope word, which the next crvq_sync on the
 *    device reports (CRVQ_ERR_DEVICE, CRVQ_ERR_NUMERIC) and clears, like the other calls'
 *    reports.
 */
crvq_status crvq_update_codebook_noalloc(const float* T, int64_t ldT, int64_t M, int64_t G_sub,
                                         int32_t d, const float* H_blocks,
                                         const crvq_codebook* cbs, int32_t n_cb, int32_t which,
                                         float* C_out, int32_t* counts, crvq_stream_t stream);

/*
 * S7. Reconstruction, reverse reorder and losses (Alg. 1 QuantLoss; Sec. 4.3 "restored to
 * their original order"). The set is all of W_sorted (M x N, G = N/d groups).
 *   perm         [N] or NULL (identity).
 *   W_hat        [M x N] out or NULL: the reconstruction in the original channel order.
 *   X            [n_tok x N] or NULL (then losses[2] = NaN).
 *   losses       HOST out [3]: loss_block = sum over vectors of err; loss_crit = the same
 *                over groups g < n_crit_groups; loss_full = ||(W - W_hat) X^T||^2 / n_tok
 *                + damp_delta ||W - W_hat||^2 = tr(dW H dW^T). Synchronizes `stream`.
 */
crvq_status crvq_reconstruct_error(const float* W_sorted, int64_t M, int64_t N, int32_t d,
                                   const float* H_blocks, const int32_t* perm,
                                   const crvq_codebook* cbs, int32_t n_cb,
                                   int64_t n_crit_groups, const float* X, int64_t n_tok,
                                   double damp_delta, float* W_hat, double* losses,
                                   crvq_stream_t stream);

/*
 * Code search under the full Alg. 1 loss (QuantLoss ||W X - W_enc X||^2 = tr(dW H dW^T),
 * cross-group terms included; the encode calls above score each vector with its own diagonal
 * block only). Gauss-Seidel over the groups of codebook `which`, every other codebook fixed:
 * for g = 0 .. G_cov-1 in order, each row's code of group g becomes the arg-min (as
 * crvq_encode_beam decides it, ties to the smaller index) of err(t', c) = (t' - c)^T H_gg (t' - c)
 * for the shifted target t' = t + H_gg^-1 b_g, where t is the row segment minus the other
 * codebooks' codewords, b_g = sum_{g' != g} H_gg' D_g' and D = W - W_enc with every code
 * decided so far (completing the square of the row loss in D_g). The full loss never rises.
 *   W_sorted  [M x N] weights in the channel order of H (row-major, 16-byte aligned).
 *   H_sorted  [N x N] the damped Hessian proxy in the same channel order (symmetric; e.g.
 *             crvq_hessian's H taken through the layer's perm).
 *   cbs       the n_cb codebooks of the M x (N/d) vector set; the codes of `which` are read
 *             and rewritten in place.
 *   sweeps    >= 0 passes over the groups.
 *   loss      HOST out [sweeps + 1] or NULL: tr(dW H dW^T) before the first sweep and after
 *             each (3xTF32 products, fp64 sums). Synchronizes `stream` when given.
 * b_g comes from tensor-core products of H with D^T taken per block of 256 channels at the
 * block's start plus the block's own earlier changes; the shift is solved in fp32 with a
 * Cholesky factor of H_gg computed in fp64. A block without a factor is reported as
 * CRVQ_ERR_NUMERIC by crvq_sync. Requires N % d == 0, N <= 49152; d = 8.
 */
crvq_status crvq_coupled_sweep(const float* W_sorted, int64_t M, int64_t N, int32_t d,
                               const float* H_sorted, const crvq_codebook* cbs, int32_t n_cb,
                               int32_t which, int32_t sweeps, double* loss,
                               crvq_stream_t stream);

/*
 * Inference product of a quantized matrix, from its codes (App. "Inference Speed", Table
 * speed: the matrix-vector product with a CRVQ layer). Y = X_in W_hat^T for b inputs, W_hat
 * being the reconstruction in the original channel order that crvq_reconstruct_error returns,
 * without forming it:
 *   Y[bi][i] = sum over codebooks s and groups g < G_cov(s) of
 *              <C_s[code_s(i, g)], x_sorted[bi][g d .. g d + d)>,  x_sorted[bi][p] = X_in[bi][perm[p]].
 *   X_in   [b x N] device, row stride ldx >= N (floats).
 *   perm   [N] device channel order (perm[new] = old), or NULL for the identity.
 *   cbs    the n_cb codebooks of the M x (N/d) vector set (base first, as the layer returns
 *          them; codes int32 on the device).
 *   Y      [b x M] out, row stride ldy >= M.
 * fp32 arithmetic: every codeword-input product is an 8-term FMA chain and the sums over
 * groups follow a fixed order (no atomics), so results are identical run to run. Codes
 * outside [0, K) and perm entries outside [0, N) are skipped and reported by crvq_sync.
 * Requires 1 <= b <= 8, N % d == 0, 1 <= n_cb <= 8; d = 8.
 */
crvq_status crvq_lut_matvec(const float* X_in, int64_t ldx, int64_t b, int64_t N, int32_t d,
                            const int32_t* perm, const crvq_codebook* cbs, int32_t n_cb,
                            int64_t M, float* Y, int64_t ldy, crvq_stream_t stream);

/* Average bits per weight (Sec. 3.2 Eq. (bitwidth); App. A.1): e-bit codes for all M N / d
 * vectors, plus m-1 extended codebooks on the lambda fraction, plus m codebooks of 2^e
 * fp16 vectors of length d, plus (include_perm) a 16-bit reorder index per channel. */
double crvq_avg_bits(int32_t e, int32_t d, int32_t m, double lambda, int64_t M, int64_t N,
                     int32_t include_perm);

/* The same with n_base base codebooks (crvq_config.n_base) and n_ext extended ones: e-bit codes
 * for all vectors per base codebook (Sec. 3.2 Eq. (bitwidth) counts m of them), n_ext on the
 * lambda fraction, n_base + n_ext codebooks of 2^e fp16 vectors of length d, and (include_perm)
 * the reorder index. n_base = 1 equals crvq_avg_bits with m = 1 + n_ext. NaN for d, M, N or
 * n_base below 1, or e or n_ext below 0. */
double crvq_avg_bits_bases(int32_t e, int32_t d, int32_t n_base, int32_t n_ext, double lambda,
                           int64_t M, int64_t N, int32_t include_perm);

/* G_c = min(N/d, ceil(crit_frac * N / d)) (0 when crit_frac == 0). */
int64_t crvq_n_crit_groups(int64_t N, int32_t d, float crit_frac);

/* Hyper-parameters of one matrix (Alg. 1 inputs m, lambda, epsilon; Sec. 3.2 e, d). */
typedef struct crvq_config {
  int32_t d;               /* vector length (8) */
  int32_t K_base;          /* base codebook size 2^e */
  int32_t n_ext;           /* extended codebooks (m - 1), 0..7, n_base + n_ext <= 8 */
  int32_t K_ext;           /* extended codebook size */
  float crit_frac;         /* lambda */
  int32_t B;               /* beam width of the refinement re-encode, 1..16 */
  int32_t kmeans_iters;    /* Lloyd iterations per codebook fit */
  int32_t refine_rounds;   /* maximum FineTuneCodebook + BeamSearch rounds */
  float eps_rel;           /* stop refining when loss_block > (1 - eps_rel) * previous */
  float damp_rel;          /* Hessian damping, relative to the mean diagonal */
  int32_t importance_mode; /* CRVQ_IMPORTANCE_* */
  int32_t n_base;          /* base codebooks over every group, 0 or 1 = one (Sec. 6.4 uses
                              two, "m = 2"); n_base + n_ext <= 8 */
  uint64_t seed;
} crvq_config;

/* Outputs of one matrix. Pointers may be device or host memory (host buffers are staged
 * through the device inside the call). */
typedef struct crvq_layer_outputs {
  int32_t* perm;       /* [N] channel order, perm[new] = old */
  float* C_base;       /* [n_base x K_base x d] */
  int32_t* codes_base; /* [n_base x M x N/d], vector (i, g) in the sorted order */
  float* C_ext;        /* [n_ext x K_ext x d] */
  int32_t* codes_ext;  /* [n_ext x M x G_c] */
  float* W_hat;        /* [M x N] reconstruction in the original order, or NULL */
  float* importance;   /* [N] or NULL */
} crvq_layer_outputs;

typedef struct crvq_layer_report {
  double loss_pre;       /* loss_block of the prequantized W (original order) */
  double loss_block;     /* final losses (see crvq_reconstruct_error) */
  double loss_crit;
  double loss_full;
  double loss_before_refine;
  double scores;         /* (hypothesis, codeword) pairs scored by the encode passes */
  int64_t n_crit_groups;
  int64_t flagged;       /* encode decisions re-taken exactly (fp32 bound not conclusive) */
  int32_t refine_rounds_done;
  int32_t _pad;
} crvq_layer_report;

/*
 * One weight matrix through Alg. 1, prequantization through the refinement loop (everything
 * but block / end-to-end fine-tuning):
 * S1 Hessian; S2 prequantize (k-means + encode in the original order); S3 importance and
 * reorder; S4 base codebook (k-means over all vectors; with n_base > 1 each further base
 * codebook is fitted the same way on the residual of the earlier ones over every vector);
 * S5 each extended codebook (k-means on the critical residual of every earlier codebook,
 * greedy encode); S6 up to refine_rounds rounds of
 * least-squares updates of every codebook followed by a joint beam re-encode (keep-if-better);
 * S7 losses and the reconstruction in the original order. Per-phase seeds are
 * SplitMix64(cfg->seed, phase * 1024 + codebook) with phase 1 = prequantize, 2 = base
 * (codebook b = 0 .. n_base - 1), 3 = extended (codebook t = 1 .. n_ext), 4 = random
 * importance. The refinement updates the base codebooks, then the extended ones, in order. W [M x N], X [n_tok x N] may be host or device
 * pointers. Synchronizes `stream` (the report is host memory).
 * When W, X and every output are device pointers and refine_rounds <= 1, the schedule has no
 * host synchronisation inside: it is captured into a CUDA graph on the first call for a given
 * (device, stream, shapes, configuration, pointers, profiling state) and replayed on later
 * calls, which reads the current contents of W and X (up to 48 graphs are kept per process,
 * least recently used evicted, never one being replayed; their scratch stays reserved while
 * they are kept). Setting CRVQ_GRAPHS=0 in the environment runs every call directly. Results
 * are identical either way.
 * Calls for different matrices may run concurrently from different host threads, each on its
 * own stream and with its own output buffers: a replay does not hold the library's graph lock,
 * and a host-buffer call stages its data in buffers no running call holds (up to eight sets
 * kept). Their results equal those of the same calls one after another. Concurrent calls that
 * share output buffers race; calls on one stream run one after another.
 * What the kernels report on the device (a non-finite input, a refused index, a bounded wait
 * that ran out) is returned by the next crvq_sync on the device, not by this call.
 */
crvq_status crvq_quantize_layer(const float* W, const float* X, int64_t M, int64_t N,
                                int64_t n_tok, const crvq_config* cfg,
                                const crvq_layer_outputs* out, crvq_layer_report* report,
                                crvq_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* CRVQ_H */
