// Host side of the tcgen05 3xTF32 GEMM (tc_gemm.cuh) and the fixed-order reductions of its
// split-K partial products. The tensor core accumulates fp32 with a small systematic
// rounding bias per accumulation step, so K is cut into chunks of at most kKChunk and the
// few chunk partials of an element are summed afterwards in fp32, in chunk order (a relative
// error of a few u); the sums of squares over elements are reduced in fp64.
#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "tc_gemm.cuh"

namespace crvq {

namespace {

constexpr int64_t kKChunk = 1024;

// scale * sum_c P[c * stride + e], chunks in order (the one rounding sequence every split-K
// product of this file uses, so its dense and block-only forms agree bit for bit)
__device__ __forceinline__ float chunk_sum(const float* __restrict__ P, int chunks,
                                           int64_t stride, int64_t e, float scale) {
  float s = 0.f;
  for (int c = 0; c < chunks; ++c) s += P[c * stride + e];
  return s * scale;
}

__global__ void __launch_bounds__(256)
sum_partials_kernel(const float* __restrict__ P, int64_t count, int chunks, int64_t stride,
                    float scale, float* __restrict__ out) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < count;
       e += (int64_t)gridDim.x * blockDim.x)
    out[e] = chunk_sum(P, chunks, stride, e, scale);
}

// Original-order blocks, one CTA: xsq[i] = the undamped diagonal, delta = damp_rel * mean(xsq)
// by the dense path's fixed-order fp64 reduction (1024 strided partials, then a tree), and the
// blocks with delta added on their diagonals (rounded once from fp64, as the dense path does).
__global__ void __launch_bounds__(1024)
blocks_finalize_kernel(const float* __restrict__ P, int chunks, int64_t stride, float scale,
                       int64_t N, float damp_rel, float* __restrict__ xsq,
                       float* __restrict__ delta_out, double* __restrict__ delta64,
                       float* __restrict__ Hb) {
  __shared__ double part[1024];
  double s = 0.0;
  for (int64_t i = threadIdx.x; i < N; i += blockDim.x) {
    const float v = chunk_sum(P, chunks, stride, i * 8 + (i & 7), scale);
    xsq[i] = v;
    s += (double)v;
  }
  part[threadIdx.x] = s;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) part[threadIdx.x] += part[threadIdx.x + w];
    __syncthreads();
  }
  const double delta = (double)damp_rel * (part[0] / (double)N);
  for (int64_t e = threadIdx.x; e < N * 8; e += blockDim.x) {
    const float v = chunk_sum(P, chunks, stride, e, scale);
    Hb[e] = ((e >> 3) & 7) == (e & 7) ? (float)((double)v + delta) : v;
  }
  if (threadIdx.x == 0) {
    if (delta_out) *delta_out = (float)delta;
    *delta64 = delta;
  }
}

// Blocks of a given channel order with a known delta.
__global__ void __launch_bounds__(256)
blocks_damp_kernel(const float* __restrict__ P, int chunks, int64_t stride, float scale,
                   int64_t N, const double* __restrict__ delta64, float* __restrict__ Hb) {
  const double delta = *delta64;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < N * 8;
       e += (int64_t)gridDim.x * blockDim.x) {
    const float v = chunk_sum(P, chunks, stride, e, scale);
    Hb[e] = ((e >> 3) & 7) == (e & 7) ? (float)((double)v + delta) : v;
  }
}

// part[block] = sum over this block's elements e of (sum_c P[c * stride + e])^2
__global__ void __launch_bounds__(256)
sumsq_partials_kernel(const float* __restrict__ P, int64_t count, int chunks, int64_t stride,
                      double* __restrict__ part) {
  __shared__ double red[256];
  float acc_f = 0.f;  // a few hundred non-negative terms per thread
  double acc;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < count;
       e += (int64_t)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int c = 0; c < chunks; ++c) s += P[c * stride + e];
    acc_f = fmaf(s, s, acc_f);
  }
  acc = (double)acc_f;
  red[threadIdx.x] = acc;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) part[blockIdx.x] = red[0];
}

// out[a][k] = X[k][a] (X: n x N row-major) for a < N, k < n; columns k in [n, ldt) are 0.
__global__ void __launch_bounds__(256)
transpose_kernel(const float* __restrict__ X, int64_t n, int64_t N, float* __restrict__ out,
                 int64_t ldt) {
  __shared__ float t[32][33];
  const int64_t k0 = (int64_t)blockIdx.x * 32, a0 = (int64_t)blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 32 x 8
#pragma unroll
  for (int r = ty; r < 32; r += 8) {
    const int64_t k = k0 + r, a = a0 + tx;
    t[r][tx] = (k < n && a < N) ? X[k * N + a] : 0.f;
  }
  __syncthreads();
#pragma unroll
  for (int r = ty; r < 32; r += 8) {
    const int64_t a = a0 + r, k = k0 + tx;
    if (a < N && k < ldt) out[a * ldt + k] = t[tx][r];
  }
}

crvq_status launch_gemm(tc::GemmArgs g, int64_t chunks, cudaStream_t stream) {
  static bool attr_set[64] = {};
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  if (dev < 64 && !attr_set[dev]) {
    CRVQ_CUDA(cudaFuncSetAttribute(tc::gemm3xtf32_kernel,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, tc::kSmemBytes));
    attr_set[dev] = true;
  }
  const int64_t tm = ceil_div(g.A.rows, tc::kBM), tn = ceil_div(g.B.rows, tc::kBN);
  g.tiles_n = (int)tn;
  dim3 grid((unsigned)(tm * tn), (unsigned)chunks);
  tc::gemm3xtf32_kernel<<<grid, tc::kThreads, tc::kSmemBytes, stream>>>(g);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace

// S = X^T X / n (X: n x N row-major) into S (N x N), both triangles, via split-K partials.
crvq_status launch_tc_syrk(const float* X, int64_t n, int64_t N, float* S, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const int64_t chunks = ceil_div(n, kKChunk);
  Scratch mem, xt_mem;
  float* P = S;
  if (chunks > 1) {
    CRVQ_TRY(mem.alloc((size_t)chunks * N * N * sizeof(float), stream));
    P = mem.as<float>();
  }
  // X^T with rows padded to a multiple of 4 floats: both operands K-major, loaded with 16-byte
  // loads (A(a, k) = X[k][a])
  const int64_t ldt = (n + 3) / 4 * 4;
  CRVQ_TRY(xt_mem.alloc((size_t)N * ldt * sizeof(float), stream));
  CRVQ_TRY(launch_transpose(X, n, N, xt_mem.as<float>(), ldt, stream));
  tc::GemmArgs g{};
  g.A = tc::Operand{xt_mem.as<float>(), ldt, N, true};
  g.B = g.A;
  g.K = n;
  g.k_chunk = kKChunk;
  g.c_chunk_stride = N * N;
  g.mode = tc::kStoreSymmetric;
  g.C = P;
  g.ldc = N;
  g.alpha = chunks > 1 ? 1.f : (float)(1.0 / (double)n);
  g.err = err;
  {
    ProfScope ps("hessian_gemm_tc", stream, 2.0 * (double)n * N * N);
    CRVQ_TRY(launch_gemm(g, chunks, stream));
  }
  if (chunks > 1) {
    ProfScope ps("hessian_sum_partials", stream, (double)chunks * N * N * 4.0);
    const int blocks = (int)std::min<int64_t>(ceil_div(N * N, 256), 16 * sm_count());
    sum_partials_kernel<<<blocks, 256, 0, stream>>>(P, N * N, (int)chunks, N * N,
                                                    (float)(1.0 / (double)n), S);
    CRVQ_LAUNCHED();
  }
  return CRVQ_OK;
}

// part[0 .. nparts) = partial sums of ||A B^T||_F^2 with A: M x K, B: Nb x K (row-major,
// leading dimension K); returns the number of partials written.
crvq_status launch_tc_sumsq(const float* A, int64_t M, const float* B, int64_t Nb, int64_t K,
                            double* part, int64_t part_cap, int64_t* nparts,
                            cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const int64_t chunks = ceil_div(K, kKChunk);
  Scratch mem;
  CRVQ_TRY(mem.alloc((size_t)chunks * M * Nb * sizeof(float), stream));
  float* P = mem.as<float>();
  tc::GemmArgs g{};
  g.A = tc::Operand{A, K, M, true};
  g.B = tc::Operand{B, K, Nb, true};
  g.K = K;
  g.k_chunk = kKChunk;
  g.c_chunk_stride = M * Nb;
  g.mode = tc::kStore;
  g.C = P;
  g.ldc = Nb;
  g.alpha = 1.f;
  g.err = err;
  {
    ProfScope ps("loss_gemm_tc", stream, 2.0 * (double)M * Nb * K);
    CRVQ_TRY(launch_gemm(g, chunks, stream));
  }
  const int blocks = (int)std::min<int64_t>(part_cap, std::min<int64_t>(
                                                          ceil_div(M * Nb, 256), 8 * sm_count()));
  ProfScope ps("loss_sumsq", stream, (double)chunks * M * Nb * 4.0);
  sumsq_partials_kernel<<<blocks, 256, 0, stream>>>(P, M * Nb, (int)chunks, M * Nb, part);
  CRVQ_LAUNCHED();
  *nparts = blocks;
  return CRVQ_OK;
}

crvq_status launch_transpose(const float* X, int64_t n, int64_t N, float* Xt, int64_t ldt,
                             cudaStream_t stream) {
  ProfScope ps("hessian_transpose", stream, 8.0 * (double)n * N);
  transpose_kernel<<<dim3((unsigned)ceil_div(ldt, 32), (unsigned)ceil_div(N, 32)), 256, 0,
                     stream>>>(X, n, N, Xt, ldt);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

// Diagonal 8 x 8 blocks of X^T X / n (+ delta I) for the channel order `perm` (NULL = the
// stored order), from Xt = X^T (N x ldt, ldt a multiple of 4). delta_known: delta64 (fp64) is
// read; otherwise perm must be NULL and xsq, delta (float, may be NULL) and delta64 are
// written. The entries equal those of launch_tc_syrk's dense S plus the damping bit for bit.
crvq_status launch_tc_hessian_blocks(const float* Xt, int64_t ldt, int64_t n, int64_t N,
                                     const int32_t* perm, bool delta_known, float damp_rel,
                                     float* xsq, float* delta, double* delta64, float* Hb,
                                     cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  static bool attr_set[64] = {};
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  if (dev < 64 && !attr_set[dev]) {
    CRVQ_CUDA(cudaFuncSetAttribute(tc::syrk_diag_kernel,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   tc::kDiagSmemBytes));
    attr_set[dev] = true;
  }
  const int64_t chunks = std::max<int64_t>(1, ceil_div(n, kKChunk));
  const int64_t stride = N * 8;
  Scratch mem;
  CRVQ_TRY(mem.alloc((size_t)chunks * stride * sizeof(float), stream));
  tc::DiagArgs a{};
  a.A = tc::Operand{Xt, ldt, N, true, perm};
  a.K = n;
  a.k_chunk = kKChunk;
  a.out = mem.as<float>();
  a.chunk_stride = stride;
  a.alpha = chunks > 1 ? 1.f : (float)(1.0 / (double)n);
  a.err = err;
  const float scale = chunks > 1 ? (float)(1.0 / (double)n) : 1.f;
  {
    ProfScope ps(perm ? "reorder_blocks_tc" : "hessian_blocks_tc", stream,
                 6.0 * (double)n * N * tc::kBM);
    dim3 grid((unsigned)ceil_div(N, tc::kBM), (unsigned)chunks);
    tc::syrk_diag_kernel<<<grid, tc::kThreads, tc::kDiagSmemBytes, stream>>>(a);
    CRVQ_LAUNCHED();
  }
  ProfScope ps("hessian_blocks_finalize", stream, (double)chunks * stride * 4.0);
  if (!delta_known) {
    if (perm) return fail(CRVQ_ERR_UNSUPPORTED, "hessian blocks: delta needs the stored order");
    blocks_finalize_kernel<<<1, 1024, 0, stream>>>(mem.as<float>(), (int)chunks, stride, scale,
                                                   N, damp_rel, xsq, delta, delta64, Hb);
  } else {
    const int blocks = (int)std::min<int64_t>(ceil_div(stride, 256), 4 * sm_count());
    blocks_damp_kernel<<<blocks, 256, 0, stream>>>(mem.as<float>(), (int)chunks, stride, scale,
                                                   N, delta64, Hb);
  }
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace crvq
