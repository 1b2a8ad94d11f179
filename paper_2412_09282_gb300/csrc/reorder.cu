// S3: channel importance (Sec. 4.1; App. A.2), the importance-order permutation and the
// column gather that makes the critical channels contiguous (Sec. 4.2, Fig. 2 left).
//
// importance: a column max over all rows, streamed with 128-bit loads (4 channels per thread),
//   reduced in shared memory and merged with an integer atomicMax on the (non-negative) float
//   bits, so the result does not depend on the order of arrival.
// ranking:    rank_i = #{j : I_j > I_i or (I_j == I_i and j < i)}; perm[rank_i] = i. An
//   O(N^2) count over shared-memory tiles (N <= 49152 channels), exact and deterministic.
// gather:     one CTA per row; the row is staged in shared memory with 128-bit loads and
//   written back in the new order with 128-bit stores.
#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

constexpr int kColThreads = 32;   // threads across columns (4 channels each) per CTA
constexpr int kRowThreads = 8;    // threads across rows per CTA

// Column max of |W - W_pre| (mode W-A) or |W| (W-only), as float bits.
__global__ void __launch_bounds__(kColThreads * kRowThreads)
colmax_kernel(const float* __restrict__ W, const float* __restrict__ W_pre, int64_t M,
              int64_t N, int64_t rows_per_block, unsigned* __restrict__ maxbits,
              unsigned* err) {
  __shared__ float part[kRowThreads][kColThreads * 4];
  const int cx = threadIdx.x % kColThreads, ry = threadIdx.x / kColThreads;
  const int64_t c0 = ((int64_t)blockIdx.x * kColThreads + cx) * 4;
  const int64_t r_begin = (int64_t)blockIdx.y * rows_per_block;
  const int64_t r_end = min(M, r_begin + rows_per_block);
  float m0 = 0.f, m1 = 0.f, m2 = 0.f, m3 = 0.f;
  bool finite = true;
  if (c0 < N) {
    for (int64_t r = r_begin + ry; r < r_end; r += kRowThreads) {
      float4 w = *reinterpret_cast<const float4*>(W + r * N + c0);
      if (W_pre) {
        const float4 p = *reinterpret_cast<const float4*>(W_pre + r * N + c0);
        w.x -= p.x; w.y -= p.y; w.z -= p.z; w.w -= p.w;
      }
      finite = finite && isfinite(w.x) && isfinite(w.y) && isfinite(w.z) && isfinite(w.w);
      m0 = fmaxf(m0, fabsf(w.x));
      m1 = fmaxf(m1, fabsf(w.y));
      m2 = fmaxf(m2, fabsf(w.z));
      m3 = fmaxf(m3, fabsf(w.w));
    }
  }
  if (!finite) raise_error(err, ERRBIT_NUMERIC);
  part[ry][cx * 4 + 0] = m0;
  part[ry][cx * 4 + 1] = m1;
  part[ry][cx * 4 + 2] = m2;
  part[ry][cx * 4 + 3] = m3;
  __syncthreads();
  if (ry == 0 && c0 < N) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float m = part[0][cx * 4 + q];
      for (int y = 1; y < kRowThreads; ++y) m = fmaxf(m, part[y][cx * 4 + q]);
      atomicMax(&maxbits[c0 + q], __float_as_uint(m));
    }
  }
}

__global__ void importance_kernel(const unsigned* __restrict__ maxbits,
                                  const float* __restrict__ xsq,
                                  const double* __restrict__ hinv, int64_t N, int mode,
                                  uint64_t seed, float* __restrict__ I) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < N;
       i += (int64_t)gridDim.x * blockDim.x) {
    float v;
    if (mode == CRVQ_IMPORTANCE_RANDOM) {
      v = (float)(splitmix64(seed, (uint64_t)i) >> 40) * 5.9604645e-08f;  // 24 bits * 2^-24
    } else if (mode == CRVQ_IMPORTANCE_WA_INV) {
      // Eq. (wa): max_j dw_ji^2 / (2 [H^-1]_ii), in fp64, rounded once
      const double m = (double)__uint_as_float(maxbits[i]);
      v = (float)(m * m / (2.0 * hinv[i]));
    } else {
      const float m = __uint_as_float(maxbits[i]);
      v = m * m;
      if (mode == CRVQ_IMPORTANCE_WA) v = (0.5f * xsq[i]) * v;
    }
    I[i] = v;
  }
}

// perm[rank(i)] = i, rank(i) = #{j : I_j > I_i or (I_j == I_i and j < i)} (descending order,
// ties to the smaller index). One warp per channel: the lanes count over j, a warp sum.
__global__ void __launch_bounds__(256)
rank_kernel(const float* __restrict__ I, int64_t N, int32_t* __restrict__ perm) {
  const int lane = threadIdx.x & 31;
  const int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (i >= N) return;  // whole warps
  const float Ii = I[i];
  int rank = 0;
  for (int64_t j = lane; j < N; j += 32) {
    const float Ij = I[j];
    rank += (Ij > Ii) || (Ij == Ii && j < i);
  }
  rank = __reduce_add_sync(0xffffffffu, rank);
  if (lane == 0) perm[rank] = (int32_t)i;
}

__global__ void __launch_bounds__(256)
gather_cols_kernel(const float* __restrict__ W, int64_t M, int64_t N,
                   const int32_t* __restrict__ perm, float* __restrict__ Ws, unsigned* err) {
  extern __shared__ __align__(16) float row[];
  for (int64_t r = blockIdx.x; r < M; r += gridDim.x) {
    __syncthreads();
    const float* src = W + r * N;
    for (int64_t c = (int64_t)threadIdx.x * 4; c < N; c += (int64_t)blockDim.x * 4)
      *reinterpret_cast<float4*>(row + c) = *reinterpret_cast<const float4*>(src + c);
    __syncthreads();
    float* dst = Ws + r * N;
    for (int64_t c = (int64_t)threadIdx.x * 4; c < N; c += (int64_t)blockDim.x * 4) {
      float v[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int32_t p = perm[c + q];
        if (p < 0 || p >= N) {
          raise_error(err, ERRBIT_INDEX);
          v[q] = 0.f;
        } else {
          v[q] = row[p];
        }
      }
      *reinterpret_cast<float4*>(dst + c) = make_float4(v[0], v[1], v[2], v[3]);
    }
  }
}

}  // namespace

crvq_status launch_select_reorder(const float* W, int64_t M, int64_t N, int d,
                                  const float* W_pre, const float* xsq, const float* H,
                                  int mode, uint64_t seed, int32_t* perm, float* importance,
                                  float* W_sorted, float* H_blocks, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const int nsm = sm_count();
  Scratch mem, mh;
  CRVQ_TRY(mem.alloc((size_t)N * (sizeof(unsigned) + sizeof(float)), stream));
  unsigned* maxbits = mem.as<unsigned>();
  float* I = importance ? importance : reinterpret_cast<float*>(maxbits + N);
  double* hinv = nullptr;
  if (mode == CRVQ_IMPORTANCE_WA_INV) {
    CRVQ_TRY(mh.alloc((size_t)N * sizeof(double), stream));
    hinv = mh.as<double>();
    CRVQ_TRY(launch_hinv_diag(H, N, hinv, stream));
  }
  const bool with_pre = mode == CRVQ_IMPORTANCE_WA || mode == CRVQ_IMPORTANCE_WA_INV;
  if (mode != CRVQ_IMPORTANCE_RANDOM) {
    CRVQ_CUDA(cudaMemsetAsync(maxbits, 0, (size_t)N * sizeof(unsigned), stream));
    const int64_t col_blocks = ceil_div(N, kColThreads * 4);
    // enough row blocks to cover ~4 CTAs per SM
    int64_t row_blocks = std::max<int64_t>(1, (4 * nsm + col_blocks - 1) / col_blocks);
    row_blocks = std::min<int64_t>(row_blocks, ceil_div(M, kRowThreads));
    const int64_t rows_per = ceil_div(M, row_blocks);
    dim3 grid((unsigned)col_blocks, (unsigned)ceil_div(M, rows_per));
    ProfScope ps("reorder_colmax", stream, (double)M * N * 4.0 * (with_pre ? 2.0 : 1.0));
    colmax_kernel<<<grid, kColThreads * kRowThreads, 0, stream>>>(
        W, with_pre ? W_pre : nullptr, M, N, rows_per, maxbits, err);
    CRVQ_LAUNCHED();
  }
  importance_kernel<<<(unsigned)ceil_div(N, 256), 256, 0, stream>>>(maxbits, xsq, hinv, N, mode,
                                                                     seed, I);
  CRVQ_LAUNCHED();
  {
    ProfScope ps("reorder_rank", stream, (double)N * N);
    rank_kernel<<<(unsigned)ceil_div(N, 8), 256, 0, stream>>>(I, N, perm);
    CRVQ_LAUNCHED();
  }
  {
    ProfScope ps("reorder_gather", stream, (double)M * N * 8.0);
    CRVQ_TRY(launch_gather_cols(W, M, N, perm, W_sorted, stream));
  }
  if (H_blocks) CRVQ_TRY(launch_extract_blocks(H, N, d, perm, H_blocks, stream));
  return CRVQ_OK;
}

crvq_status launch_gather_cols(const float* src, int64_t M, int64_t N, const int32_t* idx,
                               float* dst, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const size_t smem = (size_t)N * sizeof(float);
  if (smem > 48 * 1024)
    CRVQ_CUDA(cudaFuncSetAttribute(gather_cols_kernel,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  const int blocks = (int)std::min<int64_t>(M, (int64_t)8 * sm_count());
  gather_cols_kernel<<<blocks, 256, smem, stream>>>(src, M, N, idx, dst, err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace crvq
