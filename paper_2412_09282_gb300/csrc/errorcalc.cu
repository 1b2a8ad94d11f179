// S7: reconstruction W_enc (sum of the covering codebooks' codewords), the reverse reorder
// to the original channel order (Sec. 4.3) and the losses of Alg. 1 (QuantLoss):
//   loss_block = sum_v (t_v - r_v)^T H_g (t_v - r_v)       (block-diagonal part)
//   loss_crit  = the same over the critical groups g < G_c
//   loss_full  = ||dW X^T||^2 / n + delta ||dW||^2 = tr(dW H dW^T)   (dW in original order)
// Per-row partial sums are fp64 and reduced in a fixed order; the full loss forms dW X^T on the
// tensor cores (tc_gemm.cuh: tcgen05, 3xTF32, split K) and squares and sums it in fp64.
#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

// Reconstruction of vector (i, g) in fp64 (sum in codebook order), as fp32 values.
__device__ __forceinline__ void recon(const CbList& cbs, int64_t i, int64_t g, double r[kD],
                                      unsigned* err) {
#pragma unroll
  for (int j = 0; j < kD; ++j) r[j] = 0.0;
  for (int s = 0; s < cbs.n; ++s) {
    const CbView& cb = cbs.cb[s];
    if (g >= cb.G_cov) continue;
    const int32_t k = cb.codes[i * cb.ld + g];
    if (k < 0 || k >= cb.K) {
      raise_error(err, ERRBIT_INDEX);
      continue;
    }
    const float* c = cb.C + (int64_t)k * kD;
#pragma unroll
    for (int j = 0; j < kD; ++j) r[j] += (double)c[j];
  }
}

// One CTA per row: block/critical losses and ||dW||^2 of the row (fp64 partials), and the row
// of W_hat and of dW in the original channel order (staged in shared memory).
__global__ void __launch_bounds__(256)
decode_row_kernel(const float* __restrict__ Ws, int64_t M, int64_t N, const float* __restrict__ Hb,
                  const int32_t* __restrict__ perm, CbList cbs, int64_t n_crit_groups,
                  float* __restrict__ W_hat, float* __restrict__ dW,
                  double* __restrict__ row_part, unsigned* err) {
  extern __shared__ __align__(16) float srow[];
  __shared__ double red[3][256];
  const int64_t G = N / kD;
  for (int64_t i = blockIdx.x; i < M; i += gridDim.x) {
    double lb = 0.0, lc = 0.0, sq = 0.0;
    for (int pass = 0; pass < 2; ++pass) {
      float* out = pass == 0 ? W_hat : dW;
      if (pass == 1 && !dW) break;
      __syncthreads();
      for (int64_t g = threadIdx.x; g < G; g += blockDim.x) {
        double r[kD];
        recon(cbs, i, g, r, err);
        const float* t = Ws + i * N + g * kD;
        float dl[kD];
#pragma unroll
        for (int j = 0; j < kD; ++j) dl[j] = (float)((double)t[j] - r[j]);
        if (pass == 0) {
          const float* H = Hb + g * kD * kD;
          float e = 0.f;
#pragma unroll
          for (int b = 0; b < kD; ++b) {
            float hb = 0.f;
#pragma unroll
            for (int a = 0; a < kD; ++a) hb = fmaf(dl[a], H[a * kD + b], hb);
            e = fmaf(hb, dl[b], e);
          }
          lb += (double)e;
          if (g < n_crit_groups) lc += (double)e;
#pragma unroll
          for (int j = 0; j < kD; ++j) sq += (double)dl[j] * (double)dl[j];
        }
        if (out) {
#pragma unroll
          for (int j = 0; j < kD; ++j) {
            const int64_t p = g * kD + j;
            int64_t col = perm ? perm[p] : p;
            if (col < 0 || col >= N) {
              raise_error(err, ERRBIT_INDEX);
              continue;
            }
            srow[col] = pass == 0 ? (float)r[j] : dl[j];
          }
        }
      }
      __syncthreads();
      if (out) {
        float* dst = out + i * N;
        for (int64_t c = (int64_t)threadIdx.x * 4; c < N; c += (int64_t)blockDim.x * 4)
          *reinterpret_cast<float4*>(dst + c) = *reinterpret_cast<const float4*>(srow + c);
      }
    }
    red[0][threadIdx.x] = lb;
    red[1][threadIdx.x] = lc;
    red[2][threadIdx.x] = sq;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
      if ((int)threadIdx.x < w) {
#pragma unroll
        for (int q = 0; q < 3; ++q) red[q][threadIdx.x] += red[q][threadIdx.x + w];
      }
      __syncthreads();
    }
    if (threadIdx.x == 0) {
      row_part[i * 3 + 0] = red[0][0];
      row_part[i * 3 + 1] = red[1][0];
      row_part[i * 3 + 2] = red[2][0];
    }
  }
}

__global__ void __launch_bounds__(256)
finalize_losses_kernel(const double* __restrict__ row_part, int64_t M,
                       const double* __restrict__ gemm_part, int64_t n_gemm, int64_t n_tok,
                       double delta_host, const float* __restrict__ delta_dev,
                       double* __restrict__ losses) {
  __shared__ double red[4][256];
  double a = 0, b = 0, c = 0, e = 0;
  for (int64_t i = threadIdx.x; i < M; i += blockDim.x) {
    a += row_part[i * 3 + 0];
    b += row_part[i * 3 + 1];
    c += row_part[i * 3 + 2];
  }
  for (int64_t i = threadIdx.x; i < n_gemm; i += blockDim.x) e += gemm_part[i];
  red[0][threadIdx.x] = a;
  red[1][threadIdx.x] = b;
  red[2][threadIdx.x] = c;
  red[3][threadIdx.x] = e;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w)
      for (int q = 0; q < 4; ++q) red[q][threadIdx.x] += red[q][threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    losses[0] = red[0][0];
    losses[1] = red[1][0];
    if (gemm_part) {
      const double delta = delta_dev ? (double)*delta_dev : delta_host;
      losses[2] = red[3][0] / (double)n_tok + delta * red[2][0];
    } else {
      losses[2] = __longlong_as_double(0x7ff8000000000000ll);  // NaN: no X given
    }
  }
}

}  // namespace

crvq_status launch_reconstruct_error(const float* W_sorted, int64_t M, int64_t N,
                                     const float* Hb, const int32_t* perm, const CbList& cbs,
                                     int64_t n_crit_groups, const float* X, int64_t n_tok,
                                     double damp_delta, const float* delta_dev, float* W_hat,
                                     double* losses_dev, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const int nsm = sm_count();
  const int64_t n_gemm_cap = X ? 8 * (int64_t)nsm : 0;  // partial sums of the full loss
  int64_t n_gemm = 0;
  // Scratch: dW (16-byte aligned for the 128-bit stores), then the fp64 partial sums.
  const size_t dW_bytes = X ? align_up((size_t)M * N * sizeof(float), 256) : 0;
  const size_t part_bytes = (size_t)M * 3 * sizeof(double) + (size_t)(n_gemm_cap + 1) * sizeof(double);
  Scratch mem;
  CRVQ_TRY(mem.alloc(dW_bytes + part_bytes, stream));
  float* dW = X ? mem.as<float>() : nullptr;
  double* row_part = reinterpret_cast<double*>(mem.as<char>() + dW_bytes);
  double* gemm_part = row_part + M * 3;
  const size_t smem = (size_t)N * sizeof(float);
  if (smem > 48 * 1024)
    CRVQ_CUDA(cudaFuncSetAttribute(decode_row_kernel,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  const int blocks = (int)std::min<int64_t>(M, (int64_t)8 * nsm);
  {
  ProfScope ps("decode_rows", stream,
               (double)M * N * 4.0 * (1.0 + (W_hat ? 1.0 : 0.0) + (X ? 1.0 : 0.0)));
  decode_row_kernel<<<blocks, 256, smem, stream>>>(W_sorted, M, N, Hb, perm, cbs,
                                                   n_crit_groups, W_hat, dW, row_part, err);
  CRVQ_LAUNCHED();
  }
  if (X) {
    CRVQ_TRY(launch_tc_sumsq(dW, M, X, n_tok, N, gemm_part, n_gemm_cap, &n_gemm, stream));
  }
  finalize_losses_kernel<<<1, 256, 0, stream>>>(row_part, M, X ? gemm_part : nullptr, n_gemm,
                                                n_tok, damp_delta, delta_dev, losses_dev);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace crvq
