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

// Reconstruction of vector (i, g): the sum of the covering codebooks' codewords (codebook
// order), correctly rounded to fp32 like the fp64 sum rounded once. With at most two terms the
// fp32 sum is that value (the exact sum of two fp32 values rounds to fp32 the same way
// whether or not it first passes through fp64); three or more terms are summed in fp64.
__device__ __forceinline__ void recon(const CbList& cbs, int64_t i, int64_t g, float r[kD],
                                      unsigned* err) {
  const float* cw[kMaxCodebooks];
  int n = 0;
  for (int s = 0; s < cbs.n; ++s) {
    const CbView& cb = cbs.cb[s];
    if (g >= cb.G_cov) continue;
    const int32_t k = cb.codes[i * cb.ld + g];
    if (k < 0 || k >= cb.K) {
      raise_error(err, ERRBIT_INDEX);
      continue;
    }
    cw[n++] = cb.C + (int64_t)k * kD;
  }
  if (n <= 2) {
#pragma unroll
    for (int j = 0; j < kD; ++j) r[j] = 0.f;
    for (int q = 0; q < n; ++q) {
      const float4 a = *reinterpret_cast<const float4*>(cw[q]);
      const float4 b = *reinterpret_cast<const float4*>(cw[q] + 4);
      r[0] += a.x; r[1] += a.y; r[2] += a.z; r[3] += a.w;
      r[4] += b.x; r[5] += b.y; r[6] += b.z; r[7] += b.w;
    }
  } else {
    double d[kD];
#pragma unroll
    for (int j = 0; j < kD; ++j) d[j] = 0.0;
    for (int q = 0; q < n; ++q)
#pragma unroll
      for (int j = 0; j < kD; ++j) d[j] += (double)cw[q][j];
#pragma unroll
    for (int j = 0; j < kD; ++j) r[j] = (float)d[j];
  }
}

// Unevaluated fp32 pair (h, l) += x, and the merge of two pairs (TwoSum of the high parts).
__device__ __forceinline__ void pair_add(float& h, float& l, float x) {
  const float s = __fadd_rn(h, x);
  const float bp = __fsub_rn(s, h);
  const float e = __fadd_rn(__fsub_rn(h, __fsub_rn(s, bp)), __fsub_rn(x, bp));
  h = s;
  l = __fadd_rn(l, e);
}

__device__ __forceinline__ void pair_merge(float& h, float& l, float oh, float ol) {
  pair_add(h, l, oh);
  l = __fadd_rn(l, ol);
}

// One CTA per row (grid-strided): the row of W_hat and of dW = W - W_hat in the original
// channel order (staged in shared memory, then stored with 16-byte writes), and the row's
// block loss, critical loss and ||dW||^2. Each vector's terms are fp32 (the quadratic form as
// two FMA chains); the thread's running sums and the row reduction are fp32 pairs in a fixed
// order (about 2^-44 relative; a chain of dependent fp64 additions would cost about 180
// cycles per step on this part), rounded to fp64 once per row.
__global__ void __launch_bounds__(256)
decode_row_kernel(const float* __restrict__ Ws, int64_t M, int64_t N, const float* __restrict__ Hb,
                  const int32_t* __restrict__ perm, CbList cbs, int64_t n_crit_groups,
                  float* __restrict__ W_hat, float* __restrict__ dW,
                  double* __restrict__ row_part, unsigned* err) {
  extern __shared__ __align__(16) float srow[];  // [N] W_hat row (if any), then [N] dW row
  float* s_hat = srow;
  float* s_dw = srow + (W_hat ? N : 0);
  __shared__ float red_h[3][256 / 32], red_l[3][256 / 32];
  const int64_t G = N / kD;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int64_t i = blockIdx.x; i < M; i += gridDim.x) {
    float lb = 0.f, lbl = 0.f, lc = 0.f, lcl = 0.f, sq = 0.f, sql = 0.f;
    __syncthreads();  // the previous row's stores have read the staging rows
    for (int64_t g = threadIdx.x; g < G; g += blockDim.x) {
      float r[kD], t[kD], dl[kD];
      recon(cbs, i, g, r, err);
      const float4 t0 = *reinterpret_cast<const float4*>(Ws + i * N + g * kD);
      const float4 t1 = *reinterpret_cast<const float4*>(Ws + i * N + g * kD + 4);
      t[0] = t0.x; t[1] = t0.y; t[2] = t0.z; t[3] = t0.w;
      t[4] = t1.x; t[5] = t1.y; t[6] = t1.z; t[7] = t1.w;
      float q2 = 0.f;
#pragma unroll
      for (int j = 0; j < kD; ++j) {
        dl[j] = t[j] - r[j];
        q2 = fmaf(dl[j], dl[j], q2);
      }
      const float4* H4 = reinterpret_cast<const float4*>(Hb + g * kD * kD);
      float e = 0.f;
#pragma unroll
      for (int a = 0; a < kD; ++a) {
        const float4 h0 = __ldg(H4 + 2 * a), h1 = __ldg(H4 + 2 * a + 1);
        float hb = dl[0] * h0.x;
        hb = fmaf(dl[1], h0.y, hb);
        hb = fmaf(dl[2], h0.z, hb);
        hb = fmaf(dl[3], h0.w, hb);
        hb = fmaf(dl[4], h1.x, hb);
        hb = fmaf(dl[5], h1.y, hb);
        hb = fmaf(dl[6], h1.z, hb);
        hb = fmaf(dl[7], h1.w, hb);
        e = fmaf(hb, dl[a], e);
      }
      pair_add(lb, lbl, e);
      if (g < n_crit_groups) pair_add(lc, lcl, e);
      pair_add(sq, sql, q2);
#pragma unroll
      for (int j = 0; j < kD; ++j) {
        const int64_t p = g * kD + j;
        const int64_t col = perm ? perm[p] : p;
        if (col < 0 || col >= N) {
          raise_error(err, ERRBIT_INDEX);
          continue;
        }
        if (W_hat) s_hat[col] = r[j];
        if (dW) s_dw[col] = dl[j];
      }
    }
    __syncthreads();
    {
      if (W_hat) {
        float* dst = W_hat + i * N;
        for (int64_t c = (int64_t)threadIdx.x * 4; c < N; c += (int64_t)blockDim.x * 4)
          *reinterpret_cast<float4*>(dst + c) = *reinterpret_cast<const float4*>(s_hat + c);
      }
      if (dW) {
        float* dd = dW + i * N;
        for (int64_t c = (int64_t)threadIdx.x * 4; c < N; c += (int64_t)blockDim.x * 4)
          *reinterpret_cast<float4*>(dd + c) = *reinterpret_cast<const float4*>(s_dw + c);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float a0 = __shfl_xor_sync(0xffffffffu, lb, off);
      const float a1 = __shfl_xor_sync(0xffffffffu, lbl, off);
      const float b0 = __shfl_xor_sync(0xffffffffu, lc, off);
      const float b1 = __shfl_xor_sync(0xffffffffu, lcl, off);
      const float c0 = __shfl_xor_sync(0xffffffffu, sq, off);
      const float c1 = __shfl_xor_sync(0xffffffffu, sql, off);
      pair_merge(lb, lbl, a0, a1);
      pair_merge(lc, lcl, b0, b1);
      pair_merge(sq, sql, c0, c1);
    }
    if (lane == 0) {
      red_h[0][warp] = lb;
      red_l[0][warp] = lbl;
      red_h[1][warp] = lc;
      red_l[1][warp] = lcl;
      red_h[2][warp] = sq;
      red_l[2][warp] = sql;
    }
    __syncthreads();
    if (threadIdx.x < 3) {
      const int q = threadIdx.x;
      float h = red_h[q][0], l = red_l[q][0];
      for (int w = 1; w < (int)(blockDim.x >> 5); ++w) pair_merge(h, l, red_h[q][w], red_l[q][w]);
      row_part[i * 3 + q] = (double)h + (double)l;
    }
  }
}

// One CTA of 1024 threads (short dependent fp64 chains: strided partials, then a tree).
__global__ void __launch_bounds__(1024)
finalize_losses_kernel(const double* __restrict__ row_part, int64_t M,
                       const double* __restrict__ gemm_part, int64_t n_gemm, int64_t n_tok,
                       double delta_host, const float* __restrict__ delta_dev,
                       double* __restrict__ losses) {
  __shared__ double red[4][1024];
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
  for (int w = 512; w > 0; w >>= 1) {
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
  // partial sums of the full loss: one per 128 x 256 tile of dW X^T
  const int64_t n_gemm_cap = X ? ceil_div(M, (int64_t)128) * ceil_div(n_tok, (int64_t)256) : 0;
  int64_t n_gemm = 0;
  // Scratch: dW (16-byte aligned for the 128-bit stores), then the fp64 partial sums.
  const size_t dW_bytes = X ? align_up((size_t)M * N * sizeof(float), 256) : 0;
  const size_t part_bytes = (size_t)M * 3 * sizeof(double) + (size_t)(n_gemm_cap + 1) * sizeof(double);
  Scratch mem;
  CRVQ_TRY(mem.alloc(dW_bytes + part_bytes, stream));
  float* dW = X ? mem.as<float>() : nullptr;
  double* row_part = reinterpret_cast<double*>(mem.as<char>() + dW_bytes);
  double* gemm_part = row_part + M * 3;
  const size_t smem = (size_t)N * sizeof(float) * ((W_hat ? 1 : 0) + (dW ? 1 : 0));
  if (smem > (size_t)227 * 1024)
    return fail(CRVQ_ERR_UNSUPPORTED,
                "crvq_reconstruct_error: N = %lld channels need %zu bytes of shared memory per "
                "row (227 KB available)", (long long)N, smem);
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
  finalize_losses_kernel<<<1, 1024, 0, stream>>>(row_part, M, X ? gemm_part : nullptr, n_gemm,
                                                n_tok, damp_delta, delta_dev, losses_dev);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace crvq
