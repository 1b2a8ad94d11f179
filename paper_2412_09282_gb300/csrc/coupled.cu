// Code search under the full Alg. 1 loss (QuantLoss ||W X - W_enc X||^2 = tr(dW H dW^T)), with
// the cross-group terms that the block-diagonal search leaves out: a Gauss-Seidel sweep over
// the groups of one codebook, the others fixed (Sec. 3.1 codes; Alg. 1 QuantLoss).
//
// The loss separates over rows. For row i and group g, with every other group fixed,
//   L = D_g^T H_gg D_g + 2 D_g^T b_g + const,  b_g = sum_{g' != g} H_gg' D_g',  D = W - W_enc,
// and with D_g = t - c (t: the row segment minus the other codebooks' codewords) completing the
// square makes the best codeword the block-diagonal arg-min for the shifted target
//   t' = t + H_gg^-1 b_g,
// so each group step is the certified tensor-core arg-min of the encode path on t'. Groups are
// visited in order, each with the current codes of the others, so the loss never rises.
//
// Blocked (lazy) evaluation of b_g: the channels are taken in blocks of 256 (32 groups). At
// the start of a block one tensor-core product gives B^T = H[block rows, :] D^T for the current
// D (256 x M); inside the block each group step adds its change dD_g H[g, g'] to the columns of
// the later groups g' of the block, and later blocks see the new D through their own product.
// Every b_g therefore includes every earlier decision of the sweep, as the sequential
// definition requires, with one product of 2 M N^2 flops per sweep in total. D_g is
// recomputed from W after each decision (fp64 sum of the codewords, rounded once), so it does
// not drift.
#include <algorithm>
#include <vector>

#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

constexpr int kBlockCols = 256;                 // channels per lazy block (32 groups)
constexpr int kBlockG = kBlockCols / kD;

// D = W - sum over the covering codebooks of C[code] (fp64 sum, rounded once), M x N.
__global__ void __launch_bounds__(256)
residual_kernel(const float* __restrict__ W, int64_t M, int64_t N, CbList cbs,
                float* __restrict__ D, unsigned* err) {
  const int64_t G = N / kD;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < M * G;
       v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = v / G, g = v % G;
    double r[kD];
#pragma unroll
    for (int j = 0; j < kD; ++j) r[j] = (double)W[i * N + g * kD + j];
    for (int s = 0; s < cbs.n; ++s) {
      const CbView& cb = cbs.cb[s];
      if (g >= cb.G_cov) continue;
      const int32_t k = cb.codes[i * cb.ld + g];
      if (k < 0 || k >= cb.K) {
        raise_error(err, ERRBIT_INDEX);
        continue;
      }
#pragma unroll
      for (int j = 0; j < kD; ++j) r[j] -= (double)cb.C[(int64_t)k * kD + j];
    }
#pragma unroll
    for (int j = 0; j < kD; ++j) D[i * N + g * kD + j] = (float)r[j];
  }
}

// Per group g < G_cov: the diagonal block H_gg of H (N x N) into Hb[g] (the arg-min's Hessian
// block) and its Cholesky factor, computed in fp64 and stored in fp32 (lower triangle, row
// major) with the reciprocals of its diagonal. One thread per group; a block without a factor
// reports ERRBIT_NUMERIC and gets a zero factor (its shifted targets are then not formed).
__global__ void __launch_bounds__(128)
block_factor_kernel(const float* __restrict__ H, int64_t N, int64_t G_cov,
                    float* __restrict__ Hb, float* __restrict__ Lf, float* __restrict__ Linv,
                    unsigned* err) {
  const int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (g >= G_cov) return;
  double L[kD * kD];
  bool ok = true;
  for (int r = 0; r < kD && ok; ++r)
    for (int c = 0; c <= r; ++c) {
      double sum = (double)H[(g * kD + r) * N + g * kD + c];
      for (int m = 0; m < c; ++m) sum -= L[r * kD + m] * L[c * kD + m];
      if (r == c) {
        if (!(sum > 0.0)) {
          ok = false;
          break;
        }
        L[r * kD + r] = sqrt(sum);
      } else {
        L[r * kD + c] = sum / L[c * kD + c];
      }
    }
  if (!ok) raise_error(err, ERRBIT_NUMERIC);
  for (int r = 0; r < kD; ++r) {
    for (int c = 0; c < kD; ++c) {
      Hb[g * kD * kD + r * kD + c] = H[(g * kD + r) * N + g * kD + c];
      Lf[g * kD * kD + r * kD + c] = (ok && c <= r) ? (float)L[r * kD + c] : 0.f;
    }
    Linv[g * kD + r] = ok ? (float)(1.0 / L[r * kD + r]) : 0.f;
  }
}

// Shifted targets of group g: T'[i] = t + H_gg^-1 b_g with t = D_g + C[code_g] and
// b_g = B^T[col(g)][i] - H_gg D_g (the product at the block start plus the block's earlier
// changes, without the group's own block); the solve is a forward and a back substitution in
// fp32 with the group's factor.
__global__ void __launch_bounds__(256)
coupled_target_kernel(const float* __restrict__ D, int64_t M, int64_t N,
                      const float* __restrict__ Hb, const float* __restrict__ Lf,
                      const float* __restrict__ Linv, const float* __restrict__ Bt, int64_t ldb,
                      int col0, int64_t g, CbView cw, float* __restrict__ Tp, unsigned* err) {
  __shared__ float sH[kD * kD], sL[kD * kD], sInv[kD];
  if (threadIdx.x < kD * kD) {
    sH[threadIdx.x] = Hb[g * kD * kD + threadIdx.x];
    sL[threadIdx.x] = Lf[g * kD * kD + threadIdx.x];
  }
  if (threadIdx.x < kD) sInv[threadIdx.x] = Linv[g * kD + threadIdx.x];
  __syncthreads();
  if (sInv[0] == 0.f) return;  // no factor (reported)
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < M;
       i += (int64_t)gridDim.x * blockDim.x) {
    float dg[kD], b[kD];
#pragma unroll
    for (int j = 0; j < kD; ++j) dg[j] = D[i * N + g * kD + j];
#pragma unroll
    for (int a = 0; a < kD; ++a) {
      float hd = 0.f;
#pragma unroll
      for (int c = 0; c < kD; ++c) hd = fmaf(sH[a * kD + c], dg[c], hd);
      b[a] = Bt[(int64_t)(col0 + a) * ldb + i] - hd;
    }
    // H_gg s = b: L y = b, L^T s = y
    float y[kD], sv[kD];
#pragma unroll
    for (int r = 0; r < kD; ++r) {
      float acc = b[r];
#pragma unroll
      for (int m = 0; m < r; ++m) acc = fmaf(-sL[r * kD + m], y[m], acc);
      y[r] = acc * sInv[r];
    }
#pragma unroll
    for (int r = kD - 1; r >= 0; --r) {
      float acc = y[r];
#pragma unroll
      for (int m = r + 1; m < kD; ++m) acc = fmaf(-sL[m * kD + r], sv[m], acc);
      sv[r] = acc * sInv[r];
    }
    const int32_t k = cw.codes[i * cw.ld + g];
    const bool kok = k >= 0 && k < cw.K;
    if (!kok) raise_error(err, ERRBIT_INDEX);
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      const float c = kok ? cw.C[(int64_t)k * kD + j] : 0.f;
      Tp[i * kD + j] = (dg[j] + c) + sv[j];
    }
  }
}

// Applies the decision of group g: the new code, D_g recomputed from W (fp64 sum, rounded
// once), and its change dD_g H[g, g'] added to the columns of the later groups of the block.
__global__ void __launch_bounds__(256)
coupled_apply_kernel(const float* __restrict__ W, float* __restrict__ D, int64_t M, int64_t N,
                     const float* __restrict__ H, float* __restrict__ Bt, int64_t ldb,
                     int col_next, int col_end, int64_t g, CbList cbs, int which,
                     const int32_t* __restrict__ new_code, unsigned* err) {
  __shared__ float sHr[kBlockCols][kD];  // H[g d + a][channel of column col], col in the block
  const int ncol = col_end - col_next;
  for (int e = threadIdx.x; e < ncol * kD; e += blockDim.x) {
    const int c = e / kD, a = e % kD;
    sHr[c][a] = H[(g * kD + a) * N + (g + 1) * kD + c];
  }
  __syncthreads();
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < M;
       i += (int64_t)gridDim.x * blockDim.x) {
    const CbView& cw = cbs.cb[which];
    const int32_t kn = new_code[i];
    if (kn < 0 || kn >= cw.K) {
      raise_error(err, ERRBIT_INDEX);
      continue;
    }
    cw.codes[i * cw.ld + g] = kn;
    double r[kD];
#pragma unroll
    for (int j = 0; j < kD; ++j) r[j] = (double)W[i * N + g * kD + j];
    for (int s = 0; s < cbs.n; ++s) {
      const CbView& cb = cbs.cb[s];
      if (g >= cb.G_cov) continue;
      const int32_t k = s == which ? kn : cb.codes[i * cb.ld + g];
      if (k < 0 || k >= cb.K) {
        raise_error(err, ERRBIT_INDEX);
        continue;
      }
#pragma unroll
      for (int j = 0; j < kD; ++j) r[j] -= (double)cb.C[(int64_t)k * kD + j];
    }
    float dd[kD];
    bool changed = false;
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      const float nv = (float)r[j];
      dd[j] = nv - D[i * N + g * kD + j];
      changed |= dd[j] != 0.f;
      D[i * N + g * kD + j] = nv;
    }
    if (!changed) continue;
    for (int c = 0; c < ncol; ++c) {
      float acc = Bt[(int64_t)(col_next + c) * ldb + i];
#pragma unroll
      for (int a = 0; a < kD; ++a) acc = fmaf(dd[a], sHr[c][a], acc);
      Bt[(int64_t)(col_next + c) * ldb + i] = acc;
    }
  }
}

// sum_i sum_n Bt[n][i] D[i][c0 + n] over the block's columns (fp64 per thread, fixed order),
// into part[blockIdx.x].
__global__ void __launch_bounds__(256)
block_loss_kernel(const float* __restrict__ Bt, int64_t ldb, int ncols,
                  const float* __restrict__ D, int64_t M, int64_t N, int64_t c0,
                  double* __restrict__ part) {
  __shared__ double red[256];
  double s = 0.0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < M;
       i += (int64_t)gridDim.x * blockDim.x)
    for (int c = 0; c < ncols; ++c)
      s += (double)Bt[(int64_t)c * ldb + i] * (double)D[i * N + c0 + c];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) part[blockIdx.x] += red[0];
}

__global__ void sum_parts_kernel(const double* __restrict__ part, int n, double* out) {
  double s = 0.0;
  for (int q = 0; q < n; ++q) s += part[q];
  *out = s;
}

}  // namespace

crvq_status launch_coupled_sweep(const float* W, int64_t M, int64_t N, const float* H,
                                 const CbList& cbs_in, int which, int sweeps, double* loss_dev,
                                 cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const int nsm = sm_count();
  CbList cbs = cbs_in;
  const CbView cw = cbs.cb[which];
  const int64_t G_cov = cw.G_cov;
  const unsigned row_blocks = (unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(M, 256),
                                                                                4 * nsm));
  const int loss_blocks = (int)std::min<int64_t>(std::max<int64_t>(1, ceil_div(M, 256)), 2 * nsm);
  Scratch mD, mB, mT, mK, mW, mP, mF;
  CRVQ_TRY(mD.alloc((size_t)M * N * sizeof(float), stream));
  CRVQ_TRY(mB.alloc((size_t)kBlockCols * M * sizeof(float), stream));
  CRVQ_TRY(mT.alloc((size_t)M * kD * sizeof(float), stream));
  CRVQ_TRY(mK.alloc((size_t)M * sizeof(int32_t), stream));
  const size_t wbytes = argmin_scratch_bytes(M, 1, cw.K);
  CRVQ_TRY(mW.alloc(wbytes, stream));
  CRVQ_TRY(mP.alloc((size_t)loss_blocks * sizeof(double), stream));
  CRVQ_TRY(mF.alloc((size_t)std::max<int64_t>(G_cov, 1) * (2 * kD * kD + kD) * sizeof(float),
                    stream));
  float* D = mD.as<float>();
  float* Bt = mB.as<float>();
  float* Hb = mF.as<float>();
  float* Lf = Hb + G_cov * kD * kD;
  float* Linv = Lf + G_cov * kD * kD;
  const int64_t ldb = M;
  {
    ProfScope ps("coupled_residual", stream, (double)M * N * 8.0);
    residual_kernel<<<(unsigned)std::min<int64_t>(ceil_div(M * (N / kD), 256), 16 * nsm), 256, 0,
                      stream>>>(W, M, N, cbs, D, err);
    CRVQ_LAUNCHED();
    block_factor_kernel<<<(unsigned)ceil_div(std::max<int64_t>(G_cov, 1), 128), 128, 0,
                          stream>>>(H, N, G_cov, Hb, Lf, Linv, err);
    CRVQ_LAUNCHED();
  }
  // tr(D H D^T) by column blocks: B^T = H[block rows, :] D^T, then the block's sum of B^T . D
  auto loss_into = [&](double* out) -> crvq_status {
    CRVQ_CUDA(cudaMemsetAsync(mP.as<double>(), 0, (size_t)loss_blocks * sizeof(double), stream));
    for (int64_t c0 = 0; c0 < N; c0 += kBlockCols) {
      const int nc = (int)std::min<int64_t>(kBlockCols, N - c0);
      CRVQ_TRY(launch_tc_gemm_nt(H + c0 * N, N, nc, D, N, M, N, Bt, ldb, stream));
      ProfScope ps("coupled_loss", stream, (double)M * nc * 8.0);
      block_loss_kernel<<<loss_blocks, 256, 0, stream>>>(Bt, ldb, nc, D, M, N, c0,
                                                         mP.as<double>());
      CRVQ_LAUNCHED();
    }
    sum_parts_kernel<<<1, 1, 0, stream>>>(mP.as<double>(), loss_blocks, out);
    CRVQ_LAUNCHED();
    return CRVQ_OK;
  };
  if (loss_dev) CRVQ_TRY(loss_into(loss_dev));
  // the arg-min of one group: a vector set of one group (the shifted targets) and a codebook
  // view writing the new codes to a scratch column; one scratch for every arg-min pass
  CbList one{};
  one.n = 1;
  one.cb[0] = CbView{cw.C, mK.as<int32_t>(), 1, 1, cw.K};
  EncodeExtras ex;
  ex.work = mW.as<char>();
  ex.work_bytes = wbytes;
  for (int sw = 0; sw < sweeps; ++sw) {
    for (int64_t b0 = 0; b0 < G_cov; b0 += kBlockG) {
      const int64_t b1 = std::min<int64_t>(G_cov, b0 + kBlockG);
      const int nc = (int)((b1 - b0) * kD);
      // B^T for the block's channels, with every decision so far in D
      CRVQ_TRY(launch_tc_gemm_nt(H + b0 * kD * N, N, nc, D, N, M, N, Bt, ldb, stream));
      for (int64_t g = b0; g < b1; ++g) {
        const int col0 = (int)((g - b0) * kD);
        {
          ProfScope ps("coupled_target", stream, (double)M);
          coupled_target_kernel<<<row_blocks, 256, 0, stream>>>(D, M, N, Hb, Lf, Linv, Bt, ldb,
                                                                col0, g, cw, mT.as<float>(),
                                                                err);
          CRVQ_LAUNCHED();
        }
        const SetView set{mT.as<float>(), kD, M, 1, Hb + g * kD * kD};
        CRVQ_TRY(launch_encode_beam(set, one, 0, 1, false, nullptr, ex, stream));
        {
          ProfScope ps("coupled_apply", stream, (double)M);
          coupled_apply_kernel<<<row_blocks, 256, 0, stream>>>(W, D, M, N, H, Bt, ldb,
                                                               col0 + kD, nc, g, cbs, which,
                                                               mK.as<int32_t>(), err);
          CRVQ_LAUNCHED();
        }
      }
    }
    if (loss_dev) CRVQ_TRY(loss_into(loss_dev + 1 + sw));
  }
  return CRVQ_OK;
}

}  // namespace crvq
