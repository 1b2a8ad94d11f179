// S1: Hessian proxy H = X^T X / n + delta I (App. A.2; the paper's X is N x O and its proxy
// XX^T is the same matrix as our X^T X).
//
// The dense product X^T X (the crvq_hessian entry) runs on the tensor cores (tc_gemm.cuh:
// tcgen05, 3xTF32, tiles on or above the diagonal, mirrored; K split into 1024-token chunks
// summed in fp32 in chunk order). A single CTA then takes the diagonal, the damping and the
// original-order diagonal blocks. The layer schedule forms only the diagonal blocks
// (launch_tc_hessian_blocks in tc_gemm.cu), with the same values.
#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

// One CTA: xsq, delta = damp_rel * mean(xsq) (fixed-order fp64 sum), damped diagonal and the
// original-order diagonal blocks.
__global__ void __launch_bounds__(1024)
hessian_finalize_kernel(float* __restrict__ H, int64_t N, int d, float damp_rel,
                        float* __restrict__ xsq, float* __restrict__ delta_out) {
  __shared__ double part[1024];
  double s = 0.0;
  for (int64_t i = threadIdx.x; i < N; i += blockDim.x) s += (double)H[i * N + i];
  part[threadIdx.x] = s;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) part[threadIdx.x] += part[threadIdx.x + w];
    __syncthreads();
  }
  const double delta = (double)damp_rel * (part[0] / (double)N);
  for (int64_t i = threadIdx.x; i < N; i += blockDim.x) {
    const float v = H[i * N + i];
    xsq[i] = v;
    H[i * N + i] = (float)((double)v + delta);
  }
  if (threadIdx.x == 0 && delta_out) *delta_out = (float)delta;
}

__global__ void extract_blocks_kernel(const float* __restrict__ H, int64_t N, int d,
                                      const int32_t* __restrict__ perm,
                                      float* __restrict__ Hb, unsigned* err) {
  const int64_t G = N / d;
  const int64_t total = G * d * d;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t g = e / (d * d);
    const int r = (int)((e / d) % d), c = (int)(e % d);
    int64_t ra = g * d + r, cb = g * d + c;
    if (perm) {
      ra = perm[ra];
      cb = perm[cb];
      if (ra < 0 || ra >= N || cb < 0 || cb >= N) {
        raise_error(err, ERRBIT_INDEX);
        continue;
      }
    }
    Hb[e] = H[ra * N + cb];
  }
}

}  // namespace

crvq_status launch_hessian(const float* X, int64_t n, int64_t N, int d, float damp_rel,
                           float* H, float* xsq, float* H_blocks, float* delta,
                           cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  CRVQ_TRY(launch_tc_syrk(X, n, N, H, stream));
  {
    ProfScope ps("hessian_finalize", stream, 0.0);
    hessian_finalize_kernel<<<1, 1024, 0, stream>>>(H, N, d, damp_rel, xsq, delta);
    CRVQ_LAUNCHED();
  }
  if (H_blocks) CRVQ_TRY(launch_extract_blocks(H, N, d, nullptr, H_blocks, stream));
  return CRVQ_OK;
}

crvq_status launch_extract_blocks(const float* H, int64_t N, int d, const int32_t* perm,
                                  float* H_blocks, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const int64_t total = (N / d) * d * d;
  const int blocks = (int)std::min<int64_t>(ceil_div(total, 256), 4096);
  ProfScope ps("extract_blocks", stream, (double)total * 8.0);
  extract_blocks_kernel<<<blocks, 256, 0, stream>>>(H, N, d, perm, H_blocks, err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace crvq
