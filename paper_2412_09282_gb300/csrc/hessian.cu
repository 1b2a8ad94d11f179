// S1: Hessian proxy H = X^T X / n + delta I (App. A.2; the paper's X is N x O and its proxy
// XX^T is the same matrix as our X^T X).
//
// SIMT fp32 symmetric rank-n update: only the tiles on or above the diagonal are computed and
// mirrored. Accumulation is two-level (an inner fp32 sum over 256 tokens flushed into an
// outer fp32 sum), which bounds the rounding error by about (256 + n/256) * 2^-24 relative to
// sum_k |x_ka x_kb|.
#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

constexpr int kTile = 128;
constexpr int kBK = 16;
constexpr int kFlush = 256;  // tokens per inner accumulation

__global__ void __launch_bounds__(256)
syrk_tn_kernel(const float* __restrict__ X, int64_t n, int64_t N, float inv_n,
               float* __restrict__ S, int nb) {
  // Map the linear block id to a tile (bi <= bj) of the upper triangle.
  int64_t t = blockIdx.x;
  int bi = 0;
  while (t >= nb - bi) {
    t -= nb - bi;
    ++bi;
  }
  const int bj = bi + (int)t;
  const int64_t a0 = (int64_t)bi * kTile, b0 = (int64_t)bj * kTile;

  __shared__ __align__(16) float As[kBK][kTile];
  __shared__ __align__(16) float Bs[kBK][kTile];

  const int tid = threadIdx.x;
  const int tx = tid & 15, ty = tid >> 4;
  float acc[8][8], outer[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = outer[i][j] = 0.f;

  const bool vec_ok = (N % 4) == 0;
  int since_flush = 0;
  for (int64_t k0 = 0; k0 < n; k0 += kBK) {
    // Each thread loads 2 float4 of each operand: rows k0 + (tid / 32) * 2 + {0,1}.
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int kk = (tid >> 5) * 2 + r;
      const int c = (tid & 31) * 4;
      const int64_t k = k0 + kk;
      float4 va = make_float4(0.f, 0.f, 0.f, 0.f), vb = va;
      if (k < n) {
        const float* row = X + k * N;
        if (vec_ok && a0 + c + 3 < N) {
          va = *reinterpret_cast<const float4*>(row + a0 + c);
        } else {
          float tmp[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) tmp[q] = (a0 + c + q < N) ? row[a0 + c + q] : 0.f;
          va = make_float4(tmp[0], tmp[1], tmp[2], tmp[3]);
        }
        if (vec_ok && b0 + c + 3 < N) {
          vb = *reinterpret_cast<const float4*>(row + b0 + c);
        } else {
          float tmp[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) tmp[q] = (b0 + c + q < N) ? row[b0 + c + q] : 0.f;
          vb = make_float4(tmp[0], tmp[1], tmp[2], tmp[3]);
        }
      }
      *reinterpret_cast<float4*>(&As[kk][c]) = va;
      *reinterpret_cast<float4*>(&Bs[kk][c]) = vb;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kBK; ++kk) {
      float a[8], b[8];
      const float4 a_lo = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
      const float4 a_hi = *reinterpret_cast<const float4*>(&As[kk][64 + ty * 4]);
      const float4 b_lo = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
      const float4 b_hi = *reinterpret_cast<const float4*>(&Bs[kk][64 + tx * 4]);
      a[0] = a_lo.x; a[1] = a_lo.y; a[2] = a_lo.z; a[3] = a_lo.w;
      a[4] = a_hi.x; a[5] = a_hi.y; a[6] = a_hi.z; a[7] = a_hi.w;
      b[0] = b_lo.x; b[1] = b_lo.y; b[2] = b_lo.z; b[3] = b_lo.w;
      b[4] = b_hi.x; b[5] = b_hi.y; b[6] = b_hi.z; b[7] = b_hi.w;
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
    since_flush += kBK;
    if (since_flush >= kFlush) {
      since_flush = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          outer[i][j] += acc[i][j];
          acc[i][j] = 0.f;
        }
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t a = a0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
    if (a >= N) continue;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t b = b0 + (j < 4 ? tx * 4 + j : 64 + tx * 4 + (j - 4));
      if (b >= N) continue;
      const float v = (outer[i][j] + acc[i][j]) * inv_n;
      S[a * N + b] = v;
      if (bi != bj) S[b * N + a] = v;
    }
  }
}

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
  const int nb = (int)ceil_div(N, kTile);
  const int64_t tiles = (int64_t)nb * (nb + 1) / 2;
  {
    ProfScope ps("hessian_syrk", stream, (double)n * (double)N * (double)(N + 1));
    syrk_tn_kernel<<<(unsigned)tiles, 256, 0, stream>>>(X, n, N, (float)(1.0 / (double)n), H,
                                                        nb);
    CRVQ_LAUNCHED();
  }
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
