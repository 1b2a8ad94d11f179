// diag(H^-1) of the damped Hessian proxy, the denominator of the channel importance of
// Sec. 4.1 Eq. (wa): I_i = max_j (w_ji - VQ(w_ji))^2 / (2 [H^-1]_ii).
//
// With H = L L^T (Cholesky), H^-1 = L^-T L^-1, so [H^-1]_ii = sum_k (L^-1)_ki^2: the squared
// norm of column i of L^-1. The channel order must match an fp64 evaluation to about 1e-6
// relative while cond(H) reaches 1e4 and more, which fp32 or 3xTF32 arithmetic cannot give,
// so every step runs in fp64 (the fp64 pipe; about 2 N^3 / 3 flops):
//   1. A = H in fp64, padded to whole 64 x 64 tiles with an identity block;
//   2. blocked right-looking Cholesky: per diagonal tile k, the tile's factor and its inverse
//      in one CTA, then the panel below it times that inverse, then the trailing lower
//      triangle minus the panel's outer product;
//   3. X = L^-1 by blocked forward substitution, right-looking: block row i of X is the
//      inverse diagonal tile times block row i of B (B = I, updated), then every later block
//      row of B loses L(r, i) X(i, :);
//   4. [H^-1]_ii = the squared norm of column i of X, summed in row order.
// One 64 x 64 x 64 tile product (fp64, 256 threads, 4 x 4 outputs each) serves steps 2 and 3.
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

constexpr int kT = 64;  // tile size

__global__ void __launch_bounds__(256)
to_f64_padded_kernel(const float* __restrict__ H, int64_t N, int64_t Np,
                     double* __restrict__ A) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < Np * Np;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = e / Np, c = e % Np;
    A[e] = (r < N && c < N) ? (double)H[r * N + c] : (r == c ? 1.0 : 0.0);
  }
}

// Factor of the diagonal tile k (its lower triangle, in place) and the inverse of that factor
// into Dinv (64 x 64, lower). One CTA of 256 threads. A pivot that is not positive reports
// ERRBIT_NUMERIC and is replaced by 1 (the result is then not used by the caller).
__global__ void __launch_bounds__(256)
potrf_tile_kernel(double* __restrict__ A, int64_t Np, int64_t k, double* __restrict__ Dinv,
                  unsigned* err) {
  __shared__ double s[kT][kT + 1];
  __shared__ double inv[kT][kT + 1];
  double* base = A + k * kT * Np + k * kT;
  for (int e = threadIdx.x; e < kT * kT; e += blockDim.x) s[e / kT][e % kT] = base[(e / kT) * Np + e % kT];
  __syncthreads();
  for (int c = 0; c < kT; ++c) {
    if (threadIdx.x == 0) {
      double p = s[c][c];
      if (!(p > 0.0)) {
        raise_error(err, ERRBIT_NUMERIC);
        p = 1.0;
      }
      s[c][c] = sqrt(p);
    }
    __syncthreads();
    const double d = s[c][c];
    for (int r = c + 1 + threadIdx.x; r < kT; r += blockDim.x) s[r][c] /= d;
    __syncthreads();
    // trailing lower triangle of the tile
    const int n = kT - c - 1;
    for (int e = threadIdx.x; e < n * n; e += blockDim.x) {
      const int r = c + 1 + e / n, j = c + 1 + e % n;
      if (j <= r) s[r][j] -= s[r][c] * s[j][c];
    }
    __syncthreads();
  }
  // inverse of the lower-triangular factor: column j of inv solves L x = e_j (thread = column)
  if (threadIdx.x < kT) {
    const int j = threadIdx.x;
    for (int r = 0; r < kT; ++r) {
      double v = (r == j) ? 1.0 : 0.0;
      for (int m = j; m < r; ++m) v -= s[r][m] * inv[m][j];
      inv[r][j] = r < j ? 0.0 : v / s[r][r];
    }
  }
  __syncthreads();
  for (int e = threadIdx.x; e < kT * kT; e += blockDim.x) {
    const int r = e / kT, c = e % kT;
    base[r * Np + c] = c <= r ? s[r][c] : 0.0;
    Dinv[e] = inv[r][c];
  }
}

// One 64 x 64 output tile per CTA: C = A_tile B_tile or A_tile B_tile^T, assigned or
// subtracted, by the task's kind; the tile coordinates come from the grid: kind 0 = the Cholesky panel (rows below tile k: C = P(r, k) Dinv^T in place),
// kind 1 = the Cholesky trailing update (lower triangle of tiles k < J <= I),
// kind 2 = the inverse's diagonal step (X(i, c) = Dinv_i B(i, c) for c <= i),
// kind 3 = the inverse's update (B(r, c) -= L(r, i) X(i, c), r > i, c <= i).
struct TileTask {
  int kind;
  int64_t k;      // the step
  int64_t nblk;   // tiles per side
  int64_t Np;
  double* A;      // the factor (row-major Np x Np)
  double* X;      // the inverse / right-hand side (row-major Np x Np)
  const double* Dinv;  // inverse of diagonal tile k
};

__device__ __forceinline__ void tile_coords(const TileTask& t, int64_t b, int64_t& I,
                                            int64_t& J) {
  if (t.kind == 0) {
    I = t.k + 1 + b;
    J = t.k;
  } else if (t.kind == 1) {  // b -> (I, J) over the lower triangle of the trailing tiles
    int64_t i = (int64_t)((sqrt(8.0 * (double)b + 1.0) - 1.0) / 2.0);
    while ((i + 1) * (i + 2) / 2 <= b) ++i;
    while (i * (i + 1) / 2 > b) --i;
    I = t.k + 1 + i;
    J = t.k + 1 + (b - i * (i + 1) / 2);
  } else if (t.kind == 2) {
    I = t.k;
    J = b;
  } else {
    const int64_t cols = t.k + 1;
    I = t.k + 1 + b / cols;
    J = b % cols;
  }
}

__global__ void __launch_bounds__(256)
tile_kernel(TileTask t) {
  __shared__ double sA[kT][kT + 1];
  __shared__ double sB[kT][kT + 1];
  int64_t I, J;
  tile_coords(t, blockIdx.x, I, J);
  const int64_t Np = t.Np;
  const double* Ap;
  const double* Bp;
  double* Cp;
  bool trans_b, sub;
  if (t.kind == 0) {         // P(I, k) = P(I, k) Dinv^T
    Ap = t.A + I * kT * Np + t.k * kT;
    Bp = t.Dinv;
    Cp = t.A + I * kT * Np + t.k * kT;
    trans_b = true;
    sub = false;
  } else if (t.kind == 1) {  // A(I, J) -= P(I, k) P(J, k)^T
    Ap = t.A + I * kT * Np + t.k * kT;
    Bp = t.A + J * kT * Np + t.k * kT;
    Cp = t.A + I * kT * Np + J * kT;
    trans_b = true;
    sub = true;
  } else if (t.kind == 2) {  // X(k, J) = Dinv_k B(k, J)
    Ap = t.Dinv;
    Bp = t.X + t.k * kT * Np + J * kT;
    Cp = t.X + t.k * kT * Np + J * kT;
    trans_b = false;
    sub = false;
  } else {                   // B(I, J) -= L(I, k) X(k, J)
    Ap = t.A + I * kT * Np + t.k * kT;
    Bp = t.X + t.k * kT * Np + J * kT;
    Cp = t.X + I * kT * Np + J * kT;
    trans_b = false;
    sub = true;
  }
  const int64_t lda = (t.kind == 2) ? kT : Np;
  const int64_t ldb = (t.kind == 0) ? kT : Np;
  for (int e = threadIdx.x; e < kT * kT; e += blockDim.x) {
    const int r = e / kT, c = e % kT;
    sA[r][c] = Ap[r * lda + c];
    sB[r][c] = Bp[r * ldb + c];
  }
  __syncthreads();
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  double acc[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) acc[a][b] = 0.0;
  for (int q = 0; q < kT; ++q) {
    double av[4], bv[4];
#pragma unroll
    for (int a = 0; a < 4; ++a) av[a] = sA[ty * 4 + a][q];
#pragma unroll
    for (int b = 0; b < 4; ++b) bv[b] = trans_b ? sB[tx * 4 + b][q] : sB[q][tx * 4 + b];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) acc[a][b] = fma(av[a], bv[b], acc[a][b]);
  }
  // in-place kinds read their own tile: every thread has loaded it before any writes
  __syncthreads();
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      double* o = Cp + (int64_t)(ty * 4 + a) * Np + tx * 4 + b;
      *o = sub ? *o - acc[a][b] : acc[a][b];
    }
}

__global__ void __launch_bounds__(256)
identity_kernel(double* __restrict__ X, int64_t Np) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < Np * Np;
       e += (int64_t)gridDim.x * blockDim.x)
    X[e] = (e / Np == e % Np) ? 1.0 : 0.0;
}

// hinv[c] = sum over rows r >= c of X[r][c]^2, in row order (one thread per column).
__global__ void __launch_bounds__(256)
colnorm_kernel(const double* __restrict__ X, int64_t Np, int64_t N, double* __restrict__ hinv) {
  const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= N) return;
  double s = 0.0;
  for (int64_t r = c; r < Np; ++r) {
    const double v = X[r * Np + c];
    s = fma(v, v, s);
  }
  hinv[c] = s;
}

}  // namespace

crvq_status launch_hinv_diag(const float* H, int64_t N, double* hinv, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const int nsm = sm_count();
  const int64_t nblk = ceil_div(N, kT);
  const int64_t Np = nblk * kT;
  Scratch mA, mX, mD;
  CRVQ_TRY(mA.alloc((size_t)Np * Np * sizeof(double), stream));
  CRVQ_TRY(mX.alloc((size_t)Np * Np * sizeof(double), stream));
  CRVQ_TRY(mD.alloc((size_t)nblk * kT * kT * sizeof(double), stream));  // every L_kk^-1
  double* A = mA.as<double>();
  double* X = mX.as<double>();
  double* Dinv = mD.as<double>();
  const unsigned fill_blocks = (unsigned)std::min<int64_t>(ceil_div(Np * Np, 256), 16 * nsm);
  ProfScope ps("hinv_cholesky_inverse", stream, 2.0 / 3.0 * (double)Np * Np * Np);
  to_f64_padded_kernel<<<fill_blocks, 256, 0, stream>>>(H, N, Np, A);
  CRVQ_LAUNCHED();
  TileTask t{};
  t.nblk = nblk;
  t.Np = Np;
  t.A = A;
  t.X = X;
  t.Dinv = Dinv;
  for (int64_t k = 0; k < nblk; ++k) {
    potrf_tile_kernel<<<1, 256, 0, stream>>>(A, Np, k, Dinv + k * kT * kT, err);
    CRVQ_LAUNCHED();
    const int64_t below = nblk - k - 1;
    if (below == 0) continue;
    t.k = k;
    t.Dinv = Dinv + k * kT * kT;
    t.kind = 0;
    tile_kernel<<<(unsigned)below, 256, 0, stream>>>(t);
    CRVQ_LAUNCHED();
    t.kind = 1;
    tile_kernel<<<(unsigned)(below * (below + 1) / 2), 256, 0, stream>>>(t);
    CRVQ_LAUNCHED();
  }
  // X = L^-1: B = I, then per block row i: X(i, :) = L_ii^-1 B(i, :), B(r, :) -= L(r, i) X(i, :)
  identity_kernel<<<fill_blocks, 256, 0, stream>>>(X, Np);
  CRVQ_LAUNCHED();
  for (int64_t i = 0; i < nblk; ++i) {
    t.k = i;
    t.Dinv = Dinv + i * kT * kT;
    t.kind = 2;
    tile_kernel<<<(unsigned)(i + 1), 256, 0, stream>>>(t);
    CRVQ_LAUNCHED();
    const int64_t below = nblk - i - 1;
    if (below == 0) continue;
    t.kind = 3;
    tile_kernel<<<(unsigned)(below * (i + 1)), 256, 0, stream>>>(t);
    CRVQ_LAUNCHED();
  }
  colnorm_kernel<<<(unsigned)ceil_div(N, 256), 256, 0, stream>>>(X, Np, N, hinv);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace crvq
