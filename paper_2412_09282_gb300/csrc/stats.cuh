// Least-squares statistics of one codebook, shared by the standalone update (update.cu) and
// the Lloyd encode pass that accumulates them for the codes it writes (encode.cu).
//
//   cnt[g][k]  exact count of members of code k in group g (int32)
//   bacc[k][j] sum over members v of code k of (H_{g_v} tau_v)_j, as 64-bit fixed point
//   scale      the power of two used for the fixed point (chosen from a bound on the terms)
//
// Integer accumulation makes the sums independent of the order in which threads add, so the
// solve sees identical inputs on every run.
#pragma once

#include "common.cuh"
#include "fixed_point.cuh"
#include "kernels.h"

namespace crvq {

constexpr int kNA = 37;  // packed lower triangle of the 8 x 8 A_k (36 entries) + the count

struct StatsView {
  int32_t* cnt;     // [G_cov][K]
  long long* bacc;  // [K][d]
  double* scale;    // device scalar (followed by the maxima of the scale bound)
  float2* apair;    // [K][kNA]: A_k and the count as fp32 pairs, between the two solve kernels
  int64_t G_cov;
  int K;
};

// Memory of the statistics of one codebook: cnt | bacc | scale + maxima (256 B) | apair, each
// part 256-byte aligned.
struct StatsLayout {
  size_t cnt, bacc, head, apair, total;
};

inline StatsLayout stats_layout(int64_t G_cov, int K) {
  StatsLayout L;
  const int64_t G = G_cov > 1 ? G_cov : 1;
  L.cnt = align_up((size_t)G * K * sizeof(int32_t), 256);
  L.bacc = align_up((size_t)K * kD * sizeof(long long), 256);
  L.head = 256;
  L.apair = align_up((size_t)K * kNA * sizeof(float2), 256);
  L.total = L.cnt + L.bacc + L.head + L.apair;
  return L;
}

// Points st at the statistics laid out in `base` (stats_layout(G_cov, K).total bytes).
inline void stats_bind(void* base, int64_t G_cov, int K, StatsView* st) {
  const StatsLayout L = stats_layout(G_cov, K);
  char* p = static_cast<char*>(base);
  st->cnt = reinterpret_cast<int32_t*>(p);
  st->bacc = reinterpret_cast<long long*>(p + L.cnt);
  st->scale = reinterpret_cast<double*>(p + L.cnt + L.bacc);
  st->apair = reinterpret_cast<float2*>(p + L.cnt + L.bacc + L.head);
  st->G_cov = G_cov;
  st->K = K;
}

// 2^e with e the largest integer such that every term stays below 2^30 (bound * 2^e < 2^30,
// so that one fp32 multiply and one round-to-nearest conversion make it exact: fix_rn_small)
// and no sum of n terms can overflow (n * bound * 2^e < 2^62); e within [-126, 126] so that
// 2^e is a normal fp32 number. With terms resolved to 2^-30 of the bound, a sum's quantisation
// error is far below the fp32 precision of its terms.
__host__ __device__ inline double stats_scale_for(double bound, int64_t n) {
  const double lim = 4.611686018427387904e18;  // 2^62
  const double denom = bound * (double)(n > 0 ? n : 1);
  if (!(denom > 0.0)) return 1099511627776.0;  // 2^40: nothing to scale
  int e = (int)floor(log2(lim / denom));
  const int e_term = (int)floor(log2(1073741824.0 / bound));  // 2^30 / bound
  if (e_term < e) e = e_term;
  return ldexp(1.0, e < -126 ? -126 : (e > 126 ? 126 : e));
}

// tau = t - sum over the codebooks s != which that cover g of C_s[code] (fp32, codebook order).
__device__ __forceinline__ void stats_target(const SetView& set, const CbList& cbs, int which,
                                             int64_t i, int64_t g, float tau[kD],
                                             unsigned* err) {
  const float* t = set.T + i * set.ldT + g * kD;
  const float4 t0 = *reinterpret_cast<const float4*>(t);
  const float4 t1 = *reinterpret_cast<const float4*>(t + 4);
  tau[0] = t0.x; tau[1] = t0.y; tau[2] = t0.z; tau[3] = t0.w;
  tau[4] = t1.x; tau[5] = t1.y; tau[6] = t1.z; tau[7] = t1.w;
  for (int s = 0; s < cbs.n; ++s) {
    if (s == which) continue;
    const CbView& cb = cbs.cb[s];
    if (g >= cb.G_cov) continue;
    const int32_t k = cb.codes[i * cb.ld + g];
    if (k < 0 || k >= cb.K) {
      raise_error(err, ERRBIT_INDEX);
      continue;
    }
    const float* c = cb.C + (int64_t)k * kD;
#pragma unroll
    for (int j = 0; j < kD; ++j) tau[j] -= c[j];
  }
}

// q = H tau, each row an FMA chain over the columns in order (the encode pass evaluates
// H r the same way, so both paths produce bit-identical contributions).
__device__ __forceinline__ void stats_htau(const float* H, const float tau[kD], float q[kD]) {
#pragma unroll
  for (int r = 0; r < kD; ++r) {
    float a = 0.f;
#pragma unroll
    for (int c = 0; c < kD; ++c) a = fmaf(H[r * kD + c], tau[c], a);
    q[r] = a;
  }
}

// Exponent e of the fixed-point scale 2^e (an exact power of two, normal).
__device__ __forceinline__ int stats_scale_exp(double scale) {
  return (int)((__double_as_longlong(scale) >> 52) & 0x7ff) - 1023;
}

// The fixed-point scale as an fp32 number (an exact power of two in the normal range).
__device__ __forceinline__ float stats_scale_f(const StatsView& st) { return (float)*st.scale; }

__device__ __forceinline__ void stats_add(const StatsView& st, float scale, int64_t g, int k,
                                          const float q[kD]) {
  atomicAdd(&st.cnt[g * st.K + k], 1);
#pragma unroll
  for (int j = 0; j < kD; ++j)
    atomicAdd(reinterpret_cast<unsigned long long*>(&st.bacc[(int64_t)k * kD + j]),
              (unsigned long long)fix_rn_small(q[j], scale));
}

// Solves A x = b for a symmetric positive definite 8 x 8 A given as its packed lower
// triangle (row-major, A[r(r+1)/2 + c] for c <= r). Returns false when A is not SPD.
__device__ inline bool cholesky_solve8(const double A[36], const double b[kD], double x[kD]) {
  double L[36];
  int q = 0;
  for (int r = 0; r < kD; ++r) {
    for (int c = 0; c <= r; ++c, ++q) {
      double s = A[q];
      for (int m = 0; m < c; ++m) s -= L[r * (r + 1) / 2 + m] * L[c * (c + 1) / 2 + m];
      if (r == c) {
        if (!(s > 0.0)) return false;
        L[q] = sqrt(s);
      } else {
        L[q] = s / L[c * (c + 1) / 2 + c];
      }
    }
  }
  double y[kD];
  for (int r = 0; r < kD; ++r) {
    double s = b[r];
    for (int m = 0; m < r; ++m) s -= L[r * (r + 1) / 2 + m] * y[m];
    y[r] = s / L[r * (r + 1) / 2 + r];
  }
  for (int r = kD - 1; r >= 0; --r) {
    double s = y[r];
    for (int m = r + 1; m < kD; ++m) s -= L[m * (m + 1) / 2 + r] * x[m];
    x[r] = s / L[r * (r + 1) / 2 + r];
  }
  return true;
}

// Host side (update.cu).
crvq_status stats_alloc(Scratch& mem, int64_t G_cov, int K, StatsView* st, cudaStream_t s);
// Zeroes cnt/bacc (scale is kept).
crvq_status stats_zero(const StatsView& st, cudaStream_t s);
// Computes the fixed-point scale for accumulating codebook `which` over `set`.
crvq_status launch_stats_prepare(const SetView& set, const CbList& cbs, int which,
                                 const StatsView& st, cudaStream_t stream);
// Solves every codeword from the statistics and leaves cnt and bacc zero (each is cleared
// once read), ready for the next accumulation.
crvq_status launch_stats_solve(const SetView& set, const StatsView& st, const float* C_old,
                               float* C_out, int32_t* counts, cudaStream_t stream);

}  // namespace crvq
