// Least-squares codebook update (k-means update step; Alg. 1 FineTuneCodebook in its
// closed-form reading). For codebook `which` with all others fixed, codeword k solves
//   A_k c_k = b_k,  A_k = sum_g cnt[g][k] H_g,  b_k = sum_{v in cluster k} H_{g_v} tau_v,
//   tau_v = t_v - sum over the other covering codebooks of C[code].
//
// Deterministic by construction, with no sort and no float atomics: cnt[g][k] are integer
// counts, b_k is accumulated in 64-bit fixed point (stats.cuh), A_k is summed as fp32 pairs in
// a fixed order (partial sums over fixed slices of the groups, added in slice order), and the
// 8 x 8 system is solved by an fp32 Cholesky factor with iterative refinement whose residual
// is formed in fp32 pairs (to 2^-40 of the solution), in one kernel. GB300's fp64 pipe is a
// small fraction of its fp32 rate and a dependent fp64 operation costs about 180 cycles, so
// none of this arithmetic runs in fp64. The Lloyd encode pass (encode.cu) accumulates the
// same statistics for the codes it writes.
#include <algorithm>
#include <cmath>

#include "common.cuh"
#include "kernels.h"
#include "stats.cuh"

namespace crvq {

namespace {

// max(a, b) that keeps a NaN: fmaxf returns the other operand when one is NaN, which would
// leave the bound below finite and hide a non-finite input from the scale check.
__device__ __forceinline__ float max_keep_nan(float a, float b) {
  return (b > a || b != b) ? b : a;
}

// maxbits[0] = max |T| over the covered vectors, maxbits[1] = max row sum of |H_g|,
// maxbits[2 + s] = max |C_s| (float bits of non-negative values, merged with atomicMax; a NaN
// has larger bits than every finite value and Inf, so it survives the merge and makes the
// bound non-finite).
__global__ void __launch_bounds__(256)
maxabs_kernel(SetView set, int64_t G_cov, CbList cbs, int which, unsigned* __restrict__ maxbits) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t nth = (int64_t)gridDim.x * blockDim.x;
  float tm = 0.f;
  const int64_t nv = set.M * G_cov;
  for (int64_t v = tid; v < nv; v += nth) {
    const int64_t i = v / G_cov, g = v % G_cov;
    const float4* t = reinterpret_cast<const float4*>(set.T + i * set.ldT + g * kD);
    const float4 a = t[0], b = t[1];
    tm = max_keep_nan(tm, max_keep_nan(max_keep_nan(fabsf(a.x), fabsf(a.y)),
                                       max_keep_nan(fabsf(a.z), fabsf(a.w))));
    tm = max_keep_nan(tm, max_keep_nan(max_keep_nan(fabsf(b.x), fabsf(b.y)),
                                       max_keep_nan(fabsf(b.z), fabsf(b.w))));
  }
  float hm = 0.f;
  for (int64_t r = tid; r < G_cov * kD; r += nth) {
    const float* h = set.Hb + r * kD;
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < kD; ++j) s += fabsf(h[j]);  // a NaN entry makes the sum NaN
    hm = max_keep_nan(hm, s);
  }
  // warp max, then one atomic per warp
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    tm = max_keep_nan(tm, __shfl_xor_sync(0xffffffffu, tm, off));
    hm = max_keep_nan(hm, __shfl_xor_sync(0xffffffffu, hm, off));
  }
  if ((threadIdx.x & 31) == 0) {
    atomicMax(&maxbits[0], __float_as_uint(tm));
    atomicMax(&maxbits[1], __float_as_uint(hm));
  }
  for (int s = 0; s < cbs.n; ++s) {
    if (s == which) continue;
    float m = 0.f;
    for (int64_t e = tid; e < (int64_t)cbs.cb[s].K * kD; e += nth)
      m = max_keep_nan(m, fabsf(cbs.cb[s].C[e]));
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
      m = max_keep_nan(m, __shfl_xor_sync(0xffffffffu, m, off));
    if ((threadIdx.x & 31) == 0) atomicMax(&maxbits[2 + s], __float_as_uint(m));
  }
}

__global__ void stats_scale_kernel(const unsigned* __restrict__ maxbits, int n_cb, int which,
                                   int64_t n_members, double* __restrict__ scale,
                                   unsigned* err) {
  double cs = 0.0;
  for (int s = 0; s < n_cb; ++s)
    if (s != which) cs += (double)__uint_as_float(maxbits[2 + s]);
  // |H_g tau|_inf <= max row sum |H_g| * (max |t| + sum_s max |C_s|)
  const double bound =
      (double)__uint_as_float(maxbits[1]) * ((double)__uint_as_float(maxbits[0]) + cs) * 1.001;
  if (!isfinite(bound)) raise_error(err, ERRBIT_NUMERIC);
  *scale = stats_scale_for(bound, n_members);
}

// Statistics of every covered vector from its current code. CTA (x, y): groups y,
// y + gridDim.y, ..., rows x, x + gridDim.x, ... of each; with K <= kSmemStatsK the CTA sums
// its counts and fixed-point terms in shared memory and adds them to the global sums once;
// larger codebooks add each vector's terms to the global sums directly. A term (|v| < 2^30)
// enters shared memory as v = 2^15 vh + vl (0 <= vl < 2^15) in two 32-bit sums (native 32-bit
// atomics): exact, as accumulate_grid gives a CTA fewer than 2^16 rows of a group. Integer
// sums: the order is immaterial.
constexpr int kSmemStatsK = 256;

__global__ void __launch_bounds__(256)
accumulate_stats_kernel(SetView set, CbList cbs, int which, StatsView st, unsigned* err) {
  // [component][vh, vl][code]: lanes of a warp adding one component hit spread banks
  __shared__ int s_b32[kD * 2 * kSmemStatsK];
  __shared__ int s_cnt[kSmemStatsK];
  const CbView cw = cbs.cb[which];
  const float sscale = stats_scale_f(st);
  const bool smem = cw.K <= kSmemStatsK;
  for (int64_t g = blockIdx.y; g < cw.G_cov; g += gridDim.y) {
    if (smem) {
      __syncthreads();  // the previous group's flush has read the sums
      for (int e = threadIdx.x; e < kSmemStatsK * kD * 2; e += blockDim.x) s_b32[e] = 0;
      for (int e = threadIdx.x; e < kSmemStatsK; e += blockDim.x) s_cnt[e] = 0;
      __syncthreads();
    }
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < set.M;
         i += (int64_t)gridDim.x * blockDim.x) {
      const int32_t k = cw.codes[i * cw.ld + g];
      if (k < 0 || k >= cw.K) {
        raise_error(err, ERRBIT_INDEX);
        continue;
      }
      float tau[kD], q[kD];
      stats_target(set, cbs, which, i, g, tau, err);
      stats_htau(set.Hb + g * kD * kD, tau, q);
      if (smem) {
        atomicAdd(&s_cnt[k], 1);
#pragma unroll
        for (int j = 0; j < kD; ++j) {
          const long long v = fix_rn_small(q[j], sscale);
          atomicAdd(&s_b32[(2 * j) * kSmemStatsK + k], (int)(v >> 15));
          atomicAdd(&s_b32[(2 * j + 1) * kSmemStatsK + k], (int)(v & 0x7fff));
        }
      } else {
        stats_add(st, sscale, g, k, q);
      }
    }
    if (smem) {
      __syncthreads();
      for (int k = threadIdx.x; k < cw.K; k += blockDim.x) {
        const int c = s_cnt[k];
        if (c == 0) continue;
        atomicAdd(&st.cnt[g * st.K + k], c);
#pragma unroll
        for (int j = 0; j < kD; ++j) {
          const long long v = (long long)s_b32[(2 * j) * kSmemStatsK + k] * 32768 +
                              s_b32[(2 * j + 1) * kSmemStatsK + k];
          atomicAdd(reinterpret_cast<unsigned long long*>(&st.bacc[(int64_t)k * kD + j]),
                    (unsigned long long)v);
        }
      }
    }
  }
}

// Grid of accumulate_stats_kernel: one column of CTAs per group, enough rows per CTA that
// the flush stays small, at least ~4 CTAs per SM overall, and fewer than 2^16 rows per CTA
// (the 32-bit shared sums).
dim3 accumulate_grid(int64_t M, int64_t G_cov, int nsm) {
  const int64_t want =
      std::max<int64_t>(1, ceil_div(4 * (int64_t)nsm, std::max<int64_t>(G_cov, 1)));
  const int64_t rows_x = std::max<int64_t>(
      ceil_div(M, 65000), std::max<int64_t>(1, std::min<int64_t>(want, ceil_div(M, 1024))));
  return dim3((unsigned)rows_x, (unsigned)std::min<int64_t>(std::max<int64_t>(G_cov, 1), 65535));
}

// fp32 Cholesky factor of the packed lower triangle (false unless every pivot is positive)
// with the reciprocals of its diagonal, and the solve L L^T x = b with them: 8 divisions per
// factor, none per solve (the refinement absorbs the rounding of the reciprocals).
__device__ inline bool chol8_f32(const float A[36], float L[36], float inv[kD]) {
  int q = 0;
#pragma unroll
  for (int r = 0; r < kD; ++r)
#pragma unroll
    for (int c = 0; c <= r; ++c, ++q) {
      float s = A[q];
#pragma unroll
      for (int m = 0; m < c; ++m) s = fmaf(-L[r * (r + 1) / 2 + m], L[c * (c + 1) / 2 + m], s);
      if (r == c) {
        if (!(s > 0.f)) return false;
        L[q] = sqrtf(s);
        inv[r] = 1.f / L[q];
      } else {
        L[q] = s * inv[c];
      }
    }
  return true;
}

__device__ inline void chol8_solve_f32(const float L[36], const float inv[kD], const float b[kD],
                                       float x[kD]) {
  float y[kD];
#pragma unroll
  for (int r = 0; r < kD; ++r) {
    float s = b[r];
#pragma unroll
    for (int m = 0; m < r; ++m) s = fmaf(-L[r * (r + 1) / 2 + m], y[m], s);
    y[r] = s * inv[r];
  }
#pragma unroll
  for (int r = kD - 1; r >= 0; --r) {
    float s = y[r];
#pragma unroll
    for (int m = r + 1; m < kD; ++m) s = fmaf(-L[m * (m + 1) / 2 + r], x[m], s);
    x[r] = s * inv[r];
  }
}

__device__ __forceinline__ void pair_two_sum(float a, float b, float& s, float& e) {
  s = __fadd_rn(a, b);
  const float bp = __fsub_rn(s, a);
  e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bp)), __fsub_rn(b, bp));
}

// Solves A x = b with A (packed lower triangle) and b given as unevaluated fp32 pairs
// (hi + lo), by iterative refinement around an fp32 Cholesky factor: each step forms the
// residual r = b - A x in fp32 pairs (every product split exactly by an FMA, TwoSum
// accumulation, about 2^-44 relative), solves L L^T dx = r in fp32 and adds dx to x, which is
// kept as a pair, until the correction is below 2^-40 of x (each step gains about
// -log2(cond(A) u_32) bits) or after 12 steps. No fp64 arithmetic: a dependent fp64 operation
// costs about 180 cycles on this part, and one thread solves each codeword. Returns false
// when A has no fp32 Cholesky factor.
__device__ bool solve8_pairs(const float Ah[36], const float Al[36], const float bh[kD],
                             const float bl[kD], float x_out[kD]) {
  float Af[36], Lf[36], inv[kD];
#pragma unroll
  for (int e = 0; e < 36; ++e) Af[e] = __fadd_rn(Ah[e], Al[e]);
  if (!chol8_f32(Af, Lf, inv)) return false;
  float bf[kD], xh[kD], xl[kD];
#pragma unroll
  for (int j = 0; j < kD; ++j) {
    bf[j] = __fadd_rn(bh[j], bl[j]);
    xl[j] = 0.f;
  }
  chol8_solve_f32(Lf, inv, bf, xh);
  for (int it = 0; it < 12; ++it) {
    float rf[kD];
#pragma unroll
    for (int r = 0; r < kD; ++r) {
      float h = bh[r], l = bl[r];
#pragma unroll
      for (int c = 0; c < kD; ++c) {
        const int q = r >= c ? r * (r + 1) / 2 + c : c * (c + 1) / 2 + r;
        const float p = __fmul_rn(Ah[q], xh[c]);
        const float pe = __fmaf_rn(Ah[q], xh[c], -p);  // Ah xh = p + pe exactly
        const float cross = __fmaf_rn(Ah[q], xl[c], __fmul_rn(Al[q], xh[c]));
        float sum, t;
        pair_two_sum(h, -p, sum, t);
        h = sum;
        l = __fadd_rn(l, __fsub_rn(t, __fadd_rn(pe, cross)));
      }
      rf[r] = __fadd_rn(h, l);
    }
    float dx[kD];
    chol8_solve_f32(Lf, inv, rf, dx);
    float xm = 0.f, dm = 0.f;
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      float sum, t;
      pair_two_sum(xh[j], dx[j], sum, t);
      const float lo = __fadd_rn(xl[j], t);
      xh[j] = __fadd_rn(sum, lo);                      // renormalise the pair
      xl[j] = __fsub_rn(lo, __fsub_rn(xh[j], sum));
      xm = fmaxf(xm, fabsf(xh[j]));
      dm = fmaxf(dm, fabsf(dx[j]));
    }
    if (dm <= 9.094947e-13f * xm) break;  // 2^-40
  }
#pragma unroll
  for (int j = 0; j < kD; ++j) x_out[j] = __fadd_rn(xh[j], xl[j]);
  return true;
}

// b_j = bacc_j / 2^sexp as an fp32 pair: the int64 fixed-point sum split into three exact
// 24-bit pieces, added by TwoSum, scaled by a power of two.
__device__ __forceinline__ void fixed_to_pair(long long v, int sexp, float& h, float& l) {
  const int a2 = (int)(v >> 48);                    // |a2| < 2^15
  const int a1 = (int)((v >> 24) & 0xffffff);
  const int a0 = (int)(v & 0xffffff);
  float s, t;
  pair_two_sum((float)a2 * 281474976710656.f, (float)a1 * 16777216.f, s, t);  // 2^48, 2^24
  float s2, t2;
  pair_two_sum(s, (float)a0, s2, t2);
  h = ldexpf(s2, -sexp);
  l = ldexpf(__fadd_rn(t, t2), -sexp);
}

// The least-squares solve of every codeword, in two kernels. stats_sum_kernel: CTA = one
// codeword; thread = (entry e of A_k's packed lower triangle or the count, slice of the
// groups). Each thread sums cnt[g][k] * H_g[e] over its slice as an unevaluated fp32 pair
// (every product is split exactly: cnt < 2^24; TwoSum for the high part), so no fp64
// arithmetic runs per group; the slices are added in a fixed order as fp32 pairs, and the
// pairs of A_k go to st.apair. stats_solve_kernel: one thread per codeword solves
// A_k c_k = b_k (b_k from the fixed point) by Cholesky with refinement in fp32 pairs. The
// summing threads carry none of the solve's registers, so every codeword's CTA is resident at
// once. The fixed assignment and order make the result identical on every run. Codewords
// without members keep their old value.
constexpr int kSolveSlices = 16;  // groups split 16 ways: short dependent chains per thread
constexpr int kSumThreads = kSolveSlices * kNA;  // 592
constexpr int kSolveThreads = 128;

__global__ void __launch_bounds__(kSumThreads, 2)
stats_sum_kernel(const float* __restrict__ Hb, StatsView st) {
  pdl_trigger();  // dependents may launch; this grid waits for its predecessor first
  pdl_wait();
  __shared__ float part_h[kSolveSlices][kNA], part_l[kSolveSlices][kNA];
  const int tid = threadIdx.x;
  const int sl = tid / kNA;
  const int e = tid % kNA;
  const int K = st.K;
  const int k = blockIdx.x;
  // entry e of the packed lower triangle: row r, column c (c <= r); e = 36 is the count
  int r = 0;
  while ((r + 1) * (r + 2) / 2 <= e && r < kD - 1) ++r;
  const int c = e - r * (r + 1) / 2;
  const int hoff = r * kD + c;
  float hi = 0.f, lo = 0.f;
  const int64_t gper = (st.G_cov + kSolveSlices - 1) / kSolveSlices;
  const int64_t g0 = sl * gper, g1 = min(st.G_cov, g0 + gper);
  constexpr int kBatch = 8;  // loads of 8 groups in flight together; no branches
  for (int64_t gb = g0; gb < g1; gb += kBatch) {
    float fc[kBatch], h[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int64_t g = gb + u;
      const bool in = g < g1;
      fc[u] = in ? (float)st.cnt[g * K + k] : 0.f;  // exact: counts stay below 2^24
      h[u] = in ? (e < 36 ? __ldg(Hb + g * kD * kD + hoff) : 1.f) : 0.f;
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const float p = __fmul_rn(fc[u], h[u]);
      const float pe = __fmaf_rn(fc[u], h[u], -p);  // fc h = p + pe exactly
      const float sum = __fadd_rn(hi, p);            // TwoSum(hi, p) = sum + t exactly
      const float bp = __fsub_rn(sum, hi);
      const float t = __fadd_rn(__fsub_rn(hi, __fsub_rn(sum, bp)), __fsub_rn(p, bp));
      hi = sum;
      lo = __fadd_rn(lo, __fadd_rn(t, pe));
    }
  }
  // Slices are merged per entry by its own thread in fp32 pairs (TwoSum of the high parts, low
  // parts added), in slice order: no serial fp64 chain (a dependent fp64 operation costs
  // about 180 cycles on this part).
  part_h[sl][e] = hi;
  part_l[sl][e] = lo;
  __syncthreads();
  // Every thread of the codeword has read its counts: clear them, so that the statistics are
  // zero for the next accumulation (the Lloyd loop needs no memset between iterations).
  if (e == 0)
    for (int64_t gq = g0; gq < g1; ++gq) st.cnt[gq * K + k] = 0;
  if (sl == 0) {
    float h = part_h[0][e], l = part_l[0][e];
    for (int s2 = 1; s2 < kSolveSlices; ++s2) {
      const float p = part_h[s2][e];
      const float sum = __fadd_rn(h, p);
      const float bp = __fsub_rn(sum, h);
      const float t = __fadd_rn(__fsub_rn(h, __fsub_rn(sum, bp)), __fsub_rn(p, bp));
      h = sum;
      l = __fadd_rn(l, __fadd_rn(t, part_l[s2][e]));
    }
    st.apair[(int64_t)k * kNA + e] = make_float2(h, l);
  }
}

__global__ void __launch_bounds__(kSolveThreads)
stats_solve_kernel(StatsView st, const float* C_old, float* C_out,
                   int32_t* __restrict__ counts_out, unsigned* err) {
  pdl_trigger();
  pdl_wait();
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= st.K) return;
  float Ah[kNA], Al[kNA];
#pragma unroll
  for (int e = 0; e < kNA; ++e) {
    const float2 v = st.apair[(int64_t)k * kNA + e];
    Ah[e] = v.x;
    Al[e] = v.y;
  }
  // the count: an exact integer held by the pair
  const int64_t count = (int64_t)__float2int_rn(Ah[36]) + (int64_t)__float2int_rn(Al[36]);
  if (counts_out) counts_out[k] = (int32_t)count;
  bool keep = count == 0;
  float out[kD];
  if (!keep) {
    const int sexp = stats_scale_exp(*st.scale);
    float bh[kD], bl[kD];
#pragma unroll
    for (int j = 0; j < kD; ++j) fixed_to_pair(st.bacc[(int64_t)k * kD + j], sexp, bh[j], bl[j]);
#pragma unroll
    for (int j = 0; j < kD; ++j) st.bacc[(int64_t)k * kD + j] = 0;  // read: clear (see above)
    if (!solve8_pairs(Ah, Al, bh, bl, out)) {
      // no fp32 factor (cond(A) beyond fp32): the fp64 Cholesky solve
      double A[36], b[kD], x[kD];
#pragma unroll
      for (int q = 0; q < 36; ++q) A[q] = (double)Ah[q] + (double)Al[q];
#pragma unroll
      for (int j = 0; j < kD; ++j) b[j] = (double)bh[j] + (double)bl[j];
      if (cholesky_solve8(A, b, x)) {
#pragma unroll
        for (int j = 0; j < kD; ++j) out[j] = (float)x[j];
      } else {
        raise_error(err, ERRBIT_NUMERIC);
        keep = true;
      }
    }
  }
  if (keep)
#pragma unroll
    for (int j = 0; j < kD; ++j) out[j] = C_old[(int64_t)k * kD + j];
#pragma unroll
  for (int j = 0; j < kD; ++j) C_out[(int64_t)k * kD + j] = out[j];
}

crvq_status launch_solve_kernels(const float* Hb, const StatsView& st, const float* C_old,
                                 float* C_out, int32_t* counts, unsigned* err,
                                 cudaStream_t stream) {
  ProfScope ps("update_solve", stream, (double)st.K);
  CRVQ_CUDA(launch_pdl(stats_sum_kernel, dim3((unsigned)st.K), dim3(kSumThreads), 0, stream,
                       Hb, st));
  CRVQ_LAUNCHED();
  CRVQ_CUDA(launch_pdl(stats_solve_kernel, dim3((unsigned)ceil_div(st.K, kSolveThreads)),
                       dim3(kSolveThreads), 0, stream, st, C_old, C_out, counts, err));
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace

crvq_status stats_alloc(Scratch& mem, int64_t G_cov, int K, StatsView* st, cudaStream_t s) {
  CRVQ_TRY(mem.alloc(stats_layout(G_cov, K).total, s));
  stats_bind(mem.as<char>(), G_cov, K, st);
  return stats_zero(*st, s);
}

crvq_status stats_zero(const StatsView& st, cudaStream_t s) {
  const StatsLayout L = stats_layout(st.G_cov, st.K);
  CRVQ_CUDA(cudaMemsetAsync(st.cnt, 0, L.cnt + L.bacc, s));
  return CRVQ_OK;
}

crvq_status launch_stats_prepare(const SetView& set, const CbList& cbs, int which,
                                 const StatsView& st, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const CbView& cw = cbs.cb[which];
  // maxbits live right after the scale (same 256-byte block).
  unsigned* maxbits = reinterpret_cast<unsigned*>(st.scale + 1);
  CRVQ_CUDA(cudaMemsetAsync(maxbits, 0, (2 + kMaxCodebooks) * sizeof(unsigned), stream));
  const int64_t n = set.M * cw.G_cov;
  const int nsm = sm_count();
  ProfScope ps("update_bound", stream, (double)n * kD * 4.0);
  maxabs_kernel<<<(unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(n, 256), 4 * nsm)),
                  256, 0, stream>>>(set, cw.G_cov, cbs, which, maxbits);
  CRVQ_LAUNCHED();
  stats_scale_kernel<<<1, 1, 0, stream>>>(maxbits, cbs.n, which, std::max<int64_t>(1, n),
                                          st.scale, err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

crvq_status launch_stats_solve(const SetView& set, const StatsView& st, const float* C_old,
                               float* C_out, int32_t* counts, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  return launch_solve_kernels(set.Hb, st, C_old, C_out, counts, err, stream);
}

crvq_status launch_update_codebook(const SetView& set, const CbList& cbs, int which,
                                   float* C_out, int32_t* counts, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const CbView& cw = cbs.cb[which];
  const int64_t n = set.M * cw.G_cov;
  Scratch mem;
  StatsView st;
  CRVQ_TRY(stats_alloc(mem, cw.G_cov, cw.K, &st, stream));
  CRVQ_TRY(launch_stats_prepare(set, cbs, which, st, stream));
  if (n > 0) {
    ProfScope ps("update_accumulate", stream, (double)n);
    const int nsm = sm_count();
    accumulate_stats_kernel<<<accumulate_grid(set.M, cw.G_cov, nsm), 256, 0, stream>>>(
        set, cbs, which, st, err);
    CRVQ_LAUNCHED();
  }
  return launch_stats_solve(set, st, cw.C, C_out, counts, stream);
}

}  // namespace crvq

namespace crvq {

// The update of launch_update_codebook on caller-provided scratch (no allocation): `scratch`
// (256-byte aligned, `bytes` long) holds cnt | bacc | scale + maxima | apair, and `err` is the error
// word the kernels report to. Returns CRVQ_ERR_UNSUPPORTED when the statistics of this
// codebook do not fit in `bytes`.
size_t update_scratch_bytes(int64_t G_cov, int K) { return stats_layout(G_cov, K).total; }

crvq_status launch_update_codebook_on(const SetView& set, const CbList& cbs, int which,
                                      float* C_out, int32_t* counts, void* scratch,
                                      size_t bytes, unsigned* err, cudaStream_t stream) {
  const CbView& cw = cbs.cb[which];
  const int64_t n = set.M * cw.G_cov;
  const size_t need = update_scratch_bytes(cw.G_cov, cw.K);
  if (need > bytes)
    return fail(CRVQ_ERR_UNSUPPORTED,
                "statistics of this codebook need %zu bytes of scratch, the limit is %zu "
                "(G_cov * K * 4 + K * 64 + 256 + K * 296 bytes, each part 256-byte aligned)",
                need, bytes);
  const StatsLayout L = stats_layout(cw.G_cov, cw.K);
  StatsView st;
  stats_bind(scratch, cw.G_cov, cw.K, &st);
  unsigned* maxbits = reinterpret_cast<unsigned*>(st.scale + 1);
  // The scratch keeps the previous call's contents: clear counts, sums and maxima.
  CRVQ_CUDA(cudaMemsetAsync(scratch, 0, L.cnt + L.bacc + L.head, stream));
  const int nsm = sm_count();
  maxabs_kernel<<<(unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(n, 256), 4 * nsm)),
                  256, 0, stream>>>(set, cw.G_cov, cbs, which, maxbits);
  CRVQ_LAUNCHED();
  stats_scale_kernel<<<1, 1, 0, stream>>>(maxbits, cbs.n, which, std::max<int64_t>(1, n),
                                          st.scale, err);
  CRVQ_LAUNCHED();
  if (n > 0) {
    accumulate_stats_kernel<<<accumulate_grid(set.M, cw.G_cov, nsm), 256, 0, stream>>>(
        set, cbs, which, st, err);
    CRVQ_LAUNCHED();
  }
  return launch_solve_kernels(set.Hb, st, cw.C, C_out, counts, err, stream);
}

}  // namespace crvq
