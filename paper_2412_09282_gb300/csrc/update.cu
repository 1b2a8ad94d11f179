// Least-squares codebook update (k-means update step; Alg. 1 FineTuneCodebook in its
// closed-form reading). For codebook `which` with all others fixed, codeword k solves
//   A_k c_k = b_k,  A_k = sum_g cnt[g][k] H_g,  b_k = sum_{v in cluster k} H_{g_v} tau_v,
//   tau_v = t_v - sum over the other covering codebooks of C[code].
//
// Deterministic by construction, with no sort and no float atomics: cnt[g][k] are integer
// counts, b_k is accumulated in 64-bit fixed point (stats.cuh), A_k is summed in fp64 in a
// fixed order (one CTA per codeword, groups split over the threads, then a fixed reduction
// tree), and the 8 x 8 system is solved by an fp64 Cholesky factorisation. The Lloyd encode
// pass (encode.cu) accumulates the same statistics for the codes it writes.
#include <algorithm>
#include <cmath>

#include "common.cuh"
#include "kernels.h"
#include "stats.cuh"

namespace crvq {

namespace {

// maxbits[0] = max |T| over the covered vectors, maxbits[1] = max row sum of |H_g|,
// maxbits[2 + s] = max |C_s| (float bits of non-negative values, merged with atomicMax).
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
    tm = fmaxf(tm, fmaxf(fmaxf(fabsf(a.x), fabsf(a.y)), fmaxf(fabsf(a.z), fabsf(a.w))));
    tm = fmaxf(tm, fmaxf(fmaxf(fabsf(b.x), fabsf(b.y)), fmaxf(fabsf(b.z), fabsf(b.w))));
  }
  float hm = 0.f;
  for (int64_t r = tid; r < G_cov * kD; r += nth) {
    const float* h = set.Hb + r * kD;
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < kD; ++j) s += fabsf(h[j]);
    hm = fmaxf(hm, s);
  }
  // warp max, then one atomic per warp
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    tm = fmaxf(tm, __shfl_xor_sync(0xffffffffu, tm, off));
    hm = fmaxf(hm, __shfl_xor_sync(0xffffffffu, hm, off));
  }
  if ((threadIdx.x & 31) == 0) {
    atomicMax(&maxbits[0], __float_as_uint(tm));
    atomicMax(&maxbits[1], __float_as_uint(hm));
  }
  for (int s = 0; s < cbs.n; ++s) {
    if (s == which) continue;
    float m = 0.f;
    for (int64_t e = tid; e < (int64_t)cbs.cb[s].K * kD; e += nth)
      m = fmaxf(m, fabsf(cbs.cb[s].C[e]));
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
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

__global__ void __launch_bounds__(256)
accumulate_stats_kernel(SetView set, CbList cbs, int which, StatsView st, unsigned* err) {
  const CbView cw = cbs.cb[which];
  const int64_t n = set.M * cw.G_cov;
  const double scale = *st.scale;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < n;
       v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = v / cw.G_cov, g = v % cw.G_cov;
    const int32_t k = cw.codes[i * cw.ld + g];
    if (k < 0 || k >= cw.K) {
      raise_error(err, ERRBIT_INDEX);
      continue;
    }
    float tau[kD], q[kD];
    stats_target(set, cbs, which, i, g, tau, err);
    stats_htau(set.Hb + g * kD * kD, tau, q);
    stats_add(st, scale, g, k, q);
  }
}

// One CTA per codeword: A_k = sum_g cnt[g][k] H_g in fp64 (groups strided over the threads,
// then a fixed warp-shuffle + shared-memory tree), b_k from the fixed point, Cholesky solve.
constexpr int kSolveThreads = 128;

__global__ void __launch_bounds__(kSolveThreads)
stats_solve_kernel(const float* __restrict__ Hb, int64_t G_cov, int K, StatsView st,
                   const float* __restrict__ C_old, float* __restrict__ C_out,
                   int32_t* __restrict__ counts_out, unsigned* err) {
  __shared__ double part[kSolveThreads / 32][37];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int k = blockIdx.x; k < K; k += gridDim.x) {
    double A[37];
#pragma unroll
    for (int j = 0; j < 37; ++j) A[j] = 0.0;
    for (int64_t g = threadIdx.x; g < G_cov; g += blockDim.x) {
      const int c = st.cnt[g * K + k];
      if (c == 0) continue;
      A[36] += (double)c;
      const float* H = Hb + g * kD * kD;
      int q = 0;
#pragma unroll
      for (int r = 0; r < kD; ++r)
#pragma unroll
        for (int cc = 0; cc <= r; ++cc) A[q++] += (double)c * (double)H[r * kD + cc];
    }
#pragma unroll
    for (int j = 0; j < 37; ++j)
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) A[j] += __shfl_xor_sync(0xffffffffu, A[j], off);
    __syncthreads();
    if (lane == 0)
      for (int j = 0; j < 37; ++j) part[warp][j] = A[j];
    __syncthreads();
    if (threadIdx.x == 0) {
      for (int w = 1; w < kSolveThreads / 32; ++w)
        for (int j = 0; j < 37; ++j) A[j] += part[w][j];
      const int64_t count = (int64_t)A[36];
      if (counts_out) counts_out[k] = (int32_t)count;
      bool keep = count == 0;
      if (!keep) {
        const double scale = *st.scale;
        double b[kD], x[kD];
        for (int j = 0; j < kD; ++j) b[j] = (double)st.bacc[(int64_t)k * kD + j] / scale;
        if (cholesky_solve8(A, b, x)) {
          for (int j = 0; j < kD; ++j) C_out[(int64_t)k * kD + j] = (float)x[j];
        } else {
          raise_error(err, ERRBIT_NUMERIC);
          keep = true;
        }
      }
      if (keep)
        for (int j = 0; j < kD; ++j) C_out[(int64_t)k * kD + j] = C_old[(int64_t)k * kD + j];
    }
  }
}

}  // namespace

crvq_status stats_alloc(Scratch& mem, int64_t G_cov, int K, StatsView* st, cudaStream_t s) {
  const size_t cnt_bytes = align_up((size_t)std::max<int64_t>(G_cov, 1) * K * sizeof(int32_t), 256);
  const size_t b_bytes = align_up((size_t)K * kD * sizeof(long long), 256);
  const size_t max_bytes = 256;  // maxbits[2 + kMaxCodebooks] + scale
  CRVQ_TRY(mem.alloc(cnt_bytes + b_bytes + max_bytes, s));
  st->cnt = mem.as<int32_t>();
  st->bacc = reinterpret_cast<long long*>(mem.as<char>() + cnt_bytes);
  st->scale = reinterpret_cast<double*>(mem.as<char>() + cnt_bytes + b_bytes);
  st->G_cov = G_cov;
  st->K = K;
  return stats_zero(*st, s);
}

crvq_status stats_zero(const StatsView& st, cudaStream_t s) {
  const size_t cnt_bytes = align_up((size_t)std::max<int64_t>(st.G_cov, 1) * st.K * sizeof(int32_t), 256);
  const size_t b_bytes = align_up((size_t)st.K * kD * sizeof(long long), 256);
  CRVQ_CUDA(cudaMemsetAsync(st.cnt, 0, cnt_bytes + b_bytes, s));
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
  ProfScope ps("update_solve", stream, (double)st.K);
  const int blocks = (int)std::min<int64_t>(st.K, 64 * sm_count());
  stats_solve_kernel<<<blocks, kSolveThreads, 0, stream>>>(set.Hb, st.G_cov, st.K, st, C_old,
                                                           C_out, counts, err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
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
    accumulate_stats_kernel<<<(unsigned)std::min<int64_t>(ceil_div(n, 256), 16 * nsm), 256, 0,
                              stream>>>(set, cbs, which, st, err);
    CRVQ_LAUNCHED();
  }
  return launch_stats_solve(set, st, cw.C, C_out, counts, stream);
}

}  // namespace crvq

namespace crvq {

// The update of launch_update_codebook on caller-provided scratch (no allocation): `scratch`
// (256-byte aligned, `bytes` long) holds cnt | bacc | scale + maxima, and `err` is the error
// word the kernels report to. Returns CRVQ_ERR_UNSUPPORTED when the statistics of this
// codebook do not fit in `bytes`.
size_t update_scratch_bytes(int64_t G_cov, int K) {
  return align_up((size_t)std::max<int64_t>(G_cov, 1) * K * sizeof(int32_t), 256) +
         align_up((size_t)K * kD * sizeof(long long), 256) + 256;
}

crvq_status launch_update_codebook_on(const SetView& set, const CbList& cbs, int which,
                                      float* C_out, int32_t* counts, void* scratch,
                                      size_t bytes, unsigned* err, cudaStream_t stream) {
  const CbView& cw = cbs.cb[which];
  const int64_t n = set.M * cw.G_cov;
  const size_t need = update_scratch_bytes(cw.G_cov, cw.K);
  if (need > bytes)
    return fail(CRVQ_ERR_UNSUPPORTED,
                "statistics of this codebook need %zu bytes of scratch, the limit is %zu "
                "(G_cov * K * 4 + K * 64 + 512 bytes)",
                need, bytes);
  const size_t cnt_bytes = align_up((size_t)std::max<int64_t>(cw.G_cov, 1) * cw.K * sizeof(int32_t), 256);
  const size_t b_bytes = align_up((size_t)cw.K * kD * sizeof(long long), 256);
  StatsView st;
  st.cnt = static_cast<int32_t*>(scratch);
  st.bacc = reinterpret_cast<long long*>(static_cast<char*>(scratch) + cnt_bytes);
  st.scale = reinterpret_cast<double*>(static_cast<char*>(scratch) + cnt_bytes + b_bytes);
  st.G_cov = cw.G_cov;
  st.K = cw.K;
  unsigned* maxbits = reinterpret_cast<unsigned*>(st.scale + 1);
  // The scratch keeps the previous call's contents: clear counts, sums and maxima.
  CRVQ_CUDA(cudaMemsetAsync(scratch, 0, cnt_bytes + b_bytes + 256, stream));
  const int nsm = sm_count();
  maxabs_kernel<<<(unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(n, 256), 4 * nsm)),
                  256, 0, stream>>>(set, cw.G_cov, cbs, which, maxbits);
  CRVQ_LAUNCHED();
  stats_scale_kernel<<<1, 1, 0, stream>>>(maxbits, cbs.n, which, std::max<int64_t>(1, n),
                                          st.scale, err);
  CRVQ_LAUNCHED();
  if (n > 0) {
    accumulate_stats_kernel<<<(unsigned)std::min<int64_t>(ceil_div(n, 256), 16 * nsm), 256, 0,
                              stream>>>(set, cbs, which, st, err);
    CRVQ_LAUNCHED();
  }
  stats_solve_kernel<<<(int)std::min<int64_t>(st.K, 64 * nsm), kSolveThreads, 0, stream>>>(
      set.Hb, st.G_cov, st.K, st, cw.C, C_out, counts, err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace crvq
