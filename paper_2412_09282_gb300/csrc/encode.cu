// Vector x codeword score contraction with fused top-B selection (Sec. 3.1 Eq. (2)-(3);
// Alg. 1 VectorQuant and BeamSearchOptimize), and the k-means initial codebook draw.
//
// Score of target r against codeword c for a vector of group g:
//   err(r, c) = (r - c)^T H_g (r - c) = r^T H_g r + n_g(c) - 2 (H_g r) . c,  n_g(c) = c^T H_g c.
// The fast pass evaluates the expanded form in fp32 (8 FMAs per pair; the codewords, their
// group norms and L1 norms staged in shared memory). Every fp32 score s_k comes with an
// a-priori bound on its rounding error,
//   E_k <= Et_k = u C (Na_k + 2 Pmax L1_k),   u = 2^-24,
//   Na_k = |c_k|^T |H_g| |c_k|,  L1_k = ||c_k||_1,  Pmax = max_p sum_j |H_pj| (|t_j| + sum_f |c_f,j|),
// and the pass ranks the lower bounds low_k = s_k - Et_k, keeping the best two. The arg-min j
// is certified when low_2nd - low_j > 2 Et_j: every other codeword's exact score is then larger
// than j's. Otherwise the vector is flagged; a fallback re-scores it, keeps the codewords with
// low_k <= low_j + 2 Et_j (the exact arg-min is among them) and decides among those in fp64.
// Codes therefore equal the fp64 arg-min (ties to the smaller index) except for ties at fp64
// rounding level. Beam stages use the same bounds on a sorted top-(B+1) list.
#include <algorithm>
#include <cstdlib>
#include <type_traits>
#include <vector>

#include "common.cuh"
#include "kernels.h"
#include "stats.cuh"
#include "tc_ops.cuh"

namespace crvq {

namespace {

constexpr int kThreads = 128;
constexpr int kChunk = 256;             // codewords staged per shared-memory chunk
constexpr float kU = 5.9604645e-08f;    // 2^-24

// Error-bound multiplier: about twice the worst-case FMA-chain analysis (<= 37 + 2 n_fixed).
__host__ __device__ inline float bound_mult(int n_terms) { return 64.f + 4.f * n_terms; }

struct FlagList {
  int64_t* vec;      // vector index within the launch range (i * G_range + (g - g_begin))
  float* thr;        // decision threshold (fast-pass value units)
  unsigned* count;
  int64_t cap;
  unsigned long long* total;  // optional running total of flagged vectors
};

// --------------------------------------------------------------------------- device helpers
__device__ __forceinline__ void load_vec(const float* p, float v[kD]) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

__device__ __forceinline__ bool code_ok(int32_t k, int32_t K, unsigned* err) {
  if (k < 0 || k >= K) {
    raise_error(err, ERRBIT_INDEX);
    return false;
  }
  return true;
}

// fp32 target r = t - sum of the fixed codebooks covering g (codebook order), and the
// magnitude bound a_j = |t_j| + sum |c_fixed,j| of every term that went into r.
__device__ __forceinline__ void target32(const SetView& set, const CbList& cbs, int n_fixed,
                                         int64_t i, int64_t g, float r[kD], float a[kD],
                                         unsigned* err) {
  load_vec(set.T + i * set.ldT + g * kD, r);
#pragma unroll
  for (int j = 0; j < kD; ++j) a[j] = fabsf(r[j]);
  for (int s = 0; s < n_fixed; ++s) {
    const CbView& cb = cbs.cb[s];
    if (g >= cb.G_cov) continue;
    const int32_t k = cb.codes[i * cb.ld + g];
    if (!code_ok(k, cb.K, err)) continue;
    float c[kD];
    load_vec(cb.C + (int64_t)k * kD, c);
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      r[j] -= c[j];
      a[j] += fabsf(c[j]);
    }
  }
}

// fp64 target (the fixed reconstruction subtracted in fp64, codebook order).
__device__ void target64(const SetView& set, const CbList& cbs, int n_fixed, int64_t i,
                         int64_t g, double r[kD], unsigned* err) {
  const float* t = set.T + i * set.ldT + g * kD;
#pragma unroll
  for (int j = 0; j < kD; ++j) r[j] = (double)t[j];
  for (int s = 0; s < n_fixed; ++s) {
    const CbView& cb = cbs.cb[s];
    if (g >= cb.G_cov) continue;
    const int32_t k = cb.codes[i * cb.ld + g];
    if (!code_ok(k, cb.K, err)) continue;
    const float* c = cb.C + (int64_t)k * kD;
#pragma unroll
    for (int j = 0; j < kD; ++j) r[j] -= (double)c[j];
  }
}

// (r - c)^T H (r - c) in fp64; H row-major d x d (fp32); c fp32 or null.
__device__ double quad_err64(const double r[kD], const float* c, const float* H) {
  double dlt[kD];
#pragma unroll
  for (int j = 0; j < kD; ++j) dlt[j] = r[j] - (c ? (double)c[j] : 0.0);
  double e = 0.0;
#pragma unroll
  for (int b = 0; b < kD; ++b) {
    double hb = 0.0;
#pragma unroll
    for (int a2 = 0; a2 < kD; ++a2) hb += dlt[a2] * (double)H[a2 * kD + b];
    e += hb * dlt[b];
  }
  return e;
}

// Codeword terms of the score and of its bound: n = c^T H c (fp32, two FMA chains),
// na = |c|^T |H| |c|, l1 = ||c||_1.
__device__ __forceinline__ void codeword_terms(const float c[kD], const float* H, float& n,
                                               float& na, float& l1) {
  n = 0.f;
  na = 0.f;
  l1 = 0.f;
#pragma unroll
  for (int a = 0; a < kD; ++a) {
    float u = 0.f, ua = 0.f;
#pragma unroll
    for (int b = 0; b < kD; ++b) {
      u = fmaf(H[a * kD + b], c[b], u);
      ua = fmaf(fabsf(H[a * kD + b]), fabsf(c[b]), ua);
    }
    n = fmaf(c[a], u, n);
    na = fmaf(fabsf(c[a]), ua, na);
    l1 += fabsf(c[a]);
  }
}

// Vector terms: m2q = -2 H r (the row FMA chains of stats_htau), Pmax = max_p (|H| a)_p.
__device__ __forceinline__ void vector_terms(const float r[kD], const float a[kD],
                                             const float* H, float m2q[kD], float& pmax) {
  pmax = 0.f;
#pragma unroll
  for (int p = 0; p < kD; ++p) {
    float q = 0.f, pa = 0.f;
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      q = fmaf(H[p * kD + j], r[j], q);
      pa = fmaf(fabsf(H[p * kD + j]), a[j], pa);
    }
    m2q[p] = -2.f * q;
    pmax = fmaxf(pmax, pa);
  }
}

// vector_terms plus rr = r^T (H r) and Ra = a^T (|H| a), each row of H read once as two
// float4 (H 16-byte aligned): the same FMA chains, so the same values as computing them apart.
__device__ __forceinline__ void vector_terms_rr(const float r[kD], const float a[kD],
                                                const float* H, float m2q[kD], float& pmax,
                                                float& rr, float& ra) {
  pmax = 0.f;
  rr = 0.f;
  ra = 0.f;
#pragma unroll
  for (int p = 0; p < kD; ++p) {
    const float4 h0 = *reinterpret_cast<const float4*>(H + p * kD);
    const float4 h1 = *reinterpret_cast<const float4*>(H + p * kD + 4);
    const float hr[kD] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
    float q = 0.f, pa = 0.f;
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      q = fmaf(hr[j], r[j], q);
      pa = fmaf(fabsf(hr[j]), a[j], pa);
    }
    m2q[p] = -2.f * q;
    pmax = fmaxf(pmax, pa);
    rr = fmaf(r[p], q, rr);
    ra = fmaf(a[p], pa, ra);
  }
}

// Stage the codewords [k0, k0 + nk): sC = c, sNL = (n - u C Na, ||c||_1) (the lower-bound
// offset of the codeword part and its L1 norm), sNa = Na.
__device__ __forceinline__ void stage_chunk(const float* __restrict__ C, int k0, int nk,
                                            const float* sH, float cmul, float* sC, float2* sNL,
                                            float* sNa) {
  for (int k = threadIdx.x; k < nk; k += blockDim.x) {
    float c[kD];
    load_vec(C + (int64_t)(k0 + k) * kD, c);
    float n, na, l1;
    codeword_terms(c, sH, n, na, l1);
    *reinterpret_cast<float4*>(sC + k * kD) = make_float4(c[0], c[1], c[2], c[3]);
    *reinterpret_cast<float4*>(sC + k * kD + 4) = make_float4(c[4], c[5], c[6], c[7]);
    sNL[k] = make_float2(n - kU * cmul * na, l1);
    sNa[k] = na;
  }
}

// fp32 lower / upper bounds s_k -+ Et_k of the score of codeword k from its terms t = (n, Na,
// L1) (codeword_terms): s_k = n + sum_p m2q_p c_p, Et_k = u C (Na + 2 Pmax L1). Any
// evaluation covered by the same error analysis is a valid bound; the fallback needs no more.
__device__ __forceinline__ float low_from(float n, float na, float l1, const float c[kD],
                                          const float m2q[kD], float nbeta, float cmul) {
  float s = fmaf(-kU * cmul, na, n);
#pragma unroll
  for (int p = 0; p < kD; ++p) s = fmaf(m2q[p], c[p], s);
  return fmaf(nbeta, l1, s);
}

__device__ __forceinline__ float up_from(float n, float na, float l1, const float c[kD],
                                         const float m2q[kD], float pmax, float cmul) {
  float s = fmaf(kU * cmul, na, n);
#pragma unroll
  for (int p = 0; p < kD; ++p) s = fmaf(m2q[p], c[p], s);
  return fmaf(2.f * kU * cmul * pmax, l1, s);
}

__device__ __forceinline__ float low_score(const float c[kD], const float* H, const float m2q[kD],
                                           float nbeta, float cmul) {
  float n, na, l1;
  codeword_terms(c, H, n, na, l1);
  return low_from(n, na, l1, c, m2q, nbeta, cmul);
}

// --------------------------------------------------------------------------- arg-min pass on
// the tensor cores. The whole certified lower bound is one dot product of length 32:
//   D[v][k] = sum_p q_vp c_kp + n'_k + beta_v L1_k + off_v = low_k(v) + off_v,
//   q = -2 H_g r, n' = n - u C Na, beta = -2 u C Pmax, off >= r^T H r + bound (so D >= 0),
// with every term split into tf32 hi + lo (3xTF32: hi*hi + hi*lo + lo*hi):
//   A row (vector):   [q_hi x8 | q_hi x8 | q_lo x8 | 1 1 | beta_hi beta_hi beta_lo | off_hi off_lo | 0]
//   B row (codeword): [c_hi x8 | c_lo x8 | c_hi x8 | n'_hi n'_lo | L1_hi L1_lo L1_hi | 1 1 | 0]
// One tcgen05.mma M = 128 vectors x N = 128 codewords x K = 8, four per chunk (K = 32), fp32
// accumulator in tensor memory. The epilogue reads each row's scores in blocks of 16: per block
// its minimum (integer minima of the non-negative fp32 bit patterns); per row the block with the
// smallest minimum, kept whole, and the second smallest block minimum. The row's winner and
// second smallest score come from those 17 values, exact (no packed index). The certificate and
// the fp64 fallback are those of the fp32 pass, with the bound multiplier raised to cover the
// tensor-core products and accumulation (about 2^-22 per split product and fp32 accumulation
// over 32 terms).
namespace tcenc {

constexpr int kRows = 128;        // vectors per row tile (TMEM lanes)
constexpr int kK = 32;            // tf32 columns per row
constexpr int kATile = kRows * kK * 4;   // 16 KB
constexpr float kCmul = 256.f;           // bound multiplier (about twice the analysis)

__device__ __forceinline__ uint32_t koff(int r, int k) {
  return (uint32_t)(((r >> 3) * (kK / 4) + (k >> 2)) * 128 + (r & 7) * 16 + (k & 3) * 4);
}

// Writes the 32 tf32 values v[0..31] of row r (hi parts given as fp32 values).
__device__ __forceinline__ void put_row(char* tile, int r, const uint32_t v[kK]) {
#pragma unroll
  for (int q = 0; q < kK / 4; ++q)
    *reinterpret_cast<uint4*>(tile + koff(r, 4 * q)) =
        make_uint4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
}

__device__ __forceinline__ void split(float x, uint32_t& hi, uint32_t& lo) {
  hi = tc::to_tf32(x);
  lo = tc::to_tf32(x - __uint_as_float(hi));
}

}  // namespace tcenc

// Row of the B operand for codeword kk of C (K codewords): [c_hi | c_lo | c_hi | n'_hi n'_lo |
// L1_hi L1_lo L1_hi | 1 1 | 0]; padding rows (kk >= K) score +1e30.
__device__ __forceinline__ void build_b_row(const float* __restrict__ C, int K, int kk,
                                            const float* H, float uc, uint32_t row[tcenc::kK]) {
  using namespace tcenc;
  if (kk < K) {
    float cv[kD], n, na, l1;
    load_vec(C + (int64_t)kk * kD, cv);
    codeword_terms(cv, H, n, na, l1);
#pragma unroll
    for (int p = 0; p < kD; ++p) {
      uint32_t hh, ll;
      split(cv[p], hh, ll);
      row[p] = hh;
      row[8 + p] = ll;
      row[16 + p] = hh;
    }
    split(n - uc * na, row[24], row[25]);
    split(l1, row[26], row[27]);
    row[28] = row[26];
  } else {
#pragma unroll
    for (int p = 0; p < 24; ++p) row[p] = 0u;
    row[24] = __float_as_uint(1e30f);
    row[25] = 0u;
    row[26] = row[27] = row[28] = 0u;
  }
  row[29] = row[30] = __float_as_uint(1.f);
  row[31] = 0u;
}

// cbmax[0] = max_k ||c_k||_1 (raised by 1e-6 relative), cbmax[1] = max_k,j |c_kj|: one CTA
// of any size up to 1024 threads (maxima are order-free).
__device__ void cbmax_block(const float* __restrict__ C, int K, float* __restrict__ cbmax) {
  __shared__ float r1[32], r2[32];
  float l1m = 0.f, cm = 0.f;
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    float c[kD];
    load_vec(C + (int64_t)k * kD, c);
    float l1 = 0.f;
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      l1 += fabsf(c[j]);
      cm = fmaxf(cm, fabsf(c[j]));
    }
    l1m = fmaxf(l1m, l1);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    l1m = fmaxf(l1m, __shfl_xor_sync(0xffffffffu, l1m, off));
    cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, off));
  }
  if ((threadIdx.x & 31) == 0) {
    r1[threadIdx.x >> 5] = l1m;
    r2[threadIdx.x >> 5] = cm;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < (int)((blockDim.x + 31) >> 5); ++w) {
      l1m = fmaxf(l1m, r1[w]);
      cm = fmaxf(cm, r2[w]);
    }
    cbmax[0] = l1m * (1.f + 1e-6f);
    cbmax[1] = cm;
  }
}

constexpr int kTcCols = 128;                     // codewords per chunk (MMA N)
constexpr int kTcBTile = kTcCols * tcenc::kK * 4;  // 16 KB

// B operand images of the codebook for groups [g_begin, g_begin + G_range): block
// (g, chunk) holds 128 rows in the canonical shared-memory layout, ready for a bulk copy.
// terms[(g - g_begin) K + k] = (n, Na, L1, 0) of codeword k in group g (codeword_terms).
__global__ void __launch_bounds__(128)
prep_b_kernel(SetView set, int64_t g_begin, int64_t G_range, const float* __restrict__ C,
              int K, int nchunk, float uc, char* __restrict__ out, float4* __restrict__ terms,
              float* __restrict__ cbmax, unsigned* __restrict__ flag_count) {
  pdl_trigger();  // dependents may launch; this grid waits for its predecessor first
  pdl_wait();
  // The flag list of the arg-min pass that follows starts empty. The previous pass's exact
  // kernel, which read the count, completed before the wait above returned.
  if (blockIdx.x == 0 && threadIdx.x == 0) *flag_count = 0u;
  if (blockIdx.x == gridDim.x - 1) {  // the last CTA: the codebook maxima
    cbmax_block(C, K, cbmax);
    return;
  }
  const int64_t total = G_range * nchunk * (int64_t)kTcCols;
  const int64_t nth = (int64_t)(gridDim.x - 1) * blockDim.x;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += nth) {
    const int row = (int)(e % kTcCols);
    const int64_t blk = e / kTcCols;  // g_rel * nchunk + chunk
    const int chunk = (int)(blk % nchunk);
    const int64_t g = g_begin + blk / nchunk;
    uint32_t v[tcenc::kK];
    const int kk = chunk * kTcCols + row;
    build_b_row(C, K, kk, set.Hb + g * kD * kD, uc, v);
    tcenc::put_row(out + blk * kTcBTile, row, v);
    if (kk < K) {
      float cv[kD], n, na, l1;
      load_vec(C + (int64_t)kk * kD, cv);
      codeword_terms(cv, set.Hb + g * kD * kD, n, na, l1);
      terms[(g - g_begin) * K + kk] = make_float4(n, na, l1, 0.f);
    }
  }
}

// Exact scoring in unevaluated fp32 pairs ("double-float"): GB300's fp64 pipe is a small
// fraction of its fp32 rate, so the few decisions that the certified bounds leave open are
// settled with error-free transformations (Knuth's TwoSum, the FMA-based TwoProduct) on the
// fp32 pipe instead. The residual r = t - sum of the fixed codewords is held exactly as
// rh + rl; the err (r - c)^T H (r - c) comes out within a few 2^-48 of |r - c|^T |H| |r - c|,
// far inside the near-tie margin at which fp64 itself stops deciding.
namespace dfl {

__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
  s = __fadd_rn(a, b);
  const float bp = __fsub_rn(s, a);
  e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bp)), __fsub_rn(b, bp));
}

// (rh + rl) = t - sum of the fixed codebooks' codewords covering g (codebook order).
__device__ __forceinline__ void target(const SetView& set, const CbList& cbs, int n_fixed,
                                       int64_t i, int64_t g, float rh[kD], float rl[kD],
                                       unsigned* err) {
  load_vec(set.T + i * set.ldT + g * kD, rh);
#pragma unroll
  for (int j = 0; j < kD; ++j) rl[j] = 0.f;
  for (int s = 0; s < n_fixed; ++s) {
    const CbView& cb = cbs.cb[s];
    if (g >= cb.G_cov) continue;
    const int32_t k = cb.codes[i * cb.ld + g];
    if (!code_ok(k, cb.K, err)) continue;
    float c[kD];
    load_vec(cb.C + (int64_t)k * kD, c);
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      float sj, ej;
      two_sum(rh[j], -c[j], sj, ej);
      rh[j] = sj;
      rl[j] = __fadd_rn(rl[j], ej);
    }
  }
}

// err = (r - c)^T H (r - c) as a normalised pair (eh, el), r = rh + rl.
__device__ __forceinline__ void quad_err(const float rh[kD], const float rl[kD],
                                         const float c[kD], const float* H, float& eh,
                                         float& el) {
  float dh[kD], dl[kD];
#pragma unroll
  for (int j = 0; j < kD; ++j) {
    float e;
    two_sum(rh[j], -c[j], dh[j], e);
    dl[j] = __fadd_rn(rl[j], e);
  }
  float yh[kD], yl[kD];
#pragma unroll
  for (int b = 0; b < kD; ++b) yh[b] = yl[b] = 0.f;
#pragma unroll
  for (int a = 0; a < kD; ++a)
#pragma unroll
    for (int b = 0; b < kD; ++b) {
      const float h = H[a * kD + b];
      const float p = __fmul_rn(dh[a], h);
      const float pe = __fmaf_rn(dh[a], h, -p);  // dh h = p + pe exactly
      float s, t;
      two_sum(yh[b], p, s, t);
      yh[b] = s;
      yl[b] = __fadd_rn(yl[b], __fadd_rn(t, __fmaf_rn(dl[a], h, pe)));
    }
  float sh = 0.f, sl = 0.f;
#pragma unroll
  for (int b = 0; b < kD; ++b) {
    const float p = __fmul_rn(dh[b], yh[b]);
    const float pe = __fmaf_rn(dh[b], yh[b], -p);
    float s, t;
    two_sum(sh, p, s, t);
    sh = s;
    sl = __fadd_rn(sl, __fadd_rn(t, __fmaf_rn(dh[b], yl[b], __fmaf_rn(dl[b], yh[b], pe))));
  }
  eh = __fadd_rn(sh, sl);
  el = __fsub_rn(sl, __fsub_rn(eh, sh));
}

__device__ __forceinline__ bool less(float ah, float al, int ak, float bh, float bl, int bk) {
  return ah < bh || (ah == bh && (al < bl || (al == bl && ak < bk)));
}

}  // namespace dfl

// Per-vector terms of the arg-min's A rows that do not change while one codebook's Lloyd
// iterations run (the target, H_g and the fixed codebooks stay put): m2q = -2 H_g r and rr,
// Ra, Pmax (vector_terms_rr of target32), as three planes of M float4 per group,
// rt[(3 g + p) M + i]: p = 0, 1 the two halves of m2q, p = 2 (rr, Ra, Pmax, 0). The arg-min
// pass reads them instead of recomputing them, with bit-identical values.
__global__ void __launch_bounds__(128)
row_terms_kernel(SetView set, CbList cbs, int n_fixed, float4* __restrict__ rt,
                 unsigned* err) {
  pdl_trigger();
  pdl_wait();
  const int64_t nvec = set.M * set.G_sub;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < nvec;
       v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t g = v / set.M, i = v - g * set.M;
    float rv[kD], a[kD], m2q[kD], pmax, rr, ra;
    target32(set, cbs, n_fixed, i, g, rv, a, err);
    vector_terms_rr(rv, a, set.Hb + g * kD * kD, m2q, pmax, rr, ra);  // H_g 16-byte aligned
    rt[(3 * g) * set.M + i] = make_float4(m2q[0], m2q[1], m2q[2], m2q[3]);
    rt[(3 * g + 1) * set.M + i] = make_float4(m2q[4], m2q[5], m2q[6], m2q[7]);
    rt[(3 * g + 2) * set.M + i] = make_float4(rr, ra, pmax, 0.f);
  }
}

// Arg-min over one codebook on the tensor cores. A CTA walks `tiles` consecutive row tiles of
// one group (thread = row = tensor-memory lane) with a 128-column accumulator per tile in
// flight. HALVES = 1: 128 threads, three CTAs per SM, any codebook size (codeword chunks of 128
// come from the precomputed B images by bulk copy; with at most two chunks they stay resident
// for all the CTA's tiles). HALVES = 2 (codebooks of at most 256 codewords): 256 threads in two
// halves of 128 that run independently (each its own tiles, named barriers, MMA issue and
// accumulator) and share the resident codebook operand and the statistics; two CTAs per SM,
// so four tile pipelines per SM interleave their phases (A rows, MMA, epilogue, certificate).
// The sweep keeps per row the 16-column block with the smallest minimum and the second
// smallest block minimum. Rows the bounds do not certify go to the flag list (decided exactly
// by the exact kernels). The Lloyd statistics of certified rows are summed
// in shared memory (integer atomics, [component][code] so that a warp's lanes hit spread banks)
// and flushed once.
constexpr int kTcSmemStatsK = 256;  // codebooks up to this size aggregate statistics in smem

// Minimum of 16 non-negative fp32 values by their bit patterns (which order like the values),
// as three-input integer minima.
__device__ __forceinline__ uint32_t min16_bits(const uint32_t* x) {
  const uint32_t a = __vimin3_u32(x[0], x[1], x[2]), b = __vimin3_u32(x[3], x[4], x[5]),
                 c = __vimin3_u32(x[6], x[7], x[8]), d = __vimin3_u32(x[9], x[10], x[11]),
                 e = __vimin3_u32(x[12], x[13], x[14]);
  return min(__vimin3_u32(a, b, c), __vimin3_u32(d, e, x[15]));
}

constexpr int kBlk = 16;  // columns per block of the arg-min sweep

// dynamic shared memory of argmin_tc_kernel<HALVES>: A tiles, two B chunks, statistics, H r,
// with two halves the codeword terms (Na, L1) of the group, alignment
constexpr size_t argmin_smem(int halves) {
  return (size_t)halves * tcenc::kATile + 2 * (size_t)kTcBTile +
         (size_t)kTcSmemStatsK * (kD * 8 + 4) + (size_t)halves * tcenc::kRows * kD * 4 +
         (halves == 2 ? (size_t)kTcSmemStatsK * 8 : 0) + 1024;
}

// Barrier over this half's 128 threads (named barrier 1 + half), or the whole CTA.
template <int HALVES>
__device__ __forceinline__ void half_sync(int half) {
  if (HALVES == 1) {
    __syncthreads();
  } else {
    asm volatile("bar.sync %0, 128;" ::"r"(1 + half) : "memory");
  }
}

template <int HALVES>
__device__ __forceinline__ bool half_sync_and(int half, bool v) {
  if (HALVES == 1) return __syncthreads_and(v);
  int r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.b32 q, %1, 0;\n bar.red.and.pred p, %2, 128, q;\n"
      " selp.s32 %0, 1, 0, p;\n}\n"
      : "=r"(r)
      : "r"((int)v), "r"(1 + half)
      : "memory");
  return r != 0;
}

template <int HALVES>
__global__ void __launch_bounds__(128 * HALVES, HALVES == 1 ? 3 : 2)
argmin_tc_kernel(SetView set, int64_t g_begin, CbList cbs, int n_fixed, int s_idx,
                 int32_t* __restrict__ out_code, int64_t out_ld, int64_t out_g0,
                 FlagList flags, StatsView st, const float* __restrict__ cbmax,
                 const char* __restrict__ bpre, const float4* __restrict__ terms,
                 const float4* __restrict__ rowterms, int tiles, unsigned* err) {
  pdl_trigger();  // dependents may launch; this grid waits for its predecessor first
  pdl_wait();
  using namespace tcenc;
  extern __shared__ __align__(1024) char smem_raw[];
  // 1024-byte aligned base, derived from the shared array (keeps the shared address space)
  char* smem = smem_raw + ((1024u - (tc::smem_u32(smem_raw) & 1023u)) & 1023u);
  char* Atiles = smem;                          // HALVES x 16 KB
  char* Bbuf = smem + HALVES * kATile;          // 2 x 16 KB
  long long* s_bacc = reinterpret_cast<long long*>(Bbuf + 2 * kTcBTile);  // [8][256]
  int* s_cnt = reinterpret_cast<int*>(s_bacc + kTcSmemStatsK * kD);       // [256]
  float* sQ = reinterpret_cast<float*>(s_cnt + kTcSmemStatsK);            // [128 HALVES][8]
  float2* sNaL1 = reinterpret_cast<float2*>(sQ + HALVES * kRows * kD);     // [256] (2 halves)
  __shared__ __align__(16) float sH[kD * kD];
  __shared__ __align__(8) uint64_t bar_mma_s[HALVES], bar_b[2];
  __shared__ uint32_t tmem_slot;

  const int64_t g = g_begin + blockIdx.y;
  const int64_t G_range = gridDim.y;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int half = HALVES == 1 ? 0 : (tid >> 7), rrow = tid & (kRows - 1);
  char* Atile = Atiles + half * kATile;
  uint64_t& bar_mma = bar_mma_s[half];
  const CbView cw = cbs.cb[s_idx];
  const float cmul = kCmul + 4.f * n_fixed;
  const float uc = kU * cmul;
  const int nchunk = (cw.K + kTcCols - 1) / kTcCols;
  const bool resident = nchunk <= 2;
  const char* bimg = bpre ? bpre + (size_t)(g - g_begin) * nchunk * kTcBTile : nullptr;
  const float4* gterms = terms ? terms + (g - g_begin) * cw.K : nullptr;
  const bool smem_stats = st.cnt && cw.K <= kTcSmemStatsK;

  if (tid < kD * kD) sH[tid] = set.Hb[g * kD * kD + tid];
  if (smem_stats) {
    for (int e = tid; e < kTcSmemStatsK * kD; e += blockDim.x) s_bacc[e] = 0;  // (= s_b32)
    for (int e = tid; e < kTcSmemStatsK; e += blockDim.x) s_cnt[e] = 0;
  }
  // Statistics terms (|v| < 2^30) split as v = 2^15 vh + vl, 0 <= vl < 2^15, into two 32-bit
  // shared sums [component][vh, vl][code] (native 32-bit atomics instead of 64-bit ones): exact,
  // since the host gives a CTA with these sums fewer than 2^16 rows (|sum| < 2^31).
  int* s_b32 = reinterpret_cast<int*>(s_bacc);  // [8][2][256] in the 64-bit sums' space
  // the winner's terms for the certificate, from shared memory (K <= 256 with two halves)
  const bool smem_terms = HALVES == 2 && gterms != nullptr;
  if (smem_terms)
    for (int k = tid; k < cw.K; k += blockDim.x) {
      const float4 tk = gterms[k];
      sNaL1[k] = make_float2(tk.y, tk.z);
    }
  if (warp == 0) tc::tmem_alloc(&tmem_slot, HALVES * kTcCols);
  if (tid == 0) {
    for (int h = 0; h < HALVES; ++h) tc::mbar_init(tc::smem_u32(&bar_mma_s[h]), 1);
    tc::mbar_init(tc::smem_u32(&bar_b[0]), 1);
    tc::mbar_init(tc::smem_u32(&bar_b[1]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  // this half's accumulator: columns [128 half, 128 half + 128)
  const uint32_t tmem = tmem_slot + (uint32_t)(half * kTcCols);
  const float sscale = st.cnt ? stats_scale_f(st) : 1.f;

  // Bound on Na_k over the codebook for this group: (max row sum |H_g|) L1max cinfmax.
  float hrow = 0.f;
#pragma unroll
  for (int a = 0; a < kD; ++a) {
    float rs = 0.f;
#pragma unroll
    for (int b = 0; b < kD; ++b) rs += fabsf(sH[a * kD + b]);
    hrow = fmaxf(hrow, rs);
  }
  const float l1max = cbmax[0], cinf = cbmax[1];
  constexpr uint32_t idesc = tc::idesc_tf32(kRows, kTcCols);

  // this CTA's row tiles (the last CTA of a column may have fewer); with two halves, half h
  // takes tiles h, h + 2, ...
  const int64_t row_tiles = (set.M + kRows - 1) / kRows;
  const int my_tiles = (int)min((int64_t)tiles, row_tiles - (int64_t)blockIdx.x * tiles);
  const int steps = (my_tiles + HALVES - 1) / HALVES;
  // Chunk uses are numbered u = t * nchunk + c. Resident chunks sit in buffer c; otherwise use u
  // reads buffer u & 1, and the copy for use u + 2 starts when use u is done (one half only).
  // At most one copy per buffer is outstanding; every thread tracks the same state.
  const int n_uses = resident ? nchunk : steps * nchunk;
  // per buffer (bit b): a copy outstanding, and the parity of its wait (registers, not arrays)
  uint32_t b_pend = 0, b_par = 0;
  auto fetch = [&](int u) {  // chunk u % nchunk into buffer u & 1 (bimg only)
    const int b = u & 1;
    if (tid == 0) {
      tc::mbar_expect_tx(tc::smem_u32(&bar_b[b]), kTcBTile);
      tc::bulk_copy_g2s(tc::smem_u32(Bbuf + b * kTcBTile),
                        bimg + (size_t)(u % nchunk) * kTcBTile, kTcBTile,
                        tc::smem_u32(&bar_b[b]));
    }
    b_pend |= 1u << b;
  };
  if (bimg) {
    fetch(0);
    if (n_uses > 1) fetch(1);
  }
  bool ok = true;
  int mma_count = 0;

  for (int t = 0; t < steps && ok; ++t) {
    const int my_tile = HALVES * t + half;  // past my_tiles: a half without rows this step
    const int64_t i = ((int64_t)blockIdx.x * tiles + my_tile) * kRows + rrow;
    const bool row_ok = my_tile < my_tiles && i < set.M;
    // Prologue: this thread's A row.
    float pmax, off;
    {
      float m2q[kD], rr, ra;
      if (rowterms) {  // precomputed for this Lloyd loop (row_terms_kernel)
        float4 q0 = make_float4(0.f, 0.f, 0.f, 0.f), q1 = q0, t2 = q0;
        if (row_ok) {
          q0 = rowterms[(3 * g) * set.M + i];
          q1 = rowterms[(3 * g + 1) * set.M + i];
          t2 = rowterms[(3 * g + 2) * set.M + i];
        }
        m2q[0] = q0.x; m2q[1] = q0.y; m2q[2] = q0.z; m2q[3] = q0.w;
        m2q[4] = q1.x; m2q[5] = q1.y; m2q[6] = q1.z; m2q[7] = q1.w;
        rr = t2.x;
        ra = t2.y;
        pmax = t2.z;
      } else {
        float rv[kD], a[kD];
        if (row_ok) {
          target32(set, cbs, n_fixed, i, g, rv, a, err);
        } else {
#pragma unroll
          for (int j = 0; j < kD; ++j) rv[j] = a[j] = 0.f;
        }
        vector_terms_rr(rv, a, sH, m2q, pmax, rr, ra);
      }
      // offset making every D = low + off >= 0, with margins for every rounding involved
      off = (rr + 32.f * kU * ra + 2.f * uc * (hrow * l1max * cinf + 2.f * pmax * l1max)) *
                (1.f + 4.f * uc) + 1e-30f;
      const float beta = -2.f * uc * pmax;
      if (st.cnt) {  // H r of this row, kept for the statistics (-m2q / 2, exact)
        *reinterpret_cast<float4*>(sQ + tid * kD) =
            make_float4(-0.5f * m2q[0], -0.5f * m2q[1], -0.5f * m2q[2], -0.5f * m2q[3]);
        *reinterpret_cast<float4*>(sQ + tid * kD + 4) =
            make_float4(-0.5f * m2q[4], -0.5f * m2q[5], -0.5f * m2q[6], -0.5f * m2q[7]);
      }
      uint32_t row[kK];
#pragma unroll
      for (int p = 0; p < kD; ++p) {
        uint32_t h, l;
        split(m2q[p], h, l);
        row[p] = h;
        row[8 + p] = h;
        row[16 + p] = l;
      }
      const uint32_t one = __float_as_uint(1.f);
      row[24] = one;
      row[25] = one;
      split(beta, row[26], row[28]);
      row[27] = row[26];
      split(off * (1.f - uc), row[29], row[30]);
      row[31] = 0u;
      put_row(Atile, rrow, row);
    }
    tc::fence_async_smem();
    half_sync<HALVES>(half);

    // as fp32 bits: the smallest block minimum, its block and the block's 16 values; the
    // second smallest block minimum
    uint32_t v1 = 0xffffffffu, v2 = 0xffffffffu;
    int b1 = 0;
    uint32_t bv[kBlk];
#pragma unroll
    for (int e = 0; e < kBlk; ++e) bv[e] = 0xffffffffu;
    for (int c = 0; c < nchunk; ++c) {
      const int u = t * nchunk + c;
      const int buf = resident ? c : (u & 1);
      char* Bt = Bbuf + buf * kTcBTile;
      if (bimg) {
        if ((b_pend >> buf) & 1u) {
          if (ok) ok = tc::mbar_wait(tc::smem_u32(&bar_b[buf]), (b_par >> buf) & 1u, err);
          b_par ^= 1u << buf;
          b_pend &= ~(1u << buf);
        }
      } else if (!resident || t == 0) {  // (one half only: the host passes B images with two)
        uint32_t v[kK];
        build_b_row(cw.C, cw.K, c * kTcCols + rrow, sH, uc, v);
        put_row(Bt, rrow, v);
        tc::fence_async_smem();
        half_sync<HALVES>(half);
      }
      ok = half_sync_and<HALVES>(half, ok);
      if (!ok) break;
      if (rrow == 0) {
        tc::tc_fence_after();
        const uint32_t a0 = tc::smem_u32(Atile), b0 = tc::smem_u32(Bt);
#pragma unroll
        for (int ks = 0; ks < kK / 8; ++ks)
          tc::mma_tf32(tmem, tc::smem_desc(a0 + ks * 256, 128, (kK / 4) * 128),
                       tc::smem_desc(b0 + ks * 256, 128, (kK / 4) * 128), idesc,
                       ks > 0 ? 1u : 0u);
        tc::mma_commit(tc::smem_u32(&bar_mma));
      }
      ok = tc::mbar_wait(tc::smem_u32(&bar_mma), (uint32_t)(mma_count & 1), err);
      ++mma_count;
      ok = half_sync_and<HALVES>(half, ok);
      if (!ok) break;
      if (bimg && !resident && u + 2 < n_uses) fetch(u + 2);  // this buffer is free again
      tc::tc_fence_after();
      // Epilogue: this warp's 32 rows x 128 columns as eight blocks of 16. Per block its
      // minimum (every D >= 0, so the bit patterns order like the values); a block whose
      // minimum is the row's smallest so far is kept whole (16 selects), the previous best
      // block's minimum moves to the second smallest. No per-score index.
      const uint32_t base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
#pragma unroll
      for (int rnd = 0; rnd < 4; ++rnd) {
        uint32_t v[32];
        tc::tmem_ld32_nowait(base + 32 * rnd, v);
        tc::tmem_wait_ld_dep(v);
#pragma unroll
        for (int q = 0; q < 32 / kBlk; ++q) {
          const uint32_t m = min16_bits(v + kBlk * q);
          v2 = min(v2, max(v1, m));
          const bool lt = m < v1;
          v1 = lt ? m : v1;
          b1 = lt ? (c * kTcCols + 32 * rnd + kBlk * q) / kBlk : b1;
#pragma unroll
          for (int e = 0; e < kBlk; ++e) bv[e] = lt ? v[kBlk * q + e] : bv[e];
        }
      }
      tc::tc_fence_before();
      half_sync<HALVES>(half);  // the accumulator is free for the next MMA
    }
    if (!ok) break;

    // Certificate, code, flag and statistics of this thread's row. j = the smallest D (ties to
    // the smaller column), k2 = the second smallest D over the row (the winning block's second
    // value or the other blocks' smallest minimum).
    if (row_ok) {
      uint32_t w1 = bv[0], w2 = 0xffffffffu;
      int jb = 0;
#pragma unroll
      for (int e = 1; e < kBlk; ++e) {
        w2 = min(w2, max(w1, bv[e]));
        const bool lt = bv[e] < w1;
        w1 = lt ? bv[e] : w1;
        jb = lt ? e : jb;
      }
      int j = b1 * kBlk + jb;
      const uint32_t s2 = min(v2, w2);
      const float k1 = __uint_as_float(w1);
      const float k2 = s2 == 0xffffffffu ? INFINITY : __uint_as_float(s2);
      bool cert = false;
      float thr = INFINITY;
      if (j < cw.K) {
        float n, na, l1;
        if (smem_terms) {
          const float2 tj = sNaL1[j];
          na = tj.x;
          l1 = tj.y;
        } else if (gterms) {
          const float4 tj = gterms[j];
          n = tj.x;
          na = tj.y;
          l1 = tj.z;
        } else {
          float cv[kD];
          load_vec(cw.C + (int64_t)j * kD, cv);
          codeword_terms(cv, sH, n, na, l1);
        }
        // D_k <= s_k + off (every k); s_j + off <= D_j + e2 (the winner): no other codeword's
        // exact score reaches s_j when k2 > D_j + e2 (the sum rounded up).
        const float e2 = 2.f * uc * (na + 2.f * pmax * l1 + off);
        const float top = __fadd_ru(k1, e2);   // >= s_j + off
        cert = cw.K == 1 || k2 > top;
        thr = top - off;
        thr += 4.f * kU * (k1 + off + e2);
      } else {
        j = 0;
      }
      if (!cert) {
        const unsigned slot = atomicAdd(flags.count, 1u);
        if (slot < flags.cap) {
          flags.vec[slot] = i * G_range + (g - g_begin);
          flags.thr[slot] = thr;
        } else {
          raise_error(err, ERRBIT_INDEX);
        }
      }
      out_code[i * out_ld + (g - out_g0)] = j;
      if (cert && st.cnt) {
        // H r from the prologue (bit-identical to the standalone update's H tau)
        float q[kD];
        const float4 q0 = *reinterpret_cast<const float4*>(sQ + tid * kD);
        const float4 q1 = *reinterpret_cast<const float4*>(sQ + tid * kD + 4);
        q[0] = q0.x; q[1] = q0.y; q[2] = q0.z; q[3] = q0.w;
        q[4] = q1.x; q[5] = q1.y; q[6] = q1.z; q[7] = q1.w;
        if (smem_stats) {
          atomicAdd(&s_cnt[j], 1);
#pragma unroll
          for (int p = 0; p < kD; ++p) {
            const long long v = fix_rn_small(q[p], sscale);
            atomicAdd(&s_b32[(2 * p) * kTcSmemStatsK + j], (int)(v >> 15));
            atomicAdd(&s_b32[(2 * p + 1) * kTcSmemStatsK + j], (int)(v & 0x7fff));
          }
        } else {
          stats_add(st, sscale, g, j, q);
        }
      }
    }
  }
  // After a timeout: let copies still in flight into this CTA's shared memory land (bounded).
  for (int b = 0; b < 2; ++b)
    if ((b_pend >> b) & 1u) {
      tc::mbar_wait(tc::smem_u32(&bar_b[b]), (b_par >> b) & 1u, err);
    }
  __syncthreads();
  if (smem_stats) {  // one flush of this CTA's statistics (integer sums: order-free)
    for (int k = tid; k < cw.K; k += blockDim.x) {
      const int c = s_cnt[k];
      if (c == 0) continue;
      atomicAdd(&st.cnt[g * st.K + k], c);
#pragma unroll
      for (int p = 0; p < kD; ++p) {
        const long long v = (long long)s_b32[(2 * p) * kTcSmemStatsK + k] * 32768 +
                            s_b32[(2 * p + 1) * kTcSmemStatsK + k];
        atomicAdd(reinterpret_cast<unsigned long long*>(&st.bacc[(int64_t)k * kD + p]),
                  (unsigned long long)v);
      }
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem_slot, HALVES * kTcCols);
}

// Exact decision for the rows the arg-min pass flagged: one CTA per flagged vector. The
// threads stride over the codebook for U = min(fast-pass threshold, smallest fp32 upper
// bound); every codeword whose fp32 lower bound is at most U is a candidate (the exact
// arg-min always is) and is re-scored exactly in fp32 pairs (dfl) by one thread; the
// smallest (err, index) wins. Adds the statistics of the decided code when requested.
__global__ void __launch_bounds__(128)
argmin_exact_kernel(SetView set, int64_t g_begin, int64_t G_range, CbList cbs, int n_fixed,
                    int s_idx, int32_t* __restrict__ out_code, int64_t out_ld, int64_t out_g0,
                    FlagList flags, StatsView st, const float4* __restrict__ terms,
                    unsigned* err) {
  pdl_trigger();  // dependents may launch; this grid waits for its predecessor first
  pdl_wait();
  __shared__ float sH[kD * kD];
  __shared__ float redf[4];
  __shared__ int cand[256];
  __shared__ int ncand;
  __shared__ float bh_s[4], bl_s[4];
  __shared__ int bk_s[4];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned cnt = min((unsigned long long)*flags.count, (unsigned long long)flags.cap);
  if (flags.total && blockIdx.x == 0 && tid == 0) atomicAdd(flags.total, cnt);
  const CbView cw = cbs.cb[s_idx];
  const float cmul = bound_mult(n_fixed);
  for (unsigned f = blockIdx.x; f < cnt; f += gridDim.x) {
    const int64_t vi = flags.vec[f];
    const int64_t i = vi / G_range, grel = vi % G_range, g = g_begin + grel;
    const float thr = flags.thr[f];
    __syncthreads();
    if (tid < kD * kD) sH[tid] = set.Hb[g * kD * kD + tid];
    if (tid == 0) ncand = 0;
    __syncthreads();
    float rv[kD], av[kD], m2q[kD], pmax;
    target32(set, cbs, n_fixed, i, g, rv, av, err);
    vector_terms(rv, av, sH, m2q, pmax);
    const float nbeta = -2.f * kU * cmul * pmax;
    const float4* gt = terms ? terms + grel * cw.K : nullptr;
    auto terms_of = [&](int k, const float cv[kD], float& nn, float& na, float& l1) {
      if (gt) {
        const float4 t = gt[k];
        nn = t.x;
        na = t.y;
        l1 = t.z;
      } else {
        codeword_terms(cv, sH, nn, na, l1);
      }
    };
    float U = thr;
    for (int k = tid; k < cw.K; k += blockDim.x) {
      float cv[kD], nn, na, l1;
      load_vec(cw.C + (int64_t)k * kD, cv);
      terms_of(k, cv, nn, na, l1);
      U = fminf(U, up_from(nn, na, l1, cv, m2q, pmax, cmul));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) U = fminf(U, __shfl_xor_sync(0xffffffffu, U, o));
    if (lane == 0) redf[warp] = U;
    __syncthreads();
    U = fminf(fminf(redf[0], redf[1]), fminf(redf[2], redf[3]));
    float rh[kD], rl[kD];
    dfl::target(set, cbs, n_fixed, i, g, rh, rl, err);
    float bh = INFINITY, bl = 0.f;
    int bk = 0x7fffffff;
    for (int k0 = 0; k0 < cw.K; k0 += 256) {
      for (int k = k0 + tid; k < min(cw.K, k0 + 256); k += blockDim.x) {
        float cv[kD], nn, na, l1;
        load_vec(cw.C + (int64_t)k * kD, cv);
        terms_of(k, cv, nn, na, l1);
        if (low_from(nn, na, l1, cv, m2q, nbeta, cmul) <= U) cand[atomicAdd(&ncand, 1)] = k;
      }
      __syncthreads();
      const int nc = ncand;
      for (int q = tid; q < nc; q += blockDim.x) {
        const int k = cand[q];
        float cv[kD], eh, el;
        load_vec(cw.C + (int64_t)k * kD, cv);
        dfl::quad_err(rh, rl, cv, sH, eh, el);
        if (dfl::less(eh, el, k, bh, bl, bk)) {
          bh = eh;
          bl = el;
          bk = k;
        }
      }
      __syncthreads();
      if (tid == 0) ncand = 0;
      __syncthreads();
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float oh = __shfl_xor_sync(0xffffffffu, bh, o);
      const float ol = __shfl_xor_sync(0xffffffffu, bl, o);
      const int ok = __shfl_xor_sync(0xffffffffu, bk, o);
      if (dfl::less(oh, ol, ok, bh, bl, bk)) {
        bh = oh;
        bl = ol;
        bk = ok;
      }
    }
    if (lane == 0) {
      bh_s[warp] = bh;
      bl_s[warp] = bl;
      bk_s[warp] = bk;
    }
    __syncthreads();
    if (tid == 0) {
      for (int w = 1; w < 4; ++w)
        if (dfl::less(bh_s[w], bl_s[w], bk_s[w], bh, bl, bk)) {
          bh = bh_s[w];
          bl = bl_s[w];
          bk = bk_s[w];
        }
      if (bk == 0x7fffffff) {
        raise_error(err, ERRBIT_NUMERIC);  // no candidate: non-finite scores
      } else {
        out_code[i * out_ld + (g - out_g0)] = bk;
        if (st.cnt) {
          float q[kD];
#pragma unroll
          for (int p = 0; p < kD; ++p) q[p] = -0.5f * m2q[p];
          stats_add(st, stats_scale_f(st), g, bk, q);
        }
      }
    }
  }
}


// Exact decision of flagged rows, one warp per row, for codebooks of up to kExactWarpK
// entries: the bounds and fp32-pair scores of argmin_exact_kernel without block barriers.
// Lane l takes codewords l, l + 32, ...; the fp32 upper bounds give U, every codeword whose
// lower bound reaches U is scored in fp32 pairs by the lane that holds it, and the best
// (value, index) is reduced across the warp with the same total order, so the decision is the
// one argmin_exact_kernel makes.
constexpr int kExactWarpK = 1024;
constexpr int kExactBatch = 2;  // codewords a lane loads before using them

__global__ void __launch_bounds__(128)
argmin_exact_warp_kernel(SetView set, int64_t g_begin, int64_t G_range, CbList cbs,
                         int n_fixed, int s_idx, int32_t* __restrict__ out_code, int64_t out_ld,
                         int64_t out_g0, FlagList flags, StatsView st,
                         const float4* __restrict__ terms, unsigned* err) {
  pdl_trigger();  // dependents may launch; this grid waits for its predecessor first
  pdl_wait();
  __shared__ float sHw[4][kD * kD];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned cnt = min((unsigned long long)*flags.count, (unsigned long long)flags.cap);
  if (flags.total && blockIdx.x == 0 && threadIdx.x == 0) atomicAdd(flags.total, cnt);
  const CbView cw = cbs.cb[s_idx];
  const float cmul = bound_mult(n_fixed);
  float* sH = sHw[warp];
  for (unsigned f = blockIdx.x * 4u + warp; f < cnt; f += gridDim.x * 4u) {
    const int64_t vi = flags.vec[f];
    const int64_t i = vi / G_range, grel = vi % G_range, g = g_begin + grel;
    const float thr = flags.thr[f];
    __syncwarp();
    sH[lane] = set.Hb[g * kD * kD + lane];
    sH[lane + 32] = set.Hb[g * kD * kD + lane + 32];
    __syncwarp();
    float rv[kD], av[kD], m2q[kD], pmax;
    target32(set, cbs, n_fixed, i, g, rv, av, err);
    vector_terms(rv, av, sH, m2q, pmax);
    const float nbeta = -2.f * kU * cmul * pmax;
    const float4* gt = terms ? terms + grel * cw.K : nullptr;
    // a lane takes codewords lane, lane + 32, ...; kExactBatch of them are loaded before any is
    // used, so their L2 round trips overlap
    float U = thr;
    for (int k0 = lane; k0 < cw.K; k0 += 32 * kExactBatch) {
      float cv[kExactBatch][kD];
      float4 tt[kExactBatch];
#pragma unroll
      for (int u = 0; u < kExactBatch; ++u) {
        const int k = k0 + 32 * u;
        if (k < cw.K) {
          load_vec(cw.C + (int64_t)k * kD, cv[u]);
          if (gt) tt[u] = gt[k];
        }
      }
#pragma unroll
      for (int u = 0; u < kExactBatch; ++u) {
        if (k0 + 32 * u >= cw.K) break;
        float nn, na, l1;
        if (gt) {
          nn = tt[u].x;
          na = tt[u].y;
          l1 = tt[u].z;
        } else {
          codeword_terms(cv[u], sH, nn, na, l1);
        }
        U = fminf(U, up_from(nn, na, l1, cv[u], m2q, pmax, cmul));
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) U = fminf(U, __shfl_xor_sync(0xffffffffu, U, o));
    float rh[kD], rl[kD];
    dfl::target(set, cbs, n_fixed, i, g, rh, rl, err);
    float bh = INFINITY, bl = 0.f;
    int bk = 0x7fffffff;
    for (int k = lane; k < cw.K; k += 32) {
      float cv[kD], nn, na, l1;
      load_vec(cw.C + (int64_t)k * kD, cv);
      if (gt) {
        const float4 t = gt[k];
        nn = t.x;
        na = t.y;
        l1 = t.z;
      } else {
        codeword_terms(cv, sH, nn, na, l1);
      }
      if (low_from(nn, na, l1, cv, m2q, nbeta, cmul) <= U) {
        float eh, el;
        dfl::quad_err(rh, rl, cv, sH, eh, el);
        if (dfl::less(eh, el, k, bh, bl, bk)) {
          bh = eh;
          bl = el;
          bk = k;
        }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float oh = __shfl_xor_sync(0xffffffffu, bh, o);
      const float ol = __shfl_xor_sync(0xffffffffu, bl, o);
      const int ok = __shfl_xor_sync(0xffffffffu, bk, o);
      if (dfl::less(oh, ol, ok, bh, bl, bk)) {
        bh = oh;
        bl = ol;
        bk = ok;
      }
    }
    if (lane == 0) {
      if (bk == 0x7fffffff) {
        raise_error(err, ERRBIT_NUMERIC);  // no candidate: non-finite scores
      } else {
        out_code[i * out_ld + (g - out_g0)] = bk;
        if (st.cnt) {
          float q[kD];
#pragma unroll
          for (int p = 0; p < kD; ++p) q[p] = -0.5f * m2q[p];
          stats_add(st, stats_scale_f(st), g, bk, q);
        }
      }
    }
  }
}

// --------------------------------------------------------------------------- beam stages
// Hypotheses of a vector: up to B partial tuples (codes of the first s+1 searched codebooks)
// in rank order. hyp layout: [vector][B][S] int32; hyp_n[vector] = number kept.
struct BeamBufs {
  const int32_t* hyp_in;
  const int32_t* n_in;
  int32_t* hyp_out;
  int32_t* n_out;
};

struct StageDesc {
  int st[kMaxCodebooks];  // indices (in cbs) of the searched codebooks, in stage order
  int S;                  // number of stages
  int s;                  // current stage
  int B;                  // beam width (hypothesis buffer stride)
  int Bs;                 // hypotheses kept by the current stage (1 at the last stage)
};

// fp64 residual of a hypothesis before stage s: target - sum_{s' < s} C_{st[s']}[code].
__device__ void hyp_residual64(const double tgt[kD], const CbList& cbs, const StageDesc& sd,
                               const int32_t* codes, double r[kD], unsigned* err) {
#pragma unroll
  for (int j = 0; j < kD; ++j) r[j] = tgt[j];
  for (int q = 0; q < sd.s; ++q) {
    const CbView& cb = cbs.cb[sd.st[q]];
    const int32_t k = codes[q];
    if (!code_ok(k, cb.K, err)) continue;
    const float* c = cb.C + (int64_t)k * kD;
#pragma unroll
    for (int j = 0; j < kD; ++j) r[j] -= (double)c[j];
  }
}

// Per-hypothesis terms of the approximate err: m2q = -2 H r, rr = r^T H r (r rounded to
// fp32), and the bound pieces Ra = |r|^T |H| |r|, Pmax = max_p (|H| |r|)_p.
__device__ __forceinline__ void hyp_terms(const double r64[kD], const float* H, float m2q[kD],
                                          float& rr, float& ra, float& pmax) {
  float r[kD];
#pragma unroll
  for (int j = 0; j < kD; ++j) r[j] = (float)r64[j];
  rr = 0.f;
  ra = 0.f;
  pmax = 0.f;
#pragma unroll
  for (int p = 0; p < kD; ++p) {
    float q = 0.f, pa = 0.f;
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      q = fmaf(H[p * kD + j], r[j], q);
      pa = fmaf(fabsf(H[p * kD + j]), fabsf(r[j]), pa);
    }
    m2q[p] = -2.f * q;
    rr = fmaf(r[p], q, rr);
    ra = fmaf(fabsf(r[p]), pa, ra);
    pmax = fmaxf(pmax, pa);
  }
}

// fp32-pair residual of a hypothesis before stage s: (rh + rl) = (th + tl) - sum_{s' < s}
// C_{st[s']}[code] (TwoSum per subtraction, about 2^-48 relative; no fp64 arithmetic).
__device__ __forceinline__ void hyp_residual_pair(const float th[kD], const float tl[kD],
                                                  const CbList& cbs, const StageDesc& sd,
                                                  const int32_t* codes, float rh[kD],
                                                  float rl[kD], unsigned* err) {
#pragma unroll
  for (int j = 0; j < kD; ++j) {
    rh[j] = th[j];
    rl[j] = tl[j];
  }
  for (int q = 0; q < sd.s; ++q) {
    const CbView& cb = cbs.cb[sd.st[q]];
    const int32_t k = codes[q];
    if (!code_ok(k, cb.K, err)) continue;
    float c[kD];
    load_vec(cb.C + (int64_t)k * kD, c);
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      float sj, ej;
      dfl::two_sum(rh[j], -c[j], sj, ej);
      rh[j] = sj;
      rl[j] = __fadd_rn(rl[j], ej);
    }
  }
}

// hyp_terms of a pair residual, rounded once to fp32.
__device__ __forceinline__ void hyp_terms_pair(const float rh[kD], const float rl[kD],
                                               const float* H, float m2q[kD], float& rr,
                                               float& ra, float& pmax) {
  float r[kD];
#pragma unroll
  for (int j = 0; j < kD; ++j) r[j] = __fadd_rn(rh[j], rl[j]);
  rr = 0.f;
  ra = 0.f;
  pmax = 0.f;
#pragma unroll
  for (int p = 0; p < kD; ++p) {
    float q = 0.f, pa = 0.f;
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      q = fmaf(H[p * kD + j], r[j], q);
      pa = fmaf(fabsf(H[p * kD + j]), fabsf(r[j]), pa);
    }
    m2q[p] = -2.f * q;
    rr = fmaf(r[p], q, rr);
    ra = fmaf(fabsf(r[p]), pa, ra);
    pmax = fmaxf(pmax, pa);
  }
}

// The end of a fast stage for one vector, given its sorted top-L list (topv, topi) of fp32
// lower bounds low = approx_err - Et built in (h, k) order: bounds of the listed entries, the
// fast certificate, the fp32-pair exact path, the flag for the fallback, and the kept tuples.
// sRa / sPm: Ra_h, Pmax_h of this thread's hypotheses at [h * stride]; sNL / sNa: the staged
// codeword terms (used when the whole codebook was staged, else recomputed).
template <int L>
__device__ __forceinline__ void beam_list_finish(
    const SetView& set, const CbList& cbs, const StageDesc& sd, const BeamBufs& bb,
    const FlagList& flags, int64_t i, int64_t g, int64_t vi, int Bh, float cmul,
    const float th[kD], const float tl[kD], const float* sH, const float2* sNL,
    const float* sNa, bool one_chunk, const float* sRa, const float* sPm, int stride,
    float topv[L], int topi[L], unsigned* err) {
  const CbView cw = cbs.cb[sd.st[sd.s]];
  const int S = sd.S, B = sd.B, Bs = sd.Bs;
  int toph[L], topk[L];
#pragma unroll
  for (int j = 0; j < L; ++j) {
    toph[j] = topi[j] == 0x7fffffff ? 0x7fffffff : (topi[j] >> 16);
    topk[j] = topi[j] == 0x7fffffff ? 0x7fffffff : (topi[j] & 0xffff);
  }
  const int64_t total = (int64_t)Bh * cw.K;
  const int nkept = (int)min((int64_t)L, total);
  const int keep = (int)min((int64_t)Bs, total);
  // Non-finite scores never enter the list; keep indices valid and report it.
#pragma unroll
  for (int j = 0; j < L; ++j) {
    if (j < nkept && (toph[j] >= Bh || topk[j] >= cw.K)) {
      raise_error(err, ERRBIT_NUMERIC);
      toph[j] = 0;
      topk[j] = 0;
    }
  }
  // Per-entry bound Et = u C (Ra_h + Na_k + 2 Pmax_h L1_k) for the listed entries, from the
  // hypothesis terms kept in the sweep and the staged codeword terms (recomputed when the
  // codebook spans several chunks).
  float et[L];
#pragma unroll
  for (int j = 0; j < L; ++j) {
    et[j] = 0.f;
    if (j < nkept) {
      const float ra = sRa[toph[j] * stride];
      const float pmax = sPm[toph[j] * stride];
      float na, l1;
      if (one_chunk) {
        na = sNa[topk[j]];
        l1 = sNL[topk[j]].y;
      } else {
        float c[kD], n;
        load_vec(cw.C + (int64_t)topk[j] * kD, c);
        codeword_terms(c, sH, n, na, l1);
      }
      et[j] = kU * cmul * (ra + na + 2.f * pmax * l1);
    }
  }
  // Fast certificate: low_{j+1} - low_j > 2 Et_j for j < min(keep, total - 1) (every
  // candidate outside the list has low >= the last list entry).
  bool ok = true;
  const int lim = (int)min((int64_t)keep, total - 1);
#pragma unroll
  for (int j = 0; j < L - 1; ++j)
    if (j < lim && !(topv[j + 1] - topv[j] > 2.f * et[j])) ok = false;

  int32_t* out = bb.hyp_out + vi * B * S;
  if (!ok) {
    // Exact path on the listed candidates: errs as fp32 pairs (about 2^-44 relative; no fp64),
    // (err, h, k) order; then every unlisted candidate must have low >= the last listed low,
    // which must exceed an upper bound of the keep-th err.
    float evh[L], evl[L];
#pragma unroll
    for (int j = 0; j < L; ++j) {
      evh[j] = INFINITY;
      evl[j] = 0.f;
      if (j < nkept) {
        float rh[kD], rl[kD], c[kD];
        const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + toph[j]) * S : nullptr;
        hyp_residual_pair(th, tl, cbs, sd, pc, rh, rl, err);
        load_vec(cw.C + (int64_t)topk[j] * kD, c);
        dfl::quad_err(rh, rl, c, sH, evh[j], evl[j]);
      }
    }
    const float last_low = topv[nkept - 1];
#pragma unroll
    for (int a = 1; a < L; ++a) {
#pragma unroll
      for (int b = a; b > 0; --b) {
        const bool sw = (evh[b] < evh[b - 1]) ||
                        (evh[b] == evh[b - 1] &&
                         (evl[b] < evl[b - 1] ||
                          (evl[b] == evl[b - 1] &&
                           (toph[b] < toph[b - 1] ||
                            (toph[b] == toph[b - 1] && topk[b] < topk[b - 1])))));
        if (sw) {
          const float t0 = evh[b]; evh[b] = evh[b - 1]; evh[b - 1] = t0;
          const float t1 = evl[b]; evl[b] = evl[b - 1]; evl[b - 1] = t1;
          const int th_ = toph[b]; toph[b] = toph[b - 1]; toph[b - 1] = th_;
          const int tk = topk[b]; topk[b] = topk[b - 1]; topk[b - 1] = tk;
        }
      }
    }
    // upper bound of the keep-th listed err (the pair's own error is far below 1e-7)
    const float ev_up = isfinite(evh[keep - 1])
                            ? __fmul_ru(__fadd_ru(evh[keep - 1], evl[keep - 1]), 1.0000002f)
                            : INFINITY;
    const bool cert = total <= L || last_low > ev_up;
    if (!cert) {
      const unsigned slot = atomicAdd(flags.count, 1u);
      if (slot < flags.cap) {
        flags.vec[slot] = vi;
        // every member of the exact top-keep has err <= the keep-th listed err
        flags.thr[slot] = ev_up;
      } else {
        raise_error(err, ERRBIT_INDEX);
      }
      return;
    }
  }
#pragma unroll
  for (int j = 0; j < L; ++j) {
    if (j >= keep) break;
    const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + toph[j]) * S : nullptr;
    for (int q = 0; q < sd.s; ++q) out[j * S + q] = pc[q];
    out[j * S + sd.s] = topk[j];
  }
  bb.n_out[vi] = keep;
}

constexpr int kBeamCand = 16;  // candidate buffer slots per thread
constexpr int kBeamScan = 8;   // scores between two overflow checks

// Fast stage: one thread per vector, the stage codebook chunked through shared memory, a
// sorted top-L list (L >= Bs + 1) of lower bounds low = approx_err - Et in registers.
template <int L>
__global__ void __launch_bounds__(kThreads, L <= 9 ? 3 : 2)
beam_stage_kernel(SetView set, int64_t g_begin, CbList cbs, int n_fixed, StageDesc sd,
                  BeamBufs bb, FlagList flags, unsigned* err) {
  const int64_t g = g_begin + blockIdx.y;
  const int64_t G_range = gridDim.y;
  const int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  const bool live = i < set.M;
  const int64_t vi = live ? i * G_range + (g - g_begin) : 0;
  __shared__ float sH[kD * kD];
  __shared__ __align__(16) float sC[kChunk * kD];
  __shared__ __align__(8) float2 sNL[kChunk];
  __shared__ float sNa[kChunk];
  // candidate buffers, [slot][thread]: (score bits, (h << 16) | k)
  __shared__ uint2 cand[kBeamCand * kThreads];
  __shared__ float sRa[16 * kThreads], sPm[16 * kThreads];  // Ra_h, Pmax_h, [h][thread]
  if (threadIdx.x < kD * kD) sH[threadIdx.x] = set.Hb[g * kD * kD + threadIdx.x];
  __syncthreads();

  const CbView cw = cbs.cb[sd.st[sd.s]];
  const int S = sd.S, B = sd.B;
  const float cmul = bound_mult(n_fixed + sd.s);
  const int Bh = (sd.s == 0) ? 1 : (live ? bb.n_in[vi] : 1);
  float th[kD], tl[kD];  // target as an fp32 pair (t - the fixed codebooks' codewords)
  if (live) {
    dfl::target(set, cbs, n_fixed, i, g, th, tl, err);
  } else {
#pragma unroll
    for (int j = 0; j < kD; ++j) th[j] = tl[j] = 0.f;
  }

  float topv[L];
  int topi[L];  // (h << 16) | k: B <= 16 hypotheses, K <= 65536 codewords
#pragma unroll
  for (int j = 0; j < L; ++j) {
    topv[j] = INFINITY;
    topi[j] = 0x7fffffff;
  }

  // Scores below the list's last entry (as of the last flush) are appended to this thread's
  // candidate buffer in shared memory: a predicated store per score, no branch. Every kBeamScan
  // scores the warp flushes when any lane's buffer could overflow within the next stretch:
  // the buffered candidates, in (h, k) order, go through the sorted insertion (ties keep the
  // earlier candidate ahead, as inserting every score in order would). The insertion network,
  // which the compiler predicates, thus runs per candidate instead of per score.
  int nc = 0;
  float thr = INFINITY;
  auto flush = [&]() {
    for (int e = 0; e < nc; ++e) {
      const uint2 ce = cand[e * kThreads + threadIdx.x];
      float sv = __uint_as_float(ce.x);
      int si = (int)ce.y;
      if (sv < topv[L - 1]) {
#pragma unroll
        for (int j = 0; j < L; ++j) {
          if (sv < topv[j]) {
            const float tv = topv[j];
            const int ti = topi[j];
            topv[j] = sv;
            topi[j] = si;
            sv = tv;
            si = ti;
          }
        }
      }
    }
    nc = 0;
    thr = topv[L - 1];
  };
  for (int k0 = 0; k0 < cw.K; k0 += kChunk) {
    const int nk = min(kChunk, cw.K - k0);
    __syncthreads();
    stage_chunk(cw.C, k0, nk, sH, cmul, sC, sNL, sNa);
    __syncthreads();
    if (!live) continue;
    for (int h = 0; h < Bh; ++h) {
      float rh[kD], rl[kD];
      const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + h) * S : nullptr;
      hyp_residual_pair(th, tl, cbs, sd, pc, rh, rl, err);
      float m2q[kD], rr, ra, pmax;
      hyp_terms_pair(rh, rl, sH, m2q, rr, ra, pmax);
      sRa[h * kThreads + threadIdx.x] = ra;  // the same values in every chunk
      sPm[h * kThreads + threadIdx.x] = pmax;
      const float base = rr - kU * cmul * ra;
      const float nbeta = -2.f * kU * cmul * pmax;
      // One score: a chain of ten dependent operations; four independent chains per step.
      // Every score is stored into slot nc, which advances only for a candidate (no branch);
      // nc <= kBeamCand - kBeamScan after each check, so the at most kBeamScan stores that
      // follow stay below kBeamCand.
      auto score_at = [&](int k) {
        const float4 c0 = *reinterpret_cast<const float4*>(sC + k * kD);
        const float4 c1 = *reinterpret_cast<const float4*>(sC + k * kD + 4);
        const float2 nl = sNL[k];
        float sc = base + nl.x;
        sc = fmaf(m2q[0], c0.x, sc);
        sc = fmaf(m2q[1], c0.y, sc);
        sc = fmaf(m2q[2], c0.z, sc);
        sc = fmaf(m2q[3], c0.w, sc);
        sc = fmaf(m2q[4], c1.x, sc);
        sc = fmaf(m2q[5], c1.y, sc);
        sc = fmaf(m2q[6], c1.z, sc);
        sc = fmaf(m2q[7], c1.w, sc);
        return fmaf(nbeta, nl.y, sc);
      };
      const uint32_t hk = ((uint32_t)h << 16) | (uint32_t)k0;
      for (int kb = 0; kb < nk; kb += kBeamScan) {
        if (__any_sync(__activemask(), nc > kBeamCand - kBeamScan)) flush();
        if (kb + kBeamScan <= nk) {
#pragma unroll
          for (int e0 = 0; e0 < kBeamScan; e0 += 4) {
            float sc[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) sc[e] = score_at(kb + e0 + e);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              cand[nc * kThreads + threadIdx.x] =
                  make_uint2(__float_as_uint(sc[e]), hk + (uint32_t)(kb + e0 + e));
              nc += sc[e] < thr ? 1 : 0;
            }
          }
        } else {
          for (int k = kb; k < nk; ++k) {
            const float s1 = score_at(k);
            cand[nc * kThreads + threadIdx.x] =
                make_uint2(__float_as_uint(s1), hk + (uint32_t)k);
            nc += s1 < thr ? 1 : 0;
          }
        }
      }
    }
  }
  if (!live) return;
  flush();
  beam_list_finish<L>(set, cbs, sd, bb, flags, i, g, vi, Bh, cmul, th, tl, sH, sNL, sNa,
                      cw.K <= kChunk, sRa + threadIdx.x, sPm + threadIdx.x, kThreads, topv,
                      topi, err);
}

// Fast stage with the scores on the tensor cores (codebooks of at most 256 codewords, L <= 9).
// Thread = vector, as in beam_stage_kernel; the CTA's 128 vectors take the hypotheses in turn:
// for hypothesis h every thread writes its A row, one tcgen05.mma pass computes
//   y(h, k) = base_h + sN_k + m2q_h . c_k + nbeta_h L1_k
// for all 128 vectors x 256 codewords (3xTF32 operands: the B images of prep_b built with the
// stage's bound multiplier), and each thread reads its row from tensor memory. y differs from
// the fast stage's fp32 chain x(h, k) (the same linear form) by at most eps_h = 2^-12 S_h,
// S_h = |base_h| + Na_max + 2 Pmax_h L1max + |nbeta_h| L1max, which bounds every term's
// magnitude (the split products lose about 2^-22 and the fp32 accumulation of 32 terms about
// 2^-19 of it). A pair whose x could enter the list has y <= (the list's last x, or the bound
// tau below) + eps_h; only those are kept (a bit mask per thread), scored again with exactly
// the fast stage's chain and inserted in (h, k) order with its rule (strictly below the last
// entry, before the first entry strictly above). Every member of the final
// top-L is among them, so the list, and everything after it (beam_list_finish), equals
// beam_stage_kernel's. tau: for h = 0, the L-th smallest of the 16-column block minima of y:
// at least L pairs have y <= tau, so the L-th smallest x is at most tau + eps_0.
constexpr size_t kBeamTcSmem = 1024 + (size_t)tcenc::kATile + 2 * (size_t)kTcBTile +
                               (size_t)kChunk * kD * 4 + (size_t)kChunk * 8 + (size_t)kChunk * 4 +
                               2 * 16 * (size_t)kThreads * 4 + 2 * 9 * (size_t)kThreads * 4;

template <int L>
__global__ void __launch_bounds__(kThreads, 2)
beam_tc_kernel(SetView set, int64_t g_begin, CbList cbs, int n_fixed, StageDesc sd,
               BeamBufs bb, const char* __restrict__ bimg, const float* __restrict__ cbmax,
               FlagList flags, unsigned* err) {
  static_assert(L <= 9, "the shared-memory list holds 9 entries");
  using namespace tcenc;
  extern __shared__ __align__(1024) char smem_raw[];
  char* smem = smem_raw + ((1024u - (tc::smem_u32(smem_raw) & 1023u)) & 1023u);
  char* Atile = smem;
  char* Bbuf = Atile + kATile;
  float* sC = reinterpret_cast<float*>(Bbuf + 2 * kTcBTile);
  float2* sNL = reinterpret_cast<float2*>(sC + kChunk * kD);
  float* sNa = reinterpret_cast<float*>(sNL + kChunk);
  float* sRa = sNa + kChunk;  // [h][thread]
  float* sPm = sRa + 16 * kThreads;
  float* sTopV = sPm + 16 * kThreads;                          // [j][thread]
  int* sTopI = reinterpret_cast<int*>(sTopV + 9 * kThreads);  // [j][thread]
  __shared__ __align__(16) float sH[kD * kD];
  __shared__ __align__(8) uint64_t bar_b, bar_mma;
  __shared__ uint32_t tmem_slot;

  const int tid = threadIdx.x, warp = tid >> 5;
  const int64_t g = g_begin + blockIdx.y;
  const int64_t G_range = gridDim.y;
  const int64_t i = (int64_t)blockIdx.x * kThreads + tid;
  const bool live = i < set.M;
  const int64_t vi = live ? i * G_range + (g - g_begin) : 0;
  const CbView cw = cbs.cb[sd.st[sd.s]];
  const int nchunk = (cw.K + kTcCols - 1) / kTcCols;  // 1 or 2
  const int S = sd.S, B = sd.B;
  const float cmul = bound_mult(n_fixed + sd.s);

  if (tid < kD * kD) sH[tid] = set.Hb[g * kD * kD + tid];
  if (warp == 0) tc::tmem_alloc(&tmem_slot, 2 * kTcCols);
  if (tid == 0) {
    tc::mbar_init(tc::smem_u32(&bar_b), 1);
    tc::mbar_init(tc::smem_u32(&bar_mma), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = tmem_slot;
  if (tid == 0) {  // this group's B images, one bulk copy per 128-codeword chunk
    tc::mbar_expect_tx(tc::smem_u32(&bar_b), (uint32_t)(nchunk * kTcBTile));
    for (int c = 0; c < nchunk; ++c)
      tc::bulk_copy_g2s(tc::smem_u32(Bbuf + c * kTcBTile),
                        bimg + ((size_t)(g - g_begin) * nchunk + c) * kTcBTile, kTcBTile,
                        tc::smem_u32(&bar_b));
  }
  stage_chunk(cw.C, 0, cw.K, sH, cmul, sC, sNL, sNa);
  __syncthreads();

  // Na <= max row sum of |H_g| * L1max * cinf over the codebook (cbmax: L1max, cinf)
  float hrow = 0.f;
#pragma unroll
  for (int a = 0; a < kD; ++a) {
    float rs = 0.f;
#pragma unroll
    for (int b = 0; b < kD; ++b) rs += fabsf(sH[a * kD + b]);
    hrow = fmaxf(hrow, rs);
  }
  const float l1max = cbmax[0], cinf = cbmax[1];
  const float na_max = hrow * l1max * cinf * (1.f + kU * cmul) * 1.0001f;
  constexpr uint32_t idesc = tc::idesc_tf32(kRows, kTcCols);

  const int Bh = (sd.s == 0) ? 1 : (live ? bb.n_in[vi] : 1);
  const int Bmax = (sd.s == 0) ? 1 : B;  // uniform hypothesis loop bound of the CTA
  float th[kD], tl[kD];
  if (live) {
    dfl::target(set, cbs, n_fixed, i, g, th, tl, err);
  } else {
#pragma unroll
    for (int j = 0; j < kD; ++j) th[j] = tl[j] = 0.f;
  }
  // The sorted top-L list lives in shared memory ([j][thread]), `last` = its last value: a
  // candidate that does not enter costs one compare, one that does only the shifts it needs
  // (a register list would be updated by a predicated network for every candidate).
#pragma unroll
  for (int j = 0; j < L; ++j) {
    sTopV[j * kThreads + tid] = INFINITY;
    sTopI[j * kThreads + tid] = 0x7fffffff;
  }
  float last = INFINITY;
  float tau_x = INFINITY;
  bool ok = true;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
  // Terms of hypothesis h (zero for a thread without it) and its A row. The terms of h + 1
  // are computed while the tensor cores run the pass of h, its row written once that pass
  // has completed.
  auto hyp_terms = [&](int h, float m2q[kD], float& base, float& nbeta, float& eps) {
#pragma unroll
    for (int p = 0; p < kD; ++p) m2q[p] = 0.f;
    base = nbeta = eps = 0.f;
    if (live && h < Bh) {
      float rh[kD], rl[kD], rr, ra, pmax;
      const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + h) * S : nullptr;
      hyp_residual_pair(th, tl, cbs, sd, pc, rh, rl, err);
      hyp_terms_pair(rh, rl, sH, m2q, rr, ra, pmax);
      sRa[h * kThreads + tid] = ra;
      sPm[h * kThreads + tid] = pmax;
      base = rr - kU * cmul * ra;
      nbeta = -2.f * kU * cmul * pmax;
      eps = 2.44140625e-04f *  // 2^-12
            (fabsf(base) + na_max + 2.f * pmax * l1max * 1.0001f + fabsf(nbeta) * l1max);
    }
  };
  auto write_a = [&](const float m2q[kD], float base, float nbeta) {
    uint32_t row[kK];
#pragma unroll
    for (int p = 0; p < kD; ++p) {
      uint32_t hh, ll;
      split(m2q[p], hh, ll);
      row[p] = hh;
      row[8 + p] = hh;
      row[16 + p] = ll;
    }
    const uint32_t one = __float_as_uint(1.f);
    row[24] = one;
    row[25] = one;
    split(nbeta, row[26], row[28]);
    row[27] = row[26];
    split(base, row[29], row[30]);
    row[31] = 0u;
    put_row(Atile, tid, row);
  };
  float m2q[kD], base, nbeta, eps;
  hyp_terms(0, m2q, base, nbeta, eps);
  write_a(m2q, base, nbeta);
  for (int h = 0; h < Bmax && ok; ++h) {
    const bool act = live && h < Bh;
    tc::fence_async_smem();
    tc::tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      bool bok = true;
      if (h == 0) bok = tc::mbar_wait(tc::smem_u32(&bar_b), 0u, err);
      if (bok) {
        tc::tc_fence_after();
        const uint32_t a0 = tc::smem_u32(Atile);
        for (int c = 0; c < nchunk; ++c) {
          const uint32_t b0 = tc::smem_u32(Bbuf + c * kTcBTile);
#pragma unroll
          for (int ks = 0; ks < kK / 8; ++ks)
            tc::mma_tf32(tmem + (uint32_t)(c * kTcCols),
                         tc::smem_desc(a0 + ks * 256, 128, (kK / 4) * 128),
                         tc::smem_desc(b0 + ks * 256, 128, (kK / 4) * 128), idesc,
                         ks > 0 ? 1u : 0u);
        }
        tc::mma_commit(tc::smem_u32(&bar_mma));
      } else {
        tc::mbar_arrive(tc::smem_u32(&bar_mma));  // release the waiters; ok turns false
      }
      if (!bok) raise_error(err, ERRBIT_TIMEOUT);
    }
    float nm2q[kD], nbase, nnbeta, neps;
    if (h + 1 < Bmax) hyp_terms(h + 1, nm2q, nbase, nnbeta, neps);
    bool wok = tc::mbar_wait(tc::smem_u32(&bar_mma), (uint32_t)(h & 1), err);
    if (h == 0 && tid == 0) wok = wok && tc::mbar_try_wait(tc::smem_u32(&bar_b), 0u);
    ok = __syncthreads_and(wok);
    if (!ok) break;
    tc::tc_fence_after();

    const int nq = nchunk * 2;  // 64-column loads
    if (h == 0) {  // tau from the block minima of y for hypothesis 0
      float bl[L];
#pragma unroll
      for (int j = 0; j < L; ++j) bl[j] = INFINITY;
#pragma unroll 1
      for (int q = 0; q < nq; ++q) {
        uint32_t v[64];
        tc::tmem_ld64_wait(trow + 64 * q, v);
#pragma unroll
        for (int b4 = 0; b4 < 4; ++b4) {
          float m = __uint_as_float(v[16 * b4]);
#pragma unroll
          for (int e = 1; e < 16; ++e) m = fminf(m, __uint_as_float(v[16 * b4 + e]));
          m = (m == m) ? m : INFINITY;  // a block of NaNs holds no bound
#pragma unroll
          for (int j = 0; j < L; ++j) {
            const float t = fmaxf(bl[j], m);
            bl[j] = fminf(bl[j], m);
            m = t;
          }
        }
      }
      if (act) tau_x = __fadd_ru(bl[L - 1], eps);
    }
    // Candidates of hypothesis h, 64 columns at a time: a mask (a compare and a predicated or
    // per score), then its members in codeword order, scored again with the fast stage's chain
    // and inserted; the threshold tightens after every 64 columns. NaN threshold for a thread
    // without this hypothesis: no value compares below it.
#pragma unroll 1
    for (int q = 0; q < nq; ++q) {
      const float thrD =
          act ? __fadd_ru(fminf(last, tau_x), eps) : __int_as_float(0x7fffffff);
      uint32_t m0 = 0u, m1 = 0u;
      {
        uint32_t v[64];
        tc::tmem_ld64_wait(trow + 64 * q, v);
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          if (__uint_as_float(v[e]) <= thrD) m0 |= 1u << e;
          if (__uint_as_float(v[32 + e]) <= thrD) m1 |= 1u << e;
        }
      }
#pragma unroll
      for (int w = 0; w < 2; ++w) {
        uint32_t m = w ? m1 : m0;
        while (m) {
          const int k = 64 * q + 32 * w + __ffs(m) - 1;
          m &= m - 1u;
          if (k >= cw.K) break;  // padding columns (only with an unbounded threshold)
          const float4 c0 = *reinterpret_cast<const float4*>(sC + k * kD);
          const float4 c1 = *reinterpret_cast<const float4*>(sC + k * kD + 4);
          const float2 nl = sNL[k];
          float sv = base + nl.x;
          sv = fmaf(m2q[0], c0.x, sv);
          sv = fmaf(m2q[1], c0.y, sv);
          sv = fmaf(m2q[2], c0.z, sv);
          sv = fmaf(m2q[3], c0.w, sv);
          sv = fmaf(m2q[4], c1.x, sv);
          sv = fmaf(m2q[5], c1.y, sv);
          sv = fmaf(m2q[6], c1.z, sv);
          sv = fmaf(m2q[7], c1.w, sv);
          sv = fmaf(nbeta, nl.y, sv);
          if (sv < last) {  // insert before the first entry strictly above sv
            int j = L - 1;
            while (j > 0) {
              const float pv = sTopV[(j - 1) * kThreads + tid];
              if (!(sv < pv)) break;
              sTopV[j * kThreads + tid] = pv;
              sTopI[j * kThreads + tid] = sTopI[(j - 1) * kThreads + tid];
              --j;
            }
            sTopV[j * kThreads + tid] = sv;
            sTopI[j * kThreads + tid] = (h << 16) | k;
            last = sTopV[(L - 1) * kThreads + tid];
          }
        }
      }
      __syncwarp();
    }
    tc::tc_fence_before();
    if (h + 1 < Bmax) {  // the pass of h has completed: its A tile is free
      write_a(nm2q, nbase, nnbeta);
#pragma unroll
      for (int p = 0; p < kD; ++p) m2q[p] = nm2q[p];
      base = nbase;
      nbeta = nnbeta;
      eps = neps;
    }
  }
  // let the codebook copy land before the CTA ends (bounded), then free the tensor memory
  if (!ok && tid == 0) tc::mbar_wait(tc::smem_u32(&bar_b), 0u, err);
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 2 * kTcCols);
  if (!live) return;
  float topv[L];
  int topi[L];
#pragma unroll
  for (int j = 0; j < L; ++j) {
    topv[j] = sTopV[j * kThreads + tid];
    topi[j] = sTopI[j * kThreads + tid];
  }
  beam_list_finish<L>(set, cbs, sd, bb, flags, i, g, vi, Bh, cmul, th, tl, sH, sNL, sNa, true,
                      sRa + tid, sPm + tid, kThreads, topv, topi, err);
}

// Exact stage for flagged vectors: one warp per vector; the lanes stride over the (h, k)
// candidates, re-score in fp64 those whose fp32 lower bound is at most the vector's
// threshold (the keep-th exact err among the fast pass's listed candidates, which bounds
// every member of the exact top-Bs) and keep a sorted local top-Bs; a warp merge then
// extracts the global top-Bs in (err, h, k) order.
__global__ void __launch_bounds__(kThreads)
beam_stage_fallback_kernel(SetView set, int64_t g_begin, int64_t G_range, CbList cbs,
                           int n_fixed, StageDesc sd, BeamBufs bb, FlagList flags,
                           unsigned* err) {
  __shared__ int queue[kThreads / 32][32], queue_h[kThreads / 32][32];
  const int lane = threadIdx.x & 31;
  int* q = queue[threadIdx.x >> 5];
  int* qh = queue_h[threadIdx.x >> 5];
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const unsigned cnt = min((unsigned long long)*flags.count, (unsigned long long)flags.cap);
  if (flags.total && blockIdx.x == 0 && threadIdx.x == 0) atomicAdd(flags.total, cnt);
  const int S = sd.S, B = sd.B, Bs = sd.Bs;
  const CbView cw = cbs.cb[sd.st[sd.s]];
  for (int64_t f = warp; f < cnt; f += nwarps) {
    const int64_t vi = flags.vec[f];
    const int64_t i = vi / G_range, g = g_begin + vi % G_range;
    const float* H = set.Hb + g * kD * kD;
    double tgt[kD];
    target64(set, cbs, n_fixed, i, g, tgt, err);
    const int Bh = (sd.s == 0) ? 1 : bb.n_in[vi];
    const float thr = flags.thr[f];
    const float cmul = bound_mult(n_fixed + sd.s);
    double be[16];
    int bh[16], bk[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) be[j] = INFINITY;
    int nb = 0;
    // Candidates (h, k) are queued in increasing (h, k) order and scored one per lane, so
    // every lane still sees its own candidates in increasing (h, k): strict comparison in
    // the insertion keeps ties in (h, k) order.
    int qn = 0;
    auto drain = [&]() {
      __syncwarp();
      if (lane < qn) {
        const int h = qh[lane], k = q[lane];
        double r64[kD];
        const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + h) * S : nullptr;
        hyp_residual64(tgt, cbs, sd, pc, r64, err);
        const double e = quad_err64(r64, cw.C + (int64_t)k * kD, H);
        if (nb < Bs || e < be[nb - 1]) {
          int pos = nb < Bs ? nb : Bs - 1;
          while (pos > 0 && e < be[pos - 1]) {
            be[pos] = be[pos - 1]; bh[pos] = bh[pos - 1]; bk[pos] = bk[pos - 1];
            --pos;
          }
          be[pos] = e; bh[pos] = h; bk[pos] = k;
          if (nb < Bs) ++nb;
        }
      }
      __syncwarp();
      qn = 0;
    };
    for (int h = 0; h < Bh; ++h) {
      double r64[kD];
      const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + h) * S : nullptr;
      hyp_residual64(tgt, cbs, sd, pc, r64, err);
      float m2q[kD], rr, ra, pmax;
      hyp_terms(r64, H, m2q, rr, ra, pmax);
      const float base = rr - kU * cmul * ra;
      const float nbeta = -2.f * kU * cmul * pmax;
      for (int k0 = 0; k0 < cw.K; k0 += 32) {
        const int k = k0 + lane;
        bool cand = false;
        if (k < cw.K) {
          float c[kD];
          load_vec(cw.C + (int64_t)k * kD, c);
          cand = base + low_score(c, H, m2q, nbeta, cmul) <= thr;
        }
        const unsigned m = __ballot_sync(0xffffffffu, cand);
        const int n = __popc(m);
        if (qn + n > 32) drain();
        if (cand) {
          const int pos = qn + __popc(m & ((1u << lane) - 1u));
          q[pos] = k;
          qh[pos] = h;
        }
        qn += n;
      }
    }
    drain();
    // Warp merge: rounds of (min over the lanes' heads by (err, h, k)); the winner pops.
    int head = 0;
    int32_t* out = bb.hyp_out + vi * B * S;
    const int total = (int)min((int64_t)Bs, (int64_t)Bh * cw.K);
    for (int j = 0; j < total; ++j) {
      double e = head < nb ? be[head] : INFINITY;
      int hh = head < nb ? bh[head] : 0x7fffffff;
      int kk = head < nb ? bk[head] : 0x7fffffff;
      int src = lane;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const double oe = __shfl_xor_sync(0xffffffffu, e, off);
        const int oh = __shfl_xor_sync(0xffffffffu, hh, off);
        const int ok = __shfl_xor_sync(0xffffffffu, kk, off);
        const int os = __shfl_xor_sync(0xffffffffu, src, off);
        const bool take = oe < e || (oe == e && (oh < hh || (oh == hh && ok < kk)));
        if (take) {
          e = oe; hh = oh; kk = ok; src = os;
        }
      }
      if (lane == src) ++head;
      if (lane == 0) {
        if (hh >= Bh || kk >= cw.K) {
          raise_error(err, ERRBIT_NUMERIC);
          hh = 0;
          kk = 0;
        }
        const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + hh) * S : nullptr;
        for (int q = 0; q < sd.s; ++q) out[j * S + q] = pc[q];
        out[j * S + sd.s] = kk;
      }
    }
    if (lane == 0) bb.n_out[vi] = total;
  }
}

// fp32 err of a whole tuple for vector (i, g): the fixed codebooks' codes, then for each
// searched stage q the code sc[q] (or, with sc null, the code already stored), with a bound
// on its distance from the exact err: the residual's rounding (m subtractions) and the two
// FMA chains of the quadratic form stay below (16 + 2 m) u a^T |H| a, a_j = |t_j| + sum of
// the |c_j| subtracted; the bound uses the multiplier of the score bounds, about twice that.
__device__ void tuple_err32(const SetView& set, const CbList& cbs, int n_fixed,
                            const StageDesc& sd, int64_t i, int64_t g, const int32_t* sc,
                            const float* H, float& e, float& bnd, unsigned* err) {
  float r[kD], a[kD];
  target32(set, cbs, n_fixed, i, g, r, a, err);
  for (int q = 0; q < sd.S; ++q) {
    const CbView& cb = cbs.cb[sd.st[q]];
    const int32_t k = sc ? sc[q] : cb.codes[i * cb.ld + g];
    if (!code_ok(k, cb.K, err)) continue;
    float c[kD];
    load_vec(cb.C + (int64_t)k * kD, c);
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      r[j] -= c[j];
      a[j] += fabsf(c[j]);
    }
  }
  float ee = 0.f, na = 0.f;
#pragma unroll
  for (int b = 0; b < kD; ++b) {
    float hb = 0.f, hab = 0.f;
#pragma unroll
    for (int a2 = 0; a2 < kD; ++a2) {
      hb = fmaf(r[a2], H[a2 * kD + b], hb);
      hab = fmaf(a[a2], fabsf(H[a2 * kD + b]), hab);
    }
    ee = fmaf(hb, r[b], ee);
    na = fmaf(hab, a[b], na);
  }
  e = ee;
  bnd = kU * bound_mult(n_fixed + sd.S + 1) * na;
}

// Final step of a multi-stage (or keep-if-better) encode: write the best tuple, or keep the
// tuple already in the codes when its err is strictly smaller. The comparison is decided by
// fp32 errs with bounds when they separate, in fp64 otherwise; an unchanged tuple needs no
// comparison. vec_err (optional) is the fp64 err of the tuple kept.
__global__ void beam_finalize_kernel(SetView set, int64_t g_begin, int64_t G_range,
                                     CbList cbs, int n_fixed, StageDesc sd,
                                     const int32_t* __restrict__ hyp, bool keep_if_better,
                                     float* __restrict__ vec_err, unsigned* err) {
  const int64_t nvec = set.M * G_range;
  const int S = sd.S, B = sd.B;
  for (int64_t vi = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; vi < nvec;
       vi += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = vi / G_range, g = g_begin + vi % G_range;
    const float* H = set.Hb + g * kD * kD;
    const int32_t* best = hyp + vi * B * S;
    bool use_old = false;
    bool exact = vec_err != nullptr;
    if (keep_if_better) {
      bool same = true;
      for (int q = 0; q < S; ++q) {
        const CbView& cb = cbs.cb[sd.st[q]];
        same = same && cb.codes[i * cb.ld + g] == best[q];
      }
      if (!same) {
        float en, bn, eo, bo;
        tuple_err32(set, cbs, n_fixed, sd, i, g, best, H, en, bn, err);
        tuple_err32(set, cbs, n_fixed, sd, i, g, nullptr, H, eo, bo, err);
        if (eo + bo < en - bn) {
          use_old = true;
        } else if (!(eo - bo >= en + bn)) {
          exact = true;  // not separated (or not finite): decide in fp64
        }
      }
    }
    if (exact) {
      double tgt[kD];
      target64(set, cbs, n_fixed, i, g, tgt, err);
      double r[kD];
#pragma unroll
      for (int j = 0; j < kD; ++j) r[j] = tgt[j];
      for (int q = 0; q < S; ++q) {
        const CbView& cb = cbs.cb[sd.st[q]];
        if (!code_ok(best[q], cb.K, err)) continue;
        const float* c = cb.C + (int64_t)best[q] * kD;
#pragma unroll
        for (int j = 0; j < kD; ++j) r[j] -= (double)c[j];
      }
      const double e_new = quad_err64(r, nullptr, H);
      double e_old = e_new;
      if (keep_if_better) {
#pragma unroll
        for (int j = 0; j < kD; ++j) r[j] = tgt[j];
        for (int q = 0; q < S; ++q) {
          const CbView& cb = cbs.cb[sd.st[q]];
          const int32_t k = cb.codes[i * cb.ld + g];
          if (!code_ok(k, cb.K, err)) continue;
          const float* c = cb.C + (int64_t)k * kD;
#pragma unroll
          for (int j = 0; j < kD; ++j) r[j] -= (double)c[j];
        }
        e_old = quad_err64(r, nullptr, H);
        use_old = e_old < e_new;
      }
      if (vec_err) vec_err[i * set.G_sub + g] = (float)(use_old ? e_old : e_new);
    }
    if (!use_old) {
      for (int q = 0; q < S; ++q) {
        const CbView& cb = cbs.cb[sd.st[q]];
        cb.codes[i * cb.ld + g] = best[q];
      }
    }
  }
}

// err of the tuple currently in the codes (all covering codebooks), fp64.
__global__ void residual_err_kernel(SetView set, int64_t g_begin, int64_t G_range, CbList cbs,
                                    float* __restrict__ vec_err, unsigned* err) {
  const int64_t nvec = set.M * G_range;
  for (int64_t vi = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; vi < nvec;
       vi += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = vi / G_range, g = g_begin + vi % G_range;
    double r[kD];
    target64(set, cbs, cbs.n, i, g, r, err);
    vec_err[i * set.G_sub + g] = (float)quad_err64(r, nullptr, set.Hb + g * kD * kD);
  }
}

// --------------------------------------------------------------------------- k-means init
__global__ void kmeans_init_kernel(SetView set, CbList fixed, int K, uint64_t seed,
                                   float* __restrict__ C_out, unsigned* err) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= K) return;
  const int64_t n = set.M * set.G_sub;
  // Stratum k of the vector index range: [floor(k n / K), floor((k+1) n / K)).
  const int64_t lo = (int64_t)(((uint64_t)k * (uint64_t)n) / (uint64_t)K);
  const int64_t hi = (int64_t)(((uint64_t)(k + 1) * (uint64_t)n) / (uint64_t)K);
  const int64_t v = lo + (int64_t)(splitmix64(seed, (uint64_t)k) % (uint64_t)(hi - lo));
  const int64_t i = v / set.G_sub, g = v % set.G_sub;
  double r[kD];
  target64(set, fixed, fixed.n, i, g, r, err);
#pragma unroll
  for (int j = 0; j < kD; ++j) C_out[(int64_t)k * kD + j] = (float)r[j];
}

}  // namespace

// =============================================================================== host side
template <class Kern>
static crvq_status set_smem_attr(Kern k, size_t bytes) {
  CRVQ_CUDA(cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes));
  return CRVQ_OK;
}

crvq_status launch_kmeans_init(const SetView& set, const CbList& fixed, int K, uint64_t seed,
                               float* C_out, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  ProfScope ps("kmeans_init", stream, (double)K);
  kmeans_init_kernel<<<(unsigned)ceil_div(K, 128), 128, 0, stream>>>(set, fixed, K, seed,
                                                                    C_out, err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

namespace {

template <int L>
crvq_status launch_beam_stage_L(const SetView& set, int64_t g_begin, int64_t G_range,
                                const CbList& cbs, int n_fixed, const StageDesc& sd,
                                const BeamBufs& bb, const FlagList& fl, unsigned* err,
                                double units, cudaStream_t stream) {
  dim3 grid((unsigned)ceil_div(set.M, kThreads), (unsigned)G_range);
  ProfScope ps("encode_beam_stage", stream, units);
  beam_stage_kernel<L><<<grid, kThreads, 0, stream>>>(set, g_begin, cbs, n_fixed, sd, bb, fl,
                                                     err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

template <int L>
crvq_status launch_beam_tc_L(const SetView& set, int64_t g_begin, int64_t G_range,
                             const CbList& cbs, int n_fixed, const StageDesc& sd,
                             const BeamBufs& bb, const char* bimg, const float* cbmax,
                             const FlagList& fl, unsigned* err, double units,
                             cudaStream_t stream) {
  CRVQ_TRY(set_smem_attr(beam_tc_kernel<L>, kBeamTcSmem));
  dim3 grid((unsigned)ceil_div(set.M, kThreads), (unsigned)G_range);
  ProfScope ps("encode_beam_stage", stream, units);
  beam_tc_kernel<L><<<grid, kThreads, kBeamTcSmem, stream>>>(set, g_begin, cbs, n_fixed, sd, bb,
                                                             bimg, cbmax, fl, err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

// The tensor-core stage for codebooks of at most 256 codewords and lists of at most 9 entries
// (beam width up to 8): B images of the stage codebook for the group range (prep_b with the
// stage's bound multiplier), then beam_tc_kernel. `work` holds beam_tc_scratch_bytes.
size_t beam_tc_scratch_bytes(int64_t G_range, int K) {
  const int nchunk = (int)ceil_div(K, kTcCols);
  return 256 + (size_t)G_range * nchunk * kTcBTile +
         align_up((size_t)G_range * K * sizeof(float4), 256) + 256;
}

// CRVQ_BEAM_TC=0 in the environment (read at every call) keeps every stage on the SIMT kernel:
// the two forms give the same lists, which tests compare.
bool beam_tc_applies(const StageDesc& sd, const CbList& cbs, int64_t G_range) {
  const char* v = getenv("CRVQ_BEAM_TC");
  if (v && v[0] == '0') return false;
  const int K = cbs.cb[sd.st[sd.s]].K;
  return K <= 2 * kTcCols && sd.Bs + 1 <= 9 &&
         (size_t)G_range * ceil_div(K, kTcCols) * kTcBTile <= (size_t(256) << 20);
}

crvq_status launch_beam_stage_tc(const SetView& set, int64_t g_begin, int64_t G_range,
                                 const CbList& cbs, int n_fixed, const StageDesc& sd,
                                 const BeamBufs& bb, const FlagList& fl, unsigned* err,
                                 char* work, double units, cudaStream_t stream) {
  const CbView& cw = cbs.cb[sd.st[sd.s]];
  const int nchunk = (int)ceil_div(cw.K, kTcCols);
  float* cbmax = reinterpret_cast<float*>(work);
  char* bimg = work + 256;
  float4* tout = reinterpret_cast<float4*>(bimg + (size_t)G_range * nchunk * kTcBTile);
  const float uc = kU * bound_mult(n_fixed + sd.s);
  {
    ProfScope pb("encode_prep_b", stream, (double)G_range * nchunk * kTcCols);
    const int64_t rows = G_range * nchunk * kTcCols;
    CRVQ_CUDA(launch_pdl(prep_b_kernel,
                         dim3((unsigned)std::min<int64_t>(ceil_div(rows, 128), 16 * sm_count()) +
                              1),
                         dim3(128), 0, stream, set, g_begin, G_range, cw.C, cw.K, nchunk, uc,
                         bimg, tout, cbmax, fl.count));
    CRVQ_LAUNCHED();
  }
  // the list length L = Bs + 1, rounded up to an instantiated size
  auto go = [&](auto L) {
    return launch_beam_tc_L<decltype(L)::value>(set, g_begin, G_range, cbs, n_fixed, sd, bb,
                                                 bimg, cbmax, fl, err, units, stream);
  };
  const int need = sd.Bs + 1;
  if (need <= 2) return go(std::integral_constant<int, 2>{});
  if (need <= 3) return go(std::integral_constant<int, 3>{});
  if (need <= 5) return go(std::integral_constant<int, 5>{});
  return go(std::integral_constant<int, 9>{});
}

crvq_status launch_beam_stage(const SetView& set, int64_t g_begin, int64_t G_range,
                              const CbList& cbs, int n_fixed, const StageDesc& sd,
                              const BeamBufs& bb, const FlagList& fl, unsigned* err,
                              double units, cudaStream_t stream) {
  auto go = [&](auto L) {
    return launch_beam_stage_L<decltype(L)::value>(set, g_begin, G_range, cbs, n_fixed, sd, bb,
                                                   fl, err, units, stream);
  };
  const int need = sd.Bs + 1;
  if (need <= 2) return go(std::integral_constant<int, 2>{});
  if (need <= 3) return go(std::integral_constant<int, 3>{});
  if (need <= 5) return go(std::integral_constant<int, 5>{});
  if (need <= 9) return go(std::integral_constant<int, 9>{});
  return go(std::integral_constant<int, 17>{});
}

// Scratch of one arg-min pass: codebook maxima (256 B) | B images of G_sub groups (groups
// in sub-ranges whose images take at most 256 MB) | codeword terms | flag count (256 B) |
// flag list (vector ids and thresholds).
struct ArgminLayout {
  int nchunk;
  int64_t G_sub;
  size_t bbytes, tbytes, fbytes, total;
};

ArgminLayout argmin_layout(int64_t M, int64_t G_range, int K) {
  ArgminLayout L;
  L.nchunk = (int)ceil_div(K, kTcCols);
  const int64_t per_group = (int64_t)L.nchunk * kTcBTile;
  L.G_sub = std::max<int64_t>(1, std::min<int64_t>(G_range, (int64_t(256) << 20) / per_group));
  L.bbytes = (size_t)L.G_sub * per_group;
  L.tbytes = align_up((size_t)L.G_sub * K * sizeof(float4), 256);
  L.fbytes = align_up((size_t)M * L.G_sub * (sizeof(int64_t) + sizeof(float)), 256);
  L.total = 256 + L.bbytes + L.tbytes + 256 + L.fbytes;
  return L;
}

// One range of groups [g_begin, g_begin + G_range) whose searched stages are sd.st[0..S).
crvq_status encode_range(const SetView& set, int64_t g_begin, int64_t G_range,
                         const CbList& cbs, int n_fixed, StageDesc sd, bool keep_if_better,
                         float* vec_err, const EncodeExtras& ex, unsigned* err,
                         cudaStream_t stream) {
  const int64_t nvec = set.M * G_range;
  if (nvec == 0) return CRVQ_OK;
  const int nsm = sm_count();
  const unsigned fin_blocks = (unsigned)std::min<int64_t>(ceil_div(nvec, 128), 8 * nsm);
  if (sd.S == 0) {
    if (vec_err) {
      residual_err_kernel<<<fin_blocks, 128, 0, stream>>>(set, g_begin, G_range, cbs, vec_err,
                                                          err);
      CRVQ_LAUNCHED();
    }
    return CRVQ_OK;
  }
  if (sd.S == 1) {
    // Arg-min over one codebook (the k-means assignment step). Written in place unless the
    // old code may be kept, in which case into a scratch tuple buffer that the finalize step
    // compares with the old tuple.
    const int s_idx = sd.st[0];
    const CbView& cw = cbs.cb[s_idx];
    Scratch tup_mem;
    int32_t* out = cw.codes;
    int64_t out_ld = cw.ld, out_g0 = 0;
    if (keep_if_better) {
      CRVQ_TRY(tup_mem.alloc((size_t)nvec * sizeof(int32_t), stream));
      out = tup_mem.as<int32_t>();
      out_ld = G_range;
      out_g0 = g_begin;
    }
    StatsView st{};
    if (ex.stats && !keep_if_better) st = *ex.stats;
    // Groups in sub-ranges whose B images (the codebook's tensor-core operand per group) take
    // at most 256 MB; per sub-range: images + per-group codeword terms (prep_b, which also
    // writes the codebook maxima), the arg-min pass, and the exact decision of flagged rows.
    const ArgminLayout AL = argmin_layout(set.M, G_range, cw.K);
    const int nchunk = AL.nchunk;
    const int64_t G_sub = AL.G_sub;
    const size_t bbytes = AL.bbytes, tbytes = AL.tbytes;
    Scratch bmem;
    char* wbase = ex.work;
    if (!wbase || ex.work_bytes < AL.total) {
      CRVQ_TRY(bmem.alloc(AL.total, stream));
      wbase = bmem.as<char>();
    }
    float* cbmax = reinterpret_cast<float*>(wbase);
    char* bimg = wbase + 256;
    float4* tout = reinterpret_cast<float4*>(bimg + bbytes);
    FlagList fl;
    fl.count = reinterpret_cast<unsigned*>(wbase + 256 + bbytes + tbytes);
    fl.vec = reinterpret_cast<int64_t*>(wbase + 256 + bbytes + tbytes + 256);
    fl.cap = set.M * G_sub;
    fl.thr = reinterpret_cast<float*>(fl.vec + fl.cap);
    fl.total = ex.flag_total;
    const float uc = kU * (tcenc::kCmul + 4.f * n_fixed);
    // two independent 128-thread halves per CTA when the codebook stays resident (K <= 256)
    const bool two_halves = nchunk <= 2;
    CRVQ_TRY(set_smem_attr(argmin_tc_kernel<1>, argmin_smem(1)));
    CRVQ_TRY(set_smem_attr(argmin_tc_kernel<2>, argmin_smem(2)));
    for (int64_t gs = g_begin; gs < g_begin + G_range; gs += G_sub) {
      const int64_t gn = std::min<int64_t>(G_sub, g_begin + G_range - gs);
      const int64_t nv = set.M * gn;
      fl.cap = nv;
      fl.thr = reinterpret_cast<float*>(fl.vec + nv);  // the count is cleared by prep_b
      {
        ProfScope pb("encode_prep_b", stream, (double)gn * nchunk * kTcCols);
        const int64_t rows = gn * nchunk * kTcCols;
        CRVQ_CUDA(launch_pdl(prep_b_kernel,
                             dim3((unsigned)std::min<int64_t>(ceil_div(rows, 128), 16 * nsm) + 1),
                             dim3(128), 0, stream, set, gs, gn, cw.C, cw.K, nchunk, uc, bimg,
                             tout, cbmax, fl.count));
        CRVQ_LAUNCHED();
      }
      {
        // row tiles per CTA: about eight waves of three CTAs per SM with one half (a
        // fine-grained tail); with two halves about four waves of two (fewer statistics
        // flushes and codebook fetches; measured 3% faster than eight waves, 10% faster than
        // sixteen), each CTA reusing its group's resident codebook operand over several tiles
        // (an even count with two halves)
        const int64_t row_tiles = ceil_div(set.M, tcenc::kRows);
        const int64_t want_ctas = (two_halves ? 8 : 24) * (int64_t)nsm;
        const int64_t per_group = std::max<int64_t>(1, want_ctas / std::max<int64_t>(1, gn));
        int tiles = (int)std::max<int64_t>(1, ceil_div(row_tiles, per_group));
        if (two_halves) tiles += tiles & 1;
        // fused statistics in 32-bit shared sums: fewer than 2^16 rows per CTA
        if (st.cnt && cw.K <= kTcSmemStatsK) tiles = std::min(tiles, 510);
        const dim3 grid((unsigned)ceil_div(row_tiles, tiles), (unsigned)gn);
        ProfScope ps(st.cnt ? "encode_argmin_lloyd" : "encode_argmin", stream,
                     (double)nv * cw.K);
        if (two_halves)
          CRVQ_CUDA(launch_pdl(argmin_tc_kernel<2>, grid, dim3(256), argmin_smem(2), stream, set,
                               gs, cbs, n_fixed, s_idx, out, out_ld, out_g0, fl, st, cbmax,
                               bimg, tout, ex.rowterms, tiles, err));
        else
          CRVQ_CUDA(launch_pdl(argmin_tc_kernel<1>, grid, dim3(128), argmin_smem(1), stream, set,
                               gs, cbs, n_fixed, s_idx, out, out_ld, out_g0, fl, st, cbmax,
                               bimg, tout, ex.rowterms, tiles, err));
        CRVQ_LAUNCHED();
      }
      {
        ProfScope pf("encode_exact", stream, 0.0);
        if (cw.K <= kExactWarpK) {
          CRVQ_CUDA(launch_pdl(argmin_exact_warp_kernel,
                               dim3((unsigned)std::min<int64_t>(ceil_div(nv, 4), 16 * nsm)),
                               dim3(128), 0, stream, set, gs, gn, cbs, n_fixed, s_idx, out,
                               out_ld, out_g0, fl, st, tout, err));
        } else {
          CRVQ_CUDA(launch_pdl(argmin_exact_kernel,
                               dim3((unsigned)std::min<int64_t>(nv, 16 * nsm)), dim3(128), 0,
                               stream, set, gs, gn, cbs, n_fixed, s_idx, out, out_ld, out_g0, fl,
                               st, tout, err));
        }
        CRVQ_LAUNCHED();
      }
    }
    if (ex.scores) *ex.scores += (double)nvec * cw.K;
    if (keep_if_better) {
      ProfScope ps3("encode_finalize", stream, 0.0);
      StageDesc one = sd;
      one.B = 1;
      one.Bs = 1;
      beam_finalize_kernel<<<fin_blocks, 128, 0, stream>>>(set, g_begin, G_range, cbs, n_fixed,
                                                           one, out, true, vec_err, err);
      CRVQ_LAUNCHED();
    } else if (vec_err) {
      ProfScope ps3("encode_finalize", stream, 0.0);
      residual_err_kernel<<<fin_blocks, 128, 0, stream>>>(set, g_begin, G_range, cbs, vec_err,
                                                          err);
      CRVQ_LAUNCHED();
    }
    return CRVQ_OK;
  }

  Scratch flag_mem;
  const size_t fl_bytes = (size_t)nvec * (sizeof(int64_t) + sizeof(float)) + 256;
  CRVQ_TRY(flag_mem.alloc(fl_bytes, stream));
  FlagList fl;
  fl.count = flag_mem.as<unsigned>();
  fl.vec = reinterpret_cast<int64_t*>(flag_mem.as<char>() + 256);
  fl.thr = reinterpret_cast<float*>(fl.vec + nvec);
  fl.cap = nvec;
  fl.total = ex.flag_total;

  // Beam over S >= 2 stages: stage kernels over double-buffered hypothesis arrays.
  Scratch hyp_mem;
  const int B = sd.B, S = sd.S;
  const size_t hyp_elems = (size_t)nvec * B * S;
  CRVQ_TRY(hyp_mem.alloc(2 * (hyp_elems + nvec) * sizeof(int32_t), stream));
  int32_t* hypA = hyp_mem.as<int32_t>();
  int32_t* hypB = hypA + hyp_elems;
  int32_t* nA = hypB + hyp_elems;
  int32_t* nB = nA + nvec;
  const int32_t* in_h = nullptr;
  const int32_t* in_n = nullptr;
  int32_t* out_h = hypA;
  int32_t* out_n = nA;
  double sc = 0.0;
  int64_t parents = 1;
  // scratch of the tensor-core stages (B images and terms of one stage codebook)
  size_t tc_bytes = 0;
  for (int s = 0; s < S; ++s) {
    StageDesc d = sd;
    d.s = s;
    d.Bs = (s == S - 1) ? 1 : B;
    if (beam_tc_applies(d, cbs, G_range))
      tc_bytes = std::max(tc_bytes, beam_tc_scratch_bytes(G_range, cbs.cb[sd.st[s]].K));
  }
  Scratch tc_mem;
  if (tc_bytes) CRVQ_TRY(tc_mem.alloc(tc_bytes, stream));
  for (int s = 0; s < S; ++s) {
    sd.s = s;
    sd.Bs = (s == S - 1) ? 1 : B;  // only the best tuple of the last stage is used
    CRVQ_CUDA(cudaMemsetAsync(fl.count, 0, sizeof(unsigned), stream));
    BeamBufs bb{in_h, in_n, out_h, out_n};
    const int K = cbs.cb[sd.st[s]].K;
    if (beam_tc_applies(sd, cbs, G_range))
      CRVQ_TRY(launch_beam_stage_tc(set, g_begin, G_range, cbs, n_fixed, sd, bb, fl, err,
                                    tc_mem.as<char>(), (double)nvec * parents * K, stream));
    else
      CRVQ_TRY(launch_beam_stage(set, g_begin, G_range, cbs, n_fixed, sd, bb, fl, err,
                                 (double)nvec * parents * K, stream));
    {
      ProfScope ps("encode_beam_fallback", stream, 0.0);
      beam_stage_fallback_kernel<<<4 * nsm, kThreads, 0, stream>>>(
          set, g_begin, G_range, cbs, n_fixed, sd, bb, fl, err);
      CRVQ_LAUNCHED();
    }
    sc += (double)nvec * parents * K;
    parents = std::min<int64_t>(B, parents * K);
    in_h = out_h;
    in_n = out_n;
    out_h = (out_h == hypA) ? hypB : hypA;
    out_n = (out_n == nA) ? nB : nA;
  }
  if (ex.scores) *ex.scores += sc;
  ProfScope ps("encode_finalize", stream, 0.0);
  beam_finalize_kernel<<<fin_blocks, 128, 0, stream>>>(set, g_begin, G_range, cbs, n_fixed, sd,
                                                       in_h, keep_if_better, vec_err, err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace

crvq_status launch_row_terms(const SetView& set, const CbList& cbs, int n_fixed, float4* rt,
                             cudaStream_t stream) {
  const int64_t nvec = set.M * set.G_sub;
  if (nvec == 0) return CRVQ_OK;
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const unsigned blocks = (unsigned)std::min<int64_t>(ceil_div(nvec, 128), 16 * sm_count());
  CRVQ_CUDA(launch_pdl(row_terms_kernel, dim3(blocks), dim3(128), 0, stream, set, cbs, n_fixed,
                       rt, err));
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

size_t argmin_scratch_bytes(int64_t M, int64_t G_range, int K) {
  return argmin_layout(M, G_range, K).total;
}

crvq_status launch_encode_beam(const SetView& set, const CbList& cbs, int n_fixed, int B,
                               bool keep_if_better, float* vec_err, const EncodeExtras& ex,
                               cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  // Group ranges with the same set of covering searched codebooks: boundaries at every G_cov.
  std::vector<int64_t> cuts = {0, set.G_sub};
  for (int s = n_fixed; s < cbs.n; ++s)
    if (cbs.cb[s].G_cov > 0 && cbs.cb[s].G_cov < set.G_sub) cuts.push_back(cbs.cb[s].G_cov);
  std::sort(cuts.begin(), cuts.end());
  cuts.erase(std::unique(cuts.begin(), cuts.end()), cuts.end());
  if (ex.stats && cuts.size() > 2)
    return fail(CRVQ_ERR_UNSUPPORTED, "fused statistics need one group range");
  for (size_t r = 0; r + 1 < cuts.size(); ++r) {
    const int64_t g0 = cuts[r], g1 = cuts[r + 1];
    StageDesc sd{};
    sd.S = 0;
    sd.B = B;
    sd.Bs = B;
    for (int s = n_fixed; s < cbs.n; ++s)
      if (g0 < cbs.cb[s].G_cov) sd.st[sd.S++] = s;
    CRVQ_TRY(encode_range(set, g0, g1 - g0, cbs, n_fixed, sd, keep_if_better, vec_err, ex, err,
                          stream));
  }
  return CRVQ_OK;
}

}  // namespace crvq
