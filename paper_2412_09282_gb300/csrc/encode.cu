// Vector x codeword score contraction with fused top-B selection (Sec. 3.1 Eq. (2)-(3);
// Alg. 1 VectorQuant and BeamSearchOptimize), and the k-means initial codebook draw.
//
// Score of target r against codeword c for a vector of group g:
//   err(r, c) = (r - c)^T H_g (r - c) = r^T H_g r + n_g(c) - 2 (H_g r) . c,  n_g(c) = c^T H_g c.
// The fast pass evaluates the expanded form in fp32 (8 FMAs per pair, the norm table of the
// group staged in shared memory) and keeps, per vector, the best and second-best values. An
// a-priori bound E on the fp32 error of every score (from the magnitudes of H_g, the target
// and the codebook) certifies the arg-min when the runner-up is more than 2E away; otherwise
// the vector goes to a fallback that re-scans it and decides among the candidates within 2E
// in fp64. The result equals the fp64 arg-min (ties to the smaller index) except for ties at
// fp64 rounding level.
#include <algorithm>
#include <vector>

#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

constexpr int kThreads = 128;
constexpr int kChunk = 1024;            // codewords staged per shared-memory chunk
constexpr float kU = 5.9604645e-08f;    // 2^-24

struct FlagList {
  int64_t* vec;      // vector index within the launch range (i * G_range + (g - g_begin))
  float* thr;        // decision threshold b1 + 2E (fast pass value units)
  unsigned* count;
  int64_t cap;
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

// fp32 target r = t - sum of the fixed codebooks covering g, and the magnitude bound
// a_j = |t_j| + sum |c_fixed,j| of every term that went into r.
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

// fp64 target (the fixed reconstruction subtracted in fp64).
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

// (r - c)^T H (r - c) in fp64; H row-major d x d (fp32), c fp32.
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

// Stage the codewords [k0, k0 + nk) of C and their group norms n_g(c) = c^T H c in shared
// memory; also the running maxima Na = max_k |c|^T |H| |c| and cmax_j = max_k |c_kj|.
__device__ __forceinline__ void stage_chunk(const float* __restrict__ C, int k0, int nk,
                                            const float* sH, float* sC, float* sN,
                                            unsigned* sNa_bits, unsigned* sCmax_bits) {
  for (int k = threadIdx.x; k < nk; k += blockDim.x) {
    float c[kD];
    load_vec(C + (int64_t)(k0 + k) * kD, c);
    float n = 0.f, na = 0.f;
#pragma unroll
    for (int a = 0; a < kD; ++a) {
      float u = 0.f, ua = 0.f;
#pragma unroll
      for (int b = 0; b < kD; ++b) {
        u = fmaf(sH[a * kD + b], c[b], u);
        ua = fmaf(fabsf(sH[a * kD + b]), fabsf(c[b]), ua);
      }
      n = fmaf(c[a], u, n);
      na = fmaf(fabsf(c[a]), ua, na);
    }
    *reinterpret_cast<float4*>(sC + k * kD) = make_float4(c[0], c[1], c[2], c[3]);
    *reinterpret_cast<float4*>(sC + k * kD + 4) = make_float4(c[4], c[5], c[6], c[7]);
    sN[k] = n;
    atomicMax(sNa_bits, __float_as_uint(na));
#pragma unroll
    for (int j = 0; j < kD; ++j) atomicMax(&sCmax_bits[j], __float_as_uint(fabsf(c[j])));
  }
}

// --------------------------------------------------------------------------- arg-min pass
// One CTA = one group g and kThreads * VPT rows. Each thread owns VPT vectors.
template <int VPT>
__global__ void __launch_bounds__(kThreads)
argmin_kernel(SetView set, int64_t g_begin, CbList cbs, int n_fixed, int s_idx,
              int32_t* __restrict__ out_code, int64_t out_ld, int64_t out_g0, FlagList flags,
              unsigned* err) {
  const int64_t g = g_begin + blockIdx.y;
  const int64_t G_range = gridDim.y;
  const int64_t row0 = (int64_t)blockIdx.x * kThreads * VPT;
  __shared__ float sH[kD * kD];
  __shared__ __align__(16) float sC[kChunk * kD];
  __shared__ float sN[kChunk];
  __shared__ unsigned sNa_bits, sCmax_bits[kD];

  if (threadIdx.x < kD * kD) sH[threadIdx.x] = set.Hb[g * kD * kD + threadIdx.x];
  if (threadIdx.x < kD) sCmax_bits[threadIdx.x] = 0u;
  if (threadIdx.x == 0) sNa_bits = 0u;
  __syncthreads();

  const CbView cw = cbs.cb[s_idx];
  float m2q[VPT][kD];
  float b1[VPT], b2[VPT];
  int i1[VPT];
  bool live[VPT];
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
    const int64_t i = row0 + threadIdx.x + (int64_t)v * kThreads;
    live[v] = i < set.M;
    float r[kD], a[kD];
    if (live[v]) {
      target32(set, cbs, n_fixed, i, g, r, a, err);
    } else {
#pragma unroll
      for (int j = 0; j < kD; ++j) r[j] = a[j] = 0.f;
    }
#pragma unroll
    for (int p = 0; p < kD; ++p) {
      float q = 0.f;
#pragma unroll
      for (int j = 0; j < kD; ++j) q = fmaf(sH[p * kD + j], r[j], q);
      m2q[v][p] = -2.f * q;
    }
    b1[v] = INFINITY;
    b2[v] = INFINITY;
    i1[v] = 0;
  }

  for (int k0 = 0; k0 < cw.K; k0 += kChunk) {
    const int nk = min(kChunk, cw.K - k0);
    __syncthreads();
    stage_chunk(cw.C, k0, nk, sH, sC, sN, &sNa_bits, sCmax_bits);
    __syncthreads();
#pragma unroll 2
    for (int k = 0; k < nk; ++k) {
      const float4 c0 = *reinterpret_cast<const float4*>(sC + k * kD);
      const float4 c1 = *reinterpret_cast<const float4*>(sC + k * kD + 4);
      const float n = sN[k];
#pragma unroll
      for (int v = 0; v < VPT; ++v) {
        float s = n;
        s = fmaf(m2q[v][0], c0.x, s);
        s = fmaf(m2q[v][1], c0.y, s);
        s = fmaf(m2q[v][2], c0.z, s);
        s = fmaf(m2q[v][3], c0.w, s);
        s = fmaf(m2q[v][4], c1.x, s);
        s = fmaf(m2q[v][5], c1.y, s);
        s = fmaf(m2q[v][6], c1.z, s);
        s = fmaf(m2q[v][7], c1.w, s);
        b2[v] = fminf(b2[v], fmaxf(s, b1[v]));
        const bool lt = s < b1[v];
        i1[v] = lt ? k0 + k : i1[v];
        b1[v] = lt ? s : b1[v];
      }
    }
  }
  __syncthreads();
  const float Na = __uint_as_float(sNa_bits);
  float cmax[kD];
#pragma unroll
  for (int j = 0; j < kD; ++j) cmax[j] = __uint_as_float(sCmax_bits[j]);
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
    if (!live[v]) continue;
    const int64_t i = row0 + threadIdx.x + (int64_t)v * kThreads;
    // Error bound E = C u (Na + 2 sum_p P_p cmax_p), P_p = sum_j |H_pj| (|t_j| + sum |c_f,j|).
    float r[kD], a[kD];
    target32(set, cbs, n_fixed, i, g, r, a, err);
    float sc = Na;
#pragma unroll
    for (int p = 0; p < kD; ++p) {
      float pa = 0.f;
#pragma unroll
      for (int j = 0; j < kD; ++j) pa = fmaf(fabsf(sH[p * kD + j]), a[j], pa);
      sc = fmaf(2.f * pa, cmax[p], sc);
    }
    const float E = (160.f + 8.f * n_fixed) * kU * sc;
    if (!(b2[v] - b1[v] > 2.f * E)) {
      const unsigned slot = atomicAdd(flags.count, 1u);
      if (slot < flags.cap) {
        flags.vec[slot] = i * G_range + (g - g_begin);
        flags.thr[slot] = b1[v] + 2.f * E;
      } else {
        raise_error(err, ERRBIT_INDEX);
      }
    }
    // Always write the fast-pass winner; the fallback overwrites uncertain ones.
    out_code[i * out_ld + (g - out_g0)] = i1[v];
  }
}

// Fallback: one warp per flagged vector. Re-scores every codeword in fp32; candidates whose
// score is within the threshold are re-scored in fp64; the smallest fp64 err wins (ties to the
// smaller index).
__global__ void __launch_bounds__(kThreads)
argmin_fallback_kernel(SetView set, int64_t g_begin, int64_t G_range, CbList cbs,
                       int n_fixed, int s_idx, int32_t* __restrict__ out_code,
                       int64_t out_ld, int64_t out_g0, FlagList flags, unsigned* err) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const unsigned cnt = min((unsigned long long)*flags.count, (unsigned long long)flags.cap);
  const CbView cw = cbs.cb[s_idx];
  for (int64_t f = warp; f < cnt; f += nwarps) {
    const int64_t vi = flags.vec[f];
    const int64_t i = vi / G_range, g = g_begin + vi % G_range;
    const float thr = flags.thr[f];
    const float* H = set.Hb + g * kD * kD;
    float r[kD], a[kD], m2q[kD];
    target32(set, cbs, n_fixed, i, g, r, a, err);
    double r64[kD];
    target64(set, cbs, n_fixed, i, g, r64, err);
#pragma unroll
    for (int p = 0; p < kD; ++p) {
      float q = 0.f;
#pragma unroll
      for (int j = 0; j < kD; ++j) q = fmaf(H[p * kD + j], r[j], q);
      m2q[p] = -2.f * q;
    }
    double best = INFINITY;
    int bestk = 0x7fffffff;
    for (int k = lane; k < cw.K; k += 32) {
      float c[kD];
      load_vec(cw.C + (int64_t)k * kD, c);
      float n = 0.f;
#pragma unroll
      for (int p = 0; p < kD; ++p) {
        float u = 0.f;
#pragma unroll
        for (int j = 0; j < kD; ++j) u = fmaf(H[p * kD + j], c[j], u);
        n = fmaf(c[p], u, n);
      }
      float s = n;
#pragma unroll
      for (int p = 0; p < kD; ++p) s = fmaf(m2q[p], c[p], s);
      if (s <= thr) {
        const double e = quad_err64(r64, cw.C + (int64_t)k * kD, H);
        if (e < best || (e == best && k < bestk)) {
          best = e;
          bestk = k;
        }
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const double ob = __shfl_xor_sync(0xffffffffu, best, off);
      const int ok = __shfl_xor_sync(0xffffffffu, bestk, off);
      if (ob < best || (ob == best && ok < bestk)) {
        best = ob;
        bestk = ok;
      }
    }
    if (lane == 0) {
      if (bestk == 0x7fffffff) {
        raise_error(err, ERRBIT_NUMERIC);  // no candidate: non-finite scores
      } else {
        out_code[i * out_ld + (g - out_g0)] = bestk;
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

// fp64 residual of hypothesis h before stage s: target - sum_{s' < s} C_{st[s']}[code].
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

// Fast stage: one thread per vector, the stage codebook chunked through shared memory, a
// sorted top-L list (L >= B + 1) of approximate errs in registers.
template <int L>
__global__ void __launch_bounds__(kThreads)
beam_stage_kernel(SetView set, int64_t g_begin, CbList cbs, int n_fixed, StageDesc sd,
                  BeamBufs bb, FlagList flags, unsigned* err) {
  const int64_t g = g_begin + blockIdx.y;
  const int64_t G_range = gridDim.y;
  const int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  const bool live = i < set.M;
  const int64_t vi = live ? i * G_range + (g - g_begin) : 0;
  __shared__ float sH[kD * kD];
  __shared__ __align__(16) float sC[kChunk * kD];
  __shared__ float sN[kChunk];
  __shared__ unsigned sNa_bits, sCmax_bits[kD];
  if (threadIdx.x < kD * kD) sH[threadIdx.x] = set.Hb[g * kD * kD + threadIdx.x];
  if (threadIdx.x < kD) sCmax_bits[threadIdx.x] = 0u;
  if (threadIdx.x == 0) sNa_bits = 0u;
  __syncthreads();

  const CbView cw = cbs.cb[sd.st[sd.s]];
  const int S = sd.S, B = sd.B, Bs = sd.Bs;
  const int Bh = (sd.s == 0) ? 1 : (live ? bb.n_in[vi] : 1);
  double tgt[kD];
  if (live) {
    target64(set, cbs, n_fixed, i, g, tgt, err);
  } else {
#pragma unroll
    for (int j = 0; j < kD; ++j) tgt[j] = 0.0;
  }

  float topv[L];
  int toph[L], topk[L];
#pragma unroll
  for (int j = 0; j < L; ++j) {
    topv[j] = INFINITY;
    toph[j] = 0x7fffffff;
    topk[j] = 0x7fffffff;
  }
  for (int k0 = 0; k0 < cw.K; k0 += kChunk) {
    const int nk = min(kChunk, cw.K - k0);
    __syncthreads();
    stage_chunk(cw.C, k0, nk, sH, sC, sN, &sNa_bits, sCmax_bits);
    __syncthreads();
    if (!live) continue;
    for (int h = 0; h < Bh; ++h) {
      double r64[kD];
      const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + h) * S : nullptr;
      hyp_residual64(tgt, cbs, sd, pc, r64, err);
      float r[kD], m2q[kD];
#pragma unroll
      for (int j = 0; j < kD; ++j) r[j] = (float)r64[j];
      float rr = 0.f;
#pragma unroll
      for (int p = 0; p < kD; ++p) {
        float q = 0.f;
#pragma unroll
        for (int j = 0; j < kD; ++j) q = fmaf(sH[p * kD + j], r[j], q);
        m2q[p] = -2.f * q;
        rr = fmaf(r[p], q, rr);
      }
      for (int k = 0; k < nk; ++k) {
        const float4 c0 = *reinterpret_cast<const float4*>(sC + k * kD);
        const float4 c1 = *reinterpret_cast<const float4*>(sC + k * kD + 4);
        float s = rr + sN[k];
        s = fmaf(m2q[0], c0.x, s);
        s = fmaf(m2q[1], c0.y, s);
        s = fmaf(m2q[2], c0.z, s);
        s = fmaf(m2q[3], c0.w, s);
        s = fmaf(m2q[4], c1.x, s);
        s = fmaf(m2q[5], c1.y, s);
        s = fmaf(m2q[6], c1.z, s);
        s = fmaf(m2q[7], c1.w, s);
        if (s < topv[L - 1]) {
          float sv = s;
          int sh = h, sk = k0 + k;
#pragma unroll
          for (int j = 0; j < L; ++j) {
            if (sv < topv[j]) {
              const float tv = topv[j];
              const int th = toph[j], tk = topk[j];
              topv[j] = sv; toph[j] = sh; topk[j] = sk;
              sv = tv; sh = th; sk = tk;
            }
          }
        }
      }
    }
  }
  __syncthreads();
  if (!live) return;

  // Error bound: E = C u (Ra + Na + 2 sum_j P_j cmax_j) maximised over parents, where
  // P_j = sum_l |H_jl| |r_l|. The P-term is recomputed here with the final cmax.
  const float Na = __uint_as_float(sNa_bits);
  float scale = 0.f;
  for (int h = 0; h < Bh; ++h) {
    double r64[kD];
    const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + h) * S : nullptr;
    hyp_residual64(tgt, cbs, sd, pc, r64, err);
    float ra = 0.f, pc2 = 0.f;
#pragma unroll
    for (int p = 0; p < kD; ++p) {
      float pa = 0.f;
#pragma unroll
      for (int j = 0; j < kD; ++j) pa = fmaf(fabsf(sH[p * kD + j]), fabsf((float)r64[j]), pa);
      ra = fmaf(fabsf((float)r64[p]), pa, ra);
      pc2 = fmaf(pa, __uint_as_float(sCmax_bits[p]), pc2);
    }
    scale = fmaxf(scale, ra + Na + 2.f * pc2);
  }
  const float E = (160.f + 8.f * (n_fixed + sd.s)) * kU * scale;

  const int64_t total = (int64_t)Bh * cw.K;
  const int keep = (int)min((int64_t)Bs, total);
  // Non-finite scores never enter the list; keep indices valid and report it.
#pragma unroll
  for (int j = 0; j < L; ++j) {
    if (j < min((int64_t)L, total) && (toph[j] >= Bh || topk[j] >= cw.K)) {
      raise_error(err, ERRBIT_NUMERIC);
      toph[j] = 0;
      topk[j] = 0;
    }
  }
  const bool all_kept = total <= L;
  // Fast certificate: the gaps between consecutive entries j -> j+1, j < min(keep, total-1),
  // exceed 2E (every candidate outside the list scores at least the last list entry).
  bool ok = true;
  const int lim = (int)min((int64_t)keep, total - 1);
#pragma unroll
  for (int j = 0; j < L - 1; ++j)
    if (j < lim && !(topv[j + 1] - topv[j] > 2.f * E)) ok = false;

  int32_t* out = bb.hyp_out + vi * B * S;
  if (ok) {
#pragma unroll
    for (int j = 0; j < L; ++j) {
      if (j >= keep) break;
      const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + toph[j]) * S : nullptr;
      for (int q = 0; q < sd.s; ++q) out[j * S + q] = pc[q];
      out[j * S + sd.s] = topk[j];
    }
    bb.n_out[vi] = keep;
    return;
  }
  // Exact path on the kept candidates: fp64 errs, exact (err, h, k) order, then the boundary
  // certificate a_L - E > e_(keep).
  const int nkept = (int)min((int64_t)L, total);
  double ev[L];
#pragma unroll
  for (int j = 0; j < L; ++j) {
    ev[j] = INFINITY;
    if (j < nkept) {
      double r64[kD];
      const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + toph[j]) * S : nullptr;
      hyp_residual64(tgt, cbs, sd, pc, r64, err);
      ev[j] = quad_err64(r64, cw.C + (int64_t)topk[j] * kD, sH);
    }
  }
  // insertion sort by (ev, h, k)
#pragma unroll
  for (int a = 1; a < L; ++a) {
#pragma unroll
    for (int b = a; b > 0; --b) {
      const bool sw = (ev[b] < ev[b - 1]) ||
                      (ev[b] == ev[b - 1] &&
                       (toph[b] < toph[b - 1] || (toph[b] == toph[b - 1] && topk[b] < topk[b - 1])));
      if (sw) {
        const double te = ev[b]; ev[b] = ev[b - 1]; ev[b - 1] = te;
        const int th = toph[b]; toph[b] = toph[b - 1]; toph[b - 1] = th;
        const int tk = topk[b]; topk[b] = topk[b - 1]; topk[b - 1] = tk;
        const float tv = topv[b]; topv[b] = topv[b - 1]; topv[b - 1] = tv;
      }
    }
  }
  float amax = -INFINITY;
#pragma unroll
  for (int j = 0; j < L; ++j)
    if (j < nkept) amax = fmaxf(amax, topv[j]);
  const bool cert = all_kept || ((double)amax - (double)E > ev[keep - 1]);
  if (!cert) {
    const unsigned slot = atomicAdd(flags.count, 1u);
    if (slot < flags.cap) {
      flags.vec[slot] = vi;
      flags.thr[slot] = 0.f;
    } else {
      raise_error(err, ERRBIT_INDEX);
    }
    return;
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

// Exact stage for flagged vectors: one thread per vector, every (h, k) candidate in fp64,
// sorted top-B by (err, h, k) kept in local memory.
__global__ void beam_stage_fallback_kernel(SetView set, int64_t g_begin, int64_t G_range,
                                           CbList cbs, int n_fixed, StageDesc sd, BeamBufs bb,
                                           FlagList flags, unsigned* err) {
  const unsigned cnt = min((unsigned long long)*flags.count, (unsigned long long)flags.cap);
  const int S = sd.S, B = sd.B, Bs = sd.Bs;
  const CbView cw = cbs.cb[sd.st[sd.s]];
  for (int64_t f = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; f < cnt;
       f += (int64_t)gridDim.x * blockDim.x) {
    const int64_t vi = flags.vec[f];
    const int64_t i = vi / G_range, g = g_begin + vi % G_range;
    const float* H = set.Hb + g * kD * kD;
    double tgt[kD];
    target64(set, cbs, n_fixed, i, g, tgt, err);
    const int Bh = (sd.s == 0) ? 1 : bb.n_in[vi];
    double be[16];
    int bh[16], bk[16];
    int nb = 0;
    for (int h = 0; h < Bh; ++h) {
      double r64[kD];
      const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + h) * S : nullptr;
      hyp_residual64(tgt, cbs, sd, pc, r64, err);
      for (int k = 0; k < cw.K; ++k) {
        const double e = quad_err64(r64, cw.C + (int64_t)k * kD, H);
        // candidates arrive in (h, k) order: strict comparison keeps the earlier on ties
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
    }
    int32_t* out = bb.hyp_out + vi * B * S;
    for (int j = 0; j < nb; ++j) {
      const int32_t* pc = bb.hyp_in ? bb.hyp_in + (vi * B + bh[j]) * S : nullptr;
      for (int q = 0; q < sd.s; ++q) out[j * S + q] = pc[q];
      out[j * S + sd.s] = bk[j];
    }
    bb.n_out[vi] = nb;
  }
}

// Final step of a multi-stage (or keep-if-better) encode: write the best tuple, or keep the
// tuple already in the codes when its fp64 err is strictly smaller; optional vec_err.
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
    double tgt[kD];
    target64(set, cbs, n_fixed, i, g, tgt, err);
    const int32_t* best = hyp + vi * B * S;
    bool use_old = false;
    double e_new = 0.0, e_old = 0.0;
    if (keep_if_better || vec_err) {
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
      e_new = quad_err64(r, nullptr, H);
    }
    if (keep_if_better) {
      double r[kD];
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
    if (!use_old) {
      for (int q = 0; q < S; ++q) {
        const CbView& cb = cbs.cb[sd.st[q]];
        cb.codes[i * cb.ld + g] = best[q];
      }
    }
    if (vec_err) vec_err[i * set.G_sub + g] = (float)(use_old ? e_old : e_new);
  }
}

// err of the tuple currently in the codes (fixed + searched) for vectors that no searched
// codebook covers.
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
                                cudaStream_t stream) {
  dim3 grid((unsigned)ceil_div(set.M, kThreads), (unsigned)G_range);
  ProfScope ps("encode_beam_stage", stream, 0.0);
  beam_stage_kernel<L><<<grid, kThreads, 0, stream>>>(set, g_begin, cbs, n_fixed, sd, bb, fl,
                                                     err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

crvq_status launch_beam_stage(const SetView& set, int64_t g_begin, int64_t G_range,
                              const CbList& cbs, int n_fixed, const StageDesc& sd,
                              const BeamBufs& bb, const FlagList& fl, unsigned* err,
                              cudaStream_t stream) {
  const int need = sd.Bs + 1;
  if (need <= 2) return launch_beam_stage_L<2>(set, g_begin, G_range, cbs, n_fixed, sd, bb, fl, err, stream);
  if (need <= 3) return launch_beam_stage_L<3>(set, g_begin, G_range, cbs, n_fixed, sd, bb, fl, err, stream);
  if (need <= 5) return launch_beam_stage_L<5>(set, g_begin, G_range, cbs, n_fixed, sd, bb, fl, err, stream);
  if (need <= 9) return launch_beam_stage_L<9>(set, g_begin, G_range, cbs, n_fixed, sd, bb, fl, err, stream);
  return launch_beam_stage_L<17>(set, g_begin, G_range, cbs, n_fixed, sd, bb, fl, err, stream);
}

// One range of groups [g_begin, g_begin + G_range) whose searched stages are sd.st[0..S).
crvq_status encode_range(const SetView& set, int64_t g_begin, int64_t G_range,
                         const CbList& cbs, int n_fixed, StageDesc sd, bool keep_if_better,
                         float* vec_err, double* scores, unsigned* err, cudaStream_t stream) {
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
  Scratch flag_mem;
  const size_t fl_bytes = (size_t)nvec * (sizeof(int64_t) + sizeof(float)) + 256;
  CRVQ_TRY(flag_mem.alloc(fl_bytes, stream));
  FlagList fl;
  fl.count = flag_mem.as<unsigned>();
  fl.vec = reinterpret_cast<int64_t*>(flag_mem.as<char>() + 256);
  fl.thr = reinterpret_cast<float*>(fl.vec + nvec);
  fl.cap = nvec;

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
    CRVQ_CUDA(cudaMemsetAsync(fl.count, 0, sizeof(unsigned), stream));
    const bool big = (ceil_div(set.M, kThreads * 4) * G_range) >= 2 * nsm;
    ProfScope ps("encode_argmin", stream, (double)nvec * cw.K);
    if (big) {
      dim3 grid((unsigned)ceil_div(set.M, kThreads * 4), (unsigned)G_range);
      argmin_kernel<4><<<grid, kThreads, 0, stream>>>(set, g_begin, cbs, n_fixed, s_idx, out,
                                                      out_ld, out_g0, fl, err);
    } else {
      dim3 grid((unsigned)ceil_div(set.M, kThreads), (unsigned)G_range);
      argmin_kernel<1><<<grid, kThreads, 0, stream>>>(set, g_begin, cbs, n_fixed, s_idx, out,
                                                      out_ld, out_g0, fl, err);
    }
    CRVQ_LAUNCHED();
    ProfScope ps2("encode_argmin_fallback", stream, 0.0);
    argmin_fallback_kernel<<<4 * nsm, kThreads, 0, stream>>>(set, g_begin, G_range, cbs,
                                                             n_fixed, s_idx, out, out_ld,
                                                             out_g0, fl, err);
    CRVQ_LAUNCHED();
    if (scores) *scores += (double)nvec * cw.K;
    ProfScope ps3("encode_finalize", stream, 0.0);
    if (keep_if_better) {
      StageDesc one = sd;
      one.B = 1;
      one.Bs = 1;
      beam_finalize_kernel<<<fin_blocks, 128, 0, stream>>>(set, g_begin, G_range, cbs, n_fixed,
                                                           one, out, true, vec_err, err);
      CRVQ_LAUNCHED();
    } else if (vec_err) {
      residual_err_kernel<<<fin_blocks, 128, 0, stream>>>(set, g_begin, G_range, cbs, vec_err,
                                                          err);
      CRVQ_LAUNCHED();
    }
    return CRVQ_OK;
  }

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
  for (int s = 0; s < S; ++s) {
    sd.s = s;
    sd.Bs = (s == S - 1) ? 1 : B;  // only the best tuple of the last stage is used
    CRVQ_CUDA(cudaMemsetAsync(fl.count, 0, sizeof(unsigned), stream));
    BeamBufs bb{in_h, in_n, out_h, out_n};
    CRVQ_TRY(launch_beam_stage(set, g_begin, G_range, cbs, n_fixed, sd, bb, fl, err, stream));
    {
      ProfScope ps("encode_beam_fallback", stream, 0.0);
      beam_stage_fallback_kernel<<<std::max(1, nsm), 128, 0, stream>>>(
          set, g_begin, G_range, cbs, n_fixed, sd, bb, fl, err);
      CRVQ_LAUNCHED();
    }
    const int K = cbs.cb[sd.st[s]].K;
    sc += (double)nvec * parents * K;
    parents = std::min<int64_t>(B, parents * K);
    in_h = out_h;
    in_n = out_n;
    out_h = (out_h == hypA) ? hypB : hypA;
    out_n = (out_n == nA) ? nB : nA;
  }
  if (scores) *scores += sc;
  ProfScope ps("encode_finalize", stream, 0.0);
  beam_finalize_kernel<<<fin_blocks, 128, 0, stream>>>(set, g_begin, G_range, cbs, n_fixed, sd,
                                                       in_h, keep_if_better, vec_err, err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace

crvq_status launch_encode_beam(const SetView& set, const CbList& cbs, int n_fixed, int B,
                               bool keep_if_better, float* vec_err, double* scores,
                               cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  // Group ranges with the same set of covering searched codebooks: boundaries at every G_cov.
  std::vector<int64_t> cuts = {0, set.G_sub};
  for (int s = n_fixed; s < cbs.n; ++s)
    if (cbs.cb[s].G_cov > 0 && cbs.cb[s].G_cov < set.G_sub) cuts.push_back(cbs.cb[s].G_cov);
  std::sort(cuts.begin(), cuts.end());
  cuts.erase(std::unique(cuts.begin(), cuts.end()), cuts.end());
  for (size_t r = 0; r + 1 < cuts.size(); ++r) {
    const int64_t g0 = cuts[r], g1 = cuts[r + 1];
    StageDesc sd{};
    sd.S = 0;
    sd.B = B;
    sd.Bs = B;
    for (int s = n_fixed; s < cbs.n; ++s)
      if (g0 < cbs.cb[s].G_cov) sd.st[sd.S++] = s;
    CRVQ_TRY(encode_range(set, g0, g1 - g0, cbs, n_fixed, sd, keep_if_better, vec_err, scores,
                          err, stream));
  }
  return CRVQ_OK;
}

}  // namespace crvq
