// Inference product with a CRVQ-quantized matrix, computed from its codes (the paper's
// inference setting, App. "Inference Speed" / Table speed): Y = X_in W_hat^T, where W_hat in the
// original channel order is the permuted sum of the codebooks' codewords (Sec. 4.3: base
// codebook on every group, extended codebooks on the first G_c groups of the reordered
// channels). W_hat is never formed:
//   y[bi][i] = sum over codebooks s and groups g < G_cov(s) of <C_s[codes_s(i, g)], xs[bi][g]>,
//   xs[bi][p] = X_in[bi][perm[p]]   (the inputs taken once in the sorted channel order).
//
// Layout: a CTA owns one slice of 32 groups and a block of rows. It gathers its slice of the
// inputs through the permutation into shared memory and, for codebooks small enough, the
// lookup tables lut[g][k][bi] = <C[k], xs[bi][g]> of its 32 groups (codewords read from L2
// once per CTA); a warp then takes one row at a time with lane l on group g0 + l, so that the
// 32 codes of a row slice are one coalesced 128-byte read and each lookup is one shared-memory
// load. Codebooks whose tables do not fit are dotted directly (the codeword from L2, eight FMAs
// per input). Each row slice is reduced across the warp (shuffles, a fixed tree) into a
// partial; a second kernel adds the partials of a row in slice order, so results are
// identical on every run. The codes are the only per-element stream from HBM (4 bytes per
// code), which makes the kernel bound by HBM bandwidth.
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

constexpr int kSliceG = 32;     // groups per CTA slice (one per lane)
constexpr int kMvThreads = 256;
constexpr int kMaxBatch = 8;
constexpr size_t kLutSmemCap = 160 * 1024;  // shared memory for lookup tables per CTA
constexpr int kRowBatch = 8;    // rows a warp reads codes for before using any

struct MatvecArgs {
  const float* X;       // b x N, row stride ldx
  int64_t ldx;
  int64_t N;
  const int32_t* perm;  // N or null (identity)
  CbList cbs;
  int64_t M;
  int b;
  int lut_mask;         // bit s: codebook s uses a shared-memory lookup table
  int64_t n_slices;
  float* part;          // [n_slices][b][M]
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

// Partial products of one (row block, group slice): part[slice][bi][i].
template <int BMAX, int MAXCB>
__global__ void __launch_bounds__(kMvThreads)
matvec_slice_kernel(MatvecArgs a, int rows_per_cta, unsigned* err) {
  extern __shared__ __align__(16) float sm[];
  float* xs = sm;                             // [b][kSliceG][8]
  float* lut = sm + a.b * kSliceG * kD;       // per LUT codebook: [kSliceG][K][b]
  const int64_t slice = blockIdx.y;
  const int64_t g0 = slice * kSliceG;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t G = a.N / kD;
  const int gn = (int)(G - g0 < kSliceG ? G - g0 : kSliceG);

  // inputs of this slice in the sorted order
  for (int e = tid; e < a.b * kSliceG * kD; e += blockDim.x) {
    const int bi = e / (kSliceG * kD), r = e % (kSliceG * kD);
    const int64_t p = g0 * kD + r;
    float v = 0.f;
    if (r < gn * kD) {
      int64_t src = p;
      if (a.perm) {
        src = a.perm[p];
        if (src < 0 || src >= a.N) {
          raise_error(err, ERRBIT_INDEX);
          src = -1;
        }
      }
      if (src >= 0) v = a.X[bi * a.ldx + src];
    }
    xs[e] = v;
  }
  __syncthreads();
  // lookup tables of the codebooks that have one: lut[g][k][bi] = <C[k], xs[bi][g]>; a thread
  // takes one codeword (loaded once) across the slice's groups
  {
    float* t = lut;
    for (int s = 0; s < a.cbs.n; ++s) {
      if (!((a.lut_mask >> s) & 1)) continue;
      const CbView& cb = a.cbs.cb[s];
      const int64_t gcov = cb.G_cov - g0;
      const int gc = gcov <= 0 ? 0 : (int)(gcov < gn ? gcov : gn);
      for (int k = tid; k < cb.K && gc > 0; k += blockDim.x) {
        const float4 c0 = __ldg(reinterpret_cast<const float4*>(cb.C + (int64_t)k * kD));
        const float4 c1 = __ldg(reinterpret_cast<const float4*>(cb.C + (int64_t)k * kD + 4));
        for (int gl = 0; gl < gc; ++gl)
          for (int bi = 0; bi < a.b; ++bi) {
            const float* x = xs + (bi * kSliceG + gl) * kD;
            float v = c0.x * x[0];
            v = fmaf(c0.y, x[1], v);
            v = fmaf(c0.z, x[2], v);
            v = fmaf(c0.w, x[3], v);
            v = fmaf(c1.x, x[4], v);
            v = fmaf(c1.y, x[5], v);
            v = fmaf(c1.z, x[6], v);
            v = fmaf(c1.w, x[7], v);
            t[((int64_t)gl * cb.K + k) * a.b + bi] = v;
          }
      }
      t += (int64_t)kSliceG * cb.K * a.b;
    }
  }
  __syncthreads();

  // rows of this block: a warp takes kRowBatch rows at a time, lane = group g0 + lane; the
  // codes of every row and codebook of the batch are loaded before any is used, so that each
  // warp keeps kRowBatch x n_cb coalesced 128-byte reads in flight (the kernel is bound by the
  // latency of these reads otherwise)
  const int64_t r0 = (int64_t)blockIdx.x * rows_per_cta;
  const int64_t r1 = a.M < r0 + rows_per_cta ? a.M : r0 + rows_per_cta;
  const int nwarps = blockDim.x >> 5;
  const int64_t g = g0 + lane;
  for (int64_t ib = r0 + (int64_t)warp * kRowBatch; ib < r1; ib += (int64_t)nwarps * kRowBatch) {
    int32_t kc[MAXCB][kRowBatch];
#pragma unroll
    for (int s = 0; s < MAXCB; ++s) {
      const bool cov = s < a.cbs.n && lane < gn && g < a.cbs.cb[s].G_cov;
#pragma unroll
      for (int u = 0; u < kRowBatch; ++u) {
        const int64_t i = ib + u;
        kc[s][u] = (cov && i < r1) ? __ldg(a.cbs.cb[s].codes + i * a.cbs.cb[s].ld + g) : -1;
      }
    }
    float acc[kRowBatch][BMAX];
#pragma unroll
    for (int u = 0; u < kRowBatch; ++u)
#pragma unroll
      for (int bi = 0; bi < BMAX; ++bi) acc[u][bi] = 0.f;
    const float* t = lut;
#pragma unroll
    for (int s = 0; s < MAXCB; ++s) {
      if (s >= a.cbs.n) break;
      const CbView& cb = a.cbs.cb[s];
      const bool cov = lane < gn && g < cb.G_cov;
      const bool has_lut = (a.lut_mask >> s) & 1;
#pragma unroll
      for (int u = 0; u < kRowBatch; ++u) {
        const int32_t k = kc[s][u];
        if (!cov || ib + u >= r1) continue;
        if (k < 0 || k >= cb.K) {
          raise_error(err, ERRBIT_INDEX);
        } else if (has_lut) {
          const float* e = t + ((int64_t)lane * cb.K + k) * a.b;
#pragma unroll
          for (int bi = 0; bi < BMAX; ++bi)
            if (bi < a.b) acc[u][bi] += e[bi];
        } else {
          const float4 c0 = __ldg(reinterpret_cast<const float4*>(cb.C + (int64_t)k * kD));
          const float4 c1 = __ldg(reinterpret_cast<const float4*>(cb.C + (int64_t)k * kD + 4));
#pragma unroll
          for (int bi = 0; bi < BMAX; ++bi) {
            if (bi >= a.b) break;
            const float* x = xs + (bi * kSliceG + lane) * kD;
            float v = c0.x * x[0];
            v = fmaf(c0.y, x[1], v);
            v = fmaf(c0.z, x[2], v);
            v = fmaf(c0.w, x[3], v);
            v = fmaf(c1.x, x[4], v);
            v = fmaf(c1.y, x[5], v);
            v = fmaf(c1.z, x[6], v);
            v = fmaf(c1.w, x[7], v);
            acc[u][bi] += v;
          }
        }
      }
      if (has_lut) t += (int64_t)kSliceG * cb.K * a.b;
    }
#pragma unroll
    for (int u = 0; u < kRowBatch; ++u) {
      const int64_t i = ib + u;
#pragma unroll
      for (int bi = 0; bi < BMAX; ++bi) {
        if (bi >= a.b) break;
        const float v = warp_sum(acc[u][bi]);
        if (lane == 0 && i < r1) a.part[(slice * a.b + bi) * a.M + i] = v;
      }
    }
  }
}

// y[bi][i] = sum of the slice partials in slice order.
__global__ void __launch_bounds__(256)
matvec_reduce_kernel(const float* __restrict__ part, int64_t n_slices, int64_t M, int b,
                     float* __restrict__ Y, int64_t ldy) {
  const int64_t n = (int64_t)b * M;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t bi = e / M, i = e % M;
    float s = 0.f;
    for (int64_t q = 0; q < n_slices; ++q) s += part[(q * b + bi) * M + i];
    Y[bi * ldy + i] = s;
  }
}

}  // namespace

size_t lut_matvec_smem(const CbList& cbs, int b, int* lut_mask) {
  size_t bytes = (size_t)b * kSliceG * kD * sizeof(float);
  int mask = 0;
  for (int s = 0; s < cbs.n; ++s) {
    const size_t t = (size_t)kSliceG * cbs.cb[s].K * b * sizeof(float);
    if (bytes + t <= kLutSmemCap) {
      bytes += t;
      mask |= 1 << s;
    }
  }
  if (lut_mask) *lut_mask = mask;
  return bytes;
}

crvq_status launch_lut_matvec(const float* X, int64_t ldx, int64_t N, int b,
                              const int32_t* perm, const CbList& cbs, int64_t M, float* Y,
                              int64_t ldy, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  if (b < 1 || b > kMaxBatch)
    return fail(CRVQ_ERR_UNSUPPORTED, "batch of %d inputs: 1 to %d are implemented", b,
                kMaxBatch);
  const int64_t G = N / kD;
  MatvecArgs a;
  a.X = X;
  a.ldx = ldx;
  a.N = N;
  a.perm = perm;
  a.cbs = cbs;
  a.M = M;
  a.b = b;
  a.n_slices = ceil_div(G, kSliceG);
  const size_t smem = lut_matvec_smem(cbs, b, &a.lut_mask);
  Scratch part;
  CRVQ_TRY(part.alloc((size_t)a.n_slices * b * M * sizeof(float), stream));
  a.part = part.as<float>();
  const int nsm = sm_count();
  const int64_t row_blocks = std::max<int64_t>(
      1, std::min<int64_t>(ceil_div(M, 8), ceil_div(2 * (int64_t)nsm, a.n_slices)));
  const int rows_per_cta = (int)ceil_div(M, row_blocks);
  const dim3 grid((unsigned)ceil_div(M, rows_per_cta), (unsigned)a.n_slices);
  {
    ProfScope ps("matvec_slices", stream, (double)M * G * cbs.n);
    auto go = [&](auto kernel) -> crvq_status {
      CRVQ_TRY(smem_limit((const void*)kernel, smem));
      kernel<<<grid, kMvThreads, smem, stream>>>(a, rows_per_cta, err);
      return CRVQ_OK;
    };
    if (b == 1 && cbs.n <= 4) {
      CRVQ_TRY(go(matvec_slice_kernel<1, 4>));
    } else if (b == 1) {
      CRVQ_TRY(go(matvec_slice_kernel<1, kMaxCodebooks>));
    } else if (b <= 4 && cbs.n <= 4) {
      CRVQ_TRY(go(matvec_slice_kernel<4, 4>));
    } else {
      CRVQ_TRY(go(matvec_slice_kernel<kMaxBatch, kMaxCodebooks>));
    }
    CRVQ_LAUNCHED();
  }
  {
    ProfScope ps("matvec_reduce", stream, (double)b * M);
    const int64_t n = (int64_t)b * M;
    matvec_reduce_kernel<<<(unsigned)std::min<int64_t>(ceil_div(n, 256), 8 * nsm), 256, 0,
                           stream>>>(a.part, a.n_slices, M, b, Y, ldy);
    CRVQ_LAUNCHED();
  }
  return CRVQ_OK;
}

}  // namespace crvq
