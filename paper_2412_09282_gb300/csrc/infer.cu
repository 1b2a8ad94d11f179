// Inference product with a CRVQ-quantized matrix, computed from its codes (the paper's
// inference setting, App. "Inference Speed" / Table speed): Y = X_in W_hat^T, where W_hat in the
// original channel order is the permuted sum of the codebooks' codewords (Sec. 4.3: base
// codebook on every group, extended codebooks on the first G_c groups of the reordered
// channels). W_hat is never formed:
//   y[bi][i] = sum over codebooks s and groups g < G_cov(s) of <C_s[codes_s(i, g)], xs[bi][g]>,
//   xs[bi][p] = X_in[bi][perm[p]]   (the inputs taken once in the sorted channel order).
//
// Layout: a CTA owns one slice of 32 groups and a block of 128 rows. It first issues every
// load it needs at once: the base codebook's codes of its tile (128 rows x 32 codes, coalesced
// 128-byte reads, into shared memory) and its slice of the inputs through the permutation.
// It then builds the slice's lookup tables lut[g][k][bi] = <C_base[k], xs[bi][g]> in shared
// memory (a thread per codeword, loaded once; tables that would not fit are skipped and the
// codewords dotted from L2). A warp takes one row at a time, lane = group: a shared-memory
// code, a shared-memory table entry; the extended codebooks, which cover only the first G_c
// groups, are dotted from L2. Each row slice is reduced across the warp (a fixed shuffle tree)
// into a partial, and the last CTA of a row block to finish adds the partials of its rows in
// slice order, so results are identical on every run. The codes are the only per-element
// stream from HBM (4 bytes per code).
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

constexpr int kSliceG = 32;     // groups per CTA slice (one per lane)
constexpr int kMvThreads = 256;
constexpr int kMvRows = 64;     // rows per CTA
constexpr int kStageCb = 4;     // codebooks whose codes of the tile are staged in shared memory
constexpr int kMaxBatch = 8;
constexpr size_t kLutSmemCap = 96 * 1024;  // the base codebook's tables per CTA at most

struct MatvecArgs {
  const float* X;       // b x N, row stride ldx
  int64_t ldx;
  int64_t N;
  const int32_t* perm;  // N or null (identity)
  CbList cbs;
  int64_t M;
  int b;
  int base_lut;         // the base codebook (cbs.cb[0]) uses shared-memory lookup tables
  int64_t n_slices;
  const float* lut;     // [G][K_base][b] base-codebook tables (when base_lut)
  float* part;          // [n_slices][b][M]
  unsigned* done;       // per row block: CTAs finished (zero on entry)
  float* Y;             // b x M, row stride ldy
  int64_t ldy;
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

__device__ __forceinline__ float dot8(const float* __restrict__ c, const float* x) {
  const float4 c0 = __ldg(reinterpret_cast<const float4*>(c));
  const float4 c1 = __ldg(reinterpret_cast<const float4*>(c + 4));
  float v = c0.x * x[0];
  v = fmaf(c0.y, x[1], v);
  v = fmaf(c0.z, x[2], v);
  v = fmaf(c0.w, x[3], v);
  v = fmaf(c1.x, x[4], v);
  v = fmaf(c1.y, x[5], v);
  v = fmaf(c1.z, x[6], v);
  v = fmaf(c1.w, x[7], v);
  return v;
}

// The base codebook's lookup tables of every group, once per call: lut[g][k][bi] =
// <C_base[k], xs[bi][g]>, one thread per (group, codeword), the group's inputs taken through
// the permutation.
__global__ void __launch_bounds__(256)
lut_build_kernel(const float* __restrict__ X, int64_t ldx, int64_t N,
                 const int32_t* __restrict__ perm, CbView cb0, int b, float* __restrict__ lut,
                 unsigned* err) {
  const int64_t G = N / kD;
  const int64_t total = G * cb0.K;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t g = e / cb0.K;
    const int k = (int)(e % cb0.K);
    int64_t src[kD];
#pragma unroll
    for (int j = 0; j < kD; ++j) {
      src[j] = g * kD + j;
      if (perm) {
        src[j] = perm[g * kD + j];
        if (src[j] < 0 || src[j] >= N) {
          if (k == 0) raise_error(err, ERRBIT_INDEX);
          src[j] = -1;
        }
      }
    }
    for (int bi = 0; bi < b; ++bi) {
      float x[kD];
#pragma unroll
      for (int j = 0; j < kD; ++j) x[j] = src[j] >= 0 ? X[bi * ldx + src[j]] : 0.f;
      lut[e * b + bi] = dot8(cb0.C + (int64_t)k * kD, x);
    }
  }
}

// Partial products of one (row block, group slice), and the ordered sum of a row block's
// partials by the last of its CTAs.
template <int BMAX>
__global__ void __launch_bounds__(kMvThreads)
matvec_slice_kernel(MatvecArgs a, unsigned* err) {
  extern __shared__ __align__(16) float sm[];
  float* xs = sm;                                          // [b][kSliceG][8]
  // codes of the tile, codebook-major: [kStageCb][rows][32]
  int32_t* scode = reinterpret_cast<int32_t*>(xs + kMaxBatch * kSliceG * kD);
  float* lut = reinterpret_cast<float*>(scode + kStageCb * kMvRows * kSliceG);  // [32][K][b]
  __shared__ int s_last;
  const int64_t slice = blockIdx.y, rblk = blockIdx.x;
  const int64_t g0 = slice * kSliceG;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t G = a.N / kD;
  const int gn = (int)(G - g0 < kSliceG ? G - g0 : kSliceG);
  const int64_t r0 = rblk * kMvRows;
  const int nr = (int)(a.M - r0 < kMvRows ? a.M - r0 : kMvRows);
  const CbView& cb0 = a.cbs.cb[0];

  // every load of the tile at once: the codes of the staged codebooks that cover the slice
  // (coalesced rows of 32 codes) and the inputs
  const int nst = a.cbs.n < kStageCb ? a.cbs.n : kStageCb;
  for (int s = 0; s < nst; ++s) {
    const CbView& cb = a.cbs.cb[s];
    if (cb.G_cov <= g0) continue;
    int32_t* sc = scode + s * kMvRows * kSliceG;
    for (int e = tid; e < nr * kSliceG; e += blockDim.x) {
      const int r = e / kSliceG, l = e % kSliceG;
      const int64_t g = g0 + l;
      sc[e] = (l < gn && g < cb.G_cov) ? cb.codes[(r0 + r) * cb.ld + g] : -1;
    }
  }
  for (int e = tid; e < a.b * kSliceG * kD; e += blockDim.x) {
    const int bi = e / (kSliceG * kD), r = e % (kSliceG * kD);
    float v = 0.f;
    if (r < gn * kD) {
      int64_t src = g0 * kD + r;
      if (a.perm) {
        src = a.perm[src];
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
  // the slice's base-codebook tables, copied from the per-call build (L2-resident)
  if (a.base_lut) {
    const int64_t n4 = (int64_t)gn * cb0.K * a.b / 4;  // K * b is a multiple of 4 here
    const float4* src = reinterpret_cast<const float4*>(a.lut + g0 * cb0.K * a.b);
    for (int64_t e = tid; e < n4; e += blockDim.x) reinterpret_cast<float4*>(lut)[e] = src[e];
    __syncthreads();
  }

  const int64_t g = g0 + lane;
  for (int r = warp; r < nr; r += kMvThreads / 32) {
    const int64_t i = r0 + r;
    float acc[BMAX];
#pragma unroll
    for (int bi = 0; bi < BMAX; ++bi) acc[bi] = 0.f;
    const int32_t k = scode[r * kSliceG + lane];
    if (lane < gn && g < cb0.G_cov) {
      if (k < 0 || k >= cb0.K) {
        raise_error(err, ERRBIT_INDEX);
      } else if (a.base_lut) {
        const float* e = lut + ((int64_t)lane * cb0.K + k) * a.b;
#pragma unroll
        for (int bi = 0; bi < BMAX; ++bi)
          if (bi < a.b) acc[bi] += e[bi];
      } else {
#pragma unroll
        for (int bi = 0; bi < BMAX; ++bi)
          if (bi < a.b) acc[bi] += dot8(cb0.C + (int64_t)k * kD, xs + (bi * kSliceG + lane) * kD);
      }
    }
    for (int s = 1; s < a.cbs.n; ++s) {  // extended codebooks: the first G_c groups only
      const CbView& cb = a.cbs.cb[s];
      if (!(lane < gn && g < cb.G_cov)) continue;
      const int32_t ke = s < kStageCb ? scode[(s * kMvRows + r) * kSliceG + lane]
                                      : cb.codes[i * cb.ld + g];
      if (ke < 0 || ke >= cb.K) {
        raise_error(err, ERRBIT_INDEX);
        continue;
      }
#pragma unroll
      for (int bi = 0; bi < BMAX; ++bi)
        if (bi < a.b) acc[bi] += dot8(cb.C + (int64_t)ke * kD, xs + (bi * kSliceG + lane) * kD);
    }
#pragma unroll
    for (int bi = 0; bi < BMAX; ++bi) {
      if (bi >= a.b) break;
      const float v = warp_sum(acc[bi]);
      if (lane == 0) a.part[(slice * a.b + bi) * a.M + i] = v;
    }
  }
  // the last CTA of this row block adds the slices' partials of its rows, in slice order
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(&a.done[rblk], 1u) == (unsigned)(a.n_slices - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int e = tid; e < nr * a.b; e += blockDim.x) {
    const int bi = e / nr;
    const int64_t i = r0 + e % nr;
    float sum = 0.f;
    int64_t q = 0;
    for (; q + 8 <= a.n_slices; q += 8) {  // eight loads in flight, added in slice order
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = __ldcg(a.part + ((q + u) * a.b + bi) * a.M + i);
#pragma unroll
      for (int u = 0; u < 8; ++u) sum += v[u];
    }
    for (; q < a.n_slices; ++q) sum += __ldcg(a.part + (q * a.b + bi) * a.M + i);
    a.Y[bi * a.ldy + i] = sum;
  }
}

}  // namespace

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
  a.Y = Y;
  a.ldy = ldy;
  const size_t lut_bytes = (size_t)kSliceG * cbs.cb[0].K * b * sizeof(float);
  a.base_lut = (lut_bytes <= kLutSmemCap && (cbs.cb[0].K * b) % 4 == 0) ? 1 : 0;
  const size_t smem = (size_t)kMaxBatch * kSliceG * kD * sizeof(float) +
                      (size_t)kStageCb * kMvRows * kSliceG * sizeof(int32_t) +
                      (a.base_lut ? lut_bytes : 0);
  const int64_t row_blocks = ceil_div(M, (int64_t)kMvRows);
  const size_t part_bytes = align_up((size_t)a.n_slices * b * M * sizeof(float), 256);
  const size_t lutg_bytes = a.base_lut ? align_up((size_t)G * cbs.cb[0].K * b * 4, 256) : 0;
  Scratch mem;
  CRVQ_TRY(mem.alloc(part_bytes + lutg_bytes + (size_t)row_blocks * sizeof(unsigned), stream));
  a.part = mem.as<float>();
  a.lut = reinterpret_cast<float*>(mem.as<char>() + part_bytes);
  a.done = reinterpret_cast<unsigned*>(mem.as<char>() + part_bytes + lutg_bytes);
  CRVQ_CUDA(cudaMemsetAsync(a.done, 0, (size_t)row_blocks * sizeof(unsigned), stream));
  const int nsm = sm_count();
  if (a.base_lut) {
    ProfScope pl("matvec_tables", stream, (double)G * cbs.cb[0].K * b);
    const int64_t total = G * cbs.cb[0].K;
    lut_build_kernel<<<(unsigned)std::min<int64_t>(ceil_div(total, 256), 8 * nsm), 256, 0,
                       stream>>>(X, ldx, N, perm, cbs.cb[0], b, const_cast<float*>(a.lut), err);
    CRVQ_LAUNCHED();
  }
  const dim3 grid((unsigned)row_blocks, (unsigned)a.n_slices);
  ProfScope ps("matvec_slices", stream, (double)M * G * cbs.n);
  auto go = [&](auto kernel) -> crvq_status {
    CRVQ_TRY(smem_limit((const void*)kernel, smem));
    kernel<<<grid, kMvThreads, smem, stream>>>(a, err);
    return CRVQ_OK;
  };
  if (b == 1)
    CRVQ_TRY(go(matvec_slice_kernel<1>));
  else if (b <= 4)
    CRVQ_TRY(go(matvec_slice_kernel<4>));
  else
    CRVQ_TRY(go(matvec_slice_kernel<kMaxBatch>));
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace crvq
