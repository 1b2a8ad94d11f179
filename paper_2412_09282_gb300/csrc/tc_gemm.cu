// Host side of the tcgen05 3xTF32 products: the dense symmetric X^T X and its diagonal blocks
// alone (tc_gemm.cuh), and the image-fed sum of squares ||(A - A_sub) B^T||^2 of the full loss
// (img:: below). The tensor core accumulates fp32 with a small systematic rounding bias per
// accumulation step, so K is cut into chunks of at most kKChunk and the few chunk partials of
// an element are summed afterwards in fp32, in chunk order (a relative error of a few u); the
// squares are summed per row in fp32 and per tile in fp64.
#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "tc_gemm.cuh"

namespace crvq {

namespace {

constexpr int64_t kKChunk = 1024;

// scale * sum_c P[c * stride + e], chunks in order (the one rounding sequence every split-K
// product of this file uses, so its dense and block-only forms agree bit for bit)
__device__ __forceinline__ float chunk_sum(const float* __restrict__ P, int chunks,
                                           int64_t stride, int64_t e, float scale) {
  float s = 0.f;
  for (int c = 0; c < chunks; ++c) s += P[c * stride + e];
  return s * scale;
}

__global__ void __launch_bounds__(256)
sum_partials_kernel(const float* __restrict__ P, int64_t count, int chunks, int64_t stride,
                    float scale, float* __restrict__ out) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < count;
       e += (int64_t)gridDim.x * blockDim.x)
    out[e] = chunk_sum(P, chunks, stride, e, scale);
}

// out[m][n] (leading dimension ldo) = sum of the chunk partials P[c][m][n] (M x Nb each), in
// chunk order.
__global__ void __launch_bounds__(256)
sum_partials_strided_kernel(const float* __restrict__ P, int64_t M, int64_t Nb, int chunks,
                            float* __restrict__ out, int64_t ldo) {
  const int64_t count = M * Nb;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < count;
       e += (int64_t)gridDim.x * blockDim.x)
    out[(e / Nb) * ldo + e % Nb] = chunk_sum(P, chunks, count, e, 1.f);
}

// Original-order blocks, one CTA: xsq[i] = the undamped diagonal, delta = damp_rel * mean(xsq)
// by the dense path's fixed-order fp64 reduction (1024 strided partials, then a tree), and the
// blocks with delta added on their diagonals (rounded once from fp64, as the dense path does).
__global__ void __launch_bounds__(1024)
blocks_finalize_kernel(const float* __restrict__ P, int chunks, int64_t stride, float scale,
                       int64_t N, float damp_rel, float* __restrict__ xsq,
                       float* __restrict__ delta_out, double* __restrict__ delta64,
                       float* __restrict__ Hb) {
  __shared__ double part[1024];
  double s = 0.0;
  for (int64_t i = threadIdx.x; i < N; i += blockDim.x) {
    const float v = chunk_sum(P, chunks, stride, i * 8 + (i & 7), scale);
    xsq[i] = v;
    s += (double)v;
  }
  part[threadIdx.x] = s;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) part[threadIdx.x] += part[threadIdx.x + w];
    __syncthreads();
  }
  const double delta = (double)damp_rel * (part[0] / (double)N);
  for (int64_t e = threadIdx.x; e < N * 8; e += blockDim.x) {
    const float v = chunk_sum(P, chunks, stride, e, scale);
    Hb[e] = ((e >> 3) & 7) == (e & 7) ? (float)((double)v + delta) : v;
  }
  if (threadIdx.x == 0) {
    if (delta_out) *delta_out = (float)delta;
    *delta64 = delta;
  }
}

// Blocks of a given channel order with a known delta.
__global__ void __launch_bounds__(256)
blocks_damp_kernel(const float* __restrict__ P, int chunks, int64_t stride, float scale,
                   int64_t N, const double* __restrict__ delta64, float* __restrict__ Hb) {
  const double delta = *delta64;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < N * 8;
       e += (int64_t)gridDim.x * blockDim.x) {
    const float v = chunk_sum(P, chunks, stride, e, scale);
    Hb[e] = ((e >> 3) & 7) == (e & 7) ? (float)((double)v + delta) : v;
  }
}

// out[a][k] = X[k][a] (X: n x N row-major) for a < N, k < n; columns k in [n, ldt) are 0.
__global__ void __launch_bounds__(256)
transpose_kernel(const float* __restrict__ X, int64_t n, int64_t N, float* __restrict__ out,
                 int64_t ldt) {
  __shared__ float t[32][33];
  const int64_t k0 = (int64_t)blockIdx.x * 32, a0 = (int64_t)blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 32 x 8
#pragma unroll
  for (int r = ty; r < 32; r += 8) {
    const int64_t k = k0 + r, a = a0 + tx;
    t[r][tx] = (k < n && a < N) ? X[k * N + a] : 0.f;
  }
  __syncthreads();
#pragma unroll
  for (int r = ty; r < 32; r += 8) {
    const int64_t a = a0 + r, k = k0 + tx;
    if (a < N && k < ldt) out[a * ldt + k] = t[tx][r];
  }
}

// ---- image-fed 3xTF32 sum of squares ||A B^T||_F^2 (the full loss of Alg. 1 QuantLoss)
// Both operands are first written once as tf32 hi / lo images in the tcgen05 canonical
// K-major layout (no swizzle): 256-row blocks, 16-column slabs of 16 KB each, slabs of a block
// consecutive. A CTA then computes one 128 x 256 tile with no work of its threads on the
// operand path: warp 0 streams the slabs by bulk copy (TMA) into a four-stage ring, warp 1
// issues the MMAs (hi.hi, hi.lo, lo.hi per 8-column step, as the split GEMM does), and warps
// 2-5 keep the K-chunk partials: after every 1024-column chunk the accumulator is added, in
// chunk order and in fp32, to a running sum kept in the other half of tensor memory; the last
// chunk's sum is squared and summed per row.
namespace img {

constexpr int kRowsBlk = 256;                      // image block rows
constexpr int kSlabK = 16;                         // image slab columns
constexpr int kSlabBytes = kRowsBlk * kSlabK * 4;  // 16 KB
constexpr int kAStage = 2 * (kSlabBytes / 2);      // A hi + lo, 128 rows: 16 KB
constexpr int kBStage = 2 * kSlabBytes;            // B hi + lo, 256 rows: 32 KB
constexpr int kStageBytes = kAStage + kBStage;     // 48 KB
constexpr int kStages = 4;
constexpr int kSmem = kStages * kStageBytes + 1024 + 256;
constexpr int kThreads = 192;
constexpr int kChunkSlabs = 1024 / kSlabK;         // slabs per K chunk
constexpr uint32_t kIdesc = tc::idesc_tf32(128, 256);

// Image byte offset of element (r, k): block r / 256, slab k / 16, then the canonical offset.
__host__ __device__ inline int64_t img_off(int64_t r, int64_t k, int64_t nslab) {
  const int64_t blk = r / kRowsBlk, rr = r % kRowsBlk, sl = k / kSlabK, kk = k % kSlabK;
  return (blk * nslab + sl) * kSlabBytes +
         (((rr >> 3) * (kSlabK / 4) + (kk >> 2)) * 128 + (rr & 7) * 16 + (kk & 3) * 4);
}

// One warp = 8 rows x one 16-column slab: reads 8 x 64 B, writes 512 contiguous bytes per
// image. Element (r, k) is src[r][k] - sub[r][k] (sub optional, same layout), or
// src[r][cols[k]] with a column order (entries outside [0, K) read as 0; the caller checks
// the order). Rows >= rows and columns >= K are written as zeros (the images' padding).
__global__ void __launch_bounds__(256)
image_kernel(const float* __restrict__ src, const float* __restrict__ sub,
             const int32_t* __restrict__ cols, int64_t rows, int64_t K, int64_t ld,
             int64_t rows_pad, int64_t nslab, char* __restrict__ hi, char* __restrict__ lo) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t r = (int64_t)blockIdx.x * 8 + (lane & 7);
  const int64_t sl = (int64_t)blockIdx.y * 8 + warp;
  if (sl >= nslab || r >= rows_pad) return;
  const int64_t k = sl * kSlabK + (lane >> 3) * 4;
  float v[4] = {0.f, 0.f, 0.f, 0.f};
  if (r < rows) {
    const float* p = src + r * ld;
    if (cols) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int32_t c = (k + j < K) ? cols[k + j] : -1;
        v[j] = (c >= 0 && c < K) ? p[c] : 0.f;
      }
    } else if (k + 4 <= K && (ld & 3) == 0 && ((uintptr_t)src & 15) == 0 &&
               (!sub || ((uintptr_t)sub & 15) == 0)) {
      const float4 x = __ldg(reinterpret_cast<const float4*>(p + k));
      v[0] = x.x; v[1] = x.y; v[2] = x.z; v[3] = x.w;
      if (sub) {
        const float4 y = __ldg(reinterpret_cast<const float4*>(sub + r * ld + k));
        v[0] -= y.x; v[1] -= y.y; v[2] -= y.z; v[3] -= y.w;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        v[j] = (k + j < K) ? (sub ? p[k + j] - sub[r * ld + k + j] : p[k + j]) : 0.f;
    }
  }
  uint32_t h[4], l[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    h[j] = tc::to_tf32(v[j]);
    l[j] = tc::to_tf32(v[j] - __uint_as_float(h[j]));
  }
  const int64_t off = img_off(r, k, nslab);
  *reinterpret_cast<uint4*>(hi + off) = make_uint4(h[0], h[1], h[2], h[3]);
  *reinterpret_cast<uint4*>(lo + off) = make_uint4(l[0], l[1], l[2], l[3]);
}

struct SumsqArgs {
  const char *a_hi, *a_lo, *b_hi, *b_lo;  // images
  int64_t nslab;                          // slabs per block (both images)
  int tiles_n;                            // 256-row tiles of B
  double* part;                           // part[tile] = sum over the tile of D^2
  unsigned* err;
};

__global__ void __launch_bounds__(kThreads, 1) sumsq_img_kernel(SumsqArgs a) {
  extern __shared__ __align__(1024) char smem_raw[];
  char* smem = smem_raw + ((1024u - (tc::smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint64_t* empty = full + kStages;
  uint64_t* acc_full = empty + kStages;
  uint64_t* acc_empty = acc_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 1);
  __shared__ double red[4];
  __shared__ int ok_s[3];

  const int tile = blockIdx.x;
  const int bm = tile / a.tiles_n, bn = tile % a.tiles_n;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t nslab = a.nslab;
  const int nchunk = (int)((nslab + kChunkSlabs - 1) / kChunkSlabs);

  if (warp == 0) tc::tmem_alloc(tmem_slot, 512);
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(tc::smem_u32(&full[s]), 1);
      tc::mbar_init(tc::smem_u32(&empty[s]), 1);
    }
    tc::mbar_init(tc::smem_u32(acc_full), 1);
    tc::mbar_init(tc::smem_u32(acc_empty), 128);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (threadIdx.x < 3) ok_s[threadIdx.x] = 1;
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_slot;   // columns [0, 256): accumulator; [256, 512): chunk sum

  if (warp == 0) {
    if (lane == 0) {  // producer
      const char* ah = a.a_hi + ((int64_t)(bm >> 1) * nslab) * kSlabBytes + (bm & 1) * (kSlabBytes / 2);
      const char* al = a.a_lo + ((int64_t)(bm >> 1) * nslab) * kSlabBytes + (bm & 1) * (kSlabBytes / 2);
      const char* bh = a.b_hi + (int64_t)bn * nslab * kSlabBytes;
      const char* bl = a.b_lo + (int64_t)bn * nslab * kSlabBytes;
      bool ok = true;
      for (int64_t it = 0; it < nslab && ok; ++it) {
        const int s = (int)(it % kStages);
        if (it >= kStages)
          ok = tc::mbar_wait(tc::smem_u32(&empty[s]), (uint32_t)((it / kStages - 1) & 1), a.err);
        if (!ok) break;
        char* st = smem + s * kStageBytes;
        const uint32_t fb = tc::smem_u32(&full[s]);
        tc::mbar_expect_tx(fb, kStageBytes);
        tc::bulk_copy_g2s(tc::smem_u32(st), ah + it * kSlabBytes, kSlabBytes / 2, fb);
        tc::bulk_copy_g2s(tc::smem_u32(st + kSlabBytes / 2), al + it * kSlabBytes, kSlabBytes / 2, fb);
        tc::bulk_copy_g2s(tc::smem_u32(st + kAStage), bh + it * kSlabBytes, kSlabBytes, fb);
        tc::bulk_copy_g2s(tc::smem_u32(st + kAStage + kSlabBytes), bl + it * kSlabBytes, kSlabBytes, fb);
      }
      if (!ok) ok_s[0] = 0;
    }
  } else if (warp == 1) {
    if (lane == 0) {  // MMA issuer
      bool ok = true;
      for (int64_t it = 0; it < nslab && ok; ++it) {
        const int s = (int)(it % kStages);
        const int64_t c = it / kChunkSlabs;
        const bool first = (it % kChunkSlabs) == 0;
        if (first && c > 0) ok = tc::mbar_wait(tc::smem_u32(acc_empty), (uint32_t)((c - 1) & 1), a.err);
        if (ok) ok = tc::mbar_wait(tc::smem_u32(&full[s]), (uint32_t)((it / kStages) & 1), a.err);
        if (!ok) break;
        tc::tc_fence_after();
        const uint32_t st = tc::smem_u32(smem + s * kStageBytes);
        constexpr uint32_t sbo = (kSlabK / 4) * 128;
#pragma unroll
        for (int ks = 0; ks < kSlabK / 8; ++ks) {
          const uint32_t koff = ks * 256;
          const uint64_t dah = tc::smem_desc(st + koff, 128, sbo);
          const uint64_t dal = tc::smem_desc(st + kSlabBytes / 2 + koff, 128, sbo);
          const uint64_t dbh = tc::smem_desc(st + kAStage + koff, 128, sbo);
          const uint64_t dbl = tc::smem_desc(st + kAStage + kSlabBytes + koff, 128, sbo);
          tc::mma_tf32(tmem, dah, dbh, kIdesc, (first && ks == 0) ? 0u : 1u);
          tc::mma_tf32(tmem, dah, dbl, kIdesc, 1u);
          tc::mma_tf32(tmem, dal, dbh, kIdesc, 1u);
        }
        tc::mma_commit(tc::smem_u32(&empty[s]));
        if ((it % kChunkSlabs) == kChunkSlabs - 1 || it == nslab - 1)
          tc::mma_commit(tc::smem_u32(acc_full));
      }
      if (!ok) ok_s[1] = 0;
    }
  } else {  // warps 2-5: one accumulator row (tensor-memory lane) per thread
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    float sq = 0.f;
    bool ok = true;
    for (int c = 0; c < nchunk && ok; ++c) {
      ok = tc::mbar_wait(tc::smem_u32(acc_full), (uint32_t)(c & 1), a.err);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc::tc_fence_after();
      const bool last = c == nchunk - 1;
#pragma unroll 1
      for (int c0 = 0; c0 < 256; c0 += 32) {
        uint32_t v[32], w[32];
        tc::tmem_ld32_nowait(tmem + lane_base + (uint32_t)c0, v);
        tc::tmem_wait_ld_dep(v);
        if (c > 0) {
          tc::tmem_ld32_nowait(tmem + lane_base + 256u + (uint32_t)c0, w);
          tc::tmem_wait_ld_dep(w);
#pragma unroll
          for (int j = 0; j < 32; ++j)
            v[j] = __float_as_uint(__fadd_rn(__uint_as_float(w[j]), __uint_as_float(v[j])));
        }
        if (last) {
#pragma unroll
          for (int j = 0; j < 32; ++j) sq = fmaf(__uint_as_float(v[j]), __uint_as_float(v[j]), sq);
        } else {
          tc::tmem_st32_wait(tmem + lane_base + 256u + (uint32_t)c0, v);
        }
      }
      tc::tc_fence_before();
      if (!last) tc::mbar_arrive(tc::smem_u32(acc_empty));
    }
    if (!ok) sq = 0.f;
    double sd = (double)sq;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sd += __shfl_xor_sync(0xffffffffu, sd, o);
    if (lane == 0) red[warp - 2] = sd;
    if (lane == 0 && !ok) ok_s[2] = 0;
  }
  tc::tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) {
    const bool ok = ok_s[0] && ok_s[1] && ok_s[2];
    a.part[tile] = ok ? ((red[0] + red[1]) + (red[2] + red[3])) : 0.0;
  }
  if (warp == 0) {
    __syncwarp();
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, 512);
  }
}

}  // namespace img

crvq_status launch_gemm(tc::GemmArgs g, int64_t chunks, cudaStream_t stream) {
  static bool attr_set[64] = {};
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  if (dev < 64 && !attr_set[dev]) {
    CRVQ_CUDA(cudaFuncSetAttribute(tc::gemm3xtf32_kernel,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, tc::kSmemBytes));
    attr_set[dev] = true;
  }
  const int64_t tm = ceil_div(g.A.rows, tc::kBM), tn = ceil_div(g.B.rows, tc::kBN);
  g.tiles_n = (int)tn;
  dim3 grid((unsigned)(tm * tn), (unsigned)chunks);
  tc::gemm3xtf32_kernel<<<grid, tc::kThreads, tc::kSmemBytes, stream>>>(g);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace

// S = X^T X / n (X: n x N row-major) into S (N x N), both triangles, via split-K partials.
crvq_status launch_tc_syrk(const float* X, int64_t n, int64_t N, float* S, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const int64_t chunks = ceil_div(n, kKChunk);
  Scratch mem, xt_mem;
  float* P = S;
  if (chunks > 1) {
    CRVQ_TRY(mem.alloc((size_t)chunks * N * N * sizeof(float), stream));
    P = mem.as<float>();
  }
  // X^T with rows padded to a multiple of 4 floats: both operands K-major, loaded with 16-byte
  // loads (A(a, k) = X[k][a])
  const int64_t ldt = (n + 3) / 4 * 4;
  CRVQ_TRY(xt_mem.alloc((size_t)N * ldt * sizeof(float), stream));
  CRVQ_TRY(launch_transpose(X, n, N, xt_mem.as<float>(), ldt, stream));
  tc::GemmArgs g{};
  g.A = tc::Operand{xt_mem.as<float>(), ldt, N, true};
  g.B = g.A;
  g.K = n;
  g.k_chunk = kKChunk;
  g.c_chunk_stride = N * N;
  g.mode = tc::kStoreSymmetric;
  g.C = P;
  g.ldc = N;
  g.alpha = chunks > 1 ? 1.f : (float)(1.0 / (double)n);
  g.err = err;
  {
    ProfScope ps("hessian_gemm_tc", stream, 2.0 * (double)n * N * N);
    CRVQ_TRY(launch_gemm(g, chunks, stream));
  }
  if (chunks > 1) {
    ProfScope ps("hessian_sum_partials", stream, (double)chunks * N * N * 4.0);
    const int blocks = (int)std::min<int64_t>(ceil_div(N * N, 256), 16 * sm_count());
    sum_partials_kernel<<<blocks, 256, 0, stream>>>(P, N * N, (int)chunks, N * N,
                                                    (float)(1.0 / (double)n), S);
    CRVQ_LAUNCHED();
  }
  return CRVQ_OK;
}

// C = A B^T (A: M x K, B: Nb x K, both row-major with leading dimensions lda, ldb; C: M x Nb
// row-major, leading dimension ldc) on the tensor cores (3xTF32), K in chunks of at most 1024
// whose partials are added in chunk order (the rounding sequence of the Hessian products).
crvq_status launch_tc_gemm_nt(const float* A, int64_t lda, int64_t M, const float* B,
                              int64_t ldb, int64_t Nb, int64_t K, float* C, int64_t ldc,
                              cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const int64_t chunks = std::max<int64_t>(1, ceil_div(K, kKChunk));
  Scratch mem;
  float* P = C;
  int64_t ldp = ldc;
  if (chunks > 1) {
    CRVQ_TRY(mem.alloc((size_t)chunks * M * Nb * sizeof(float), stream));
    P = mem.as<float>();
    ldp = Nb;
  }
  tc::GemmArgs g{};
  g.A = tc::Operand{A, lda, M, true};
  g.B = tc::Operand{B, ldb, Nb, true};
  g.K = K;
  g.k_chunk = kKChunk;
  g.c_chunk_stride = M * Nb;
  g.mode = tc::kStorePlain;
  g.C = P;
  g.ldc = ldp;
  g.alpha = 1.f;
  g.err = err;
  {
    ProfScope ps("gemm_nt_tc", stream, 2.0 * (double)M * Nb * K);
    CRVQ_TRY(launch_gemm(g, chunks, stream));
  }
  if (chunks > 1) {
    ProfScope ps("gemm_nt_sum_partials", stream, (double)chunks * M * Nb * 4.0);
    const int blocks = (int)std::min<int64_t>(ceil_div(M * Nb, 256), 16 * sm_count());
    sum_partials_strided_kernel<<<blocks, 256, 0, stream>>>(P, M, Nb, (int)chunks, C, ldc);
    CRVQ_LAUNCHED();
  }
  return CRVQ_OK;
}

// part[0 .. nparts) = partial sums of ||(A - A_sub) B'^T||_F^2 with A, A_sub: M x K, B: Nb x K
// (row-major, leading dimension K; B' = B with columns in the order B_cols when given), one
// per 128 x 256 tile; part_cap must hold ceil(M / 128) * ceil(Nb / 256) values. Returns the
// number of partials written.
crvq_status launch_tc_sumsq(const float* A, const float* A_sub, int64_t M, const float* B,
                            const int32_t* B_cols, int64_t Nb, int64_t K, double* part,
                            int64_t part_cap, int64_t* nparts, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  static bool attr_set[64] = {};
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  if (dev < 64 && !attr_set[dev]) {
    CRVQ_CUDA(cudaFuncSetAttribute(img::sumsq_img_kernel,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, img::kSmem));
    attr_set[dev] = true;
  }
  const int64_t tiles_m = ceil_div(M, 128), tiles_n = ceil_div(Nb, 256);
  if (tiles_m * tiles_n > part_cap)
    return fail(CRVQ_ERR_UNSUPPORTED, "loss product: %lld tiles exceed %lld partials",
                (long long)(tiles_m * tiles_n), (long long)part_cap);
  if (tiles_m * tiles_n > INT32_MAX)
    return fail(CRVQ_ERR_UNSUPPORTED, "loss product: too many tiles");
  const int64_t nslab = ceil_div(K, (int64_t)img::kSlabK);
  const int64_t am = ceil_div(M, (int64_t)img::kRowsBlk) * img::kRowsBlk;
  const int64_t bm = ceil_div(Nb, (int64_t)img::kRowsBlk) * img::kRowsBlk;
  const size_t a_bytes = (size_t)am * nslab * img::kSlabK * 4;
  const size_t b_bytes = (size_t)bm * nslab * img::kSlabK * 4;
  Scratch mem;
  CRVQ_TRY(mem.alloc(2 * a_bytes + 2 * b_bytes, stream));
  char* a_hi = mem.as<char>();
  char* a_lo = a_hi + a_bytes;
  char* b_hi = a_lo + a_bytes;
  char* b_lo = b_hi + b_bytes;
  {
    ProfScope ps("loss_images", stream, 12.0 * (double)(M + Nb) * K);
    img::image_kernel<<<dim3((unsigned)(am / 8), (unsigned)ceil_div(nslab, 8)), 256, 0,
                        stream>>>(A, A_sub, nullptr, M, K, K, am, nslab, a_hi, a_lo);
    CRVQ_LAUNCHED();
    img::image_kernel<<<dim3((unsigned)(bm / 8), (unsigned)ceil_div(nslab, 8)), 256, 0,
                        stream>>>(B, nullptr, B_cols, Nb, K, K, bm, nslab, b_hi, b_lo);
    CRVQ_LAUNCHED();
  }
  img::SumsqArgs g{a_hi, a_lo, b_hi, b_lo, nslab, (int)tiles_n, part, err};
  ProfScope ps("loss_gemm_tc", stream, 2.0 * (double)M * Nb * K);
  img::sumsq_img_kernel<<<(unsigned)(tiles_m * tiles_n), img::kThreads, img::kSmem, stream>>>(g);
  CRVQ_LAUNCHED();
  *nparts = tiles_m * tiles_n;
  return CRVQ_OK;
}

crvq_status launch_transpose(const float* X, int64_t n, int64_t N, float* Xt, int64_t ldt,
                             cudaStream_t stream) {
  ProfScope ps("hessian_transpose", stream, 8.0 * (double)n * N);
  transpose_kernel<<<dim3((unsigned)ceil_div(ldt, 32), (unsigned)ceil_div(N, 32)), 256, 0,
                     stream>>>(X, n, N, Xt, ldt);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

// Diagonal 8 x 8 blocks of X^T X / n (+ delta I) for the channel order `perm` (NULL = the
// stored order), from Xt = X^T (N x ldt, ldt a multiple of 4). delta_known: delta64 (fp64) is
// read; otherwise perm must be NULL and xsq, delta (float, may be NULL) and delta64 are
// written. The entries equal those of launch_tc_syrk's dense S plus the damping bit for bit.
crvq_status launch_tc_hessian_blocks(const float* Xt, int64_t ldt, int64_t n, int64_t N,
                                     const int32_t* perm, bool delta_known, float damp_rel,
                                     float* xsq, float* delta, double* delta64, float* Hb,
                                     cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  static bool attr_set[64] = {};
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  if (dev < 64 && !attr_set[dev]) {
    CRVQ_CUDA(cudaFuncSetAttribute(tc::syrk_diag_kernel,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   tc::kDiagSmemBytes));
    attr_set[dev] = true;
  }
  const int64_t chunks = std::max<int64_t>(1, ceil_div(n, kKChunk));
  const int64_t stride = N * 8;
  Scratch mem;
  CRVQ_TRY(mem.alloc((size_t)chunks * stride * sizeof(float), stream));
  tc::DiagArgs a{};
  a.A = tc::Operand{Xt, ldt, N, true, perm};
  a.K = n;
  a.k_chunk = kKChunk;
  a.out = mem.as<float>();
  a.chunk_stride = stride;
  a.alpha = chunks > 1 ? 1.f : (float)(1.0 / (double)n);
  a.err = err;
  const float scale = chunks > 1 ? (float)(1.0 / (double)n) : 1.f;
  {
    ProfScope ps(perm ? "reorder_blocks_tc" : "hessian_blocks_tc", stream,
                 6.0 * (double)n * N * tc::kBM);
    dim3 grid((unsigned)ceil_div(N, tc::kBM), (unsigned)chunks);
    tc::syrk_diag_kernel<<<grid, tc::kThreads, tc::kDiagSmemBytes, stream>>>(a);
    CRVQ_LAUNCHED();
  }
  ProfScope ps("hessian_blocks_finalize", stream, (double)chunks * stride * 4.0);
  if (!delta_known) {
    if (perm) return fail(CRVQ_ERR_UNSUPPORTED, "hessian blocks: delta needs the stored order");
    blocks_finalize_kernel<<<1, 1024, 0, stream>>>(mem.as<float>(), (int)chunks, stride, scale,
                                                   N, damp_rel, xsq, delta, delta64, Hb);
  } else {
    const int blocks = (int)std::min<int64_t>(ceil_div(stride, 256), 4 * sm_count());
    blocks_damp_kernel<<<blocks, 256, 0, stream>>>(mem.as<float>(), (int)chunks, stride, scale,
                                                   N, delta64, Hb);
  }
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace crvq
