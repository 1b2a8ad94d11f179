// Tensor-core (tcgen05, sm_103a) fp32-accurate GEMM D = A B^T via the 3xTF32 split, with the
// accumulator in tensor memory, used for the Hessian proxy X^T X (App. A.2) and for the full
// loss ||dW X^T||^2 (Alg. 1 QuantLoss).
//
// Each fp32 operand x is split into x_hi = tf32(x) and x_lo = tf32(x - x_hi); the product
// uses a_hi b_hi + a_hi b_lo + a_lo b_hi (the dropped a_lo b_lo term and the rounding of the
// lo parts are ~2^-22 relative), accumulated in fp32 by the tensor core.
//
// CTA tile 128 x 256 (one tcgen05.mma M = 128, N = 256, K = 8 per instruction), K staged 16
// at a time through two shared-memory stages. All 128 threads split and store a stage while
// the tensor core works on the previous one, with the global loads of the next stage already
// in flight in registers (software pipeline); thread 0 issues the MMAs and commits them to the
// stage's mbarrier. Operands sit in shared memory in the canonical K-major layout
// without swizzle: 8-row x 16-byte core matrices, consecutive along K (LBO = 128 B), 8-row
// groups SBO = (BK / 4) * 128 B apart. Every wait on an mbarrier is bounded (~2 s of
// %globaltimer); on expiry the kernel records ERRBIT_TIMEOUT, stops issuing and exits
// after freeing its tensor memory.
#pragma once

#include "common.cuh"
#include "tc_ops.cuh"

namespace crvq {
namespace tc {

constexpr int kBM = 128, kBN = 256, kBK = 16, kStages = 2, kThreads = 128;
constexpr int kAStageBytes = kBM * kBK * 4;            // one of hi / lo
constexpr int kBStageBytes = kBN * kBK * 4;
constexpr int kStageBytes = 2 * kAStageBytes + 2 * kBStageBytes;  // 48 KB
constexpr int kSmemBytes = kStages * kStageBytes + 1024 + 128;    // + alignment + barriers
constexpr int kTmemCols = 256;
constexpr uint32_t kIdesc = idesc_tf32(kBM, kBN);

// Byte offset of element (r, k) in a K-major no-swizzle tile with kBK columns.
__device__ __forceinline__ uint32_t tile_off(int r, int k) {
  return (uint32_t)(((r >> 3) * (kBK / 4) + (k >> 2)) * 128 + (r & 7) * 16 + (k & 3) * 4);
}

// Operand view: element (row, k) = p[row * ld + k] (K-major) or p[k * ld + row].
struct Operand {
  const float* p;
  int64_t ld;
  int64_t rows;
  bool kmajor;
};

// Loads rows [r0, r0 + R) x k [k0, k0 + kBK) of the operand into registers (zero outside the
// matrix). Thread t handles rows t, t + 128, ...
template <int R>
__device__ __forceinline__ void load_tile(const Operand& op, int64_t r0, int64_t k0, int64_t K,
                                          float v[R / kThreads][kBK]) {
#pragma unroll
  for (int rr = 0; rr < R / kThreads; ++rr) {
    const int r = threadIdx.x + rr * kThreads;
    const int64_t row = r0 + r;
    if (row < op.rows) {
      if (op.kmajor) {
        const float* src = op.p + row * op.ld + k0;
        if (k0 + kBK <= K && (op.ld & 3) == 0 && ((uintptr_t)op.p & 15) == 0) {
#pragma unroll
          for (int q = 0; q < kBK / 4; ++q) {
            const float4 x = __ldg(reinterpret_cast<const float4*>(src) + q);
            v[rr][4 * q] = x.x; v[rr][4 * q + 1] = x.y; v[rr][4 * q + 2] = x.z; v[rr][4 * q + 3] = x.w;
          }
        } else {
#pragma unroll
          for (int q = 0; q < kBK; ++q) v[rr][q] = (k0 + q < K) ? src[q] : 0.f;
        }
      } else {
#pragma unroll
        for (int q = 0; q < kBK; ++q)
          v[rr][q] = (k0 + q < K) ? op.p[(k0 + q) * op.ld + row] : 0.f;
      }
    } else {
#pragma unroll
      for (int q = 0; q < kBK; ++q) v[rr][q] = 0.f;
    }
  }
}

// Splits the loaded values into tf32 hi / lo and stores both tiles.
template <int R>
__device__ __forceinline__ void split_store(const float v[R / kThreads][kBK], char* hi, char* lo) {
#pragma unroll
  for (int rr = 0; rr < R / kThreads; ++rr) {
    const int r = threadIdx.x + rr * kThreads;
#pragma unroll
    for (int q = 0; q < kBK / 4; ++q) {
      uint32_t h[4], l[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        h[j] = to_tf32(v[rr][4 * q + j]);
        l[j] = to_tf32(v[rr][4 * q + j] - __uint_as_float(h[j]));
      }
      const uint32_t off = tile_off(r, 4 * q);
      *reinterpret_cast<uint4*>(hi + off) = make_uint4(h[0], h[1], h[2], h[3]);
      *reinterpret_cast<uint4*>(lo + off) = make_uint4(l[0], l[1], l[2], l[3]);
    }
  }
}

// Epilogues.
enum Mode { kStoreSymmetric = 0, kSumSquares = 1, kStore = 2 };

struct GemmArgs {
  Operand A, B;   // D[m][n] = sum_k A(m, k) B(n, k); M = A.rows, N = B.rows
  int64_t K;
  // Split K: blockIdx.y = chunk c covers k in [c * k_chunk, min(K, (c + 1) * k_chunk)) and
  // writes to C + c * c_chunk_stride (kStore / kStoreSymmetric) or part + c * tiles.
  int64_t k_chunk;
  int64_t c_chunk_stride;
  int mode;
  // kStoreSymmetric: C[m][n] = C[n][m] = alpha * D[m][n] for n >= m (row-major, ldc)
  // kStore: C[m][n] = alpha * D[m][n]
  float* C;
  int64_t ldc;
  float alpha;
  // kSumSquares: part[tile] = sum over the tile of D^2 (fp64)
  double* part;
  int tiles_n;    // tiles along N (grid is linear; tile = bm * tiles_n + bn)
  unsigned* err;
};

__global__ void __launch_bounds__(kThreads, 1) gemm3xtf32_kernel(GemmArgs a) {
  extern __shared__ __align__(1024) char smem_raw[];
  // 1024-byte aligned base, derived from the shared array (keeps the shared address space)
  char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + kStages);
  __shared__ double red[kThreads];

  const int tile = blockIdx.x;
  const int bm = tile / a.tiles_n, bn = tile % a.tiles_n;
  const int64_t m0 = (int64_t)bm * kBM, n0 = (int64_t)bn * kBN;
  const int64_t kbeg = (int64_t)blockIdx.y * a.k_chunk;
  const int64_t kend = min(a.K, kbeg + a.k_chunk);
  float* C = a.C ? a.C + (int64_t)blockIdx.y * a.c_chunk_stride : nullptr;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // a symmetric product needs only the tiles that reach the upper triangle
  if (a.mode == kStoreSymmetric && n0 + kBN <= m0) return;

  if (warp == 0) tmem_alloc(tmem_slot, kTmemCols);
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(smem_u32(&bars[s]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  const int64_t nkt = (kend - kbeg + kBK - 1) / kBK;
  uint32_t par = 0;  // parity of the next wait per stage (bit = stage)
  bool ok = true;
  // Software pipeline: the global loads of step kt + 1 are in flight while step kt is split,
  // stored and multiplied.
  float va[kBM / kThreads][kBK], vb[kBN / kThreads][kBK];
  if (nkt > 0) {
    load_tile<kBM>(a.A, m0, kbeg, kend, va);
    load_tile<kBN>(a.B, n0, kbeg, kend, vb);
  }
  for (int64_t kt = 0; kt < nkt; ++kt) {
    const int s = (int)(kt & 1);
    char* st = smem + s * kStageBytes;
    char* a_hi = st;
    char* a_lo = st + kAStageBytes;
    char* b_hi = st + 2 * kAStageBytes;
    char* b_lo = b_hi + kBStageBytes;
    if (kt >= kStages) {
      // the MMAs issued two stages ago read this buffer: wait for them (bounded)
      if (ok) ok = mbar_wait(smem_u32(&bars[s]), (par >> s) & 1u, a.err);
      par ^= 1u << s;
    }
    ok = __syncthreads_and(ok);
    if (!ok) break;
    split_store<kBM>(va, a_hi, a_lo);
    split_store<kBN>(vb, b_hi, b_lo);
    if (kt + 1 < nkt) {
      load_tile<kBM>(a.A, m0, kbeg + (kt + 1) * kBK, kend, va);
      load_tile<kBN>(a.B, n0, kbeg + (kt + 1) * kBK, kend, vb);
    }
    fence_async_smem();
    __syncthreads();
    if (threadIdx.x == 0) {
      tc_fence_after();
      const uint32_t sbo = (kBK / 4) * 128;
#pragma unroll
      for (int ks = 0; ks < kBK / 8; ++ks) {
        const uint32_t koff = ks * 256;  // 8 tf32 = two core matrices along K
        const uint64_t dah = smem_desc(smem_u32(a_hi) + koff, 128, sbo);
        const uint64_t dal = smem_desc(smem_u32(a_lo) + koff, 128, sbo);
        const uint64_t dbh = smem_desc(smem_u32(b_hi) + koff, 128, sbo);
        const uint64_t dbl = smem_desc(smem_u32(b_lo) + koff, 128, sbo);
        mma_tf32(tmem, dah, dbh, kIdesc, (kt > 0 || ks > 0) ? 1u : 0u);
        mma_tf32(tmem, dah, dbl, kIdesc, 1u);
        mma_tf32(tmem, dal, dbh, kIdesc, 1u);
      }
      mma_commit(smem_u32(&bars[s]));
    }
  }
  // wait for the last commit (it covers every earlier MMA of this thread)
  if (ok && nkt > 0) {
    const int s = (int)((nkt - 1) & 1);
    ok = mbar_wait(smem_u32(&bars[s]), (par >> s) & 1u, a.err);
  }
  ok = __syncthreads_and(ok);
  tc_fence_after();

  double sq = 0.0;
  if (ok) {
    const int row = warp * 32 + lane;
    const int64_t m = m0 + row;
#pragma unroll 1
    for (int c0 = 0; c0 < kBN; c0 += 32) {
      float v[32];
      tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, v);
      if (a.mode == kSumSquares) {
#pragma unroll
        for (int j = 0; j < 32; ++j) sq += (double)v[j] * (double)v[j];
      } else if (a.mode == kStore) {
        if (m < a.A.rows) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int64_t n = n0 + c0 + j;
            if (n < a.B.rows) C[m * a.ldc + n] = a.alpha * v[j];
          }
        }
      } else if (m < a.A.rows) {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int64_t n = n0 + c0 + j;
          if (n >= m && n < a.B.rows) {
            const float x = a.alpha * v[j];
            C[m * a.ldc + n] = x;
            C[n * a.ldc + m] = x;
          }
        }
      }
    }
  }
  if (a.mode == kSumSquares) {
    red[threadIdx.x] = sq;
    __syncthreads();
    for (int w = kThreads / 2; w > 0; w >>= 1) {
      if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
      __syncthreads();
    }
    if (threadIdx.x == 0)
      a.part[(int64_t)blockIdx.y * gridDim.x + tile] = ok ? red[0] : 0.0;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
}

}  // namespace tc
}  // namespace crvq
