// Tensor-core (tcgen05, sm_103a) fp32-accurate GEMM D = A B^T via the 3xTF32 split, with the
// accumulator in tensor memory, used for the Hessian proxy X^T X (App. A.2) and for the full
// loss ||dW X^T||^2 (Alg. 1 QuantLoss).
//
// Each fp32 operand x is split into x_hi = tf32(x) and x_lo = tf32(x - x_hi); the product
// uses a_hi b_hi + a_hi b_lo + a_lo b_hi (the dropped a_lo b_lo term and the rounding of the
// lo parts are ~2^-22 relative), accumulated in fp32 by the tensor core.
//
// CTA tile 128 x 256 (one tcgen05.mma M = 128, N = 256, K = 8 per instruction), K staged 16
// at a time through two shared-memory stages. All 128 threads load and split the next stage
// while the tensor core works on the previous one; thread 0 issues the MMAs and commits them
// to the stage's mbarrier. Operands sit in shared memory in the canonical K-major layout
// without swizzle: 8-row x 16-byte core matrices, consecutive along K (LBO = 128 B), 8-row
// groups SBO = (BK / 4) * 128 B apart. Every wait on an mbarrier is bounded (~2 s of
// %globaltimer); on expiry the kernel records ERRBIT_TIMEOUT, stops issuing and exits
// after freeing its tensor memory.
#pragma once

#include "common.cuh"

namespace crvq {
namespace tc {

constexpr int kBM = 128, kBN = 256, kBK = 16, kStages = 2, kThreads = 128;
constexpr int kAStageBytes = kBM * kBK * 4;            // one of hi / lo
constexpr int kBStageBytes = kBN * kBK * 4;
constexpr int kStageBytes = 2 * kAStageBytes + 2 * kBStageBytes;  // 48 KB
constexpr int kSmemBytes = kStages * kStageBytes + 1024 + 128;    // + alignment + barriers
constexpr int kTmemCols = 256;
constexpr unsigned long long kWaitNs = 2000000000ull;  // 2 s

// Instruction descriptor, kind::tf32: D fp32, A/B tf32, both K-major, N = 256, M = 128.
constexpr uint32_t kIdesc = (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(kBN >> 3) << 17) |
                            ((uint32_t)(kBM >> 4) << 24);

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Shared-memory matrix descriptor: start, LBO, SBO (bytes, multiples of 16), version 1,
// no swizzle.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((addr & 0x3FFFF) >> 4);
  d |= (uint64_t)((lbo & 0x3FFFF) >> 4) << 16;
  d |= (uint64_t)((sbo & 0x3FFFF) >> 4) << 32;
  d |= (uint64_t)1 << 46;
  return d;
}

__device__ __forceinline__ uint32_t to_tf32(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: false (and ERRBIT_TIMEOUT) when the phase did not complete within kWaitNs.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, unsigned* err) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer() - t0 > kWaitNs) {
      raise_error(err, ERRBIT_TIMEOUT);
      return false;
    }
  }
  return true;
}

__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void mma_tf32(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

// 32 consecutive accumulator columns of this thread's lane (row).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float v[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}

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

// Loads rows [r0, r0 + R) x k [k0, k0 + kBK) of the operand, splits each value into tf32
// hi / lo and stores both tiles (zero outside the matrix). Thread t handles rows t, t + 128...
template <int R>
__device__ __forceinline__ void load_split(const Operand& op, int64_t r0, int64_t k0,
                                           int64_t K, char* hi, char* lo) {
#pragma unroll
  for (int rr = 0; rr < R / kThreads; ++rr) {
    const int r = threadIdx.x + rr * kThreads;
    const int64_t row = r0 + r;
    float v[kBK];
    if (row < op.rows) {
      if (op.kmajor) {
        const float* src = op.p + row * op.ld + k0;
        if (k0 + kBK <= K && (op.ld & 3) == 0 && ((uintptr_t)op.p & 15) == 0) {
#pragma unroll
          for (int q = 0; q < kBK / 4; ++q) {
            const float4 x = reinterpret_cast<const float4*>(src)[q];
            v[4 * q] = x.x; v[4 * q + 1] = x.y; v[4 * q + 2] = x.z; v[4 * q + 3] = x.w;
          }
        } else {
#pragma unroll
          for (int q = 0; q < kBK; ++q) v[q] = (k0 + q < K) ? src[q] : 0.f;
        }
      } else {
#pragma unroll
        for (int q = 0; q < kBK; ++q) v[q] = (k0 + q < K) ? op.p[(k0 + q) * op.ld + row] : 0.f;
      }
    } else {
#pragma unroll
      for (int q = 0; q < kBK; ++q) v[q] = 0.f;
    }
#pragma unroll
    for (int q = 0; q < kBK / 4; ++q) {
      uint32_t h[4], l[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        h[j] = to_tf32(v[4 * q + j]);
        l[j] = to_tf32(v[4 * q + j] - __uint_as_float(h[j]));
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
  char* smem = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                       ~(uintptr_t)1023);
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

  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(smem_u32(&bars[s]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  const int64_t nkt = (kend - kbeg + kBK - 1) / kBK;
  uint32_t waits[kStages] = {0, 0};
  bool ok = true;
  for (int64_t kt = 0; kt < nkt; ++kt) {
    const int s = (int)(kt & 1);
    char* st = smem + s * kStageBytes;
    char* a_hi = st;
    char* a_lo = st + kAStageBytes;
    char* b_hi = st + 2 * kAStageBytes;
    char* b_lo = b_hi + kBStageBytes;
    if (kt >= kStages) {
      // the MMAs issued two stages ago read this buffer: wait for them (bounded)
      if (ok) ok = mbar_wait(smem_u32(&bars[s]), waits[s] & 1, a.err);
      ++waits[s];
    }
    ok = __syncthreads_and(ok);
    if (!ok) break;
    load_split<kBM>(a.A, m0, kbeg + kt * kBK, kend, a_hi, a_lo);
    load_split<kBN>(a.B, n0, kbeg + kt * kBK, kend, b_hi, b_lo);
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
        mma_tf32(tmem, dah, dbh, (kt > 0 || ks > 0) ? 1u : 0u);
        mma_tf32(tmem, dah, dbl, 1u);
        mma_tf32(tmem, dal, dbh, 1u);
      }
      mma_commit(smem_u32(&bars[s]));
    }
  }
  // wait for the last commit (it covers every earlier MMA of this thread)
  if (ok && nkt > 0) {
    const int s = (int)((nkt - 1) & 1);
    ok = mbar_wait(smem_u32(&bars[s]), waits[s] & 1, a.err);
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
  if (warp == 0) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols)
                 : "memory");
  }
}

}  // namespace tc
}  // namespace crvq
