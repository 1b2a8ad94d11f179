// Tensor-core (tcgen05, sm_103a) fp32-accurate GEMM D = A B^T via the 3xTF32 split, with the
// accumulator in tensor memory, used for the dense Hessian proxy X^T X (App. A.2) and, in a
// block-diagonal form, for its d x d diagonal blocks alone.
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

// Operand view: element (row, k) = p[row * ld + k] (K-major) or p[k * ld + row]. With `idx`
// (K-major only) logical row r reads stored row idx[r]; an entry outside [0, rows) reads as 0.
struct Operand {
  const float* p;
  int64_t ld;
  int64_t rows;
  bool kmajor;
  const int32_t* idx = nullptr;
};

// Loads rows [r0, r0 + R) x k [k0, k0 + kBK) of the operand into registers (zero outside the
// matrix). Thread t handles rows t, t + 128, ...
template <int R>
__device__ __forceinline__ void load_tile(const Operand& op, int64_t r0, int64_t k0, int64_t K,
                                          float v[R / kThreads][kBK]) {
#pragma unroll
  for (int rr = 0; rr < R / kThreads; ++rr) {
    const int r = threadIdx.x + rr * kThreads;
    int64_t row = r0 + r;
    if (row < op.rows && op.idx) {
      row = op.idx[row];
      if (row < 0) row = op.rows;  // out of range: zero row (the caller reports it)
    }
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
enum Mode { kStoreSymmetric = 0, kStorePlain = 1 };

struct GemmArgs {
  Operand A, B;   // D[m][n] = sum_k A(m, k) B(n, k); M = A.rows, N = B.rows
  int64_t K;
  // Split K: blockIdx.y = chunk c covers k in [c * k_chunk, min(K, (c + 1) * k_chunk)) and
  // writes to C + c * c_chunk_stride.
  int64_t k_chunk;
  int64_t c_chunk_stride;
  int mode;
  // kStoreSymmetric: C[m][n] = C[n][m] = alpha * D[m][n] for n >= m (row-major, ldc)
  // kStorePlain:     C[m][n] = alpha * D[m][n] (row-major, ldc)
  float* C;
  int64_t ldc;
  float alpha;
  int tiles_n;    // tiles along N (grid is linear; tile = bm * tiles_n + bn)
  unsigned* err;
};

__global__ void __launch_bounds__(kThreads, 1) gemm3xtf32_kernel(GemmArgs a) {
  extern __shared__ __align__(1024) char smem_raw[];
  // 1024-byte aligned base, derived from the shared array (keeps the shared address space)
  char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + kStages);

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

  if (ok) {
    const int row = warp * 32 + lane;
    const int64_t m = m0 + row;
#pragma unroll 1
    for (int c0 = 0; c0 < kBN; c0 += 32) {
      float v[32];
      tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, v);
      if (m < a.A.rows && a.mode == kStorePlain) {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int64_t n = n0 + c0 + j;
          if (n < a.B.rows) C[m * a.ldc + n] = a.alpha * v[j];
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
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
}

// Diagonal d x d blocks (d = 8) of S = A A^T for the rows of A taken in a given order (the
// Hessian blocks of the original or of the importance-sorted channel groups): one CTA per
// 128-row tile and K chunk. A block only pairs rows of the same tile, so the tile's operand is
// split once and is both MMA operands (M = N = 128, half the shared memory and staging work of
// a 128 x 256 tile). Entry (a, b) of a block is taken as the dense product's tile path takes
// it: the dense S keeps D(A row min(p, q), B row max(p, q)) for stored rows p, q (its upper
// triangle, mirrored), so here too the row with the smaller stored index is the A side. Every
// tcgen05 output element is the same function of its A row, B row and K order wherever it sits
// in a tile, so the blocks equal the dense S's entries bit for bit.
constexpr int kDiagStageBytes = 2 * kAStageBytes;                      // hi + lo, 16 KB
constexpr int kDiagSmemBytes = kStages * kDiagStageBytes + 1024 + 128;  // + alignment + barriers
constexpr int kDiagTmemCols = kBM;
constexpr uint32_t kIdescDiag = idesc_tf32(kBM, kBM);

struct DiagArgs {
  Operand A;            // rows = channels (A.idx: the order, NULL = stored order)
  int64_t K;
  int64_t k_chunk;      // blockIdx.y = chunk c covers k in [c * k_chunk, (c + 1) * k_chunk)
  float* out;           // out[c * chunk_stride + (r / 8) * 64 + (r % 8) * 8 + b]
  int64_t chunk_stride;
  float alpha;
  unsigned* err;
};

__global__ void __launch_bounds__(kThreads, 1) syrk_diag_kernel(DiagArgs a) {
  extern __shared__ __align__(1024) char smem_raw[];
  char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * kDiagStageBytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + kStages);
  __shared__ float blk[kBM][9];   // each tile row: the 8 entries of its own block row
  __shared__ int32_t src[kBM];    // stored row of each tile row (-1 past the end)

  const int64_t m0 = (int64_t)blockIdx.x * kBM;
  const int64_t kbeg = (int64_t)blockIdx.y * a.k_chunk;
  const int64_t kend = min(a.K, kbeg + a.k_chunk);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  {
    const int64_t r = m0 + threadIdx.x;
    int32_t p = -1;
    if (r < a.A.rows) {
      p = a.A.idx ? a.A.idx[r] : (int32_t)r;
      if (p < 0 || p >= a.A.rows) {
        raise_error(a.err, ERRBIT_INDEX);
        p = -1;
      }
    }
    src[threadIdx.x] = p;
  }
  if (warp == 0) tmem_alloc(tmem_slot, kDiagTmemCols);
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(smem_u32(&bars[s]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  const int64_t nkt = (kend - kbeg + kBK - 1) / kBK;
  uint32_t par = 0;
  bool ok = true;
  float va[kBM / kThreads][kBK];
  if (nkt > 0) load_tile<kBM>(a.A, m0, kbeg, kend, va);
  for (int64_t kt = 0; kt < nkt; ++kt) {
    const int s = (int)(kt & 1);
    char* a_hi = smem + s * kDiagStageBytes;
    char* a_lo = a_hi + kAStageBytes;
    if (kt >= kStages) {
      if (ok) ok = mbar_wait(smem_u32(&bars[s]), (par >> s) & 1u, a.err);
      par ^= 1u << s;
    }
    ok = __syncthreads_and(ok);
    if (!ok) break;
    split_store<kBM>(va, a_hi, a_lo);
    if (kt + 1 < nkt) load_tile<kBM>(a.A, m0, kbeg + (kt + 1) * kBK, kend, va);
    fence_async_smem();
    __syncthreads();
    if (threadIdx.x == 0) {
      tc_fence_after();
      const uint32_t sbo = (kBK / 4) * 128;
#pragma unroll
      for (int ks = 0; ks < kBK / 8; ++ks) {
        const uint32_t koff = ks * 256;
        const uint64_t dh = smem_desc(smem_u32(a_hi) + koff, 128, sbo);
        const uint64_t dl = smem_desc(smem_u32(a_lo) + koff, 128, sbo);
        // same order as the dense tile: hi.hi, hi.lo, lo.hi
        mma_tf32(tmem, dh, dh, kIdescDiag, (kt > 0 || ks > 0) ? 1u : 0u);
        mma_tf32(tmem, dh, dl, kIdescDiag, 1u);
        mma_tf32(tmem, dl, dh, kIdescDiag, 1u);
      }
      mma_commit(smem_u32(&bars[s]));
    }
  }
  if (ok && nkt > 0) {
    const int s = (int)((nkt - 1) & 1);
    ok = mbar_wait(smem_u32(&bars[s]), (par >> s) & 1u, a.err);
  }
  ok = __syncthreads_and(ok);
  tc_fence_after();

  const int row = warp * 32 + lane;
  if (ok) {
    // the warp's rows meet their block partners in columns [32 warp, 32 warp + 32)
    float v[32];
    tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(warp * 32), v);
    const int q = lane >> 3;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      float x = v[j];
#pragma unroll
      for (int qq = 1; qq < 4; ++qq)
        if (q == qq) x = v[8 * qq + j];
      blk[row][j] = x;
    }
  }
  __syncthreads();
  if (ok && m0 + row < a.A.rows && src[row] >= 0) {
    const int ra = row & 7, g0 = row & ~7;
    const int32_t pa = src[row];
    float* o = a.out + (int64_t)blockIdx.y * a.chunk_stride + (m0 + row) * 8;
    float w[8];
#pragma unroll
    for (int b = 0; b < 8; ++b) {
      const int32_t pb = src[g0 + b];
      w[b] = a.alpha * (pa <= pb ? blk[row][b] : blk[g0 + b][ra]);
    }
    *reinterpret_cast<float4*>(o) = make_float4(w[0], w[1], w[2], w[3]);
    *reinterpret_cast<float4*>(o + 4) = make_float4(w[4], w[5], w[6], w[7]);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, kDiagTmemCols);
}

}  // namespace tc
}  // namespace crvq
