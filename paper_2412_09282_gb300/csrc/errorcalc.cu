// S7: reconstruction W_enc (sum of the covering codebooks' codewords), the reverse reorder
// to the original channel order (Sec. 4.3) and the losses of Alg. 1 (QuantLoss):
//   loss_block = sum_v (t_v - r_v)^T H_g (t_v - r_v)       (block-diagonal part)
//   loss_crit  = the same over the critical groups g < G_c
//   loss_full  = ||dW X^T||^2 / n + delta ||dW||^2 = tr(dW H dW^T)
// The reconstruction is formed in the sorted channel order and gathered back to the original
// order; per-(row, group slice) sums are fp32 pairs, reduced as fp32 pairs in a fixed order
// and rounded to fp64 once. The full loss takes dW and X's columns in the sorted order (a
// permutation of the channel sum) on the tensor cores (tc_gemm.cu: tf32 operand images,
// tcgen05 3xTF32).
#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

// Unevaluated fp32 pair (h, l) += x, and the merge of two pairs (TwoSum of the high parts).
__device__ __forceinline__ void pair_add(float& h, float& l, float x) {
  const float s = __fadd_rn(h, x);
  const float bp = __fsub_rn(s, h);
  const float e = __fadd_rn(__fsub_rn(h, __fsub_rn(s, bp)), __fsub_rn(x, bp));
  h = s;
  l = __fadd_rn(l, e);
}

__device__ __forceinline__ void pair_merge(float& h, float& l, float oh, float ol) {
  pair_add(h, l, oh);
  l = __fadd_rn(l, ol);
}

constexpr int kDecRows = 16;     // rows per warp (the CTA's H blocks are staged once for all)
constexpr int kDecBatch = 2;     // rows whose codes and vectors are loaded together
constexpr int kDecWarps = 8;     // warps per CTA
constexpr int kDecHStride = 260; // floats per staged H block (256 + 4: conflict-free float4)
constexpr int kDecSmemCb = 48 * 1024;  // codebooks staged in shared memory up to this size

// Reconstruction of a vector from its codes (k[s] < 0: codebook s does not cover it), with the
// codewords read from `cw[s]` (shared memory or global): the sum in codebook order, correctly
// rounded to fp32 like the fp64 sum rounded once (two terms in fp32 give that value exactly;
// three or more are summed in fp64).
template <int MAXCB>
__device__ __forceinline__ void recon_codes(const float* const* cw, const int32_t* k, int ncb,
                                            float r[kD]) {
  int n = 0;
#pragma unroll
  for (int s = 0; s < MAXCB; ++s) n += (s < ncb && k[s] >= 0) ? 1 : 0;
  if (n <= 2) {
#pragma unroll
    for (int j = 0; j < kD; ++j) r[j] = 0.f;
#pragma unroll
    for (int s = 0; s < MAXCB; ++s) {
      if (s >= ncb || k[s] < 0) continue;
      const float4 a = *reinterpret_cast<const float4*>(cw[s] + (int64_t)k[s] * kD);
      const float4 b = *reinterpret_cast<const float4*>(cw[s] + (int64_t)k[s] * kD + 4);
      r[0] += a.x; r[1] += a.y; r[2] += a.z; r[3] += a.w;
      r[4] += b.x; r[5] += b.y; r[6] += b.z; r[7] += b.w;
    }
  } else {
    double d[kD];
#pragma unroll
    for (int j = 0; j < kD; ++j) d[j] = 0.0;
#pragma unroll
    for (int s = 0; s < MAXCB; ++s) {
      if (s >= ncb || k[s] < 0) continue;
      const float* c = cw[s] + (int64_t)k[s] * kD;
#pragma unroll
      for (int j = 0; j < kD; ++j) d[j] += (double)c[j];
    }
#pragma unroll
    for (int j = 0; j < kD; ++j) r[j] = (float)d[j];
  }
}

// One warp = kDecRows rows x one slice of 32 groups, lane = group: the reconstruction in the
// sorted order (32-byte stores, consecutive lanes on consecutive vectors) and, per (row block,
// slice), the block loss, the critical loss and ||dW||^2 as fp32 pairs in a fixed order:
// row_part[(row_block * slices + slice) * 3 + {0, 1, 2}] = (hi, lo). A lane sums its group's
// S = sum over its rows of dl dl^T (dl = w - w_hat; the 36 entries of the symmetric 8 x 8), then
// takes the loss as tr(H_g S) = sum_v dl_v^T H_g dl_v once, and ||dW||^2 as tr(S). A CTA's warps
// share one slice: its H blocks are staged in shared memory once; the codebooks sit in shared
// memory when they fit, so the codeword lookup is not a dependent global load; the codes of
// kDecBatch rows are loaded before any is used.
template <int MAXCB>
__global__ void __launch_bounds__(kDecWarps * 32)
decode_vec_kernel(const float* __restrict__ Ws, int64_t M, int64_t N,
                  const float* __restrict__ Hb, CbList cbs, int64_t n_crit_groups, int slices,
                  int cb_in_smem, float* __restrict__ W_rec, float2* __restrict__ row_part,
                  unsigned* err) {
  extern __shared__ __align__(16) float s_dyn[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float* sH = s_dyn;                         // the CTA slice's 32 H blocks
  float* s_cb = s_dyn + 32 * kDecHStride;    // codebooks (when staged)
  const float* cw[MAXCB];
  {
    int64_t off = 0;
#pragma unroll
    for (int s = 0; s < MAXCB; ++s) {
      if (s >= cbs.n) break;
      const int64_t n = (int64_t)cbs.cb[s].K * kD;
      if (cb_in_smem) {
        for (int64_t e = threadIdx.x * 4; e < n; e += blockDim.x * 4)
          *reinterpret_cast<float4*>(s_cb + off + e) =
              __ldg(reinterpret_cast<const float4*>(cbs.cb[s].C + e));
        cw[s] = s_cb + off;
        off += n;
      } else {
        cw[s] = cbs.cb[s].C;
      }
    }
    if (cb_in_smem) __syncthreads();
  }
  // CTA = (slice of 32 groups, kDecWarps x kDecRows rows); warp w takes kDecRows rows
  const int64_t G = N / kD;
  const int sl = (int)(blockIdx.x % slices);
  const int64_t rb = (int64_t)(blockIdx.x / slices) * kDecWarps + warp;
  const int64_t g = (int64_t)sl * 32 + lane;
  const bool gok = g < G;
  // stage the H blocks of the slice (256 bytes per group, 16 floats of padding between)
  for (int e = threadIdx.x; e < 32 * 2 * kD; e += blockDim.x) {
    const int gl = e / (2 * kD), q = e % (2 * kD);
    if ((int64_t)sl * 32 + gl < G)
      *reinterpret_cast<float4*>(sH + gl * kDecHStride + 4 * q) =
          __ldg(reinterpret_cast<const float4*>(Hb + ((int64_t)sl * 32 + gl) * kD * kD) + q);
  }
  __syncthreads();
  const int64_t i0 = rb * kDecRows;
  if (i0 >= M) return;  // whole warps (no block barrier follows)
  const int nr = (int)min((int64_t)kDecRows, M - i0);
  float S[kD * (kD + 1) / 2];  // sum of dl dl^T over this warp's rows, packed lower triangle
#pragma unroll
  for (int e = 0; e < kD * (kD + 1) / 2; ++e) S[e] = 0.f;
  for (int r0 = 0; r0 < nr; r0 += kDecBatch) {
    int32_t kc[kDecBatch][MAXCB];
    float4 tv[kDecBatch][2];
#pragma unroll
    for (int u = 0; u < kDecBatch; ++u) {
      const int64_t i = i0 + min(r0 + u, nr - 1);
#pragma unroll
      for (int s = 0; s < MAXCB; ++s) {
        kc[u][s] = -1;
        if (gok && s < cbs.n && g < cbs.cb[s].G_cov)
          kc[u][s] = cbs.cb[s].codes[i * cbs.cb[s].ld + g];
      }
      tv[u][0] = tv[u][1] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (gok) {
        tv[u][0] = *reinterpret_cast<const float4*>(Ws + i * N + g * kD);
        tv[u][1] = *reinterpret_cast<const float4*>(Ws + i * N + g * kD + 4);
      }
    }
#pragma unroll
    for (int u = 0; u < kDecBatch; ++u) {
      if (r0 + u >= nr || !gok) break;
      const int64_t i = i0 + r0 + u;
#pragma unroll
      for (int s = 0; s < MAXCB; ++s) {
        if (s >= cbs.n || g >= cbs.cb[s].G_cov) continue;
        if (kc[u][s] < 0 || kc[u][s] >= cbs.cb[s].K) {
          raise_error(err, ERRBIT_INDEX);
          kc[u][s] = -1;
        }
      }
      float rv[kD], dl[kD];
      recon_codes<MAXCB>(cw, kc[u], cbs.n, rv);
      const float t[kD] = {tv[u][0].x, tv[u][0].y, tv[u][0].z, tv[u][0].w,
                           tv[u][1].x, tv[u][1].y, tv[u][1].z, tv[u][1].w};
#pragma unroll
      for (int j = 0; j < kD; ++j) dl[j] = t[j] - rv[j];
      int e = 0;
#pragma unroll
      for (int a2 = 0; a2 < kD; ++a2)
#pragma unroll
        for (int b2 = 0; b2 <= a2; ++b2, ++e) S[e] = fmaf(dl[a2], dl[b2], S[e]);
      if (W_rec) {
        float* o = W_rec + i * N + g * kD;
        *reinterpret_cast<float4*>(o) = make_float4(rv[0], rv[1], rv[2], rv[3]);
        *reinterpret_cast<float4*>(o + 4) = make_float4(rv[4], rv[5], rv[6], rv[7]);
      }
    }
  }
  // lb = tr(H_g S) (H_g symmetric: diagonal once, each off-diagonal pair twice), sq = tr(S)
  float lb = 0.f, lc = 0.f, sq = 0.f;
  if (gok) {
    const float* Hl = sH + lane * kDecHStride;
    float off = 0.f;
    int e = 0;
#pragma unroll
    for (int a2 = 0; a2 < kD; ++a2)
#pragma unroll
      for (int b2 = 0; b2 <= a2; ++b2, ++e) {
        if (a2 == b2) {
          lb = fmaf(Hl[a2 * kD + b2], S[e], lb);
          sq += S[e];
        } else {
          off = fmaf(Hl[a2 * kD + b2], S[e], off);
        }
      }
    lb = fmaf(2.f, off, lb);
    if (g < n_crit_groups) lc = lb;
  }
  // the 32 groups of this (row block, slice) summed as fp32 pairs in a fixed tree
  float lbl = 0.f, lcl = 0.f, sql = 0.f;
#pragma unroll
  for (int o2 = 16; o2 > 0; o2 >>= 1) {
    const float a0 = __shfl_xor_sync(0xffffffffu, lb, o2);
    const float a1 = __shfl_xor_sync(0xffffffffu, lbl, o2);
    const float b0 = __shfl_xor_sync(0xffffffffu, lc, o2);
    const float b1 = __shfl_xor_sync(0xffffffffu, lcl, o2);
    const float c0 = __shfl_xor_sync(0xffffffffu, sq, o2);
    const float c1 = __shfl_xor_sync(0xffffffffu, sql, o2);
    pair_merge(lb, lbl, a0, a1);
    pair_merge(lc, lcl, b0, b1);
    pair_merge(sq, sql, c0, c1);
  }
  if (lane == 0) {
    float2* o = row_part + (rb * slices + sl) * 3;
    o[0] = make_float2(lb, lbl);
    o[1] = make_float2(lc, lcl);
    o[2] = make_float2(sq, sql);
  }
}

// inv[perm[p]] = p; entries outside [0, N) are reported and skipped.
__global__ void invert_perm_kernel(const int32_t* __restrict__ perm, int64_t N,
                                   int32_t* __restrict__ inv, unsigned* err) {
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < N;
       p += (int64_t)gridDim.x * blockDim.x) {
    const int32_t c = perm[p];
    if (c < 0 || c >= N) {
      raise_error(err, ERRBIT_INDEX);
      continue;
    }
    inv[c] = (int32_t)p;
  }
}

// One CTA of 1024 threads: the (row block, slice) partials summed as fp32 pairs (strided, then a
// tree; no dependent fp64 chain), the loss-product partials in fp64 (a few per thread).
__global__ void __launch_bounds__(1024)
finalize_losses_kernel(const float2* __restrict__ row_part, int64_t n_rows,
                       const double* __restrict__ gemm_part, int64_t n_gemm, int64_t n_tok,
                       double delta_host, const float* __restrict__ delta_dev,
                       double* __restrict__ losses) {
  __shared__ float red_h[3][1024], red_l[3][1024];
  __shared__ double red_e[1024];
  float h[3] = {0.f, 0.f, 0.f}, l[3] = {0.f, 0.f, 0.f};
  for (int64_t i = threadIdx.x; i < n_rows; i += blockDim.x) {
#pragma unroll
    for (int q = 0; q < 3; ++q) {
      const float2 v = row_part[i * 3 + q];
      pair_merge(h[q], l[q], v.x, v.y);
    }
  }
  double e = 0.0;
  for (int64_t i = threadIdx.x; i < n_gemm; i += blockDim.x) e += gemm_part[i];
#pragma unroll
  for (int q = 0; q < 3; ++q) {
    red_h[q][threadIdx.x] = h[q];
    red_l[q][threadIdx.x] = l[q];
  }
  red_e[threadIdx.x] = e;
  __syncthreads();
  for (int w = 512; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) {
#pragma unroll
      for (int q = 0; q < 3; ++q) {
        float hh = red_h[q][threadIdx.x], ll = red_l[q][threadIdx.x];
        pair_merge(hh, ll, red_h[q][threadIdx.x + w], red_l[q][threadIdx.x + w]);
        red_h[q][threadIdx.x] = hh;
        red_l[q][threadIdx.x] = ll;
      }
      red_e[threadIdx.x] += red_e[threadIdx.x + w];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    losses[0] = (double)red_h[0][0] + (double)red_l[0][0];
    losses[1] = (double)red_h[1][0] + (double)red_l[1][0];
    if (gemm_part) {
      const double delta = delta_dev ? (double)*delta_dev : delta_host;
      losses[2] = red_e[0] / (double)n_tok + delta * ((double)red_h[2][0] + (double)red_l[2][0]);
    } else {
      losses[2] = __longlong_as_double(0x7ff8000000000000ll);  // NaN: no X given
    }
  }
}

}  // namespace

crvq_status launch_reconstruct_error(const float* W_sorted, int64_t M, int64_t N,
                                     const float* Hb, const int32_t* perm, const CbList& cbs,
                                     int64_t n_crit_groups, const float* X, int64_t n_tok,
                                     double damp_delta, const float* delta_dev, float* W_hat,
                                     double* losses_dev, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const int nsm = sm_count();
  const int64_t G = N / kD;
  // warps: kDecRows rows x a slice of 32 groups
  const int64_t row_blocks = ceil_div(M, (int64_t)kDecRows);
  const int slices = (int)ceil_div(G, (int64_t)32);
  // partial sums of the full loss: one per 128 x 256 tile of dW X^T
  const int64_t n_gemm_cap = X ? ceil_div(M, (int64_t)128) * ceil_div(n_tok, (int64_t)256) : 0;
  int64_t n_gemm = 0;
  // Scratch: the reconstruction in the sorted order when it is not W_hat itself, the inverse
  // order, and the fp64 partial sums.
  const bool need_rec = W_hat || X;
  const bool rec_is_out = W_hat && !perm;
  const size_t rec_bytes = (need_rec && !rec_is_out) ? align_up((size_t)M * N * 4, 256) : 0;
  const size_t inv_bytes = (W_hat && perm) ? align_up((size_t)N * 4, 256) : 0;
  const size_t part_bytes = align_up((size_t)row_blocks * slices * 3 * sizeof(float2), 256) +
                            (size_t)(n_gemm_cap + 1) * sizeof(double);
  Scratch mem;
  CRVQ_TRY(mem.alloc(rec_bytes + inv_bytes + part_bytes, stream));
  float* W_rec = rec_is_out ? W_hat : (need_rec ? mem.as<float>() : nullptr);
  int32_t* inv = inv_bytes ? reinterpret_cast<int32_t*>(mem.as<char>() + rec_bytes) : nullptr;
  float2* row_part = reinterpret_cast<float2*>(mem.as<char>() + rec_bytes + inv_bytes);
  double* gemm_part = reinterpret_cast<double*>(
      reinterpret_cast<char*>(row_part) +
      align_up((size_t)row_blocks * slices * 3 * sizeof(float2), 256));
  {
    ProfScope ps("decode_rows", stream,
                 (double)M * N * 4.0 * (1.0 + (W_rec ? 1.0 : 0.0)));
    const int64_t ctas = ceil_div(row_blocks, (int64_t)kDecWarps) * slices;
    int64_t cb_bytes = 0;
    for (int s = 0; s < cbs.n; ++s) cb_bytes += (int64_t)cbs.cb[s].K * kD * sizeof(float);
    const int in_smem = cb_bytes <= kDecSmemCb ? 1 : 0;
    const size_t smem = (size_t)32 * kDecHStride * sizeof(float) +
                        (in_smem ? (size_t)cb_bytes : 0);
    const dim3 grid((unsigned)ctas);
    if (cbs.n <= 4) {
      CRVQ_TRY(smem_limit((const void*)decode_vec_kernel<4>, smem));
      decode_vec_kernel<4><<<grid, kDecWarps * 32, smem, stream>>>(
          W_sorted, M, N, Hb, cbs, n_crit_groups, slices, in_smem, W_rec, row_part, err);
    } else {
      CRVQ_TRY(smem_limit((const void*)decode_vec_kernel<kMaxCodebooks>, smem));
      decode_vec_kernel<kMaxCodebooks><<<grid, kDecWarps * 32, smem, stream>>>(
          W_sorted, M, N, Hb, cbs, n_crit_groups, slices, in_smem, W_rec, row_part, err);
    }
    CRVQ_LAUNCHED();
  }
  if (W_hat && perm) {  // back to the original channel order: W_hat[:, c] = W_rec[:, inv[c]]
    ProfScope ps("decode_unpermute", stream, (double)M * N * 8.0);
    invert_perm_kernel<<<(unsigned)std::min<int64_t>(ceil_div(N, 256), 4 * nsm), 256, 0,
                         stream>>>(perm, N, inv, err);
    CRVQ_LAUNCHED();
    CRVQ_TRY(launch_gather_cols(W_rec, M, N, inv, W_hat, stream));
  }
  if (X) {
    // ||dW X^T||^2 with dW and X's columns both in the sorted order (the same sum over the
    // channels, in another order)
    CRVQ_TRY(launch_tc_sumsq(W_sorted, W_rec, M, X, perm, n_tok, N, gemm_part, n_gemm_cap,
                             &n_gemm, stream));
  }
  finalize_losses_kernel<<<1, 1024, 0, stream>>>(row_part, row_blocks * slices,
                                                 X ? gemm_part : nullptr,
                                                 n_gemm, n_tok, damp_delta, delta_dev,
                                                 losses_dev);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

}  // namespace crvq
