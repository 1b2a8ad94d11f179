// Least-squares codebook update (k-means update step; Alg. 1 FineTuneCodebook in its
// closed-form reading). For codebook `which` with all others fixed, codeword k solves
//   (sum_{v in cluster k} H_{g_v}) c_k = sum_{v in cluster k} H_{g_v} tau_v,
//   tau_v = t_v - sum over the other covering codebooks of C[code].
//
// Deterministic by construction: members are ordered by a stable LSD radix sort of the codes
// (8-bit digits, per-tile warp-match ranks, no float atomics), every cluster is reduced by
// one warp in a fixed lane/flush order (fp32 partials flushed into fp64 every 32 members),
// and the 8 x 8 normal equations are solved by an fp64 Cholesky factorisation.
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace crvq {

namespace {

constexpr int kRadixThreads = 256;
constexpr int kRadixItems = 8;
constexpr int kTileElems = kRadixThreads * kRadixItems;  // 2048
constexpr int kDigits = 256;
constexpr int kWarps = kRadixThreads / 32;

// keys[v] = code of member v (v = i * G_cov + g), vals[v] = v.
__global__ void gather_keys_kernel(const int32_t* __restrict__ codes, int64_t ld, int64_t M,
                                   int64_t G_cov, int32_t K, uint32_t* __restrict__ keys,
                                   uint32_t* __restrict__ vals, int32_t* __restrict__ counts,
                                   unsigned* err) {
  const int64_t n = M * G_cov;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < n;
       v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = v / G_cov, g = v % G_cov;
    int32_t k = codes[i * ld + g];
    if (k < 0 || k >= K) {
      raise_error(err, ERRBIT_INDEX);
      k = 0;
    }
    keys[v] = (uint32_t)k;
    vals[v] = (uint32_t)v;
    atomicAdd(&counts[k], 1);  // integer counts: order-independent
  }
}

__global__ void __launch_bounds__(kRadixThreads)
radix_hist_kernel(const uint32_t* __restrict__ keys, int64_t n, int shift,
                  uint32_t* __restrict__ tile_hist, int64_t num_tiles) {
  __shared__ uint32_t h[kDigits];
  const int64_t tile = blockIdx.x;
  h[threadIdx.x] = 0;
  __syncthreads();
  const int64_t base = tile * kTileElems;
  for (int r = 0; r < kRadixItems; ++r) {
    const int64_t e = base + (int64_t)r * kRadixThreads + threadIdx.x;
    if (e < n) atomicAdd(&h[(keys[e] >> shift) & 0xFF], 1u);
  }
  __syncthreads();
  tile_hist[(int64_t)threadIdx.x * num_tiles + tile] = h[threadIdx.x];
}

// Exclusive scan of a uint32 array in place: one CTA walks the array in coalesced blocks of
// 4096 values (warp-shuffle scans, then a scan of the warp totals) carrying the running sum.
__global__ void __launch_bounds__(1024)
exclusive_scan_kernel(uint32_t* __restrict__ a, int64_t n) {
  __shared__ uint32_t warp_sums[32];
  __shared__ uint32_t carry;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) carry = 0;
  __syncthreads();
  for (int64_t base = 0; base < n; base += 4096) {
    const int64_t e0 = base + (int64_t)tid * 4;
    uint32_t v[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) v[j] = (e0 + j < n) ? a[e0 + j] : 0u;
    const uint32_t s = v[0] + v[1] + v[2] + v[3];
    uint32_t x = s;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, x, off);
      if (lane >= off) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
      uint32_t w = warp_sums[lane];
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, w, off);
        if (lane >= off) w += y;
      }
      warp_sums[lane] = w;
    }
    __syncthreads();
    uint32_t excl = carry + (warp ? warp_sums[warp - 1] : 0u) + x - s;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (e0 + j < n) a[e0 + j] = excl;
      excl += v[j];
    }
    __syncthreads();
    if (tid == 1023) carry = excl;
    __syncthreads();
  }
}

__global__ void __launch_bounds__(kRadixThreads)
radix_scatter_kernel(const uint32_t* __restrict__ keys_in, const uint32_t* __restrict__ vals_in,
                     int64_t n, int shift, const uint32_t* __restrict__ tile_off,
                     int64_t num_tiles, uint32_t* __restrict__ keys_out,
                     uint32_t* __restrict__ vals_out) {
  __shared__ uint32_t cnt[kWarps][kDigits];
  __shared__ uint32_t run[kDigits];
  const int64_t tile = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  run[threadIdx.x] = tile_off[(int64_t)threadIdx.x * num_tiles + tile];
  const int64_t base = tile * kTileElems;
  const unsigned lt_mask = (1u << lane) - 1u;
  for (int r = 0; r < kRadixItems; ++r) {
#pragma unroll
    for (int w = 0; w < kWarps; ++w) cnt[w][threadIdx.x] = 0;
    __syncthreads();
    const int64_t e = base + (int64_t)r * kRadixThreads + threadIdx.x;
    const bool act = e < n;
    const unsigned amask = __ballot_sync(0xffffffffu, act);
    uint32_t key = 0, val = 0, dig = 0, rank = 0;
    if (act) {
      key = keys_in[e];
      val = vals_in[e];
      dig = (key >> shift) & 0xFF;
      const unsigned peers = __match_any_sync(amask, dig);
      rank = __popc(peers & lt_mask);
      if ((peers & lt_mask) == 0) cnt[warp][dig] = __popc(peers);
    }
    __syncthreads();
    {  // exclusive prefix over warps for digit = threadIdx.x, continuing the running offset
      uint32_t p = run[threadIdx.x];
#pragma unroll
      for (int w = 0; w < kWarps; ++w) {
        const uint32_t t = cnt[w][threadIdx.x];
        cnt[w][threadIdx.x] = p;
        p += t;
      }
      run[threadIdx.x] = p;
    }
    __syncthreads();
    if (act) {
      const uint32_t pos = cnt[warp][dig] + rank;
      keys_out[pos] = key;
      vals_out[pos] = val;
    }
    __syncthreads();
  }
}

// One warp per codeword: ordered reduction of its members, then the fp64 Cholesky solve.
__global__ void __launch_bounds__(128)
cluster_solve_kernel(SetView set, CbList cbs, int which, const uint32_t* __restrict__ members,
                     const uint32_t* __restrict__ seg_start, const int32_t* __restrict__ counts,
                     float* __restrict__ C_out, unsigned* err) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const CbView cw = cbs.cb[which];
  const int64_t G_cov = cw.G_cov;
  for (int64_t k = warp; k < cw.K; k += nwarps) {
    const int64_t beg = seg_start[k];
    const int64_t cnt = counts[k];
    if (cnt == 0) {
      if (lane < kD) C_out[k * kD + lane] = cw.C[k * kD + lane];
      continue;
    }
    double A[36], b[kD];
    float Af[36], bf[kD];
#pragma unroll
    for (int j = 0; j < 36; ++j) { A[j] = 0.0; Af[j] = 0.f; }
#pragma unroll
    for (int j = 0; j < kD; ++j) { b[j] = 0.0; bf[j] = 0.f; }
    int since = 0;
    for (int64_t p = beg + lane; p < beg + cnt; p += 32) {
      const int64_t v = members[p];
      const int64_t i = v / G_cov, g = v % G_cov;
      const float* H = set.Hb + g * kD * kD;
      float tau[kD];
      const float* t = set.T + i * set.ldT + g * kD;
      const float4 t0 = *reinterpret_cast<const float4*>(t);
      const float4 t1 = *reinterpret_cast<const float4*>(t + 4);
      tau[0] = t0.x; tau[1] = t0.y; tau[2] = t0.z; tau[3] = t0.w;
      tau[4] = t1.x; tau[5] = t1.y; tau[6] = t1.z; tau[7] = t1.w;
      for (int s = 0; s < cbs.n; ++s) {
        if (s == which) continue;
        const CbView& cb = cbs.cb[s];
        if (g >= cb.G_cov) continue;
        const int32_t kk = cb.codes[i * cb.ld + g];
        if (kk < 0 || kk >= cb.K) {
          raise_error(err, ERRBIT_INDEX);
          continue;
        }
        const float* c = cb.C + (int64_t)kk * kD;
#pragma unroll
        for (int j = 0; j < kD; ++j) tau[j] -= c[j];
      }
      float h[kD * kD];
#pragma unroll
      for (int j = 0; j < kD * kD; ++j) h[j] = H[j];
      int q = 0;
#pragma unroll
      for (int r = 0; r < kD; ++r) {
        float acc = 0.f;
#pragma unroll
        for (int c = 0; c < kD; ++c) acc = fmaf(h[r * kD + c], tau[c], acc);
        bf[r] += acc;
#pragma unroll
        for (int c = 0; c <= r; ++c) Af[q++] += h[r * kD + c];
      }
      if (++since == 32) {
        since = 0;
#pragma unroll
        for (int j = 0; j < 36; ++j) { A[j] += (double)Af[j]; Af[j] = 0.f; }
#pragma unroll
        for (int j = 0; j < kD; ++j) { b[j] += (double)bf[j]; bf[j] = 0.f; }
      }
    }
#pragma unroll
    for (int j = 0; j < 36; ++j) A[j] += (double)Af[j];
#pragma unroll
    for (int j = 0; j < kD; ++j) b[j] += (double)bf[j];
    // Fixed butterfly reduction across the warp.
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
      for (int j = 0; j < 36; ++j) A[j] += __shfl_xor_sync(0xffffffffu, A[j], off);
#pragma unroll
      for (int j = 0; j < kD; ++j) b[j] += __shfl_xor_sync(0xffffffffu, b[j], off);
    }
    if (lane == 0) {
      // Cholesky A = L L^T (packed lower triangle, row-major), then two triangular solves.
      double L[36];
      bool spd = true;
      int q = 0;
      for (int r = 0; r < kD; ++r) {
        for (int c = 0; c <= r; ++c, ++q) {
          double s = A[q];
          for (int m = 0; m < c; ++m) s -= L[r * (r + 1) / 2 + m] * L[c * (c + 1) / 2 + m];
          if (r == c) {
            if (!(s > 0.0)) { spd = false; s = 1.0; }
            L[q] = sqrt(s);
          } else {
            L[q] = s / L[c * (c + 1) / 2 + c];
          }
        }
      }
      if (!spd) {
        raise_error(err, ERRBIT_NUMERIC);
        for (int j = 0; j < kD; ++j) C_out[k * kD + j] = cw.C[k * kD + j];
      } else {
        double y[kD], x[kD];
        for (int r = 0; r < kD; ++r) {
          double s = b[r];
          for (int m = 0; m < r; ++m) s -= L[r * (r + 1) / 2 + m] * y[m];
          y[r] = s / L[r * (r + 1) / 2 + r];
        }
        for (int r = kD - 1; r >= 0; --r) {
          double s = y[r];
          for (int m = r + 1; m < kD; ++m) s -= L[m * (m + 1) / 2 + r] * x[m];
          x[r] = s / L[r * (r + 1) / 2 + r];
        }
        for (int j = 0; j < kD; ++j) C_out[k * kD + j] = (float)x[j];
      }
    }
  }
}

}  // namespace

crvq_status launch_update_codebook(const SetView& set, const CbList& cbs, int which,
                                   float* C_out, int32_t* counts_out, cudaStream_t stream) {
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  const CbView& cw = cbs.cb[which];
  const int64_t n = set.M * cw.G_cov;
  const int K = cw.K;
  const int nsm = sm_count();
  const int64_t num_tiles = std::max<int64_t>(1, ceil_div(n, kTileElems));
  const int passes = K > 256 ? 2 : 1;
  // scratch: keys/vals x2, tile histogram, counts, segment starts
  Scratch mem;
  const size_t nn = (size_t)std::max<int64_t>(n, 1);
  const size_t bytes = 4 * nn * sizeof(uint32_t) + (size_t)kDigits * num_tiles * sizeof(uint32_t) +
                       2 * (size_t)K * sizeof(uint32_t) + 256;
  CRVQ_TRY(mem.alloc(bytes, stream));
  uint32_t* keysA = mem.as<uint32_t>();
  uint32_t* valsA = keysA + nn;
  uint32_t* keysB = valsA + nn;
  uint32_t* valsB = keysB + nn;
  uint32_t* tile_hist = valsB + nn;
  int32_t* counts = reinterpret_cast<int32_t*>(tile_hist + (size_t)kDigits * num_tiles);
  uint32_t* seg = reinterpret_cast<uint32_t*>(counts + K);

  CRVQ_CUDA(cudaMemsetAsync(counts, 0, (size_t)K * sizeof(int32_t), stream));
  if (n > 0) {
    ProfScope ps("update_sort", stream, (double)n);
    gather_keys_kernel<<<(unsigned)std::min<int64_t>(ceil_div(n, 256), 16 * nsm), 256, 0,
                         stream>>>(cw.codes, cw.ld, set.M, cw.G_cov, K, keysA, valsA, counts,
                                   err);
    CRVQ_LAUNCHED();
    uint32_t *kin = keysA, *vin = valsA, *kout = keysB, *vout = valsB;
    for (int pass = 0; pass < passes; ++pass) {
      const int shift = 8 * pass;
      radix_hist_kernel<<<(unsigned)num_tiles, kRadixThreads, 0, stream>>>(kin, n, shift,
                                                                          tile_hist, num_tiles);
      CRVQ_LAUNCHED();
      exclusive_scan_kernel<<<1, 1024, 0, stream>>>(tile_hist, (int64_t)kDigits * num_tiles);
      CRVQ_LAUNCHED();
      radix_scatter_kernel<<<(unsigned)num_tiles, kRadixThreads, 0, stream>>>(
          kin, vin, n, shift, tile_hist, num_tiles, kout, vout);
      CRVQ_LAUNCHED();
      std::swap(kin, kout);
      std::swap(vin, vout);
    }
    // sorted member list is now in (kin, vin)
    CRVQ_CUDA(cudaMemcpyAsync(seg, counts, (size_t)K * sizeof(int32_t), cudaMemcpyDeviceToDevice,
                              stream));
    exclusive_scan_kernel<<<1, 1024, 0, stream>>>(seg, K);
    CRVQ_LAUNCHED();
    ProfScope ps2("update_solve", stream, (double)n);
    cluster_solve_kernel<<<(unsigned)std::min<int64_t>(ceil_div((int64_t)K * 32, 128), 64 * nsm),
                           128, 0, stream>>>(set, cbs, which, vin, seg, counts, C_out, err);
    CRVQ_LAUNCHED();
  } else {
    CRVQ_CUDA(cudaMemcpyAsync(C_out, cw.C, (size_t)K * kD * sizeof(float),
                              cudaMemcpyDeviceToDevice, stream));
  }
  if (counts_out)
    CRVQ_CUDA(cudaMemcpyAsync(counts_out, counts, (size_t)K * sizeof(int32_t),
                              cudaMemcpyDeviceToDevice, stream));
  return CRVQ_OK;
}

}  // namespace crvq
