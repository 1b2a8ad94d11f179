// crvq_update_codebook_noalloc: the least-squares codebook update without any device memory
// allocation, for callers that cannot allocate. Examples are code running while a CUDA graph
// is being captured into a pool they do not own, runtimes that hand out fixed memory arenas
// and forbid cudaMalloc after start-up, and callers that must not synchronise (cudaFree
// does). The update's scratch (per-group code counts, fixed-point sums, the scale) lives in
// a file-scope device array of fixed size that every GPU loading the library holds until the
// process exits.
#include <mutex>
#include <vector>

#include "common.cuh"
#include "kernels.h"

namespace crvq {
size_t update_scratch_bytes(int64_t G_cov, int K);
crvq_status launch_update_codebook_on(const SetView& set, const CbList& cbs, int which,
                                      float* C_out, int32_t* counts, void* scratch,
                                      size_t bytes, unsigned* err, cudaStream_t stream);
}  // namespace crvq

namespace {

// 4 MiB: counts for G_cov * K <= ~1M (group, code) pairs, e.g. K = 256 with up to ~4000
// covered groups. The last 256 bytes hold this entry point's own error word.
constexpr size_t kNoAllocBytes = size_t(4) << 20;
constexpr size_t kNoAllocUsable = kNoAllocBytes - 256;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

std::mutex g_na_mu;
std::vector<void*> g_na_ptr;  // device address of g_noalloc_scratch, per device

// Device address of the static scratch on the current device. The array's name in host code
// is only a host-side stand-in, so the address is looked up once per device (with that
// device current) and cached.
crvq_status noalloc_scratch(void** out) {
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  std::lock_guard<std::mutex> lk(g_na_mu);
  if ((int)g_na_ptr.size() <= dev) g_na_ptr.resize(dev + 1, nullptr);
  if (!g_na_ptr[dev]) {
    void* p = nullptr;
    CRVQ_CUDA(cudaGetSymbolAddress(&p, g_noalloc_scratch));
    g_na_ptr[dev] = p;
  }
  *out = g_na_ptr[dev];
  return CRVQ_OK;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace

using namespace crvq;

extern "C" crvq_status crvq_update_codebook_noalloc(const float* T, int64_t ldT, int64_t M,
                                                    int64_t G_sub, int32_t d,
                                                    const float* H_blocks,
                                                    const crvq_codebook* cbs, int32_t n_cb,
                                                    int32_t which, float* C_out,
                                                    int32_t* counts, crvq_stream_t stream) {
  clear_last_error();
  if (d != kD) return fail(d <= 0 ? CRVQ_ERR_INVALID_ARG : CRVQ_ERR_UNSUPPORTED,
                           "only d = 8 is implemented (got %d)", d);
  CRVQ_CHECK_ARG(T && H_blocks && C_out, "T, H_blocks and C_out must not be NULL");
  CRVQ_CHECK_ARG(M >= 1 && G_sub >= 1 && ldT >= G_sub * kD && ldT % 4 == 0,
                 "bad vector set (M, G_sub, ldT)");
  CRVQ_CHECK_ARG(aligned16(T) && aligned16(H_blocks), "T and H_blocks must be 16-byte aligned");
  CRVQ_CHECK_ARG(M * G_sub < (int64_t)1 << 31, "too many vectors in one set");
  CRVQ_CHECK_ARG(n_cb >= 1 && n_cb <= kMaxCodebooks && cbs, "n_cb must be in [1, %d]",
                 kMaxCodebooks);
  CRVQ_CHECK_ARG(which >= 0 && which < n_cb, "which must be in [0, n_cb)");
  CbList cl;
  cl.n = n_cb;
  for (int s = 0; s < n_cb; ++s) {
    const crvq_codebook& c = cbs[s];
    CRVQ_CHECK_ARG(c.C && aligned16(c.C), "codebook %d: C is NULL or not 16-byte aligned", s);
    CRVQ_CHECK_ARG(c.K >= 1 && c.K <= 65536, "codebook %d: K must be in [1, 65536]", s);
    CRVQ_CHECK_ARG(c.G_cov >= 0 && c.G_cov <= G_sub, "codebook %d: G_cov out of [0, G_sub]", s);
    CRVQ_CHECK_ARG(c.G_cov == 0 || (c.codes && c.ld >= c.G_cov),
                   "codebook %d: codes NULL or ld < G_cov", s);
    cl.cb[s] = CbView{c.C, c.codes, c.ld, c.G_cov, c.K};
  }
  const size_t need = update_scratch_bytes(cl.cb[which].G_cov, cl.cb[which].K);
  if (need > kNoAllocUsable)
    return fail(CRVQ_ERR_UNSUPPORTED,
                "crvq_update_codebook_noalloc: G_cov * K = %lld (group, code) pairs need %zu "
                "bytes of scratch; the static limit is %zu bytes",
                (long long)(cl.cb[which].G_cov * cl.cb[which].K), need, kNoAllocUsable);
  void* scratch = nullptr;
  CRVQ_TRY(noalloc_scratch(&scratch));
  unsigned* err = reinterpret_cast<unsigned*>(static_cast<char*>(scratch) + kNoAllocUsable);
  cudaStream_t s = (cudaStream_t)stream;
  CRVQ_CUDA(cudaMemsetAsync(err, 0, sizeof(unsigned), s));
  SetView set{T, ldT, M, G_sub, H_blocks};
  return launch_update_codebook_on(set, cl, which, C_out, counts, scratch, kNoAllocUsable, err,
                                   s);
}
