// crvq_update_codebook_noalloc: the least-squares codebook update without any device memory
// allocation, for callers that cannot allocate: runtimes that hand out a fixed memory arena
// and forbid cudaMalloc after start-up, plugins whose host owns every device allocation, and
// latency-critical callers that must not synchronise (cudaFree synchronises the device). The
// update's scratch (per-group code counts, fixed-point sums, the scale) lives in a file-scope
// device array of fixed size that every GPU loading the library holds until the process
// exits; its error word is a second file-scope device variable that crvq_sync reads.
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
// covered groups.
constexpr size_t kNoAllocBytes = size_t(4) << 20;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];
// ERRBIT_* of the kernels this entry point launches: set by them, read and cleared by
// crvq_sync (zero when the module loads).
static __device__ unsigned g_noalloc_err;

struct DevAddrs {
  void* scratch = nullptr;
  unsigned* err = nullptr;
};
std::mutex g_na_mu;
std::vector<DevAddrs> g_na;  // device addresses of the two variables, per device

// Device addresses of the static scratch and error word on the current device. Their names
// in host code are only host-side stand-ins, so the addresses are looked up once per device
// (with that device current) and cached.
crvq_status noalloc_addrs(DevAddrs* out) {
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  std::lock_guard<std::mutex> lk(g_na_mu);
  if ((int)g_na.size() <= dev) g_na.resize(dev + 1);
  if (!g_na[dev].scratch) {
    DevAddrs a;
    CRVQ_CUDA(cudaGetSymbolAddress(&a.scratch, g_noalloc_scratch));
    void* e = nullptr;
    CRVQ_CUDA(cudaGetSymbolAddress(&e, g_noalloc_err));
    a.err = static_cast<unsigned*>(e);
    g_na[dev] = a;
  }
  *out = g_na[dev];
  return CRVQ_OK;
}

}  // namespace

namespace crvq {

crvq_status noalloc_take_error(unsigned* bits) {
  *bits = 0;
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  unsigned* w = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_na_mu);
    if (dev < (int)g_na.size()) w = g_na[dev].err;
  }
  if (!w) return CRVQ_OK;  // the entry point never ran on this device
  CRVQ_CUDA(cudaMemcpy(bits, w, sizeof(unsigned), cudaMemcpyDeviceToHost));
  if (*bits) CRVQ_CUDA(cudaMemset(w, 0, sizeof(unsigned)));
  return CRVQ_OK;
}

}  // namespace crvq

using namespace crvq;

extern "C" crvq_status crvq_update_codebook_noalloc(const float* T, int64_t ldT, int64_t M,
                                                    int64_t G_sub, int32_t d,
                                                    const float* H_blocks,
                                                    const crvq_codebook* cbs, int32_t n_cb,
                                                    int32_t which, float* C_out,
                                                    int32_t* counts, crvq_stream_t stream) {
  clear_last_error();
  // the same checks as crvq_update_codebook, host pointers refused before any launch
  CRVQ_TRY(check_d(d));
  CRVQ_TRY(check_set(T, ldT, M, G_sub, H_blocks));
  CRVQ_CHECK_ARG(n_cb >= 1 && which >= 0 && which < n_cb, "which must be in [0, n_cb)");
  CRVQ_CHECK_ARG(C_out != nullptr, "C_out is NULL");
  CbList cl;
  CRVQ_TRY(make_cblist(cbs, n_cb, G_sub, true, &cl));
  CRVQ_TRY(check_dev({{T, "T"}, {H_blocks, "H_blocks"}, {C_out, "C_out"}, {counts, "counts"}}));
  CRVQ_TRY(check_dev_cbs(cbs, n_cb));
  const size_t need = update_scratch_bytes(cl.cb[which].G_cov, cl.cb[which].K);
  if (need > kNoAllocBytes)
    return fail(CRVQ_ERR_UNSUPPORTED,
                "crvq_update_codebook_noalloc: G_cov * K = %lld (group, code) pairs need %zu "
                "bytes of scratch; the static limit is %zu bytes",
                (long long)(cl.cb[which].G_cov * cl.cb[which].K), need, kNoAllocBytes);
  DevAddrs a;
  CRVQ_TRY(noalloc_addrs(&a));
  SetView set{T, ldT, M, G_sub, H_blocks};
  return launch_update_codebook_on(set, cl, which, C_out, counts, a.scratch, kNoAllocBytes,
                                   a.err, (cudaStream_t)stream);
}
