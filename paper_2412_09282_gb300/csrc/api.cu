// C ABI of libcrvq: argument validation, status / error-word handling and the per-matrix
// schedule (Alg. 1, prequantization through the refinement loop) that strings the kernels
// together on one stream.
#include <atomic>
#include <cmath>
#include <cstring>
#include <initializer_list>
#include <mutex>
#include <type_traits>
#include <string>
#include <utility>
#include <vector>

#include "common.cuh"
#include "kernels.h"
#include "stats.cuh"
#include "tc_ops.cuh"

namespace crvq {

// ------------------------------------------------------------------------- status helpers
static thread_local std::string t_last_error;

void set_last_error(const char* fmt, ...) {
  char buf[1024];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  t_last_error = buf;
}

crvq_status fail(crvq_status st, const char* fmt, ...) {
  char buf[1024];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  t_last_error = buf;
  return st;
}

void clear_last_error() { t_last_error.clear(); }

namespace {
std::mutex g_mu;
std::vector<unsigned*> g_err_words;  // per device
std::vector<int> g_sm;               // per device
}  // namespace

crvq_status device_error_word(unsigned** out) {
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  std::lock_guard<std::mutex> lk(g_mu);
  if ((int)g_err_words.size() <= dev) g_err_words.resize(dev + 1, nullptr);
  if (!g_err_words[dev]) {
    unsigned* p = nullptr;
    CRVQ_CUDA(cudaMalloc(&p, sizeof(unsigned)));
    CRVQ_CUDA(cudaMemset(p, 0, sizeof(unsigned)));
    g_err_words[dev] = p;
  }
  *out = g_err_words[dev];
  return CRVQ_OK;
}

int sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  std::lock_guard<std::mutex> lk(g_mu);
  if ((int)g_sm.size() <= dev) g_sm.resize(dev + 1, 0);
  if (!g_sm[dev]) {
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    g_sm[dev] = n > 0 ? n : 1;
  }
  return g_sm[dev];
}

namespace {
struct SmemLimit {
  const void* kernel;
  int dev;
  size_t bytes;
};
std::vector<SmemLimit> g_smem_limits;
}  // namespace

crvq_status smem_limit(const void* kernel, size_t bytes) {
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  std::lock_guard<std::mutex> lk(g_mu);
  for (auto& e : g_smem_limits)
    if (e.kernel == kernel && e.dev == dev) {
      if (e.bytes >= bytes) return CRVQ_OK;
      CRVQ_CUDA(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)bytes));
      e.bytes = bytes;
      return CRVQ_OK;
    }
  CRVQ_CUDA(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)bytes));
  g_smem_limits.push_back(SmemLimit{kernel, dev, bytes});
  return CRVQ_OK;
}

// ------------------------------------------------------------------------- launch stats
namespace {
std::atomic<long long> g_launches{0};
std::atomic<bool> g_prof{false};
std::mutex g_pmu;
char g_filter[64] = {0};  // profiled name prefix ("" = all); changed only between sessions
struct ProfRec {
  const char* name;
  cudaEvent_t a, b;
  double units;
};
std::vector<ProfRec> g_recs;
struct ProfDone {  // a launch timed inside a replayed layer graph
  const char* name;
  float ms;
  double units;
};
std::vector<ProfDone> g_graph_recs;
std::vector<cudaEvent_t> g_pool;  // events reused across profiling sessions

cudaEvent_t pool_get() {
  std::lock_guard<std::mutex> lk(g_pmu);
  if (!g_pool.empty()) {
    cudaEvent_t e = g_pool.back();
    g_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return e;
}
}  // namespace

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

// Layer graph being captured on this thread (ProfScope then records external event nodes
// owned by it instead of pooled events).
struct CapturedEvents {
  std::vector<ProfRec> recs;
};
thread_local CapturedEvents* t_capture = nullptr;

ProfScope::ProfScope(const char* name, cudaStream_t s, double units)
    : name_(name), s_(s), units_(units) {
  if (g_prof.load(std::memory_order_relaxed) &&
      strncmp(name, g_filter, strlen(g_filter)) == 0) {
    if (t_capture) {  // an event node of the graph, recorded on every replay
      if (cudaEventCreate(&a_) != cudaSuccess ||
          cudaEventRecordWithFlags(a_, s_, cudaEventRecordExternal) != cudaSuccess) {
        cudaGetLastError();
        a_ = nullptr;
      }
      return;
    }
    a_ = pool_get();
    if (a_ && cudaEventRecord(a_, s_) != cudaSuccess) {
      cudaGetLastError();
      a_ = nullptr;
    }
  }
}

ProfScope::~ProfScope() {
  if (!a_) return;
  if (t_capture) {
    cudaEvent_t b = nullptr;
    if (cudaEventCreate(&b) != cudaSuccess ||
        cudaEventRecordWithFlags(b, s_, cudaEventRecordExternal) != cudaSuccess) {
      cudaGetLastError();
      return;
    }
    t_capture->recs.push_back(ProfRec{name_, a_, b, units_});
    return;
  }
  cudaEvent_t b = pool_get();
  if (!b || cudaEventRecord(b, s_) != cudaSuccess) {
    cudaGetLastError();
    return;
  }
  std::lock_guard<std::mutex> lk(g_pmu);
  g_recs.push_back(ProfRec{name_, a_, b, units_});
}

// ------------------------------------------------------------------------- validation
static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

crvq_status check_d(int32_t d) {
  if (d <= 0) return fail(CRVQ_ERR_INVALID_ARG, "d must be positive (got %d)", d);
  if (d != kD) return fail(CRVQ_ERR_UNSUPPORTED, "only d = 8 is implemented (got %d)", d);
  return CRVQ_OK;
}

crvq_status check_set(const float* T, int64_t ldT, int64_t M, int64_t G_sub,
                      const float* Hb) {
  CRVQ_CHECK_ARG(T != nullptr, "T is NULL");
  CRVQ_CHECK_ARG(Hb != nullptr, "H_blocks is NULL");
  CRVQ_CHECK_ARG(M >= 1 && G_sub >= 1, "empty vector set (M=%lld, G_sub=%lld)", (long long)M,
                 (long long)G_sub);
  CRVQ_CHECK_ARG(ldT >= G_sub * kD, "ldT (%lld) < G_sub * d (%lld)", (long long)ldT,
                 (long long)(G_sub * kD));
  CRVQ_CHECK_ARG(ldT % 4 == 0, "ldT must be a multiple of 4 floats");
  CRVQ_CHECK_ARG(aligned16(T) && aligned16(Hb), "T and H_blocks must be 16-byte aligned");
  CRVQ_CHECK_ARG(M * G_sub < (int64_t)1 << 31, "too many vectors in one set");
  return CRVQ_OK;
}

crvq_status make_cblist(const crvq_codebook* cbs, int32_t n_cb, int64_t G_sub,
                        bool need_codes_all, CbList* out) {
  CRVQ_CHECK_ARG(n_cb >= 0 && n_cb <= kMaxCodebooks, "n_cb must be in [0, %d]", kMaxCodebooks);
  CRVQ_CHECK_ARG(n_cb == 0 || cbs != nullptr, "codebook array is NULL");
  out->n = n_cb;
  for (int s = 0; s < n_cb; ++s) {
    const crvq_codebook& c = cbs[s];
    CRVQ_CHECK_ARG(c.C != nullptr && aligned16(c.C), "codebook %d: C is NULL or not 16-byte aligned", s);
    CRVQ_CHECK_ARG(c.K >= 1 && c.K <= 65536, "codebook %d: K must be in [1, 65536]", s);
    CRVQ_CHECK_ARG(c.G_cov >= 0 && c.G_cov <= G_sub, "codebook %d: G_cov out of [0, G_sub]", s);
    CRVQ_CHECK_ARG(c.G_cov == 0 || c.ld >= c.G_cov, "codebook %d: ld < G_cov", s);
    if (need_codes_all && c.G_cov > 0)
      CRVQ_CHECK_ARG(c.codes != nullptr, "codebook %d: codes is NULL", s);
    out->cb[s] = CbView{c.C, c.codes, c.ld, c.G_cov, c.K};
  }
  return CRVQ_OK;
}

static bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

// The kernels dereference these pointers: each non-null one must be device (or managed)
// memory. A host pointer is refused here instead of reaching a kernel.
crvq_status check_dev(std::initializer_list<std::pair<const void*, const char*>> ps) {
  for (const auto& p : ps)
    if (p.first && !is_device_ptr(p.first))
      return fail(CRVQ_ERR_INVALID_ARG, "%s is not device memory", p.second);
  return CRVQ_OK;
}

crvq_status check_dev_cbs(const crvq_codebook* cbs, int32_t n) {
  for (int32_t s = 0; s < n; ++s) {
    if (!is_device_ptr(cbs[s].C))
      return fail(CRVQ_ERR_INVALID_ARG, "codebook %d: C is not device memory", s);
    if (cbs[s].codes && !is_device_ptr(cbs[s].codes))
      return fail(CRVQ_ERR_INVALID_ARG, "codebook %d: codes is not device memory", s);
  }
  return CRVQ_OK;
}

namespace {

// One thread waits on an mbarrier nothing arrives on (crvq_selftest_bounded_wait).
__global__ void selftest_wait_kernel(unsigned* err) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    tc::mbar_init(tc::smem_u32(&bar), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    tc::mbar_wait(tc::smem_u32(&bar), 0u, err);  // gives up after the bound: ERRBIT_TIMEOUT
  }
}

}  // namespace

}  // namespace crvq

using namespace crvq;

#define CRVQ_STR_(x) #x
#define CRVQ_XSTR(x) CRVQ_STR_(x)

// =========================================================================== C entry points
extern "C" {

const char* crvq_last_error(void) { return t_last_error.c_str(); }

const char* crvq_version(void) {
  return "libcrvq (sm_103a, CUDA " CRVQ_XSTR(__CUDACC_VER_MAJOR__) "." CRVQ_XSTR(__CUDACC_VER_MINOR__) ")";
}

int64_t crvq_launch_count(void) { return (int64_t)g_launches.load(); }

crvq_status crvq_profile_begin(void) {
  {
    std::lock_guard<std::mutex> lk(g_pmu);
    for (auto& r : g_recs) {
      g_pool.push_back(r.a);
      g_pool.push_back(r.b);
    }
    g_recs.clear();
    g_graph_recs.clear();
  }
  // pre-create events so that recording inside the profiled region does not create any
  std::vector<cudaEvent_t> fresh;
  for (int i = 0; i < 1024; ++i) fresh.push_back(pool_get());
  {
    std::lock_guard<std::mutex> lk(g_pmu);
    for (auto e : fresh)
      if (e) g_pool.push_back(e);
  }
  g_prof.store(true);
  return CRVQ_OK;
}

crvq_status crvq_profile_filter(const char* prefix) {
  if (g_prof.load()) return fail(CRVQ_ERR_INVALID_ARG, "crvq_profile_filter: a session is running");
  const size_t n = prefix ? strlen(prefix) : 0;
  if (n >= sizeof(g_filter))
    return fail(CRVQ_ERR_INVALID_ARG, "crvq_profile_filter: prefix longer than %zu characters",
                sizeof(g_filter) - 1);
  std::lock_guard<std::mutex> lk(g_pmu);
  memset(g_filter, 0, sizeof(g_filter));
  if (n) memcpy(g_filter, prefix, n);
  return CRVQ_OK;
}

crvq_status crvq_profile_end(crvq_kernel_stat* stats, int32_t cap, int32_t* n_stats) {
  g_prof.store(false);
  std::vector<ProfRec> recs;
  std::vector<ProfDone> done;
  {
    std::lock_guard<std::mutex> lk(g_pmu);
    recs.swap(g_recs);
    done.swap(g_graph_recs);
  }
  std::vector<crvq_kernel_stat> agg;
  crvq_status st = CRVQ_OK;
  auto add = [&](const char* name, double ms, double units) {
    size_t j = 0;
    for (; j < agg.size(); ++j)
      if (strncmp(agg[j].name, name, sizeof(agg[j].name)) == 0) break;
    if (j == agg.size()) {
      crvq_kernel_stat z;
      memset(&z, 0, sizeof(z));
      strncpy(z.name, name, sizeof(z.name) - 1);
      agg.push_back(z);
    }
    agg[j].launches += 1;
    agg[j].ms += ms;
    agg[j].units += units;
  };
  for (auto& r : done) add(r.name, r.ms, r.units);
  for (auto& r : recs) {
    float ms = 0.f;
    if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) {
      st = fail(CRVQ_ERR_CUDA, "profiling event failed: %s", cudaGetErrorString(cudaGetLastError()));
    }
    {
      std::lock_guard<std::mutex> lk(g_pmu);
      g_pool.push_back(r.a);
      g_pool.push_back(r.b);
    }
    add(r.name, ms, r.units);
  }
  const int n = (int)std::min<size_t>(agg.size(), cap > 0 ? (size_t)cap : 0);
  for (int i = 0; i < n; ++i) stats[i] = agg[i];
  if (n_stats) *n_stats = n;
  return st;
}

crvq_status crvq_selftest_bounded_wait(crvq_stream_t stream) {
  clear_last_error();
  unsigned* err = nullptr;
  CRVQ_TRY(device_error_word(&err));
  selftest_wait_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(err);
  CRVQ_LAUNCHED();
  return CRVQ_OK;
}

crvq_status crvq_sync(crvq_stream_t stream) {
  CRVQ_CUDA(cudaStreamSynchronize((cudaStream_t)stream));
  unsigned* w = nullptr;
  CRVQ_TRY(device_error_word(&w));
  unsigned h = 0;
  CRVQ_CUDA(cudaMemcpy(&h, w, sizeof(unsigned), cudaMemcpyDeviceToHost));
  unsigned h_na = 0;  // the no-allocation update's own word (read and cleared here too)
  CRVQ_TRY(noalloc_take_error(&h_na));
  if (h) CRVQ_CUDA(cudaMemset(w, 0, sizeof(unsigned)));
  h |= h_na;
  if (h) {
    if (h & ERRBIT_TIMEOUT) return fail(CRVQ_ERR_TIMEOUT, "a bounded device wait ran out");
    if (h & ERRBIT_INDEX) return fail(CRVQ_ERR_DEVICE, "a device-side index check failed");
    return fail(CRVQ_ERR_NUMERIC, "non-finite value or non-SPD normal matrix on the device");
  }
  return CRVQ_OK;
}

crvq_status crvq_hessian(const float* X, int64_t n_tok, int64_t N, int32_t d, float damp_rel,
                         float* H, float* xsq, float* H_blocks, float* delta,
                         crvq_stream_t stream) {
  clear_last_error();
  CRVQ_TRY(check_d(d));
  CRVQ_CHECK_ARG(X && H && xsq, "X, H and xsq must not be NULL");
  CRVQ_CHECK_ARG(n_tok >= 1 && N >= 1 && N % d == 0, "need n_tok >= 1, N >= 1, N %% d == 0");
  CRVQ_CHECK_ARG(std::isfinite(damp_rel) && damp_rel >= 0.f, "damp_rel must be finite, >= 0");
  CRVQ_CHECK_ARG(aligned16(X), "X must be 16-byte aligned");
  CRVQ_TRY(check_dev({{X, "X"}, {H, "H"}, {xsq, "xsq"}, {H_blocks, "H_blocks"},
                      {delta, "delta"}}));
  return launch_hessian(X, n_tok, N, d, damp_rel, H, xsq, H_blocks, delta,
                        (cudaStream_t)stream);
}

crvq_status crvq_hessian_blocks(const float* X, int64_t n_tok, int64_t N, int32_t d,
                                float damp_rel, const int32_t* perm, float* xsq, float* delta,
                                float* H_blocks, crvq_stream_t stream) {
  clear_last_error();
  CRVQ_TRY(check_d(d));
  CRVQ_CHECK_ARG(X && H_blocks, "X and H_blocks must not be NULL");
  CRVQ_CHECK_ARG(n_tok >= 1 && N >= 1 && N % d == 0, "need n_tok >= 1, N >= 1, N %% d == 0");
  CRVQ_CHECK_ARG(N <= INT32_MAX, "N must fit in int32");
  CRVQ_CHECK_ARG(std::isfinite(damp_rel) && damp_rel >= 0.f, "damp_rel must be finite, >= 0");
  CRVQ_CHECK_ARG(aligned16(X), "X must be 16-byte aligned");
  CRVQ_TRY(check_dev({{X, "X"}, {perm, "perm"}, {xsq, "xsq"}, {delta, "delta"},
                      {H_blocks, "H_blocks"}}));
  cudaStream_t s = (cudaStream_t)stream;
  const int64_t ldt = (n_tok + 3) / 4 * 4;
  Scratch mXt, md64, mxsq, mHb;
  CRVQ_TRY(mXt.alloc((size_t)N * ldt * sizeof(float), s));
  CRVQ_TRY(md64.alloc(sizeof(double), s));
  float* Xt = mXt.as<float>();
  double* delta64 = md64.as<double>();
  if (!xsq) {
    CRVQ_TRY(mxsq.alloc((size_t)N * sizeof(float), s));
    xsq = mxsq.as<float>();
  }
  float* Hb0 = H_blocks;
  if (perm) {
    CRVQ_TRY(mHb.alloc((size_t)N * d * sizeof(float), s));
    Hb0 = mHb.as<float>();
  }
  CRVQ_TRY(launch_transpose(X, n_tok, N, Xt, ldt, s));
  CRVQ_TRY(launch_tc_hessian_blocks(Xt, ldt, n_tok, N, nullptr, false, damp_rel, xsq, delta,
                                    delta64, Hb0, s));
  if (perm)
    CRVQ_TRY(launch_tc_hessian_blocks(Xt, ldt, n_tok, N, perm, true, 0.f, nullptr, nullptr,
                                      delta64, H_blocks, s));
  return CRVQ_OK;
}

crvq_status crvq_hessian_inverse_diag(const float* H, int64_t N, double* hinv,
                                      crvq_stream_t stream) {
  clear_last_error();
  CRVQ_CHECK_ARG(H && hinv, "H and hinv must not be NULL");
  CRVQ_CHECK_ARG(N >= 1 && N <= 49152, "N must be in [1, 49152]");
  CRVQ_TRY(check_dev({{H, "H"}, {hinv, "hinv"}}));
  return launch_hinv_diag(H, N, hinv, (cudaStream_t)stream);
}

int64_t crvq_n_crit_groups(int64_t N, int32_t d, float crit_frac) {
  if (d <= 0 || N <= 0 || !(crit_frac > 0.f)) return 0;
  const int64_t G = N / d;
  const double x = std::ceil((double)crit_frac * (double)N / (double)d - 1e-12);
  return std::min<int64_t>(G, (int64_t)x);
}

crvq_status crvq_select_reorder_channels(const float* W, int64_t M, int64_t N, int32_t d,
                                         const float* W_pre, const float* xsq, const float* H,
                                         float crit_frac, int32_t mode, uint64_t seed,
                                         int32_t* perm, float* importance, float* W_sorted,
                                         float* H_blocks, int64_t* n_crit_groups,
                                         crvq_stream_t stream) {
  clear_last_error();
  CRVQ_TRY(check_d(d));
  CRVQ_CHECK_ARG(W && H && perm && W_sorted && H_blocks, "required pointer is NULL");
  CRVQ_CHECK_ARG(M >= 1 && N >= 1 && N % d == 0, "need M >= 1, N >= 1, N %% d == 0");
  CRVQ_CHECK_ARG(N <= 49152, "N must be <= 49152");
  CRVQ_CHECK_ARG(crit_frac >= 0.f && crit_frac <= 1.f, "crit_frac must be in [0, 1]");
  CRVQ_CHECK_ARG(mode >= 0 && mode <= 3, "unknown importance mode %d", mode);
  if (mode == CRVQ_IMPORTANCE_WA) CRVQ_CHECK_ARG(W_pre && xsq, "W-A mode needs W_pre and xsq");
  if (mode == CRVQ_IMPORTANCE_WA_INV) CRVQ_CHECK_ARG(W_pre, "W-A inverse mode needs W_pre");
  CRVQ_CHECK_ARG(aligned16(W) && aligned16(W_sorted) && (!W_pre || aligned16(W_pre)),
                 "W, W_pre and W_sorted must be 16-byte aligned");
  CRVQ_TRY(check_dev({{W, "W"}, {W_pre, "W_pre"}, {xsq, "xsq"}, {H, "H"}, {perm, "perm"},
                      {importance, "importance"}, {W_sorted, "W_sorted"},
                      {H_blocks, "H_blocks"}}));
  if (n_crit_groups) *n_crit_groups = crvq_n_crit_groups(N, d, crit_frac);
  return launch_select_reorder(W, M, N, d, W_pre, xsq, H, mode, seed, perm, importance,
                               W_sorted, H_blocks, (cudaStream_t)stream);
}

crvq_status crvq_kmeans_init(const float* T, int64_t ldT, int64_t M, int64_t G_sub, int32_t d,
                             const crvq_codebook* fixed, int32_t n_fixed, int32_t K,
                             uint64_t seed, float* C_out, crvq_stream_t stream) {
  clear_last_error();
  CRVQ_TRY(check_d(d));
  CRVQ_CHECK_ARG(T && C_out, "T and C_out must not be NULL");
  CRVQ_CHECK_ARG(M >= 1 && G_sub >= 1 && ldT >= G_sub * d && ldT % 4 == 0 && aligned16(T),
                 "bad vector set");
  CRVQ_CHECK_ARG(K >= 1 && K <= 65536 && (int64_t)K <= M * G_sub,
                 "K must be in [1, min(65536, M * G_sub)]");
  CbList fl;
  CRVQ_TRY(make_cblist(fixed, n_fixed, G_sub, true, &fl));
  CRVQ_TRY(check_dev({{T, "T"}, {C_out, "C_out"}}));
  CRVQ_TRY(check_dev_cbs(fixed, n_fixed));
  SetView set{T, ldT, M, G_sub, nullptr};
  return launch_kmeans_init(set, fl, K, seed, C_out, (cudaStream_t)stream);
}

crvq_status crvq_encode_beam(const float* T, int64_t ldT, int64_t M, int64_t G_sub, int32_t d,
                             const float* H_blocks, const crvq_codebook* cbs, int32_t n_cb,
                             int32_t n_fixed, int32_t B, int32_t keep_if_better,
                             float* vec_err, crvq_stream_t stream) {
  clear_last_error();
  CRVQ_TRY(check_d(d));
  CRVQ_TRY(check_set(T, ldT, M, G_sub, H_blocks));
  if (G_sub > 65535)  // beam stages launch one grid row (gridDim.y) per group
    return fail(CRVQ_ERR_UNSUPPORTED, "vector sets of more than 65535 groups are not implemented "
                "(got %lld)", (long long)G_sub);
  CRVQ_CHECK_ARG(n_cb >= 1 && n_cb <= kMaxCodebooks, "n_cb must be in [1, %d]", kMaxCodebooks);
  CRVQ_CHECK_ARG(n_fixed >= 0 && n_fixed < n_cb, "n_fixed must be in [0, n_cb)");
  CRVQ_CHECK_ARG(B >= 1, "B must be >= 1");
  if (B > 16) return fail(CRVQ_ERR_UNSUPPORTED, "beam width B > 16 is not implemented");
  CbList cl;
  CRVQ_TRY(make_cblist(cbs, n_cb, G_sub, true, &cl));
  CRVQ_TRY(check_dev({{T, "T"}, {H_blocks, "H_blocks"}, {vec_err, "vec_err"}}));
  CRVQ_TRY(check_dev_cbs(cbs, n_cb));
  SetView set{T, ldT, M, G_sub, H_blocks};
  return launch_encode_beam(set, cl, n_fixed, B, keep_if_better != 0, vec_err, EncodeExtras{},
                            (cudaStream_t)stream);
}

crvq_status crvq_update_codebook(const float* T, int64_t ldT, int64_t M, int64_t G_sub,
                                 int32_t d, const float* H_blocks, const crvq_codebook* cbs,
                                 int32_t n_cb, int32_t which, float* C_out, int32_t* counts,
                                 crvq_stream_t stream) {
  clear_last_error();
  CRVQ_TRY(check_d(d));
  CRVQ_TRY(check_set(T, ldT, M, G_sub, H_blocks));
  CRVQ_CHECK_ARG(n_cb >= 1 && which >= 0 && which < n_cb, "which must be in [0, n_cb)");
  CRVQ_CHECK_ARG(C_out != nullptr, "C_out is NULL");
  CbList cl;
  CRVQ_TRY(make_cblist(cbs, n_cb, G_sub, true, &cl));
  CRVQ_TRY(check_dev({{T, "T"}, {H_blocks, "H_blocks"}, {C_out, "C_out"}, {counts, "counts"}}));
  CRVQ_TRY(check_dev_cbs(cbs, n_cb));
  SetView set{T, ldT, M, G_sub, H_blocks};
  return launch_update_codebook(set, cl, which, C_out, counts, (cudaStream_t)stream);
}

crvq_status crvq_reconstruct_error(const float* W_sorted, int64_t M, int64_t N, int32_t d,
                                   const float* H_blocks, const int32_t* perm,
                                   const crvq_codebook* cbs, int32_t n_cb,
                                   int64_t n_crit_groups, const float* X, int64_t n_tok,
                                   double damp_delta, float* W_hat, double* losses,
                                   crvq_stream_t stream) {
  clear_last_error();
  CRVQ_TRY(check_d(d));
  CRVQ_CHECK_ARG(N >= 1 && N % d == 0, "N must be a positive multiple of d");
  CRVQ_TRY(check_set(W_sorted, N, M, N / d, H_blocks));
  CRVQ_CHECK_ARG(losses != nullptr, "losses is NULL");
  CRVQ_CHECK_ARG(N <= 49152, "N must be <= 49152");
  CRVQ_CHECK_ARG(n_crit_groups >= 0 && n_crit_groups <= N / d, "n_crit_groups out of range");
  CRVQ_CHECK_ARG(!X || n_tok >= 1, "n_tok must be >= 1 when X is given");
  CRVQ_CHECK_ARG(!W_hat || aligned16(W_hat), "W_hat must be 16-byte aligned");
  CbList cl;
  CRVQ_TRY(make_cblist(cbs, n_cb, N / d, true, &cl));
  CRVQ_TRY(check_dev({{W_sorted, "W_sorted"}, {H_blocks, "H_blocks"}, {perm, "perm"},
                      {X, "X"}, {W_hat, "W_hat"}}));
  CRVQ_TRY(check_dev_cbs(cbs, n_cb));
  cudaStream_t s = (cudaStream_t)stream;
  Scratch mem;
  CRVQ_TRY(mem.alloc(3 * sizeof(double), s));
  CRVQ_TRY(launch_reconstruct_error(W_sorted, M, N, H_blocks, perm, cl, n_crit_groups, X, n_tok,
                                    damp_delta, nullptr, W_hat, mem.as<double>(), s));
  CRVQ_CUDA(cudaMemcpyAsync(losses, mem.as<double>(), 3 * sizeof(double),
                            cudaMemcpyDeviceToHost, s));
  CRVQ_CUDA(cudaStreamSynchronize(s));
  return CRVQ_OK;
}

crvq_status crvq_coupled_sweep(const float* W_sorted, int64_t M, int64_t N, int32_t d,
                               const float* H_sorted, const crvq_codebook* cbs, int32_t n_cb,
                               int32_t which, int32_t sweeps, double* loss,
                               crvq_stream_t stream) {
  clear_last_error();
  CRVQ_TRY(check_d(d));
  CRVQ_CHECK_ARG(N >= 1 && N % d == 0, "N must be a positive multiple of d");
  CRVQ_CHECK_ARG(N <= 49152, "N must be <= 49152");
  CRVQ_TRY(check_set(W_sorted, N, M, N / d, H_sorted));
  CRVQ_CHECK_ARG(n_cb >= 1 && which >= 0 && which < n_cb, "which must be in [0, n_cb)");
  CRVQ_CHECK_ARG(sweeps >= 0, "sweeps must be >= 0");
  CbList cl;
  CRVQ_TRY(make_cblist(cbs, n_cb, N / d, true, &cl));
  CRVQ_TRY(check_dev({{W_sorted, "W_sorted"}, {H_sorted, "H_sorted"}}));
  CRVQ_TRY(check_dev_cbs(cbs, n_cb));
  cudaStream_t s = (cudaStream_t)stream;
  Scratch mem;
  double* ld = nullptr;
  if (loss) {
    CRVQ_TRY(mem.alloc((size_t)(sweeps + 1) * sizeof(double), s));
    ld = mem.as<double>();
  }
  CRVQ_TRY(launch_coupled_sweep(W_sorted, M, N, H_sorted, cl, which, sweeps, ld, s));
  if (loss) {
    CRVQ_CUDA(cudaMemcpyAsync(loss, ld, (size_t)(sweeps + 1) * sizeof(double),
                              cudaMemcpyDeviceToHost, s));
    CRVQ_CUDA(cudaStreamSynchronize(s));
  }
  return CRVQ_OK;
}

crvq_status crvq_lut_matvec(const float* X_in, int64_t ldx, int64_t b, int64_t N, int32_t d,
                            const int32_t* perm, const crvq_codebook* cbs, int32_t n_cb,
                            int64_t M, float* Y, int64_t ldy, crvq_stream_t stream) {
  clear_last_error();
  CRVQ_TRY(check_d(d));
  CRVQ_CHECK_ARG(X_in && Y, "X_in and Y must not be NULL");
  CRVQ_CHECK_ARG(N >= 1 && N % d == 0 && M >= 1, "need N >= 1, N %% d == 0, M >= 1");
  CRVQ_CHECK_ARG(b >= 1 && ldx >= N && ldy >= M, "need b >= 1, ldx >= N, ldy >= M");
  if (b > 8) return fail(CRVQ_ERR_UNSUPPORTED, "batches of more than 8 inputs are not implemented");
  CRVQ_CHECK_ARG(n_cb >= 1, "n_cb must be >= 1");
  CbList cl;
  CRVQ_TRY(make_cblist(cbs, n_cb, N / d, true, &cl));
  CRVQ_TRY(check_dev({{X_in, "X_in"}, {perm, "perm"}, {Y, "Y"}}));
  CRVQ_TRY(check_dev_cbs(cbs, n_cb));
  return launch_lut_matvec(X_in, ldx, N, (int)b, perm, cl, M, Y, ldy, (cudaStream_t)stream);
}

double crvq_avg_bits(int32_t e, int32_t d, int32_t m, double lambda, int64_t M, int64_t N,
                     int32_t include_perm) {
  if (d <= 0 || M <= 0 || N <= 0 || m < 1 || e < 0) return std::nan("");
  const double nvec = (double)M * (double)N / (double)d;
  double bits = nvec * e + (double)(m - 1) * lambda * nvec * e +
                (double)m * std::ldexp(1.0, e) * d * 16.0;
  if (include_perm) bits += 16.0 * (double)N;
  return bits / ((double)M * (double)N);
}

double crvq_avg_bits_bases(int32_t e, int32_t d, int32_t n_base, int32_t n_ext, double lambda,
                           int64_t M, int64_t N, int32_t include_perm) {
  if (d <= 0 || M <= 0 || N <= 0 || n_base < 1 || n_ext < 0 || e < 0) return std::nan("");
  const double nvec = (double)M * (double)N / (double)d;
  double bits = (double)n_base * nvec * e + (double)n_ext * lambda * nvec * e +
                (double)(n_base + n_ext) * std::ldexp(1.0, e) * d * 16.0;
  if (include_perm) bits += 16.0 * (double)N;
  return bits / ((double)M * (double)N);
}

}  // extern "C"

// ------------------------------------------------------------------------- layer schedule
namespace {

struct Buf {
  Scratch s;
  template <class T>
  crvq_status get(T** p, size_t count, cudaStream_t st) {
    CRVQ_TRY(s.alloc(count * sizeof(T), st));
    *p = s.as<T>();
    return CRVQ_OK;
  }
};

uint64_t phase_seed(uint64_t seed, int phase, int cb) {
  return splitmix64(seed, (uint64_t)phase * 1024u + (uint64_t)cb);
}

// Lloyd iterations for the last codebook of `cbs` (all earlier ones fixed), then a final
// encode: T x (encode, LS update) + encode. Each encode accumulates the least-squares
// statistics of the codes it writes, so the update is only the per-codeword solve, which
// also clears the statistics it read. One scratch serves every pass, so an iteration is
// kernels only (no allocation or memset between them in the stream).
crvq_status lloyd(const SetView& set, CbList cbs, int iters, const EncodeExtras& ex0,
                  cudaStream_t s) {
  const int j = cbs.n - 1;
  float* C = const_cast<float*>(cbs.cb[j].C);
  Scratch mem, wmem;
  StatsView st;
  CRVQ_TRY(stats_alloc(mem, cbs.cb[j].G_cov, cbs.cb[j].K, &st, s));
  CRVQ_TRY(launch_stats_prepare(set, cbs, j, st, s));  // T, H and fixed codebooks stay put
  const size_t wbytes = argmin_scratch_bytes(set.M, cbs.cb[j].G_cov, cbs.cb[j].K);
  CRVQ_TRY(wmem.alloc(wbytes, s));
  // the arg-min's per-vector terms, once for all iterations
  Scratch rmem;
  CRVQ_TRY(rmem.alloc((size_t)3 * set.M * set.G_sub * sizeof(float4), s));
  CRVQ_TRY(launch_row_terms(set, cbs, j, rmem.as<float4>(), s));
  EncodeExtras ex = ex0;
  ex.work = wmem.as<char>();
  ex.work_bytes = wbytes;
  ex.rowterms = rmem.as<float4>();
  EncodeExtras ex_last = ex;
  ex.stats = &st;
  for (int it = 0; it < iters; ++it) {
    CRVQ_TRY(launch_encode_beam(set, cbs, j, 1, false, nullptr, ex, s));
    CRVQ_TRY(launch_stats_solve(set, st, C, C, nullptr, s));
  }
  return launch_encode_beam(set, cbs, j, 1, false, nullptr, ex_last, s);
}

template <class T>
crvq_status to_device(const T* host_or_dev, size_t count, Buf& b, const T** out,
                      cudaStream_t s) {
  if (is_device_ptr(host_or_dev)) {
    *out = host_or_dev;
    return CRVQ_OK;
  }
  T* d = nullptr;
  CRVQ_TRY(b.get(&d, count, s));
  CRVQ_CUDA(cudaMemcpyAsync(d, host_or_dev, count * sizeof(T), cudaMemcpyHostToDevice, s));
  *out = d;
  return CRVQ_OK;
}

// Output buffer: the caller's device pointer, or a device staging buffer copied back at the end.
template <class T>
struct OutBuf {
  T* user = nullptr;
  T* dev = nullptr;
  size_t count = 0;
  Buf b;
  crvq_status init(T* u, size_t n, cudaStream_t s) {
    user = u;
    count = n;
    if (u && is_device_ptr(u)) {
      dev = u;
      return CRVQ_OK;
    }
    return b.get(&dev, std::max<size_t>(n, 1), s);
  }
  crvq_status flush(cudaStream_t s) {
    if (user && dev != user && count)
      CRVQ_CUDA(cudaMemcpyAsync(user, dev, count * sizeof(T), cudaMemcpyDeviceToHost, s));
    return CRVQ_OK;
  }
};

}  // namespace

namespace {

// Base codebooks of a configuration (n_base 0 reads as one).
int n_base_of(const crvq_config* cfg) { return cfg->n_base > 1 ? cfg->n_base : 1; }

// Device outputs of one layer (every pointer on the device; C_ext / codes_ext NULL when
// n_ext = 0, W_hat and imp may be NULL). C_base / codes_base hold n_base codebooks back to back.
struct LayerDev {
  int32_t* perm;
  float* C_base;
  int32_t* codes_base;
  float* C_ext;
  int32_t* codes_ext;
  float* W_hat;
  float* imp;
};

// S1-S7 on device pointers: losses[0..11] (block, crit, full | pre | before refinement) and
// *flag_total are written on the device; *scores and *rounds on the host. No host
// synchronisation unless cfg->refine_rounds > 1 (the early stop reads the loss).
crvq_status run_schedule(const float* W, const float* X, int64_t M, int64_t N, int64_t n_tok,
                         const crvq_config* cfg, int64_t Gc, const LayerDev& o, double* losses,
                         unsigned long long* flag_total, double* scores_out, int* rounds_out,
                         cudaStream_t s) {
  const int d = cfg->d;
  const int64_t G = N / d;
  double scores = 0.0;
  CRVQ_CUDA(cudaMemsetAsync(flag_total, 0, sizeof(unsigned long long), s));
  EncodeExtras ex;
  ex.scores = &scores;
  ex.flag_total = flag_total;

  // Only the 8 x 8 diagonal blocks of H (original and sorted order) and its diagonal are read,
  // so the dense N x N product is never formed: X^T is kept from S1 to S3 and each order's
  // blocks are taken on the tensor cores from it (the same values as the dense H's).
  const int64_t ldt = (n_tok + 3) / 4 * 4;
  Buf bXt, bd64, bxsq, bHb0, bdelta, bC0, bcodes0, bWpre, bWs, bHb;
  float *Xt, *xsq, *Hb0, *delta, *C0, *Wpre, *Ws, *Hb;
  double* delta64;
  int32_t* codes0;
  CRVQ_TRY(bXt.get(&Xt, (size_t)N * ldt, s));
  CRVQ_TRY(bd64.get(&delta64, 1, s));
  CRVQ_TRY(bxsq.get(&xsq, N, s));
  CRVQ_TRY(bHb0.get(&Hb0, (size_t)G * d * d, s));
  CRVQ_TRY(bdelta.get(&delta, 4, s));
  CRVQ_TRY(bC0.get(&C0, (size_t)cfg->K_base * d, s));
  CRVQ_TRY(bcodes0.get(&codes0, (size_t)M * G, s));
  CRVQ_TRY(bWpre.get(&Wpre, (size_t)M * N, s));
  CRVQ_TRY(bWs.get(&Ws, (size_t)M * N, s));
  CRVQ_TRY(bHb.get(&Hb, (size_t)G * d * d, s));

  // S1: Hessian proxy (diagonal blocks, xsq and delta)
  CRVQ_TRY(launch_transpose(X, n_tok, N, Xt, ldt, s));
  CRVQ_TRY(launch_tc_hessian_blocks(Xt, ldt, n_tok, N, nullptr, false, cfg->damp_rel, xsq,
                                    delta, delta64, Hb0, s));
  // S2: prequantize in the original order (Alg. 1, prequantization step)
  {
    SetView set{W, N, M, G, Hb0};
    CbList cl{};
    cl.n = 1;
    cl.cb[0] = CbView{C0, codes0, G, G, cfg->K_base};
    CRVQ_TRY(launch_kmeans_init(set, CbList{}, cfg->K_base,
                                phase_seed(cfg->seed, 1, 0), C0, s));
    CRVQ_TRY(lloyd(set, cl, cfg->kmeans_iters, ex, s));
    CRVQ_TRY(launch_reconstruct_error(W, M, N, Hb0, nullptr, cl, 0, nullptr, 0, 0.0, nullptr,
                                      Wpre, losses + 3, s));
  }
  // S3: importance and reordering (Alg. 1, importance and reordering steps); Eq. (wa) as
  // printed needs diag(H^-1), hence the dense H
  Buf bHd;
  float* Hd = nullptr;
  if (cfg->importance_mode == CRVQ_IMPORTANCE_WA_INV) {
    CRVQ_TRY(bHd.get(&Hd, (size_t)N * N, s));
    Buf bx2;
    float* xsq2 = nullptr;
    CRVQ_TRY(bx2.get(&xsq2, N, s));
    CRVQ_TRY(launch_hessian(X, n_tok, N, d, cfg->damp_rel, Hd, xsq2, nullptr, nullptr, s));
  }
  CRVQ_TRY(launch_select_reorder(W, M, N, d, Wpre, xsq, Hd, cfg->importance_mode,
                                 phase_seed(cfg->seed, 4, 0), o.perm, o.imp, Ws, nullptr, s));
  CRVQ_TRY(launch_tc_hessian_blocks(Xt, ldt, n_tok, N, o.perm, true, 0.f, nullptr, nullptr,
                                    delta64, Hb, s));
  // S4: base codebooks over all vectors (Alg. 1, base codebook steps). With several (Sec. 6.4,
  // the m = 2 setting) base b is fitted on the residual of bases 0..b-1 over every group.
  const int nb = n_base_of(cfg);
  CbList all{};
  all.n = nb + cfg->n_ext;
  for (int b = 0; b < nb; ++b)
    all.cb[b] = CbView{o.C_base + (size_t)b * cfg->K_base * d, o.codes_base + (size_t)b * M * G,
                       G, G, cfg->K_base};
  for (int t = 1; t <= cfg->n_ext; ++t)
    all.cb[nb + t - 1] = CbView{o.C_ext + (size_t)(t - 1) * cfg->K_ext * d,
                                o.codes_ext + (size_t)(t - 1) * M * Gc, Gc, Gc, cfg->K_ext};
  const SetView full{Ws, N, M, G, Hb};
  for (int b = 0; b < nb; ++b) {
    CbList cl{};
    cl.n = b + 1;
    for (int q = 0; q <= b; ++q) cl.cb[q] = all.cb[q];
    CbList fixed{};
    fixed.n = b;
    for (int q = 0; q < b; ++q) fixed.cb[q] = all.cb[q];
    CRVQ_TRY(launch_kmeans_init(full, fixed, cfg->K_base, phase_seed(cfg->seed, 2, b),
                                const_cast<float*>(all.cb[b].C), s));
    CRVQ_TRY(lloyd(full, cl, cfg->kmeans_iters, ex, s));
  }
  // S5: extended codebooks on the critical residual of every earlier codebook (Alg. 1,
  // extended-codebook loop)
  if (cfg->n_ext > 0) {
    const SetView crit{Ws, N, M, Gc, Hb};
    for (int t = 1; t <= cfg->n_ext; ++t) {
      const int j = nb + t - 1;
      CbList cl{};
      cl.n = j + 1;
      for (int q = 0; q <= j; ++q) {
        cl.cb[q] = all.cb[q];
        cl.cb[q].G_cov = Gc;
      }
      CbList fixed{};
      fixed.n = j;
      for (int q = 0; q < j; ++q) fixed.cb[q] = cl.cb[q];
      CRVQ_TRY(launch_kmeans_init(crit, fixed, cfg->K_ext, phase_seed(cfg->seed, 3, t),
                                  const_cast<float*>(all.cb[j].C), s));
      CRVQ_TRY(lloyd(crit, cl, cfg->kmeans_iters, ex, s));
    }
  }
  // S6: least-squares codebook updates + joint beam re-encode (Alg. 1, refinement loop)
  CRVQ_TRY(launch_reconstruct_error(Ws, M, N, Hb, o.perm, all, Gc, nullptr, 0, 0.0, nullptr,
                                    nullptr, losses + 6, s));
  double prev = 0.0;
  if (cfg->refine_rounds > 1) {
    CRVQ_CUDA(cudaMemcpyAsync(&prev, losses + 6, sizeof(double), cudaMemcpyDeviceToHost, s));
    CRVQ_CUDA(cudaStreamSynchronize(s));
  }
  int rounds = 0;
  for (int r = 0; r < cfg->refine_rounds; ++r) {
    for (int j = 0; j < all.n; ++j)
      CRVQ_TRY(launch_update_codebook(full, all, j, const_cast<float*>(all.cb[j].C), nullptr, s));
    CRVQ_TRY(launch_encode_beam(full, all, 0, cfg->B, true, nullptr, ex, s));
    ++rounds;
    if (cfg->refine_rounds > 1 && r + 1 < cfg->refine_rounds) {
      CRVQ_TRY(launch_reconstruct_error(Ws, M, N, Hb, o.perm, all, Gc, nullptr, 0, 0.0,
                                        nullptr, nullptr, losses + 9, s));
      double cur = 0.0;
      CRVQ_CUDA(cudaMemcpyAsync(&cur, losses + 9, sizeof(double), cudaMemcpyDeviceToHost, s));
      CRVQ_CUDA(cudaStreamSynchronize(s));
      if (cur > (1.0 - (double)cfg->eps_rel) * prev) break;
      prev = cur;
    }
  }
  // S7: losses and the reconstruction in the original order
  CRVQ_TRY(launch_reconstruct_error(Ws, M, N, Hb, o.perm, all, Gc, X, n_tok, 0.0, delta,
                                    o.W_hat, losses, s));
  *scores_out = scores;
  *rounds_out = rounds;
  return CRVQ_OK;
}

void fill_report(crvq_layer_report* report, const double hl[12], unsigned long long flagged,
                 double scores, int rounds) {
  report->flagged = (int64_t)flagged;
  report->loss_block = hl[0];
  report->loss_crit = hl[1];
  report->loss_full = hl[2];
  report->loss_pre = hl[3];
  report->loss_before_refine = hl[6];
  report->scores = scores;
  report->refine_rounds_done = rounds;
}

// ---- replay of whole-layer CUDA graphs
// A layer whose inputs and outputs all live on the device, with at most one refinement round,
// runs without host synchronisation between its ~240 launches; it is captured once into a
// CUDA graph per (device, stream, shapes, configuration, pointers, profiling state) and
// replayed, which removes the host launch gaps. Up to kGraphs graphs are kept (least recently
// used evicted, never one being replayed). Calls on different streams from different host
// threads run concurrently: the cache lock covers the lookup (and a capture), not the replay.
// CRVQ_GRAPHS=0 in the environment turns this off.
struct LayerGraph {
  int dev = -1;
  cudaStream_t stream = nullptr;
  int64_t M = 0, N = 0, n_tok = 0;
  crvq_config cfg;
  const float* W = nullptr;
  const float* X = nullptr;
  LayerDev o{};
  bool prof = false;
  char filter[64] = {0};
  cudaGraphExec_t exec = nullptr;
  double* losses = nullptr;                 // persistent device buffers read after a replay
  unsigned long long* flag_total = nullptr;
  double scores = 0.0;
  int rounds = 0;
  int64_t launches = 0;                     // kernels in the graph
  CapturedEvents events;                    // arg-min event nodes when captured while profiling
  uint64_t used = 0;
  int users = 0;                            // replays in flight (never evicted meanwhile)
};
// A 7-matrix decoder block in both profiling states on its streams, plus the host-buffer and
// single-stream variants of the same matrices.
constexpr int kGraphs = 48;
std::mutex g_graph_mu;
std::vector<LayerGraph*> g_graphs;
uint64_t g_graph_clock = 0;

void destroy_graph(LayerGraph* e) {
  if (e->exec) cudaGraphExecDestroy(e->exec);
  if (e->losses) cudaFree(e->losses);
  for (auto& r : e->events.recs) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  cudaGetLastError();
  delete e;
}

bool graphs_enabled() {
  const char* v = getenv("CRVQ_GRAPHS");
  return !(v && v[0] == '0');
}

bool same_key(const LayerGraph& e, int dev, cudaStream_t st, int64_t M, int64_t N, int64_t n_tok,
              const crvq_config* cfg, const float* W, const float* X, const LayerDev& o,
              bool prof) {
  return e.dev == dev && e.stream == st && e.M == M && e.N == N && e.n_tok == n_tok &&
         memcmp(&e.cfg, cfg, sizeof(crvq_config)) == 0 && e.W == W && e.X == X &&
         memcmp(&e.o, &o, sizeof(LayerDev)) == 0 && e.prof == prof &&
         (!prof || strncmp(e.filter, g_filter, sizeof(e.filter)) == 0);
}

// A device-to-host copy enqueued after a replay, before its synchronisation.
struct HostCopy {
  void* dst;
  const void* src;
  size_t bytes;
};

crvq_status run_graph(const float* W, const float* X, int64_t M, int64_t N, int64_t n_tok,
                      const crvq_config* cfg, int64_t Gc, const LayerDev& o,
                      crvq_layer_report* report, cudaStream_t s, bool* done,
                      const HostCopy* d2h = nullptr, int n_d2h = 0) {
  *done = false;
  int dev = 0;
  CRVQ_CUDA(cudaGetDevice(&dev));
  const bool prof = g_prof.load();
  std::unique_lock<std::mutex> lk(g_graph_mu);
  LayerGraph* e = nullptr;
  for (auto* c : g_graphs)
    if (same_key(*c, dev, s, M, N, n_tok, cfg, W, X, o, prof)) e = c;
  if (!e) {
    // Everything that allocates or initialises lazily happens before the capture.
    unsigned* err = nullptr;
    CRVQ_TRY(device_error_word(&err));
    sm_count();
    e = new LayerGraph;
    e->dev = dev;
    e->stream = s;
    e->M = M;
    e->N = N;
    e->n_tok = n_tok;
    e->cfg = *cfg;
    e->W = W;
    e->X = X;
    e->o = o;
    e->prof = prof;
    strncpy(e->filter, g_filter, sizeof(e->filter) - 1);
    if (cudaMalloc(&e->losses, 16 * sizeof(double) + 64) != cudaSuccess) {
      cudaGetLastError();
      delete e;
      return CRVQ_OK;  // not done: the caller runs the schedule directly
    }
    e->flag_total = reinterpret_cast<unsigned long long*>(e->losses + 16);
    const long long l0 = g_launches.load();
    cudaGraph_t graph = nullptr;
    crvq_status st = CRVQ_OK;
    if (cudaStreamBeginCapture(s, cudaStreamCaptureModeRelaxed) == cudaSuccess) {
      t_capture = &e->events;
      st = run_schedule(W, X, M, N, n_tok, cfg, Gc, o, e->losses, e->flag_total, &e->scores,
                        &e->rounds, s);
      t_capture = nullptr;
      const cudaError_t ce = cudaStreamEndCapture(s, &graph);
      if (ce != cudaSuccess) st = CRVQ_ERR_CUDA;
    } else {
      st = CRVQ_ERR_CUDA;
    }
    e->launches = g_launches.load() - l0;
    g_launches.fetch_sub(e->launches);  // counted when replayed
    if (st == CRVQ_OK && cudaGraphInstantiate(&e->exec, graph, 0) != cudaSuccess) st = CRVQ_ERR_CUDA;
    if (graph) cudaGraphDestroy(graph);
    cudaGetLastError();
    if (st != CRVQ_OK) {  // capture not possible here: run the schedule directly
      destroy_graph(e);
      clear_last_error();
      return CRVQ_OK;
    }
    if ((int)g_graphs.size() >= kGraphs) {
      int lru = -1;
      for (int q = 0; q < (int)g_graphs.size(); ++q)
        if (g_graphs[q]->users == 0 && (lru < 0 || g_graphs[q]->used < g_graphs[lru]->used))
          lru = q;
      if (lru >= 0) {
        destroy_graph(g_graphs[lru]);
        g_graphs.erase(g_graphs.begin() + lru);
      }
    }
    g_graphs.push_back(e);
  }
  e->used = ++g_graph_clock;
  ++e->users;
  lk.unlock();
  struct Unpin {  // the entry may be evicted again once this replay is done
    LayerGraph* e;
    ~Unpin() {
      std::lock_guard<std::mutex> l(g_graph_mu);
      --e->users;
    }
  } unpin{e};
  CRVQ_CUDA(cudaGraphLaunch(e->exec, s));
  g_launches.fetch_add(e->launches);
  double hl[12];
  unsigned long long flagged = 0;
  CRVQ_CUDA(cudaMemcpyAsync(hl, e->losses, sizeof(hl), cudaMemcpyDeviceToHost, s));
  CRVQ_CUDA(cudaMemcpyAsync(&flagged, e->flag_total, sizeof(flagged), cudaMemcpyDeviceToHost, s));
  for (int q = 0; q < n_d2h; ++q)
    if (d2h[q].bytes)
      CRVQ_CUDA(cudaMemcpyAsync(d2h[q].dst, d2h[q].src, d2h[q].bytes, cudaMemcpyDeviceToHost, s));
  CRVQ_CUDA(cudaStreamSynchronize(s));
  if (prof && g_prof.load()) {  // the event nodes of this replay have completed
    std::lock_guard<std::mutex> lk2(g_pmu);
    for (auto& r : e->events.recs) {
      float ms = 0.f;
      if (cudaEventElapsedTime(&ms, r.a, r.b) == cudaSuccess)
        g_graph_recs.push_back(ProfDone{r.name, ms, r.units});
      else
        cudaGetLastError();
    }
  }
  fill_report(report, hl, flagged, e->scores, e->rounds);
  *done = true;
  return CRVQ_OK;
}

// Persistent device staging for layers called with host inputs or outputs: the host data is
// copied into buffers that outlive the call, so that the graph captured on them (keyed by
// pointers) is replayed by later calls of the same shapes, as for device buffers. Up to
// kStagings sets are kept (least recently used freed; never one a call is using): calls of one
// shape running concurrently on several streams each take their own set.
struct Staging {
  int dev = -1;
  int64_t M = 0, N = 0, n_tok = 0, n_base = 0, K_base = 0, n_ext = 0, K_ext = 0, Gc = 0;
  float *W = nullptr, *X = nullptr, *C_base = nullptr, *C_ext = nullptr, *W_hat = nullptr,
        *imp = nullptr;
  int32_t *perm = nullptr, *codes_base = nullptr, *codes_ext = nullptr;
  uint64_t used = 0;
  int users = 0;
};
constexpr int kStagings = 8;
std::mutex g_stage_mu;
std::vector<Staging*> g_stagings;
uint64_t g_stage_clock = 0;

void free_staging(Staging* sg) {
  for (void* p : {(void*)sg->W, (void*)sg->X, (void*)sg->C_base, (void*)sg->C_ext,
                  (void*)sg->W_hat, (void*)sg->imp, (void*)sg->perm, (void*)sg->codes_base,
                  (void*)sg->codes_ext})
    if (p) cudaFree(p);
  cudaGetLastError();
  delete sg;
}

crvq_status acquire_staging(int dev, int64_t M, int64_t N, int64_t n_tok, const crvq_config* cfg,
                            int64_t Gc, Staging** out) {
  std::lock_guard<std::mutex> lk(g_stage_mu);
  const int d = cfg->d;
  const int nb = n_base_of(cfg);
  for (auto* sg : g_stagings)
    if (sg->dev == dev && sg->M == M && sg->N == N && sg->n_tok == n_tok &&
        sg->n_base == nb && sg->K_base == cfg->K_base && sg->n_ext == cfg->n_ext &&
        sg->K_ext == (cfg->n_ext ? cfg->K_ext : 0) && sg->Gc == Gc && sg->users == 0) {
      sg->used = ++g_stage_clock;
      sg->users = 1;
      *out = sg;
      return CRVQ_OK;
    }
  if ((int)g_stagings.size() >= kStagings) {
    int lru = -1;
    for (int q = 0; q < (int)g_stagings.size(); ++q)
      if (g_stagings[q]->users == 0 && (lru < 0 || g_stagings[q]->used < g_stagings[lru]->used))
        lru = q;
    if (lru >= 0) {
      free_staging(g_stagings[lru]);
      g_stagings.erase(g_stagings.begin() + lru);
    }
  }
  Staging* sg = new Staging;
  sg->dev = dev;
  sg->M = M;
  sg->N = N;
  sg->n_tok = n_tok;
  sg->n_base = nb;
  sg->K_base = cfg->K_base;
  sg->n_ext = cfg->n_ext;
  sg->K_ext = cfg->n_ext ? cfg->K_ext : 0;
  sg->Gc = Gc;
  const int64_t G = N / d;
  bool ok = cudaMalloc(&sg->W, (size_t)M * N * 4) == cudaSuccess &&
            cudaMalloc(&sg->X, (size_t)n_tok * N * 4) == cudaSuccess &&
            cudaMalloc(&sg->C_base, (size_t)nb * cfg->K_base * d * 4) == cudaSuccess &&
            cudaMalloc(&sg->W_hat, (size_t)M * N * 4) == cudaSuccess &&
            cudaMalloc(&sg->imp, (size_t)N * 4) == cudaSuccess &&
            cudaMalloc(&sg->perm, (size_t)N * 4) == cudaSuccess &&
            cudaMalloc(&sg->codes_base, (size_t)nb * M * G * 4) == cudaSuccess;
  if (ok && cfg->n_ext > 0)
    ok = cudaMalloc(&sg->C_ext, (size_t)cfg->n_ext * cfg->K_ext * d * 4) == cudaSuccess &&
         cudaMalloc(&sg->codes_ext, (size_t)cfg->n_ext * M * Gc * 4) == cudaSuccess;
  if (!ok) {
    free_staging(sg);
    return fail(CRVQ_ERR_NOMEM, "staging buffers for a host-buffer layer call");
  }
  sg->used = ++g_stage_clock;
  sg->users = 1;
  g_stagings.push_back(sg);
  *out = sg;
  return CRVQ_OK;
}

void release_staging(Staging* sg) {
  std::lock_guard<std::mutex> lk(g_stage_mu);
  sg->users = 0;
}

}  // namespace

extern "C" {

crvq_status crvq_quantize_layer(const float* W_in, const float* X_in, int64_t M, int64_t N,
                                int64_t n_tok, const crvq_config* cfg,
                                const crvq_layer_outputs* out, crvq_layer_report* report,
                                crvq_stream_t stream) {
  clear_last_error();
  CRVQ_CHECK_ARG(cfg && out && report && W_in && X_in, "required pointer is NULL");
  CRVQ_TRY(check_d(cfg->d));
  const int d = cfg->d;
  CRVQ_CHECK_ARG(M >= 1 && N >= 1 && N % d == 0 && n_tok >= 1, "bad matrix shape");
  CRVQ_CHECK_ARG(N <= 49152, "N must be <= 49152");
  const int64_t G = N / d;
  CRVQ_CHECK_ARG(cfg->K_base >= 1 && cfg->K_base <= 65536 && cfg->K_base <= M * G,
                 "K_base out of range");
  CRVQ_CHECK_ARG(cfg->n_ext >= 0 && cfg->n_ext <= kMaxCodebooks - 1, "n_ext must be in [0, 7]");
  CRVQ_CHECK_ARG(cfg->n_base >= 0 && cfg->n_base <= kMaxCodebooks &&
                     n_base_of(cfg) + cfg->n_ext <= kMaxCodebooks,
                 "n_base must be >= 0 with n_base + n_ext <= 8");
  const int nb = n_base_of(cfg);
  CRVQ_CHECK_ARG(cfg->crit_frac >= 0.f && cfg->crit_frac <= 1.f, "crit_frac must be in [0, 1]");
  CRVQ_CHECK_ARG(cfg->B >= 1 && cfg->B <= 16, "B must be in [1, 16]");
  CRVQ_CHECK_ARG(cfg->kmeans_iters >= 0 && cfg->refine_rounds >= 0, "negative iteration count");
  CRVQ_CHECK_ARG(cfg->importance_mode >= 0 && cfg->importance_mode <= 3, "bad importance mode");
  CRVQ_CHECK_ARG(std::isfinite(cfg->damp_rel) && cfg->damp_rel >= 0.f, "bad damp_rel");
  const int64_t Gc = crvq_n_crit_groups(N, d, cfg->crit_frac);
  if (cfg->n_ext > 0) {
    CRVQ_CHECK_ARG(Gc >= 1, "extended codebooks need at least one critical group");
    CRVQ_CHECK_ARG(cfg->K_ext >= 1 && cfg->K_ext <= 65536 && cfg->K_ext <= M * Gc,
                   "K_ext out of range");
  }
  CRVQ_CHECK_ARG(out->perm && out->C_base && out->codes_base, "perm, C_base, codes_base needed");
  CRVQ_CHECK_ARG(cfg->n_ext == 0 || (out->C_ext && out->codes_ext), "C_ext, codes_ext needed");
  cudaStream_t s = (cudaStream_t)stream;
  memset(report, 0, sizeof(*report));
  report->n_crit_groups = Gc;

  const bool dev_in = is_device_ptr(W_in) && is_device_ptr(X_in);
  const bool dev_out = is_device_ptr(out->perm) && is_device_ptr(out->C_base) &&
                       is_device_ptr(out->codes_base) &&
                       (cfg->n_ext == 0 || (is_device_ptr(out->C_ext) &&
                                            is_device_ptr(out->codes_ext))) &&
                       (!out->W_hat || is_device_ptr(out->W_hat)) &&
                       (!out->importance || is_device_ptr(out->importance));
  if (dev_in && dev_out && cfg->refine_rounds <= 1 && graphs_enabled() &&
      aligned16(W_in) && aligned16(X_in) && aligned16(out->C_base) &&
      (cfg->n_ext == 0 || aligned16(out->C_ext)) && (!out->W_hat || aligned16(out->W_hat))) {
    const LayerDev o{out->perm, out->C_base, out->codes_base,
                     cfg->n_ext ? out->C_ext : nullptr, cfg->n_ext ? out->codes_ext : nullptr,
                     out->W_hat, out->importance};
    bool done = false;
    CRVQ_TRY(run_graph(W_in, X_in, M, N, n_tok, cfg, Gc, o, report, s, &done));
    if (done) {
      report->n_crit_groups = Gc;
      return CRVQ_OK;
    }
  } else if (cfg->refine_rounds <= 1 && graphs_enabled()) {
    // Host inputs or outputs: the same graph replay on persistent staging buffers, with the
    // host copies around it (device pointers of the caller are used in place).
    const bool ok_align = (!is_device_ptr(W_in) || aligned16(W_in)) &&
                          (!is_device_ptr(X_in) || aligned16(X_in)) &&
                          (!is_device_ptr(out->C_base) || aligned16(out->C_base)) &&
                          (cfg->n_ext == 0 || !is_device_ptr(out->C_ext) ||
                           aligned16(out->C_ext)) &&
                          (!out->W_hat || !is_device_ptr(out->W_hat) || aligned16(out->W_hat));
    int dev = 0;
    CRVQ_CUDA(cudaGetDevice(&dev));
    Staging* sg = nullptr;
    if (ok_align && acquire_staging(dev, M, N, n_tok, cfg, Gc, &sg) == CRVQ_OK) {
      struct Release {
        Staging* p;
        ~Release() { release_staging(p); }
      } rel{sg};
      const float* Wd = W_in;
      const float* Xd = X_in;
      if (!is_device_ptr(W_in)) {
        CRVQ_CUDA(cudaMemcpyAsync(sg->W, W_in, (size_t)M * N * 4, cudaMemcpyHostToDevice, s));
        Wd = sg->W;
      }
      if (!is_device_ptr(X_in)) {
        CRVQ_CUDA(cudaMemcpyAsync(sg->X, X_in, (size_t)n_tok * N * 4, cudaMemcpyHostToDevice,
                                  s));
        Xd = sg->X;
      }
      HostCopy cp[7];
      int ncp = 0;
      auto place = [&](auto* user, auto* stage, size_t count) {
        using T = std::remove_pointer_t<decltype(stage)>;
        if (!user) return (T*)nullptr;
        if (is_device_ptr(user)) return (T*)user;
        cp[ncp++] = HostCopy{(void*)user, (const void*)stage, count * sizeof(T)};
        return stage;
      };
      LayerDev o{};
      o.perm = place(out->perm, sg->perm, (size_t)N);
      o.C_base = place(out->C_base, sg->C_base, (size_t)nb * cfg->K_base * d);
      o.codes_base = place(out->codes_base, sg->codes_base, (size_t)nb * M * G);
      if (cfg->n_ext) {
        o.C_ext = place(out->C_ext, sg->C_ext, (size_t)cfg->n_ext * cfg->K_ext * d);
        o.codes_ext = place(out->codes_ext, sg->codes_ext, (size_t)cfg->n_ext * M * Gc);
      }
      o.W_hat = place(out->W_hat, sg->W_hat, (size_t)M * N);
      o.imp = out->importance ? place(out->importance, sg->imp, (size_t)N) : sg->imp;
      bool done = false;
      CRVQ_TRY(run_graph(Wd, Xd, M, N, n_tok, cfg, Gc, o, report, s, &done, cp, ncp));
      if (done) {
        report->n_crit_groups = Gc;
        return CRVQ_OK;
      }
    }
    clear_last_error();
  }

  // Direct path: host inputs / outputs are staged through device buffers.
  Buf bW, bX, bloss;
  const float *W = nullptr, *X = nullptr;
  CRVQ_TRY(to_device(W_in, (size_t)M * N, bW, &W, s));
  CRVQ_TRY(to_device(X_in, (size_t)n_tok * N, bX, &X, s));
  CRVQ_CHECK_ARG(aligned16(W) && aligned16(X), "W and X must be 16-byte aligned");
  OutBuf<int32_t> o_perm, o_codes_base, o_codes_ext;
  OutBuf<float> o_C_base, o_C_ext, o_W_hat, o_imp;
  CRVQ_TRY(o_perm.init(out->perm, N, s));
  CRVQ_TRY(o_C_base.init(out->C_base, (size_t)nb * cfg->K_base * d, s));
  CRVQ_TRY(o_codes_base.init(out->codes_base, (size_t)nb * M * G, s));
  CRVQ_TRY(o_C_ext.init(out->C_ext, (size_t)cfg->n_ext * cfg->K_ext * d, s));
  CRVQ_TRY(o_codes_ext.init(out->codes_ext, (size_t)cfg->n_ext * M * Gc, s));
  if (out->W_hat) CRVQ_TRY(o_W_hat.init(out->W_hat, (size_t)M * N, s));
  CRVQ_TRY(o_imp.init(out->importance, N, s));
  CRVQ_CHECK_ARG(aligned16(o_C_base.dev) && aligned16(o_C_ext.dev) &&
                     (!out->W_hat || aligned16(o_W_hat.dev)),
                 "C_base, C_ext and W_hat must be 16-byte aligned");
  double* losses = nullptr;
  CRVQ_TRY(bloss.get(&losses, 16 + 8, s));
  unsigned long long* flag_total = reinterpret_cast<unsigned long long*>(losses + 16);
  const LayerDev o{o_perm.dev, o_C_base.dev, o_codes_base.dev, o_C_ext.dev, o_codes_ext.dev,
                   out->W_hat ? o_W_hat.dev : nullptr, o_imp.dev};
  double scores = 0.0;
  int rounds = 0;
  CRVQ_TRY(run_schedule(W, X, M, N, n_tok, cfg, Gc, o, losses, flag_total, &scores, &rounds, s));
  CRVQ_TRY(o_perm.flush(s));
  CRVQ_TRY(o_C_base.flush(s));
  CRVQ_TRY(o_codes_base.flush(s));
  CRVQ_TRY(o_C_ext.flush(s));
  CRVQ_TRY(o_codes_ext.flush(s));
  if (out->W_hat) CRVQ_TRY(o_W_hat.flush(s));
  if (out->importance) CRVQ_TRY(o_imp.flush(s));
  double hl[12];
  unsigned long long flagged = 0;
  CRVQ_CUDA(cudaMemcpyAsync(hl, losses, sizeof(hl), cudaMemcpyDeviceToHost, s));
  CRVQ_CUDA(cudaMemcpyAsync(&flagged, flag_total, sizeof(flagged), cudaMemcpyDeviceToHost, s));
  CRVQ_CUDA(cudaStreamSynchronize(s));
  fill_report(report, hl, flagged, scores, rounds);
  return CRVQ_OK;
}

}  // extern "C"
