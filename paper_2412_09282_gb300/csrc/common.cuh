// Shared host/device helpers of libcrvq: status handling, the device error word, stream-
// ordered scratch, SplitMix64 and small device utilities.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <cstdarg>
#include <cstdio>
#include <initializer_list>
#include <string>
#include <utility>

#include "crvq.h"

namespace crvq {

// ---------------------------------------------------------------- host-side status
void set_last_error(const char* fmt, ...);
crvq_status fail(crvq_status st, const char* fmt, ...);
void clear_last_error();

#define CRVQ_CHECK_ARG(cond, ...)                                        \
  do {                                                                   \
    if (!(cond)) return ::crvq::fail(CRVQ_ERR_INVALID_ARG, __VA_ARGS__); \
  } while (0)

#define CRVQ_CUDA(call)                                                                     \
  do {                                                                                      \
    cudaError_t e_ = (call);                                                                \
    if (e_ != cudaSuccess)                                                                  \
      return ::crvq::fail(e_ == cudaErrorMemoryAllocation ? CRVQ_ERR_NOMEM : CRVQ_ERR_CUDA, \
                          "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_), __FILE__, \
                          __LINE__);                                                        \
  } while (0)

#define CRVQ_TRY(expr)                    \
  do {                                    \
    crvq_status s_ = (expr);              \
    if (s_ != CRVQ_OK) return s_;         \
  } while (0)

// Launch bookkeeping: counts the launch and reports a launch-configuration failure right
// after a <<<>>> launch.
void count_launch();
#define CRVQ_LAUNCHED()              \
  do {                               \
    ::crvq::count_launch();          \
    CRVQ_CUDA(cudaGetLastError());   \
  } while (0)

// Programmatic dependent launch. A kernel launched by launch_pdl may be scheduled while its
// stream predecessor (a kernel) is still running: it lets its own dependents launch
// (pdl_trigger) and then waits for the predecessor to complete with its memory visible
// (pdl_wait) before it reads anything or allocates tensor memory. Both are no-ops in a kernel
// launched without the attribute. Removes the launch gap between dependent kernels of a layer.
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Brackets the launches in its scope with CUDA events when profiling is on.
class ProfScope {
 public:
  ProfScope(const char* name, cudaStream_t s, double units);
  ~ProfScope();
  ProfScope(const ProfScope&) = delete;
  ProfScope& operator=(const ProfScope&) = delete;

 private:
  const char* name_;
  cudaStream_t s_;
  double units_;
  cudaEvent_t a_ = nullptr;
};

// Error-word bits set by kernels (never a trap): decoded by crvq_sync().
enum : unsigned { ERRBIT_INDEX = 1u, ERRBIT_NUMERIC = 2u, ERRBIT_TIMEOUT = 4u };

// Device error word of the current device (allocated once per device, zeroed).
crvq_status device_error_word(unsigned** out);

// Stream-ordered scratch buffer; freed (stream-ordered) when it goes out of scope.
class Scratch {
 public:
  Scratch() = default;
  Scratch(const Scratch&) = delete;
  Scratch& operator=(const Scratch&) = delete;
  ~Scratch() { release(); }
  crvq_status alloc(size_t bytes, cudaStream_t s) {
    release();
    stream_ = s;
    if (bytes == 0) return CRVQ_OK;
    CRVQ_CUDA(cudaMallocAsync(&p_, bytes, s));
    return CRVQ_OK;
  }
  void release() {
    if (p_) cudaFreeAsync(p_, stream_);
    p_ = nullptr;
  }
  template <class T>
  T* as() const { return static_cast<T*>(p_); }

 private:
  void* p_ = nullptr;
  cudaStream_t stream_ = nullptr;
};

inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Number of SMs of the current device (cached per device).
int sm_count();

// Raises `kernel`'s dynamic shared-memory limit on the current device to at least `bytes`,
// calling cudaFuncSetAttribute only when a larger limit than before is needed (remembered per
// kernel address and device).
crvq_status smem_limit(const void* kernel, size_t bytes);

// ---------------------------------------------------------------- device helpers
// SplitMix64 (Steele, Lea & Flood 2014): output `ctr` (0-based) of the stream `stream`.
__host__ __device__ inline uint64_t splitmix64(uint64_t stream, uint64_t ctr) {
  uint64_t z = stream + (ctr + 1ull) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ inline void raise_error(unsigned* err, unsigned bit) {
  if (err) atomicOr(err, bit);
}

// Codebook view passed to kernels by value (fits in kernel parameter space).
constexpr int kMaxCodebooks = 8;
struct CbView {
  const float* C;
  int32_t* codes;
  int64_t ld;
  int64_t G_cov;
  int32_t K;
};
struct CbList {
  CbView cb[kMaxCodebooks];
  int n;
};

// ---------------------------------------------------------------- argument validation
// Shared by every entry point (api.cu): each returns CRVQ_OK or sets the last error and
// returns CRVQ_ERR_INVALID_ARG (CRVQ_ERR_UNSUPPORTED for d != 8).
crvq_status check_d(int32_t d);
// A vector set: non-null, non-empty, ldT >= G_sub * 8 and a multiple of 4, 16-byte aligned.
crvq_status check_set(const float* T, int64_t ldT, int64_t M, int64_t G_sub, const float* Hb);
// Codebook array -> CbList, with the range checks of crvq_codebook's fields.
crvq_status make_cblist(const crvq_codebook* cbs, int32_t n_cb, int64_t G_sub,
                        bool need_codes_all, CbList* out);
// Each non-null pointer must be device (or managed) memory: a host pointer is refused here
// instead of reaching a kernel.
crvq_status check_dev(std::initializer_list<std::pair<const void*, const char*>> ps);
crvq_status check_dev_cbs(const crvq_codebook* cbs, int32_t n);

// The error word of crvq_update_codebook_noalloc on the current device (noalloc.cu): *bits
// receives its ERRBIT_* bits, which are then cleared. Reads nothing on a device where that
// entry point has not run.
crvq_status noalloc_take_error(unsigned* bits);

}  // namespace crvq
