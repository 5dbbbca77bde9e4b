// Error reporting, device queries, the bounded-wait status word and its
// self-test kernel.
#include <atomic>
#include <cstdlib>
#include <mutex>
#include <string>
#include <vector>

#include "decomoe_internal.cuh"

namespace decomoe {

static thread_local std::string t_last_error;
static std::atomic<int64_t> g_wait_limit_ns{2000000000LL};

void set_error(const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  t_last_error = buf;
}

void clear_error() { t_last_error.clear(); }

int64_t wait_limit_ns() { return g_wait_limit_ns.load(std::memory_order_relaxed); }

static std::atomic<int> g_discard_scratch{1};
bool discard_scratch() { return g_discard_scratch.load(std::memory_order_relaxed) != 0; }

// Programmatic launch pays for grids of at most one block per SM (the
// persistent GEMMs and the decode-size kernels); kernels of many blocks ran
// slower with it, so they launch plainly. decomoe_set_pdl(0) turns it off.
static std::atomic<int> g_pdl{1};
bool pdl_enabled(int64_t blocks) {
  return g_pdl.load(std::memory_order_relaxed) != 0 && blocks <= static_cast<int64_t>(sm_count());
}

int sm_count() {
  static std::mutex mu;
  static std::vector<int> cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  std::lock_guard<std::mutex> lk(mu);
  if (static_cast<int>(cache.size()) <= dev) cache.resize(dev + 1, 0);
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 1;
    cache[dev] = n;
  }
  return cache[dev];
}

// One thread waits on an mbarrier that nothing ever arrives at; the bounded
// wait must give up after limit_ns and record DECOMOE_ERR_TIMEOUT.
__global__ void k_selftest_wait(int32_t* status, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    abort_flag = 0;
    mbar_init(smem_u32(&bar), 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (!mbar_wait(smem_u32(&bar), 0, limit_ns, &abort_flag)) report_status(status, DECOMOE_ERR_TIMEOUT);
  }
}

}  // namespace decomoe

using namespace decomoe;

extern "C" {

// C-callable setter for the host C sources of the library (not exported).
__attribute__((visibility("hidden"))) void decomoe_internal_set_error(const char* msg) {
  set_error("%s", msg);
}

const char* decomoe_last_error(void) { return t_last_error.c_str(); }

int decomoe_version(void) { return 100; }

int decomoe_device_info(int* sm_count_host, int* cc_major_host, int* cc_minor_host) {
  int dev = 0;
  DM_CUDA_CHECK(cudaGetDevice(&dev));
  if (sm_count_host) *sm_count_host = sm_count();
  if (cc_major_host) DM_CUDA_CHECK(cudaDeviceGetAttribute(cc_major_host, cudaDevAttrComputeCapabilityMajor, dev));
  if (cc_minor_host) DM_CUDA_CHECK(cudaDeviceGetAttribute(cc_minor_host, cudaDevAttrComputeCapabilityMinor, dev));
  return DECOMOE_OK;
}

int decomoe_read_status(int32_t* status_dev, int32_t* code_host, decomoe_stream_t stream) {
  DM_ARG_CHECK(status_dev != nullptr && code_host != nullptr, "read_status: null pointer");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int32_t v = 0;
  DM_CUDA_CHECK(cudaMemcpyAsync(&v, status_dev, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
  DM_CUDA_CHECK(cudaStreamSynchronize(s));
  DM_CUDA_CHECK(cudaMemsetAsync(status_dev, 0, sizeof(int32_t), s));
  *code_host = v;
  return DECOMOE_OK;
}

int decomoe_set_wait_limit_ns(int64_t limit_ns) {
  DM_ARG_CHECK(limit_ns > 0, "set_wait_limit_ns: limit must be positive");
  g_wait_limit_ns.store(limit_ns, std::memory_order_relaxed);
  return DECOMOE_OK;
}

int decomoe_set_pdl(int on) {
  g_pdl.store(on != 0 ? 1 : 0, std::memory_order_relaxed);
  return DECOMOE_OK;
}

int decomoe_set_discard_scratch(int on) {
  g_discard_scratch.store(on != 0 ? 1 : 0, std::memory_order_relaxed);
  return DECOMOE_OK;
}

int decomoe_selftest_wait(int32_t* status_dev, int64_t limit_ns, decomoe_stream_t stream) {
  DM_ARG_CHECK(status_dev != nullptr, "selftest_wait: status_dev is null");
  DM_ARG_CHECK(limit_ns > 0 && limit_ns <= 10000000000LL, "selftest_wait: limit out of (0, 10 s]");
  k_selftest_wait<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(status_dev,
                                                                         static_cast<uint64_t>(limit_ns));
  DM_LAUNCH_CHECK("k_selftest_wait");
  return DECOMOE_OK;
}

}  // extern "C"
