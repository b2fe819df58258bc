// api.cu -- library-wide entry points: status strings, version, the last
// CUDA error, and the cached SM count used to size grids.
#include <atomic>
#include <mutex>
#include <map>
#include <utility>

#include "common.cuh"

namespace dreams {

namespace {
thread_local int32_t g_last_cuda_error = 0;
std::mutex g_sm_mutex;
int g_sm_count[64] = {0};
std::mutex g_attr_mutex;
std::map<std::pair<const void *, int>, int> g_attr_done;  // (kernel, device) -> the largest limit set
constexpr uint64_t DEFAULT_WAIT_NS = 2000000000ull;
std::atomic<int32_t> g_stall_kernels{0};
std::atomic<int32_t> g_stall_at{-1};
std::atomic<uint64_t> g_stall_wait_ns{DEFAULT_WAIT_NS};
}  // namespace

void test_stall(int32_t kernel, int32_t *stall_at, uint64_t *wait_ns) {
  if ((g_stall_kernels.load() & kernel) != 0 && g_stall_at.load() >= 0) {
    *stall_at = g_stall_at.load();
    *wait_ns = g_stall_wait_ns.load();
  } else {
    *stall_at = -1;
    *wait_ns = DEFAULT_WAIT_NS;
  }
}

void set_last_cuda_error(cudaError_t e) { g_last_cuda_error = static_cast<int32_t>(e); }

int num_sms() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152;
  std::lock_guard<std::mutex> lock(g_sm_mutex);
  if (g_sm_count[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 152;
    g_sm_count[dev] = n;
  }
  return g_sm_count[dev];
}

dreams_status_t ensure_max_dynamic_smem(const void *func, int bytes) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  std::lock_guard<std::mutex> lock(g_attr_mutex);
  const auto it = g_attr_done.find({func, dev});
  if (it != g_attr_done.end() && it->second >= bytes) return DREAMS_OK;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  g_attr_done[{func, dev}] = bytes;
  return DREAMS_OK;
}

}  // namespace dreams

extern "C" const char *dreams_status_string(dreams_status_t status) {
  switch (status) {
    case DREAMS_OK: return "ok";
    case DREAMS_ERR_INVALID_ARG: return "invalid argument";
    case DREAMS_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case DREAMS_ERR_WORKSPACE: return "workspace missing or too small";
    case DREAMS_ERR_CUDA: return "CUDA error";
    case DREAMS_ERR_SCRATCH_LIMIT: return "problem larger than the fixed scratch of a no-allocation entry point";
  }
  return "unknown status";
}

extern "C" int32_t dreams_version(void) { return DREAMS_VERSION; }

extern "C" dreams_status_t dreams_test_set_stall(int32_t kernels, int32_t stall_at, int64_t wait_limit_ns) {
  if (stall_at < 0) {
    dreams::g_stall_at.store(-1);
    dreams::g_stall_kernels.store(0);
    dreams::g_stall_wait_ns.store(dreams::DEFAULT_WAIT_NS);
    return DREAMS_OK;
  }
  if ((kernels & ~(DREAMS_TEST_ATTENTION | DREAMS_TEST_LM_HEAD)) != 0 || kernels == 0 || wait_limit_ns < 1000 ||
      wait_limit_ns > int64_t(dreams::DEFAULT_WAIT_NS))
    return DREAMS_ERR_INVALID_ARG;
  dreams::g_stall_wait_ns.store(uint64_t(wait_limit_ns));
  dreams::g_stall_kernels.store(kernels);
  dreams::g_stall_at.store(stall_at);
  return DREAMS_OK;
}

extern "C" int32_t dreams_last_cuda_error(void) { return dreams::g_last_cuda_error; }
