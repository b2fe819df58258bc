// api.cu -- library-wide entry points: status strings, version, the last
// CUDA error, and the cached SM count used to size grids.
#include <mutex>

#include "common.cuh"

namespace dreams {

namespace {
thread_local int32_t g_last_cuda_error = 0;
std::mutex g_sm_mutex;
int g_sm_count[64] = {0};
}  // namespace

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

extern "C" int32_t dreams_last_cuda_error(void) { return dreams::g_last_cuda_error; }
