// common.cuh -- device helpers shared by the library's kernels (sm_103a).
#pragma once
#include <limits.h>

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dreams.h"

namespace dreams {

// Thread-local record of the last failing CUDA call (dreams_last_cuda_error).
void set_last_cuda_error(cudaError_t e);

// Streaming multiprocessors of the current device (cached per device).
int num_sms();

// Raises a kernel's maximum dynamic shared memory on the current device to at
// least `bytes` (the attribute is set again only for a larger request); safe
// to call from several host threads.
dreams_status_t ensure_max_dynamic_smem(const void *func, int bytes);

// The stall test hook (dreams_test_set_stall) as it applies to one kernel
// family: the index of the first withheld copy (-1: none) and the limit of
// every pipeline wait (2 s unless the hook shortens it).
void test_stall(int32_t kernel, int32_t *stall_at, uint64_t *wait_ns);

inline dreams_status_t check_launch() {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  return DREAMS_OK;
}

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

__device__ __forceinline__ void flag(int32_t *status_word, int32_t bits) {
  if (status_word != nullptr) atomicOr(status_word, bits);
}

// ---------------------------------------------------------------- tree checks
// A tree row is valid when 1 <= T <= T_max, parent[0] == -1 and
// 0 <= parent[i] < i for 0 < i < T.

// ---------------------------------------------------------------- PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// 16-byte global -> shared copy; src_bytes == 0 zero-fills the destination.
// Order-preserving integer key of an f32 bit pattern for the argmax order:
// greater value -> greater key, +0 == -0, NaN above every number.
__device__ __forceinline__ int order_key(uint32_t u) {
  const uint32_t mag = u & 0x7fffffffu;
  if (mag > 0x7f800000u) return INT_MAX;  // NaN
  if (mag == 0u) return 0;                // +0 and -0
  const int s = static_cast<int>(u);
  return s ^ ((s >> 31) & 0x7fffffff);
}

// (key, index) packed so that a 64-bit max keeps the greater key, then the
// lower index.
__device__ __forceinline__ unsigned long long pack_key_idx(int key, int idx) {
  return (static_cast<unsigned long long>(static_cast<uint32_t>(key) ^ 0x80000000u) << 32) |
         static_cast<unsigned long long>(~static_cast<uint32_t>(idx));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

}  // namespace dreams
