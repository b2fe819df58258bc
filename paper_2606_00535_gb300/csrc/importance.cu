// importance.cu -- visual-token importance and top-r selection (paper Sec. 3.2,
// "Visual Token Compression", Eq. 2): from the target's final-layer attention
// weights A [B, H, Q, K] of the prefill, the importance of visual token j is
// the mean of its attention column over heads and query positions,
//     I_j = 1 / (H Q) * sum_h sum_i A[h, i, j],
// and only the r visual tokens of highest importance are kept (the budget r
// is drawn from the pool R per forward pass; here it is an argument).
//
// Three launches, chained by programmatic dependent launch:
//   1. partial column sums, an HBM-bound reduction over the H Q rows of the
//      visual column range: CTAs over (column block, row range, sequence),
//      each thread owning 8 consecutive columns (16-byte loads from v0 rounded
//      down to 8 columns, eight rows of bf16 in flight); a CTA spans the whole
//      visual range of its rows when it fits in 1024 threads, so it reads
//      whole row segments;
//   2. the partials of each column added in a fixed tree over the row ranges
//      (the result does not depend on scheduling), scaled by 1 / (H Q);
//   3. one CTA per sequence selects the r largest by a radix select on
//      order-preserving keys (equal importances: the lower position wins) and
//      writes the kept positions in increasing order.
#include <limits.h>

#include <algorithm>

#include "common.cuh"

namespace dreams {
namespace {

constexpr int COLS_PER_THREAD = 8;
constexpr int MAX_PART_THREADS = 1024;  // a CTA covers up to 8192 columns of its rows
constexpr int SEL_THREADS = 1024;

struct ImpParams {
  const void *attn;
  int64_t H, Q, K, v0, n_vis;
  int64_t c0;         // first column read: v0 rounded down to 8, so 16-byte loads stay aligned
  int32_t col_block;  // columns per CTA (8 per thread)
  int64_t rows;       // H * Q rows per sequence
  int32_t nchunk;     // row ranges per sequence
  int64_t chunk;      // rows per range
  bool vec_ok;
  float *partial;     // [B][nchunk][n_vis]
};

template <typename T>
__device__ __forceinline__ void load8(const T *p, bool vec, int64_t n_left, float (&x)[8]) {
  if (vec && n_left >= 8) {
    if (sizeof(T) == 2) {
      const uint4 v = __ldcs(reinterpret_cast<const uint4 *>(p));
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        x[2 * i] = __uint_as_float(w[i] << 16);
        x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
      }
    } else {
      const uint4 a = __ldcs(reinterpret_cast<const uint4 *>(p));
      const uint4 b = __ldcs(reinterpret_cast<const uint4 *>(p) + 1);
      x[0] = __uint_as_float(a.x), x[1] = __uint_as_float(a.y), x[2] = __uint_as_float(a.z);
      x[3] = __uint_as_float(a.w), x[4] = __uint_as_float(b.x), x[5] = __uint_as_float(b.y);
      x[6] = __uint_as_float(b.z), x[7] = __uint_as_float(b.w);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if (i < n_left) {
        if (sizeof(T) == 2) x[i] = __uint_as_float(uint32_t(reinterpret_cast<const uint16_t *>(p)[i]) << 16);
        else x[i] = reinterpret_cast<const float *>(p)[i];
      } else {
        x[i] = 0.f;
      }
    }
  }
}

// Adds the 8 values of one 16-byte group (bf16: one word; f32: two) to acc.
template <typename T>
__device__ __forceinline__ void add_words(const uint4 *w, float (&acc)[8]) {
  if (sizeof(T) == 2) {
    const uint32_t v[4] = {w[0].x, w[0].y, w[0].z, w[0].w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      acc[2 * i] += __uint_as_float(v[i] << 16);
      acc[2 * i + 1] += __uint_as_float(v[i] & 0xffff0000u);
    }
  } else {
    acc[0] += __uint_as_float(w[0].x), acc[1] += __uint_as_float(w[0].y);
    acc[2] += __uint_as_float(w[0].z), acc[3] += __uint_as_float(w[0].w);
    acc[4] += __uint_as_float(w[1].x), acc[5] += __uint_as_float(w[1].y);
    acc[6] += __uint_as_float(w[1].z), acc[7] += __uint_as_float(w[1].w);
  }
}

// grid (column blocks, row ranges, B): partial column sums of one row range.
// Rows are loaded as raw 16-byte words, 32 words per thread in flight.
template <typename T>
__global__ void __launch_bounds__(MAX_PART_THREADS) importance_partial_kernel(const ImpParams p) {
  constexpr int WPG = int(sizeof(T)) / 2;  // words per 8-column group
  constexpr int U = 8 / WPG;               // rows in flight
  const int b = blockIdx.z, c = blockIdx.y;
  // this thread's 8 columns, absolute: col .. col + 7 (those before v0 are read, not kept)
  const int64_t col = p.c0 + int64_t(blockIdx.x) * p.col_block + threadIdx.x * COLS_PER_THREAD;
  const int64_t r0 = int64_t(c) * p.chunk, r1 = std::min<int64_t>(p.rows, r0 + p.chunk);
  const int64_t n_left = p.v0 + p.n_vis - col;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (n_left > 0) {
    const T *base = static_cast<const T *>(p.attn) + (int64_t(b) * p.rows) * p.K + col;
    int64_t r = r0;
    // 16-byte loads whenever the 8 columns lie inside the row (columns past the
    // visual range are read and not kept)
    if (p.vec_ok && col + 8 <= p.K) {
      for (; r + U <= r1; r += U) {
        uint4 w[U][WPG];
#pragma unroll
        for (int u = 0; u < U; ++u)
#pragma unroll
          for (int q = 0; q < WPG; ++q) w[u][q] = __ldcs(reinterpret_cast<const uint4 *>(base + (r + u) * p.K) + q);
#pragma unroll
        for (int u = 0; u < U; ++u) add_words<T>(w[u], acc);
      }
    }
    // the remainder (and a group cut by the end of the row): scalar loads,
    // still four rows in flight
    for (; r + 4 <= r1; r += 4) {
      float x[4][8];
#pragma unroll
      for (int u = 0; u < 4; ++u) load8<T>(base + (r + u) * p.K, p.vec_ok, n_left, x[u]);
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] += x[u][i];
    }
    for (; r < r1; ++r) {
      float x[8];
      load8<T>(base + r * p.K, p.vec_ok, n_left, x);
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] += x[i];
    }
    float *out = p.partial + (int64_t(b) * p.nchunk + c) * p.n_vis;
#pragma unroll
    for (int i = 0; i < 8; ++i)
      if (i < n_left && col + i >= p.v0) out[col + i - p.v0] = acc[i];
  }
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Block-wide exclusive prefix sum of one int per thread (SEL_THREADS threads);
// also returns the total.
__device__ int block_exclusive_scan(int v, int &total) {
  __shared__ int s_w[SEL_THREADS / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) s_w[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = s_w[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    s_w[lane] = w;
  }
  __syncthreads();
  total = s_w[SEL_THREADS / 32 - 1];
  const int ex = x - v + (warp > 0 ? s_w[warp - 1] : 0);
  __syncthreads();
  return ex;
}

// grid (column groups of 32, B), block 32 x 32: importance = the sum of the
// row-range partials / (H Q). Thread (x, y) adds ranges y, y + 32, ... of
// column x; the 32 sums meet in a fixed tree.
__global__ void __launch_bounds__(1024) importance_reduce_kernel(const ImpParams p, float *importance) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  __shared__ float red[32][33];
  const int b = blockIdx.y, tx = threadIdx.x, ty = threadIdx.y;
  const int64_t n = p.n_vis;
  const int64_t j = int64_t(blockIdx.x) * 32 + tx;
  float s = 0.f;
  if (j < n) {
    const float *col = p.partial + int64_t(b) * p.nchunk * n + j;
#pragma unroll 4
    for (int c = ty; c < p.nchunk; c += 32) s += __ldcg(col + int64_t(c) * n);
  }
  red[ty][tx] = s;
  __syncthreads();
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    if (ty < o) red[ty][tx] += red[ty + o][tx];
    __syncthreads();
  }
  if (ty == 0 && j < n) importance[int64_t(b) * n + j] = red[0][tx] * (1.f / float(double(p.H) * double(p.Q)));
}

// One CTA per sequence: the r largest importances (order-preserving keys;
// equal keys: lower position first), kept positions written in increasing
// order. s_key holds n_vis keys (dynamic shared memory).
__global__ void __launch_bounds__(SEL_THREADS) importance_select_kernel(const ImpParams p, int32_t r,
                                                                        const float *importance, int32_t *keep) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  extern __shared__ uint32_t s_key[];
  __shared__ int s_hist[256];
  __shared__ uint32_t s_prefix;
  __shared__ int s_need;
  const int b = blockIdx.x, tid = threadIdx.x;
  const int64_t n = p.n_vis;
  for (int64_t j = tid; j < n; j += SEL_THREADS) {
    const float v = __ldcg(importance + int64_t(b) * n + j);
    // unsigned order key: larger value -> larger key (NaN above everything)
    s_key[j] = uint32_t(order_key(__float_as_uint(v))) ^ 0x80000000u;
  }
  __syncthreads();
  // radix select of the r-th largest key, 8 bits at a time from the top
  if (tid == 0) {
    s_prefix = 0u;
    s_need = r;
  }
  uint32_t mask = 0u;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += SEL_THREADS) s_hist[i] = 0;
    __syncthreads();
    const uint32_t prefix = s_prefix;
    for (int64_t j = tid; j < n; j += SEL_THREADS) {
      const uint32_t k = s_key[j];
      if ((k & mask) == prefix) atomicAdd(&s_hist[(k >> shift) & 255u], 1);
    }
    __syncthreads();
    if (tid < 32) {
      // the digit d where the count of keys with digits >= d first reaches
      // need, scanned from the top: lane l holds digits 8l .. 8l + 7, and the
      // lanes above it hold the larger digits
      const int lane = tid;
      int h[8], tot = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        h[i] = s_hist[8 * lane + i];
        tot += h[i];
      }
      int above = tot;  // becomes: keys with a digit in a lane above this one
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_down_sync(0xffffffffu, above, o);
        if (lane + o < 32) above += y;
      }
      above -= tot;
      const int need = s_need;
      __syncwarp();  // every lane has read s_need before one rewrites it
      const bool mine = above < need && above + tot >= need;
      if (mine) {
        int cum = above, d = 8 * lane + 7;
        for (int i = 7; i >= 0; --i) {
          d = 8 * lane + i;
          if (cum + h[i] >= need) break;
          cum += h[i];
        }
        s_need = need - cum;  // how many keys with this digit are kept
        s_prefix = prefix | (uint32_t(d) << shift);
      }
    }
    mask |= 255u << shift;
    __syncthreads();
  }
  const uint32_t thr = s_prefix;
  const int need_eq = s_need;
  // keys above the threshold are kept; of those equal to it, the need_eq
  // lowest positions. Positions go out in increasing order.
  const int64_t per = (n + SEL_THREADS - 1) / SEL_THREADS;  // contiguous positions per thread
  const int64_t j0 = std::min<int64_t>(n, tid * per), j1 = std::min<int64_t>(n, j0 + per);
  int n_eq = 0;
  for (int64_t j = j0; j < j1; ++j) n_eq += s_key[j] == thr;
  int tot_eq;
  const int eq_before = block_exclusive_scan(n_eq, tot_eq);
  int n_keep = 0, e = eq_before;
  for (int64_t j = j0; j < j1; ++j) {
    const uint32_t k = s_key[j];
    if (k > thr) ++n_keep;
    else if (k == thr) n_keep += (e++ < need_eq);
  }
  int tot_keep;
  int pos = block_exclusive_scan(n_keep, tot_keep);
  e = eq_before;
  for (int64_t j = j0; j < j1; ++j) {
    const uint32_t k = s_key[j];
    bool take = k > thr;
    if (k == thr) take = (e++ < need_eq);
    if (take) keep[int64_t(b) * r + pos++] = int32_t(p.v0 + j);
  }
}

}  // namespace
}  // namespace dreams

using namespace dreams;

namespace {
// Threads per CTA: one per 8 columns of the visual range (plus the rounding
// of v0), so that a CTA reads whole row segments, at most 1024.
int32_t part_threads(int64_t n_vis) {
  const int64_t groups = (n_vis + 7 + 7) / 8;
  return int32_t(std::min<int64_t>(MAX_PART_THREADS, (groups + 31) / 32 * 32));
}

int32_t plan_chunks(int64_t B, int64_t n_vis, int64_t rows) {
  const int64_t tpb = part_threads(n_vis);
  const int64_t cblocks = (n_vis + 7 + tpb * 8 - 1) / (tpb * 8);
  // about 48 resident warps per SM across the grid
  const int64_t target = std::max<int64_t>(1, int64_t(num_sms()) * 48 * 32 / tpb);
  int64_t nchunk = (target + B * cblocks - 1) / (B * cblocks);
  nchunk = std::max<int64_t>(1, std::min<int64_t>(nchunk, (rows + 63) / 64));  // >= 64 rows per range
  return int32_t(nchunk);
}
}  // namespace

extern "C" size_t dreams_visual_importance_workspace_size(int64_t B, int64_t H, int64_t Q, int64_t n_vis) {
  if (B < 1 || H < 1 || Q < 1 || n_vis < 1) return 0;
  const int64_t nchunk = plan_chunks(B, n_vis, H * Q);
  return (size_t(B) * size_t(nchunk) * size_t(n_vis) * 4 + 255) / 256 * 256;
}

extern "C" dreams_status_t dreams_visual_importance(const void *attn, dreams_dtype_t dtype, int64_t B, int64_t H,
                                                    int64_t Q, int64_t K, int64_t v0, int64_t n_vis, int32_t r,
                                                    float *importance, int32_t *keep, void *workspace,
                                                    size_t workspace_bytes, dreams_stream_t stream) {
  if (attn == nullptr || importance == nullptr || keep == nullptr || B < 1 || H < 1 || Q < 1 || K < 1 ||
      v0 < 0 || n_vis < 1 || v0 + n_vis > K || r < 1 || r > n_vis)
    return DREAMS_ERR_INVALID_ARG;
  if (dtype != DREAMS_F32 && dtype != DREAMS_BF16) return DREAMS_ERR_UNSUPPORTED;
  const size_t esz = dtype == DREAMS_F32 ? 4 : 2;
  if (reinterpret_cast<uintptr_t>(attn) % esz) return DREAMS_ERR_INVALID_ARG;
  if (B > 65535 || n_vis > 48 * 1024 || n_vis > INT_MAX) return DREAMS_ERR_UNSUPPORTED;  // keys in shared memory
  const size_t need = dreams_visual_importance_workspace_size(B, H, Q, n_vis);
  if (workspace == nullptr || workspace_bytes < need || !aligned16(workspace)) return DREAMS_ERR_WORKSPACE;
  ImpParams p{};
  p.attn = attn;
  p.H = H;
  p.Q = Q;
  p.K = K;
  p.v0 = v0;
  p.n_vis = n_vis;
  p.rows = H * Q;
  p.nchunk = plan_chunks(B, n_vis, p.rows);
  p.chunk = (p.rows + p.nchunk - 1) / p.nchunk;
  p.c0 = v0 & ~int64_t(7);
  p.vec_ok = aligned16(attn) && (K * int64_t(esz)) % 16 == 0;
  p.partial = static_cast<float *>(workspace);
  const int32_t tpb = part_threads(n_vis);
  p.col_block = tpb * COLS_PER_THREAD;
  const int64_t cblocks = (v0 + n_vis - p.c0 + p.col_block - 1) / p.col_block;
  if (cblocks > INT_MAX || p.nchunk > 65535) return DREAMS_ERR_UNSUPPORTED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const dim3 grid(unsigned(cblocks), unsigned(p.nchunk), unsigned(B));
  if (dtype == DREAMS_F32) importance_partial_kernel<float><<<grid, tpb, 0, s>>>(p);
  else importance_partial_kernel<__nv_bfloat16><<<grid, tpb, 0, s>>>(p);
  dreams_status_t st = check_launch();
  if (st != DREAMS_OK) return st;
  {
    cudaLaunchConfig_t rc = {};
    rc.gridDim = dim3(unsigned((n_vis + 31) / 32), unsigned(B));
    rc.blockDim = dim3(32, 32);
    rc.stream = s;
    cudaLaunchAttribute ra[1];
    ra[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    ra[0].val.programmaticStreamSerializationAllowed = 1;
    rc.attrs = ra;
    rc.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&rc, importance_reduce_kernel, p, importance);
    if (e != cudaSuccess) {
      set_last_cuda_error(e);
      return DREAMS_ERR_CUDA;
    }
    st = check_launch();
    if (st != DREAMS_OK) return st;
  }
  const size_t smem = size_t(n_vis) * 4;
  st = ensure_max_dynamic_smem(reinterpret_cast<const void *>(importance_select_kernel), 48 * 1024 * 4);
  if (st != DREAMS_OK) return st;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(B));
  cfg.blockDim = dim3(SEL_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e =
      cudaLaunchKernelEx(&cfg, importance_select_kernel, p, r, static_cast<const float *>(importance), keep);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  return check_launch();
}
