// verify.cu -- the verification tail: per-node vocabulary argmax (the target's
// greedy prediction, paper Sec. 2 "Speculative decoding" at temperature 0),
// greedy acceptance over the draft tree (Sec. 2, generalised from a chain to
// the longest matching root path), and KV compaction of the accepted nodes
// (the cache persists across decoding steps, Sec. 2 "Vision-Language Models").
//
// Argmax: one CTA per (row, vocabulary chunk). Each thread walks 16-byte
// vectors in increasing order, reduces a vector to its maximum with
// NaN-propagating max instructions, and keeps the first vector holding its
// best value; the winning element inside that vector is found by re-reading it
// at the end. Values are compared through an order-preserving integer key
// (NaN above +inf, -0 equal to +0); ties go to the lower index, so any
// reduction tree gives the same answer. Chunks of one row meet in a 64-bit
// atomicMax of (key, ~index); the last chunk to finish (ticket counter, no
// waiting) writes the index and resets the slot and the counter.
//
// Acceptance: one warp per sequence. Pointer jumping gives every node its
// depth, whether its whole root path matches, and its ancestor set; the
// longest matching depth n is a warp max; the lexicographically smallest path
// to depth n is walked top-down through the union of the candidate paths.
//
// Compaction: one thread per (layer, K or V, KV head, 16-byte column). A path
// from the walk starts at 0 and increases, so source slot path[x] >= x and a
// thread that reads its sources before writing them (batches of 8, batch by
// batch in increasing x) never overwrites a slot it still has to read.
//
// The fused step is two launches: the argmax over the rows of real tree nodes,
// then, one CTA per sequence and chained by programmatic dependent launch, the
// walk and the compaction. Kept apart, the argmax kernel needs few registers,
// so every CTA of a large batch is resident at once.
#include <limits.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"

namespace dreams {
namespace {

constexpr int ARGMAX_THREADS = 256;
constexpr int TAIL_THREADS = 256;

// ------------------------------------------------------------------ keys
__device__ __forceinline__ int order_key(uint32_t u) {
  const uint32_t mag = u & 0x7fffffffu;
  if (mag > 0x7f800000u) return INT_MAX;  // NaN
  if (mag == 0u) return 0;                // +0 and -0
  const int s = static_cast<int>(u);
  return s ^ ((s >> 31) & 0x7fffffff);
}

__device__ __forceinline__ bool better(int ka, int ia, int kb, int ib) {
  return ka > kb || (ka == kb && ia < ib);
}

__device__ __forceinline__ uint32_t bmax2_nan(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float d;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
  return d;
}
// 2^x by the hardware approximation (ex2.approx, subnormals flushed to zero).
__device__ __forceinline__ float exp2f_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <typename T>
struct Elem;
template <>
struct Elem<float> {
  static constexpr int VEC = 4;
  __device__ static uint32_t bits(const float *p, int64_t i) { return __float_as_uint(p[i]); }
  __device__ static int vec_key(const uint4 &v) {
    const float m = fmax_nan(fmax_nan(__uint_as_float(v.x), __uint_as_float(v.y)),
                             fmax_nan(__uint_as_float(v.z), __uint_as_float(v.w)));
    return order_key(__float_as_uint(m));
  }
  __device__ static uint32_t lane_bits(const uint4 &v, int j) {
    return j == 0 ? v.x : j == 1 ? v.y : j == 2 ? v.z : v.w;
  }
};
template <>
struct Elem<__nv_bfloat16> {
  static constexpr int VEC = 8;
  __device__ static uint32_t bits(const __nv_bfloat16 *p, int64_t i) {
    return uint32_t(reinterpret_cast<const uint16_t *>(p)[i]) << 16;
  }
  __device__ static int vec_key(const uint4 &v) {
    uint32_t m = bmax2_nan(bmax2_nan(v.x, v.y), bmax2_nan(v.z, v.w));
    m = bmax2_nan(m, __byte_perm(m, 0, 0x1032));
    return order_key(m << 16);
  }
  __device__ static uint32_t lane_bits(const uint4 &v, int j) {
    const uint32_t w = j < 2 ? v.x : j < 4 ? v.y : j < 6 ? v.z : v.w;
    return (j & 1) ? (w & 0xffff0000u) : (w << 16);
  }
};

// Best (key, index) of row[begin, end) over the CTA; every thread gets it.
template <typename T>
__device__ void block_argmax(const T *row, int64_t begin, int64_t end, bool vec_ok, int &out_key,
                             int &out_idx) {
  using E = Elem<T>;
  constexpr int VEC = E::VEC;
  const int tid = threadIdx.x;
  int bk = INT_MIN, bi = INT_MAX;
  int64_t vend = begin;
  if (vec_ok) {
    const int64_t nvec = (end - begin) / VEC;
    vend = begin + nvec * VEC;
    const uint4 *vp = reinterpret_cast<const uint4 *>(row + begin);
    int64_t best_v = -1;
    int64_t vi = tid;
    constexpr int U = 4;
    for (; vi + (U - 1) * ARGMAX_THREADS < nvec; vi += U * ARGMAX_THREADS) {
      uint4 x[U];
#pragma unroll
      for (int u = 0; u < U; ++u) x[u] = __ldcs(vp + vi + u * ARGMAX_THREADS);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int k = E::vec_key(x[u]);
        if (k > bk) {
          bk = k;
          best_v = vi + u * ARGMAX_THREADS;
        }
      }
    }
    for (; vi < nvec; vi += ARGMAX_THREADS) {
      const int k = E::vec_key(__ldcs(vp + vi));
      if (k > bk) {
        bk = k;
        best_v = vi;
      }
    }
    if (best_v >= 0) {
      const uint4 x = __ldg(vp + best_v);
#pragma unroll
      for (int j = VEC - 1; j >= 0; --j)
        if (order_key(E::lane_bits(x, j)) == bk) bi = int(begin + best_v * VEC + j);
    }
  }
  for (int64_t i = vend + tid; i < end; i += ARGMAX_THREADS) {
    const int k = order_key(E::bits(row, i));
    if (better(k, int(i), bk, bi)) {
      bk = k;
      bi = int(i);
    }
  }
  // warp, then block reduction
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const int ok = __shfl_xor_sync(0xffffffffu, bk, off);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
    if (better(ok, oi, bk, bi)) {
      bk = ok;
      bi = oi;
    }
  }
  __shared__ int s_k[ARGMAX_THREADS / 32], s_i[ARGMAX_THREADS / 32];
  const int warp = tid >> 5, lane = tid & 31;
  if (lane == 0) {
    s_k[warp] = bk;
    s_i[warp] = bi;
  }
  __syncthreads();
  if (warp == 0) {
    bk = lane < ARGMAX_THREADS / 32 ? s_k[lane] : INT_MIN;
    bi = lane < ARGMAX_THREADS / 32 ? s_i[lane] : INT_MAX;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const int ok = __shfl_xor_sync(0xffffffffu, bk, off);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
      if (better(ok, oi, bk, bi)) {
        bk = ok;
        bi = oi;
      }
    }
    if (lane == 0) {
      s_k[0] = bk;
      s_i[0] = bi;
    }
  }
  __syncthreads();
  out_key = s_k[0];
  out_idx = s_i[0];
  __syncthreads();
}

__device__ __forceinline__ unsigned long long pack_key_idx(int key, int idx) {
  return (static_cast<unsigned long long>(static_cast<uint32_t>(key) ^ 0x80000000u) << 32) |
         static_cast<unsigned long long>(~static_cast<uint32_t>(idx));
}

// Combines one chunk's winner into the row's slot. Returns true (and the
// row's index) in the CTA that finished the row last.
__device__ bool row_combine(int nchunk, unsigned long long *slot, int32_t *cnt, int key, int idx,
                            int &row_idx) {
  __shared__ int s_last;
  if (nchunk == 1) {
    row_idx = idx;
    return true;
  }
  if (threadIdx.x == 0) {
    atomicMax(slot, pack_key_idx(key, idx));
    __threadfence();
    const int last = atomicAdd(cnt, 1) == nchunk - 1;
    if (last) {
      __threadfence();
      const unsigned long long v = atomicExch(slot, 0ull);
      *cnt = 0;
      s_last = ~static_cast<uint32_t>(v & 0xffffffffull);
    } else {
      s_last = -1;
    }
  }
  __syncthreads();
  row_idx = s_last;
  return row_idx >= 0;
}

struct ArgmaxParams {
  const void *logits;
  int64_t V, row_stride, chunk;
  int32_t nchunk;
  bool vec_ok;
  int32_t *out;
  unsigned long long *slot;
  int32_t *cnt;
};

template <typename T>
__global__ void __launch_bounds__(ARGMAX_THREADS) vocab_argmax_kernel(const ArgmaxParams p) {
  const int64_t row = blockIdx.x / p.nchunk;
  const int c = blockIdx.x % p.nchunk;
  const T *base = static_cast<const T *>(p.logits) + row * p.row_stride;
  const int64_t begin = c * p.chunk, end = std::min<int64_t>(p.V, begin + p.chunk);
  int key, idx, row_idx;
  block_argmax<T>(base, begin, end, p.vec_ok, key, idx);
  if (row_combine(p.nchunk, p.slot + row, p.cnt + row, key, idx, row_idx) && threadIdx.x == 0)
    p.out[row] = row_idx;
}


// ------------------------------------------------------------------ temperature sampling
// One draw per row from softmax(x / tau) by inverse transform with the row's
// uniform u (the target's own sample, paper Sec. 2 "Speculative decoding";
// Table 2, Temperature = 1). A row is cut into segments of SEG consecutive
// values, one warp per segment, 8 values per lane.
//   stage 1 (data-parallel over rows x segment ranges): per segment its
//     maximum m (NaN-propagating) and s = sum of 2^((x - m) k), k = log2(e) /
//     tau, each lane summing its 8 values in index order, then a xor-shuffle
//     tree over the lanes;
//   stage 2 (one warp per row): the row maximum M over the segments; Z = the
//     segments' s scaled by 2^((m - M) k), summed in segment order (each lane
//     a contiguous block, then an inclusive warp scan); the segment where the
//     running sum first exceeds u Z; that segment re-read in index order and
//     the value where the running sum crosses.
// Where fp32 rounding leaves the crossing just past a segment's total, the
// draw is the segment's last value of positive weight. Rows holding a NaN, with
// maximum +inf, or with every value -inf take their argmax.
constexpr int SEG = 256;
constexpr int SAMPLE_THREADS = 256;  // stage 1: 8 warps, each one segment at a time

struct SampleParams {
  const void *logits;
  int64_t V, row_stride;
  int32_t nseg;         // segments per row
  int32_t seg_per_cta;  // segments per stage-1 CTA
  int32_t ncta_row;     // stage-1 CTAs per row
  float k2;             // log2(e) / tau
  bool vec_ok;          // rows start 16-byte aligned
  const float *u;       // [rows]
  float2 *seg;          // [rows][nseg] (m, s)
};

// The 8 values of this lane in segment g (elements g * SEG + 8 lane + i), as
// floats; values at or past V read as -inf.
template <typename T>
__device__ __forceinline__ void seg_load(const T *row, int64_t V, bool vec_ok, int64_t g, float (&x)[8]) {
  const int lane = threadIdx.x & 31;
  const int64_t e0 = g * SEG + 8 * lane;
  if (vec_ok && e0 + 8 <= V) {
    if (sizeof(T) == 2) {
      const uint4 v = __ldcs(reinterpret_cast<const uint4 *>(row + e0));
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        x[2 * i] = __uint_as_float(w[i] << 16);
        x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
      }
    } else {
      const uint4 a = __ldcs(reinterpret_cast<const uint4 *>(row + e0));
      const uint4 b = __ldcs(reinterpret_cast<const uint4 *>(row + e0) + 1);
      x[0] = __uint_as_float(a.x), x[1] = __uint_as_float(a.y), x[2] = __uint_as_float(a.z);
      x[3] = __uint_as_float(a.w), x[4] = __uint_as_float(b.x), x[5] = __uint_as_float(b.y);
      x[6] = __uint_as_float(b.z), x[7] = __uint_as_float(b.w);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) x[i] = e0 + i < V ? __uint_as_float(Elem<T>::bits(row, e0 + i)) : -INFINITY;
  }
}

// Lane sum of 2^((x - m) k) over its 8 values, in index order.
__device__ __forceinline__ float seg_lane_sum(const float (&x)[8], float m, float k2) {
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) s += exp2f_approx((x[i] - m) * k2);
  return s;
}

// Stage 1 for segments [g0, g1) of one row: warp w takes g0 + w, g0 + w + 8, ...
template <typename T>
__device__ void sample_stats(const SampleParams &p, const T *row, float2 *seg_row, int64_t g0, int64_t g1) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int NW = SAMPLE_THREADS / 32;
  int64_t g = g0 + warp;
  for (; g + NW < g1; g += 2 * NW) {  // two segments in flight per warp
    float xa[8], xb[8];
    seg_load<T>(row, p.V, p.vec_ok, g, xa);
    seg_load<T>(row, p.V, p.vec_ok, g + NW, xb);
    float ma = xa[0], mb = xb[0];
#pragma unroll
    for (int i = 1; i < 8; ++i) {
      ma = fmax_nan(ma, xa[i]);
      mb = fmax_nan(mb, xb[i]);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      ma = fmax_nan(ma, __shfl_xor_sync(0xffffffffu, ma, off));
      mb = fmax_nan(mb, __shfl_xor_sync(0xffffffffu, mb, off));
    }
    float sa = seg_lane_sum(xa, ma, p.k2), sb = seg_lane_sum(xb, mb, p.k2);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      sa += __shfl_xor_sync(0xffffffffu, sa, off);
      sb += __shfl_xor_sync(0xffffffffu, sb, off);
    }
    if (lane == 0) {
      seg_row[g] = make_float2(ma, sa);
      seg_row[g + NW] = make_float2(mb, sb);
    }
  }
  for (; g < g1; g += NW) {
    float x[8];
    seg_load<T>(row, p.V, p.vec_ok, g, x);
    float m = x[0];
#pragma unroll
    for (int i = 1; i < 8; ++i) m = fmax_nan(m, x[i]);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = fmax_nan(m, __shfl_xor_sync(0xffffffffu, m, off));
    float s = seg_lane_sum(x, m, p.k2);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) seg_row[g] = make_float2(m, s);
  }
}

// Stage 2 for one row (one warp): returns the draw. seg_row was written by
// stage 1 (possibly by other CTAs of a completed grid: read through L2).
template <typename T>
__device__ int sample_select_warp(const SampleParams &p, const T *row, const float2 *seg_row, float u) {
  const int lane = threadIdx.x & 31;
  const int nseg = p.nseg;
  const int q = (nseg + 31) / 32;
  const int gb = min(nseg, lane * q), ge = min(nseg, gb + q);  // this lane's block of segments
  float lm = -INFINITY;
  for (int g = gb; g < ge; ++g) lm = fmax_nan(lm, __ldcg(seg_row + g).x);
  float M = lm;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) M = fmax_nan(M, __shfl_xor_sync(0xffffffffu, M, off));
  if (M == -INFINITY) return 0;  // every value -inf: the argmax is index 0
  if (isnan(M) || M == INFINITY) {
    // degenerate: the first NaN, else the first +inf (the argmax order)
    int first = INT_MAX;
    for (int g = gb; g < ge && first == INT_MAX; ++g) {
      const float m = __ldcg(seg_row + g).x;
      if (isnan(M) ? isnan(m) : m == INFINITY) first = g;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) first = min(first, __shfl_xor_sync(0xffffffffu, first, off));
    if (first == INT_MAX) return 0;
    float x[8];
    seg_load<T>(row, p.V, false, first, x);
    int hit = 8;
#pragma unroll
    for (int i = 7; i >= 0; --i)
      if (isnan(M) ? isnan(x[i]) : x[i] == INFINITY) hit = i;
    const unsigned bal = __ballot_sync(0xffffffffu, hit < 8);
    const int l0 = __ffs(bal) - 1;
    return first * SEG + 8 * l0 + __shfl_sync(0xffffffffu, hit, l0);
  }
  // weights of this lane's segments in the row's scale, their block sum, and
  // an inclusive scan over the lanes (segment order)
  float wsum = 0.f;
  for (int g = gb; g < ge; ++g) {
    const float2 ms = __ldcg(seg_row + g);
    if (ms.x != -INFINITY) wsum += ms.y * exp2f_approx((ms.x - M) * p.k2);
  }
  float inc = wsum;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, inc, off);
    if (lane >= off) inc += y;
  }
  const float Z = __shfl_sync(0xffffffffu, inc, 31);
  const float uc = u > 0.f ? fminf(u, 1.f) : 0.f;  // NaN and negatives count as 0
  const float t = uc * Z;
  const unsigned cross = __ballot_sync(0xffffffffu, inc > t);
  int gs = -1;         // segment holding the draw
  float r = 0.f;       // what is left of t at the start of that segment, in its own scale
  bool tail = false;   // no crossing: take the last value of positive weight
  if (cross) {
    const int L = __ffs(cross) - 1;
    if (lane == L) {
      float acc = inc - wsum;
      int last = -1;
      float last_r = 0.f;
      for (int g = gb; g < ge; ++g) {
        const float2 ms = __ldcg(seg_row + g);
        if (ms.x == -INFINITY) continue;
        const float sc = exp2f_approx((ms.x - M) * p.k2);
        const float c = ms.y * sc;
        if (c > 0.f) {
          last = g;
          last_r = fmaxf(t - acc, 0.f) / sc;
        }
        if (acc + c > t) {
          gs = g;
          r = fmaxf(t - acc, 0.f) / sc;  // >= 0: the draw has positive weight
          break;
        }
        acc += c;
      }
      if (gs < 0) {
        gs = last;
        r = last_r;
        tail = true;
      }
    }
    gs = __shfl_sync(0xffffffffu, gs, L);
    r = __shfl_sync(0xffffffffu, r, L);
    tail = __shfl_sync(0xffffffffu, tail, L);
  } else {
    // t >= Z (u = 1, or rounding): the last segment of positive weight
    int last = -1;
    for (int g = gb; g < ge; ++g) {
      const float2 ms = __ldcg(seg_row + g);
      if (ms.x != -INFINITY && ms.y * exp2f_approx((ms.x - M) * p.k2) > 0.f) last = g;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) last = max(last, __shfl_xor_sync(0xffffffffu, last, off));
    gs = last;
    tail = true;
  }
  if (gs < 0) return 0;
  // the segment again, in index order, in its own scale
  const float m = __ldcg(seg_row + gs).x;
  float x[8];
  seg_load<T>(row, p.V, p.vec_ok, gs, x);
  float w[8], ls = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    w[i] = exp2f_approx((x[i] - m) * p.k2);
    ls += w[i];
  }
  float linc = ls;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, linc, off);
    if (lane >= off) linc += y;
  }
  int pick = -1;
  const unsigned lc = tail ? 0u : __ballot_sync(0xffffffffu, linc > r);
  if (lc) {
    const int L = __ffs(lc) - 1;
    if (lane == L) {
      float acc = linc - ls;
      for (int i = 0; i < 8; ++i) {
        acc += w[i];
        if (w[i] > 0.f) pick = i;
        if (acc > r) {
          pick = i;
          break;
        }
      }
    }
    pick = __shfl_sync(0xffffffffu, pick, L);
    return gs * SEG + 8 * (__ffs(lc) - 1) + pick;
  }
  // the segment's last value of positive weight
  int li = -1;
#pragma unroll
  for (int i = 0; i < 8; ++i)
    if (w[i] > 0.f) li = i;
  const unsigned has = __ballot_sync(0xffffffffu, li >= 0);
  if (!has) return gs * SEG;
  const int L = 31 - __clz(has);
  return gs * SEG + 8 * L + __shfl_sync(0xffffffffu, li, L);
}

template <typename T>
__global__ void __launch_bounds__(SAMPLE_THREADS) vocab_sample_stats_kernel(const SampleParams p) {
  const int64_t row = blockIdx.x / p.ncta_row;
  const int c = blockIdx.x % p.ncta_row;
  const T *base = static_cast<const T *>(p.logits) + row * p.row_stride;
  const int64_t g0 = int64_t(c) * p.seg_per_cta, g1 = std::min<int64_t>(p.nseg, g0 + p.seg_per_cta);
  sample_stats<T>(p, base, p.seg + row * p.nseg, g0, g1);
}

template <typename T>
__global__ void __launch_bounds__(256) vocab_sample_select_kernel(const SampleParams p, int64_t rows, int32_t *out) {
  const int64_t row = int64_t(blockIdx.x) * 8 + (threadIdx.x >> 5);
  if (row >= rows) return;
  const T *base = static_cast<const T *>(p.logits) + row * p.row_stride;
  const int idx = sample_select_warp<T>(p, base, p.seg + row * p.nseg, __ldg(p.u + row));
  if ((threadIdx.x & 31) == 0) out[row] = idx;
}

// ------------------------------------------------------------------ tree walk
struct WalkOut {
  int n;    // drafts accepted (-1: bad sequence)
  int bad;  // data-error bits
};

// One warp. Reads the sequence's parent / tokens / predictions, writes the
// accepted path into s_path[0..n]. Pred rows may have been written by other
// CTAs of this grid, so they are read through L2.
__device__ WalkOut tree_walk_warp(const int32_t *par_row, const int32_t *tok_row, const int32_t *pred_row, int T,
                                  int max_path, int32_t *s_path) {
  __shared__ int s_good[64], s_dist[64], s_jump[64];
  __shared__ unsigned long long s_anc[64];
  const int lane = threadIdx.x & 31;
  int par[2], tok[2], pred[2], bad = 0;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int i = lane + 32 * h;
    par[h] = (i < T) ? __ldg(par_row + i) : -1;
    tok[h] = (i < T) ? __ldg(tok_row + i) : 0;
    pred[h] = (i < T) ? __ldcg(pred_row + i) : 0;
    if (i == 0) bad |= (par[h] != -1);
    else if (i < T) bad |= (par[h] < 0 || par[h] >= i);
  }
  if (__any_sync(0xffffffffu, bad)) return {-1, DREAMS_DATA_BAD_PARENT};
  // pred of each node's parent, through shared memory
  __shared__ int s_pred[64];
  s_pred[lane] = pred[0];
  s_pred[lane + 32] = pred[1];
  __syncwarp();
  int good[2], dist[2], jump[2];
  unsigned long long anc[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int i = lane + 32 * h;
    const bool live = i < T;
    good[h] = (i == 0) ? 1 : (live && tok[h] == s_pred[par[h]]);
    dist[h] = (i == 0 || !live) ? 0 : 1;
    jump[h] = live ? par[h] : -1;
    anc[h] = 1ull << i;
    s_good[i] = good[h];
    s_dist[i] = dist[h];
    s_jump[i] = jump[h];
    s_anc[i] = anc[h];
  }
  __syncwarp();
  for (int r = 0; r < 6; ++r) {
    int gg[2], dd[2], jj[2];
    unsigned long long aa[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int j = jump[h];
      gg[h] = j >= 0 ? s_good[j] : 1;
      dd[h] = j >= 0 ? s_dist[j] : 0;
      jj[h] = j >= 0 ? s_jump[j] : -1;
      aa[h] = j >= 0 ? s_anc[j] : 0ull;
    }
    __syncwarp();
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int i = lane + 32 * h;
      good[h] &= gg[h];
      dist[h] += dd[h];
      jump[h] = jj[h];
      anc[h] |= aa[h];
      s_good[i] = good[h];
      s_dist[i] = dist[h];
      s_jump[i] = jump[h];
      s_anc[i] = anc[h];
    }
    __syncwarp();
  }
  // longest matching depth, cut to max_path - 1 drafts
  int n = 0;
#pragma unroll
  for (int h = 0; h < 2; ++h)
    if (lane + 32 * h < T && good[h]) n = max(n, dist[h]);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) n = max(n, __shfl_xor_sync(0xffffffffu, n, off));
  n = min(n, max_path - 1);
  // union of the root paths of the candidates (matching nodes at depth >= n)
  unsigned long long mark = 0ull;
#pragma unroll
  for (int h = 0; h < 2; ++h)
    if (lane + 32 * h < T && good[h] && dist[h] >= n) mark |= anc[h];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mark |= __shfl_xor_sync(0xffffffffu, mark, off);
  // top-down: lowest marked child at each level
  int cur = 0;
  if (lane == 0) s_path[0] = 0;
  for (int k = 1; k <= n; ++k) {
    const unsigned lo = __ballot_sync(0xffffffffu, par[0] == cur && ((mark >> lane) & 1ull));
    const unsigned hi = __ballot_sync(0xffffffffu, par[1] == cur && ((mark >> (lane + 32)) & 1ull));
    cur = lo ? (__ffs(lo) - 1) : (__ffs(hi) + 31);
    if (lane == 0) s_path[k] = cur;
  }
  __syncwarp();
  return {n, 0};
}

// Writes accept_len, path, out_tokens and new_kv_len of sequence b (warp).
__device__ void write_walk(int b, int n, int L, const int32_t *tok_row, const int32_t *pred_row, const int32_t *s_path,
                           int max_path, int32_t *accept_len, int32_t *path, int32_t *out_tokens,
                           int32_t *new_kv_len) {
  const int lane = threadIdx.x & 31;
  for (int k = lane; k < max_path; k += 32) {
    int pv = -1, ov = -1;
    if (n >= 0 && k <= n) {
      pv = s_path[k];
      ov = (k < n) ? __ldg(tok_row + s_path[k + 1]) : __ldcg(pred_row + s_path[n]);
    }
    path[int64_t(b) * max_path + k] = pv;
    out_tokens[int64_t(b) * max_path + k] = ov;
  }
  if (lane == 0) {
    accept_len[b] = n >= 0 ? n + 1 : 0;
    new_kv_len[b] = n >= 0 ? L + n + 1 : L;
  }
}

// ------------------------------------------------------------------ compaction
struct KVParams {
  uint4 *k;  // 16-byte columns
  uint4 *v;
  int32_t n_layers;
  int64_t layer_stride16;  // in 16-byte units
  int32_t Hkv, ch;         // ch = D / 8 columns per head row
  int32_t capacity;
  const int32_t *page_table;
  int32_t pages_per_seq, num_pages;
};

// 16-byte unit offset of (b, slot s, head 0, column 0); -1 for a bad page.
__device__ __forceinline__ int64_t slot_off16(const KVParams &kv, int b, int s) {
  if (kv.page_table == nullptr) return (int64_t(b) * kv.capacity + s) * kv.Hkv * kv.ch;
  const int pg = __ldg(kv.page_table + int64_t(b) * kv.pages_per_seq + (s >> 6));
  if (pg < 0 || pg >= kv.num_pages) return -1;
  return (int64_t(pg) * 64 + (s & 63)) * kv.Hkv * kv.ch;
}

// Slot offsets of the moves of sequence b into s_src / s_dst (x = 1 .. n),
// computed by one warp; returns false (and flags) on a bad page.
__device__ bool move_offsets(const KVParams &kv, int b, int L, int n, const int32_t *s_path, int64_t *s_src,
                             int64_t *s_dst, int32_t *status) {
  const int lane = threadIdx.x & 31;
  int bad = 0;
  for (int x = 1 + lane; x <= n; x += 32) {
    const int64_t so = slot_off16(kv, b, L + s_path[x]);
    const int64_t dst = slot_off16(kv, b, L + x);
    bad |= (so < 0 || dst < 0);
    s_src[x] = so;
    s_dst[x] = dst;
  }
  bad = __any_sync(0xffffffffu, bad);
  if (bad && lane == 0) flag(status, DREAMS_DATA_BAD_PAGE);
  __syncwarp();
  return !bad;
}

// Moves of one sequence over units [u0, u_end) with stride ustep.
__device__ void compact_units(const KVParams &kv, int n, const int64_t *s_src, const int64_t *s_dst, int64_t u0,
                              int64_t ustep) {
  const int64_t per_layer = int64_t(2) * kv.Hkv * kv.ch;
  const int64_t units = per_layer * kv.n_layers;
  for (int64_t u = u0; u < units; u += ustep) {
    const int layer = int(u / per_layer);
    int64_t r = u - layer * per_layer;
    const int which = int(r / (int64_t(kv.Hkv) * kv.ch));
    r -= int64_t(which) * kv.Hkv * kv.ch;  // head * ch + column
    uint4 *base = (which ? kv.v : kv.k) + layer * kv.layer_stride16 + r;
    for (int x0 = 1; x0 <= n; x0 += 8) {
      uint4 tmp[8];
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (x0 + j <= n) tmp[j] = __ldcg(base + s_src[x0 + j]);
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (x0 + j <= n) base[s_dst[x0 + j]] = tmp[j];
    }
  }
}

// ------------------------------------------------------------------ kernels
struct TreeParams {
  const int32_t *parent, *tokens, *tree_len, *kv_len;
  int32_t B, T_max;
};

__global__ void __launch_bounds__(32) accept_path_kernel(const int32_t *pred, const TreeParams tr, int max_path,
                                                         int32_t *accept_len, int32_t *path, int32_t *out_tokens,
                                                         int32_t *new_kv_len, int32_t *status) {
  __shared__ int32_t s_path[65];
  const int b = blockIdx.x;
  const int T = __ldg(tr.tree_len + b), L = __ldg(tr.kv_len + b);
  const int64_t rb = int64_t(b) * tr.T_max;
  WalkOut w{-1, 0};
  if (T < 1 || T > tr.T_max) w.bad = DREAMS_DATA_BAD_TREE_LEN;
  else if (L < 0) w.bad = DREAMS_DATA_BAD_KV_LEN;
  else w = tree_walk_warp(tr.parent + rb, tr.tokens + rb, pred + rb, T, max_path, s_path);
  if (w.bad) {
    w.n = -1;
    if (threadIdx.x == 0) flag(status, w.bad);
  }
  write_walk(b, w.n, L, tr.tokens + rb, pred + rb, s_path, max_path, accept_len, path, out_tokens, new_kv_len);
}

__global__ void __launch_bounds__(TAIL_THREADS) kv_compact_kernel(const KVParams kv, const int32_t *kv_len,
                                                                  const int32_t *accept_len, const int32_t *path,
                                                                  int max_path, int32_t *status) {
  __shared__ int32_t s_path[65];
  __shared__ int64_t s_src[65], s_dst[65];
  __shared__ int s_ok;
  const int b = blockIdx.y;
  const int A = __ldg(accept_len + b), L = __ldg(kv_len + b);
  if (A <= 0) return;
  const bool report = blockIdx.x == 0;
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    int bad = 0;
    if (A > max_path || L < 0) {
      bad = DREAMS_DATA_BAD_KV_LEN;
    } else {
      for (int x = lane; x < A; x += 32) {
        const int pv = __ldg(path + int64_t(b) * max_path + x);
        const int prev = x ? __ldg(path + int64_t(b) * max_path + x - 1) : -1;
        s_path[x] = pv;
        if ((x == 0 && pv != 0) || (x > 0 && pv <= prev)) bad |= DREAMS_DATA_BAD_PATH;
      }
      bad = __reduce_or_sync(0xffffffffu, bad);
      if (!bad && int64_t(L) + __ldg(path + int64_t(b) * max_path + A - 1) >= kv.capacity)
        bad = DREAMS_DATA_BAD_KV_LEN;
    }
    __syncwarp();
    if (bad) {
      if (lane == 0 && report) flag(status, bad);
    } else if (!move_offsets(kv, b, L, A - 1, s_path, s_src, s_dst, report ? status : nullptr)) {
      bad = DREAMS_DATA_BAD_PAGE;
    }
    if (lane == 0) s_ok = !bad;
  }
  __syncthreads();
  if (!s_ok) return;
  compact_units(kv, A - 1, s_src, s_dst, int64_t(blockIdx.x) * blockDim.x + threadIdx.x,
                int64_t(gridDim.x) * blockDim.x);
}

struct StepParams {
  ArgmaxParams am;
  SampleParams sp;
  bool sampled;  // predictions are draws at temperature tau (sp), not argmaxes (am)
  TreeParams tr;
  KVParams kv;
  int32_t max_path;
  int32_t *pred;  // [B, T_max] predictions (caller's argmax_out or workspace)
  bool pred_in_ws;
  int32_t *accept_len, *path, *out_tokens, *new_kv_len;
  int32_t *status;
};

// Launch 1 of the verification tail. grid.x = B * T_max * nchunk: (sequence,
// tree node, vocabulary chunk); CTAs of padding nodes return at once. The CTA
// that completes a node's row writes the node's prediction.
template <typename T>
__global__ void __launch_bounds__(ARGMAX_THREADS) verify_rows_kernel(const StepParams p) {
  // the walk kernel may start now: it waits for this grid to complete
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int nchunk = p.am.nchunk;
  const int c = blockIdx.x % nchunk;
  const int rowg = blockIdx.x / nchunk;
  const int b = rowg / p.tr.T_max, i = rowg % p.tr.T_max;
  const int tl = __ldg(p.tr.tree_len + b);
  if (tl < 1 || tl > p.tr.T_max || i >= tl) return;
  const int64_t rb = int64_t(b) * p.tr.T_max;
  const T *row = static_cast<const T *>(p.am.logits) + (rb + i) * p.am.row_stride;
  const int64_t begin = c * p.am.chunk, end = std::min<int64_t>(p.am.V, begin + p.am.chunk);
  int key, idx, row_idx;
  block_argmax<T>(row, begin, end, p.am.vec_ok, key, idx);
  if (row_combine(nchunk, p.am.slot + rb + i, p.am.cnt + rb + i, key, idx, row_idx) && threadIdx.x == 0)
    p.pred[rb + i] = row_idx;
}

// Launch 1 of the sampled verification tail. grid.x = B * T_max * ncta_row:
// (sequence, tree node, segment range); padding nodes return at once. Stage 1
// of the draw (segment statistics) of the node's row.
template <typename T>
__global__ void __launch_bounds__(SAMPLE_THREADS) verify_sample_rows_kernel(const StepParams p) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int ncta = p.sp.ncta_row;
  const int c = blockIdx.x % ncta;
  const int rowg = blockIdx.x / ncta;
  const int b = rowg / p.tr.T_max, i = rowg % p.tr.T_max;
  const int tl = __ldg(p.tr.tree_len + b);
  if (tl < 1 || tl > p.tr.T_max || i >= tl) return;
  const int64_t r = int64_t(b) * p.tr.T_max + i;
  const T *row = static_cast<const T *>(p.sp.logits) + r * p.sp.row_stride;
  const int64_t g0 = int64_t(c) * p.sp.seg_per_cta, g1 = std::min<int64_t>(p.sp.nseg, g0 + p.sp.seg_per_cta);
  sample_stats<T>(p.sp, row, p.sp.seg + r * p.sp.nseg, g0, g1);
}

// Launch 2 of the verification tail, one CTA per sequence, chained to launch 1
// by programmatic dependent launch (it may start early and waits until launch
// 1 has completed): the acceptance walk, its outputs, and the KV compaction.
template <typename LT>
__global__ void __launch_bounds__(TAIL_THREADS) verify_tail_kernel(const StepParams p) {
  __shared__ int32_t s_path[65];
  __shared__ int64_t s_src[65], s_dst[65];
  __shared__ int s_n;
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int b = blockIdx.x, Tm = p.tr.T_max;
  const int64_t rb = int64_t(b) * Tm;
  const int T = __ldg(p.tr.tree_len + b);
  const int L = __ldg(p.tr.kv_len + b);
  if (p.sampled && T >= 1 && T <= Tm) {
    // stage 2 of the draws: one warp per node row
    for (int i = threadIdx.x >> 5; i < T; i += TAIL_THREADS / 32) {
      const int64_t r = rb + i;
      const LT *row = static_cast<const LT *>(p.sp.logits) + r * p.sp.row_stride;
      const int idx = sample_select_warp<LT>(p.sp, row, p.sp.seg + r * p.sp.nseg, __ldg(p.sp.u + r));
      if ((threadIdx.x & 31) == 0) p.pred[r] = idx;
    }
    __syncthreads();
  }
  if (threadIdx.x < 32) {
    WalkOut w{-1, 0};
    if (T < 1 || T > Tm) w.bad = DREAMS_DATA_BAD_TREE_LEN;
    else if (L < 0 || L > p.kv.capacity - T) w.bad = DREAMS_DATA_BAD_KV_LEN;
    else w = tree_walk_warp(p.tr.parent + rb, p.tr.tokens + rb, p.pred + rb, T, p.max_path, s_path);
    if (w.bad) {
      w.n = -1;
      if (threadIdx.x == 0) flag(p.status, w.bad);
    }
    write_walk(b, w.n, L, p.tr.tokens + rb, p.pred + rb, s_path, p.max_path, p.accept_len, p.path, p.out_tokens,
               p.new_kv_len);
    if (p.pred_in_ws && T >= 1 && T <= Tm) {  // leave the workspace zero-filled
      __syncwarp();
      for (int x = threadIdx.x; x < T; x += 32) p.pred[rb + x] = 0;
    }
    bool ok = w.n > 0;
    if (ok) ok = move_offsets(p.kv, b, L, w.n, s_path, s_src, s_dst, p.status);
    if (threadIdx.x == 0) s_n = ok ? w.n : 0;
  }
  __syncthreads();
  const int n = s_n;
  if (n > 0) compact_units(p.kv, n, s_src, s_dst, threadIdx.x, blockDim.x);
}

// ------------------------------------------------------------------ host side
inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct ArgmaxPlan {
  int64_t chunk;
  int32_t nchunk;
};

ArgmaxPlan plan_argmax(int64_t rows, int64_t V) {
  // aim for about four CTAs per SM across the grid, chunks of >= 4096 elements
  const int64_t target = int64_t(num_sms()) * 4;
  int64_t nchunk = (target + rows - 1) / std::max<int64_t>(rows, 1);
  nchunk = std::max<int64_t>(1, std::min<int64_t>(nchunk, (V + 4095) / 4096));
  int64_t chunk = (V + nchunk - 1) / nchunk;
  chunk = (chunk + 7) / 8 * 8;  // keep chunk starts on 16-byte boundaries
  nchunk = (V + chunk - 1) / chunk;
  return {chunk, int32_t(nchunk)};
}

size_t argmax_ws(int64_t rows) { return align_up(size_t(rows) * 8, 256) + align_up(size_t(rows) * 4, 256); }

struct SamplePlan {
  int32_t nseg, seg_per_cta, ncta_row;
};

SamplePlan plan_sample(int64_t rows, int64_t V) {
  // about four stage-1 CTAs per SM across the grid, >= 8 segments per CTA
  const int64_t nseg = (V + SEG - 1) / SEG;
  const int64_t target = int64_t(num_sms()) * 4;
  int64_t ncta = (target + rows - 1) / std::max<int64_t>(rows, 1);
  ncta = std::max<int64_t>(1, std::min<int64_t>(ncta, (nseg + 7) / 8));
  const int64_t per = (nseg + ncta - 1) / ncta;
  return {int32_t(nseg), int32_t(per), int32_t((nseg + per - 1) / per)};
}

size_t sample_ws(int64_t rows, int64_t V) { return align_up(size_t(rows) * size_t((V + SEG - 1) / SEG) * 8, 256); }

// Checks and fills the sampling parameters shared by both entry points.
bool sample_params(const void *logits, dreams_dtype_t dtype, int64_t rows, int64_t V, int64_t row_stride,
                   float temperature, const float *uniforms, void *seg_ws, SampleParams &p, int64_t &ctas) {
  const float k2 = 1.4426950408889634f / temperature;
  if (!(temperature > 0.f) || !isfinite(temperature) || !isfinite(k2) || uniforms == nullptr) return false;
  const size_t esz = dtype == DREAMS_F32 ? 4 : 2;
  const SamplePlan pl = plan_sample(rows, V);
  p.logits = logits;
  p.V = V;
  p.row_stride = row_stride;
  p.nseg = pl.nseg;
  p.seg_per_cta = pl.seg_per_cta;
  p.ncta_row = pl.ncta_row;
  p.k2 = k2;
  p.vec_ok = aligned16(logits) && (row_stride * int64_t(esz)) % 16 == 0;
  p.u = uniforms;
  p.seg = static_cast<float2 *>(seg_ws);
  ctas = rows * pl.ncta_row;
  return true;
}

bool kv_params(const dreams_kv_cache_t *kv, KVParams &out) {
  if (kv == nullptr || kv->k == nullptr || kv->v == nullptr || kv->n_layers < 1 || kv->Hkv < 1 ||
      kv->capacity < 1 || kv->layer_stride < 0)
    return false;
  if (kv->D < 8 || kv->D % 8 != 0) return false;
  if (!aligned16(kv->k) || !aligned16(kv->v) || (kv->layer_stride * 2) % 16 != 0) return false;
  if (kv->page_table != nullptr &&
      (kv->page_size != 64 || kv->pages_per_seq < 1 || kv->num_pages < 1 ||
       int64_t(kv->pages_per_seq) * 64 != kv->capacity))
    return false;
  out.k = static_cast<uint4 *>(kv->k);
  out.v = static_cast<uint4 *>(kv->v);
  out.n_layers = kv->n_layers;
  out.layer_stride16 = kv->layer_stride * 2 / 16;
  out.Hkv = kv->Hkv;
  out.ch = kv->D / 8;
  out.capacity = kv->capacity;
  out.page_table = kv->page_table;
  out.pages_per_seq = kv->pages_per_seq;
  out.num_pages = kv->num_pages;
  return true;
}

bool tree_params(const dreams_tree_t *tree, bool need_tokens, TreeParams &out) {
  if (tree == nullptr || tree->parent == nullptr || tree->tree_len == nullptr || tree->kv_len == nullptr ||
      (need_tokens && tree->tokens == nullptr) || tree->B < 1 || tree->T_max < 1 || tree->T_max > 64)
    return false;
  out = {tree->parent, tree->tokens, tree->tree_len, tree->kv_len, tree->B, tree->T_max};
  return true;
}

}  // namespace
}  // namespace dreams

using namespace dreams;

extern "C" size_t dreams_vocab_argmax_workspace_size(int64_t rows, int64_t V) {
  if (rows < 1 || V < 1) return 0;
  return plan_argmax(rows, V).nchunk > 1 ? argmax_ws(rows) : 0;
}

extern "C" dreams_status_t dreams_vocab_argmax(const void *logits, dreams_dtype_t dtype, int64_t rows, int64_t V,
                                               int64_t row_stride, int32_t *out_idx, void *workspace,
                                               size_t workspace_bytes, dreams_stream_t stream) {
  if (logits == nullptr || out_idx == nullptr || rows < 1 || V < 1 || V > INT_MAX || row_stride < V)
    return DREAMS_ERR_INVALID_ARG;
  if (dtype != DREAMS_F32 && dtype != DREAMS_BF16) return DREAMS_ERR_UNSUPPORTED;
  const size_t esz = dtype == DREAMS_F32 ? 4 : 2;
  if (reinterpret_cast<uintptr_t>(logits) % esz) return DREAMS_ERR_INVALID_ARG;
  const ArgmaxPlan pl = plan_argmax(rows, V);
  if (rows * pl.nchunk > INT_MAX) return DREAMS_ERR_UNSUPPORTED;
  ArgmaxParams p{};
  p.logits = logits;
  p.V = V;
  p.row_stride = row_stride;
  p.chunk = pl.chunk;
  p.nchunk = pl.nchunk;
  p.vec_ok = aligned16(logits) && (row_stride * int64_t(esz)) % 16 == 0;
  p.out = out_idx;
  if (pl.nchunk > 1) {
    if (workspace == nullptr || workspace_bytes < argmax_ws(rows) || !aligned16(workspace))
      return DREAMS_ERR_WORKSPACE;
    p.slot = static_cast<unsigned long long *>(workspace);
    p.cnt = reinterpret_cast<int32_t *>(static_cast<uint8_t *>(workspace) + align_up(size_t(rows) * 8, 256));
  }
  const dim3 grid(unsigned(rows * pl.nchunk));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (dtype == DREAMS_F32) vocab_argmax_kernel<float><<<grid, ARGMAX_THREADS, 0, s>>>(p);
  else vocab_argmax_kernel<__nv_bfloat16><<<grid, ARGMAX_THREADS, 0, s>>>(p);
  return check_launch();
}

extern "C" dreams_status_t dreams_accept_path(const int32_t *argmax, const dreams_tree_t *tree, int32_t max_path,
                                              int32_t *accept_len, int32_t *path, int32_t *out_tokens,
                                              int32_t *new_kv_len, int32_t *status_word, dreams_stream_t stream) {
  TreeParams tr;
  if (argmax == nullptr || !tree_params(tree, true, tr) || max_path < 1 || accept_len == nullptr ||
      path == nullptr || out_tokens == nullptr || new_kv_len == nullptr)
    return DREAMS_ERR_INVALID_ARG;
  accept_path_kernel<<<tree->B, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      argmax, tr, max_path, accept_len, path, out_tokens, new_kv_len, status_word);
  return check_launch();
}

extern "C" dreams_status_t dreams_kv_compact(const dreams_kv_cache_t *kv, int32_t B, const int32_t *kv_len,
                                             const int32_t *accept_len, const int32_t *path, int32_t max_path,
                                             int32_t *status_word, dreams_stream_t stream) {
  KVParams kp;
  if (!kv_params(kv, kp) || B < 1 || B > 65535 || kv_len == nullptr || accept_len == nullptr ||
      path == nullptr || max_path < 1 || max_path > 65)
    return DREAMS_ERR_INVALID_ARG;
  const int64_t units = int64_t(2) * kv->n_layers * kv->Hkv * (kv->D / 8);
  const int64_t blocks = std::min<int64_t>((units + TAIL_THREADS - 1) / TAIL_THREADS, 1024);
  kv_compact_kernel<<<dim3(unsigned(blocks), B), TAIL_THREADS, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      kp, kv_len, accept_len, path, max_path, status_word);
  return check_launch();
}

extern "C" size_t dreams_verify_step_workspace_size(const dreams_tree_t *tree, int64_t V) {
  if (tree == nullptr || tree->B < 1 || tree->T_max < 1 || V < 1) return 0;
  const int64_t rows = int64_t(tree->B) * tree->T_max;
  return argmax_ws(rows) + align_up(size_t(rows) * 4, 256);
}

extern "C" dreams_status_t dreams_verify_step(const void *logits, dreams_dtype_t dtype, int64_t V,
                                              int64_t row_stride, const dreams_tree_t *tree,
                                              const dreams_kv_cache_t *kv, int32_t max_path, int32_t *argmax_out,
                                              int32_t *accept_len, int32_t *path, int32_t *out_tokens,
                                              int32_t *new_kv_len, void *workspace, size_t workspace_bytes,
                                              int32_t *status_word, dreams_stream_t stream) {
  StepParams p{};
  if (logits == nullptr || V < 1 || V > INT_MAX || row_stride < V || !tree_params(tree, true, p.tr) ||
      !kv_params(kv, p.kv) || max_path < 1 || max_path > 65 || accept_len == nullptr || path == nullptr ||
      out_tokens == nullptr || new_kv_len == nullptr)
    return DREAMS_ERR_INVALID_ARG;
  if (dtype != DREAMS_F32 && dtype != DREAMS_BF16) return DREAMS_ERR_UNSUPPORTED;
  const size_t esz = dtype == DREAMS_F32 ? 4 : 2;
  if (reinterpret_cast<uintptr_t>(logits) % esz) return DREAMS_ERR_INVALID_ARG;
  const int64_t rows = int64_t(tree->B) * tree->T_max;
  const size_t need = dreams_verify_step_workspace_size(tree, V);
  if (workspace == nullptr || workspace_bytes < need || !aligned16(workspace)) return DREAMS_ERR_WORKSPACE;
  const ArgmaxPlan pl = plan_argmax(rows, V);
  if (rows * pl.nchunk > INT_MAX) return DREAMS_ERR_UNSUPPORTED;
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  p.am.logits = logits;
  p.am.V = V;
  p.am.row_stride = row_stride;
  p.am.chunk = pl.chunk;
  p.am.nchunk = pl.nchunk;
  p.am.vec_ok = aligned16(logits) && (row_stride * int64_t(esz)) % 16 == 0;
  p.am.slot = reinterpret_cast<unsigned long long *>(ws);
  p.am.cnt = reinterpret_cast<int32_t *>(ws + align_up(size_t(rows) * 8, 256));
  int32_t *ws_pred = reinterpret_cast<int32_t *>(ws + argmax_ws(rows));
  p.pred = argmax_out != nullptr ? argmax_out : ws_pred;
  p.pred_in_ws = argmax_out == nullptr;
  p.max_path = max_path;
  p.accept_len = accept_len;
  p.path = path;
  p.out_tokens = out_tokens;
  p.new_kv_len = new_kv_len;
  p.status = status_word;
  const dim3 grid(unsigned(rows * pl.nchunk));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (dtype == DREAMS_F32) verify_rows_kernel<float><<<grid, ARGMAX_THREADS, 0, s>>>(p);
  else verify_rows_kernel<__nv_bfloat16><<<grid, ARGMAX_THREADS, 0, s>>>(p);
  dreams_status_t st = check_launch();
  if (st != DREAMS_OK) return st;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(tree->B));
  cfg.blockDim = dim3(TAIL_THREADS);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = dtype == DREAMS_F32 ? cudaLaunchKernelEx(&cfg, verify_tail_kernel<float>, p)
                                             : cudaLaunchKernelEx(&cfg, verify_tail_kernel<__nv_bfloat16>, p);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  return check_launch();
}

extern "C" size_t dreams_vocab_sample_workspace_size(int64_t rows, int64_t V) {
  if (rows < 1 || V < 1) return 0;
  return sample_ws(rows, V);
}

extern "C" dreams_status_t dreams_vocab_sample(const void *logits, dreams_dtype_t dtype, int64_t rows, int64_t V,
                                               int64_t row_stride, float temperature, const float *uniforms,
                                               int32_t *out_idx, void *workspace, size_t workspace_bytes,
                                               dreams_stream_t stream) {
  if (logits == nullptr || out_idx == nullptr || rows < 1 || V < 1 || V > INT_MAX - SEG || row_stride < V)
    return DREAMS_ERR_INVALID_ARG;
  if (dtype != DREAMS_F32 && dtype != DREAMS_BF16) return DREAMS_ERR_UNSUPPORTED;
  const size_t esz = dtype == DREAMS_F32 ? 4 : 2;
  if (reinterpret_cast<uintptr_t>(logits) % esz || (reinterpret_cast<uintptr_t>(uniforms) & 3))
    return DREAMS_ERR_INVALID_ARG;
  if (workspace == nullptr || workspace_bytes < sample_ws(rows, V) || !aligned16(workspace))
    return DREAMS_ERR_WORKSPACE;
  SampleParams p{};
  int64_t ctas = 0;
  if (!sample_params(logits, dtype, rows, V, row_stride, temperature, uniforms, workspace, p, ctas))
    return DREAMS_ERR_INVALID_ARG;
  if (ctas > INT_MAX || (rows + 7) / 8 > INT_MAX) return DREAMS_ERR_UNSUPPORTED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const dim3 g1(static_cast<unsigned>(ctas)), g2(static_cast<unsigned>((rows + 7) / 8));
  if (dtype == DREAMS_F32) {
    vocab_sample_stats_kernel<float><<<g1, SAMPLE_THREADS, 0, s>>>(p);
    vocab_sample_select_kernel<float><<<g2, 256, 0, s>>>(p, rows, out_idx);
  } else {
    vocab_sample_stats_kernel<__nv_bfloat16><<<g1, SAMPLE_THREADS, 0, s>>>(p);
    vocab_sample_select_kernel<__nv_bfloat16><<<g2, 256, 0, s>>>(p, rows, out_idx);
  }
  return check_launch();
}

extern "C" size_t dreams_verify_step_sampled_workspace_size(const dreams_tree_t *tree, int64_t V) {
  if (tree == nullptr || tree->B < 1 || tree->T_max < 1 || V < 1) return 0;
  const int64_t rows = int64_t(tree->B) * tree->T_max;
  return sample_ws(rows, V) + align_up(size_t(rows) * 4, 256);
}

extern "C" dreams_status_t dreams_verify_step_sampled(
    const void *logits, dreams_dtype_t dtype, int64_t V, int64_t row_stride, const dreams_tree_t *tree,
    const dreams_kv_cache_t *kv, int32_t max_path, float temperature, const float *uniforms, int32_t *sample_out,
    int32_t *accept_len, int32_t *path, int32_t *out_tokens, int32_t *new_kv_len, void *workspace,
    size_t workspace_bytes, int32_t *status_word, dreams_stream_t stream) {
  StepParams p{};
  if (logits == nullptr || V < 1 || V > INT_MAX - SEG || row_stride < V || !tree_params(tree, true, p.tr) ||
      !kv_params(kv, p.kv) || max_path < 1 || max_path > 65 || accept_len == nullptr || path == nullptr ||
      out_tokens == nullptr || new_kv_len == nullptr)
    return DREAMS_ERR_INVALID_ARG;
  if (dtype != DREAMS_F32 && dtype != DREAMS_BF16) return DREAMS_ERR_UNSUPPORTED;
  const size_t esz = dtype == DREAMS_F32 ? 4 : 2;
  if (reinterpret_cast<uintptr_t>(logits) % esz || (reinterpret_cast<uintptr_t>(uniforms) & 3))
    return DREAMS_ERR_INVALID_ARG;
  const int64_t rows = int64_t(tree->B) * tree->T_max;
  const size_t need = dreams_verify_step_sampled_workspace_size(tree, V);
  if (workspace == nullptr || workspace_bytes < need || !aligned16(workspace)) return DREAMS_ERR_WORKSPACE;
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  int64_t ctas = 0;
  if (!sample_params(logits, dtype, rows, V, row_stride, temperature, uniforms, ws, p.sp, ctas))
    return DREAMS_ERR_INVALID_ARG;
  if (ctas > INT_MAX) return DREAMS_ERR_UNSUPPORTED;
  p.sampled = true;
  int32_t *ws_pred = reinterpret_cast<int32_t *>(ws + sample_ws(rows, V));
  p.pred = sample_out != nullptr ? sample_out : ws_pred;
  p.pred_in_ws = false;
  p.max_path = max_path;
  p.accept_len = accept_len;
  p.path = path;
  p.out_tokens = out_tokens;
  p.new_kv_len = new_kv_len;
  p.status = status_word;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const dim3 grid(static_cast<unsigned>(ctas));
  if (dtype == DREAMS_F32) verify_sample_rows_kernel<float><<<grid, SAMPLE_THREADS, 0, s>>>(p);
  else verify_sample_rows_kernel<__nv_bfloat16><<<grid, SAMPLE_THREADS, 0, s>>>(p);
  dreams_status_t st = check_launch();
  if (st != DREAMS_OK) return st;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(tree->B));
  cfg.blockDim = dim3(TAIL_THREADS);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = dtype == DREAMS_F32 ? cudaLaunchKernelEx(&cfg, verify_tail_kernel<float>, p)
                                             : cudaLaunchKernelEx(&cfg, verify_tail_kernel<__nv_bfloat16>, p);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  return check_launch();
}

// ------------------------------------------------------------------ no-allocation argmax
// Scratch of dreams_vocab_argmax_noalloc: a fixed file-scope device array that
// every GPU loading this library holds until the process exits. Host code
// must not hand g_noalloc_scratch to a kernel directly (in host code that
// name is a host-side stand-in, not a device address): its device address is
// looked up with cudaGetSymbolAddress once per device.
namespace {
constexpr int64_t NOALLOC_ROWS = DREAMS_NOALLOC_ARGMAX_MAX_ROWS;
constexpr size_t NOALLOC_SLOT_BYTES = size_t(NOALLOC_ROWS) * 8;  // one (key, index) word per row
constexpr size_t NOALLOC_BYTES = NOALLOC_SLOT_BYTES + size_t(NOALLOC_ROWS) * 4;
static __device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_BYTES];

std::mutex g_noalloc_mutex;
void *g_noalloc_ptr[64] = {nullptr};

// Device address of the scratch on the current device (looked up on the first
// call per device, which must happen outside any stream capture).
dreams_status_t noalloc_scratch(void **out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  if (dev < 0 || dev >= 64) return DREAMS_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  if (g_noalloc_ptr[dev] == nullptr) {
    void *ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess || ptr == nullptr) {
      set_last_cuda_error(e);
      return DREAMS_ERR_CUDA;
    }
    g_noalloc_ptr[dev] = ptr;
  }
  *out = g_noalloc_ptr[dev];
  return DREAMS_OK;
}
}  // namespace

extern "C" dreams_status_t dreams_vocab_argmax_noalloc(const void *logits, dreams_dtype_t dtype, int64_t rows,
                                                       int64_t V, int64_t row_stride, int32_t *out_idx,
                                                       dreams_stream_t stream) {
  if (logits == nullptr || out_idx == nullptr || rows < 1 || V < 1 || V > INT_MAX || row_stride < V)
    return DREAMS_ERR_INVALID_ARG;
  if (dtype != DREAMS_F32 && dtype != DREAMS_BF16) return DREAMS_ERR_UNSUPPORTED;
  if (rows > NOALLOC_ROWS) return DREAMS_ERR_SCRATCH_LIMIT;
  const size_t esz = dtype == DREAMS_F32 ? 4 : 2;
  if (reinterpret_cast<uintptr_t>(logits) % esz) return DREAMS_ERR_INVALID_ARG;
  const ArgmaxPlan pl = plan_argmax(rows, V);
  if (rows * pl.nchunk > INT_MAX) return DREAMS_ERR_UNSUPPORTED;
  void *scratch = nullptr;
  dreams_status_t st = noalloc_scratch(&scratch);
  if (st != DREAMS_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  ArgmaxParams p{};
  p.logits = logits;
  p.V = V;
  p.row_stride = row_stride;
  p.chunk = pl.chunk;
  p.nchunk = pl.nchunk;
  p.vec_ok = aligned16(logits) && (row_stride * int64_t(esz)) % 16 == 0;
  p.out = out_idx;
  p.slot = static_cast<unsigned long long *>(scratch);
  p.cnt = reinterpret_cast<int32_t *>(static_cast<uint8_t *>(scratch) + NOALLOC_SLOT_BYTES);
  if (pl.nchunk > 1) {
    // the row slots and counters must start at zero
    cudaError_t e = cudaMemsetAsync(p.slot, 0, size_t(rows) * 8, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(p.cnt, 0, size_t(rows) * 4, s);
    if (e != cudaSuccess) {
      set_last_cuda_error(e);
      return DREAMS_ERR_CUDA;
    }
  }
  const dim3 grid(unsigned(rows * pl.nchunk));
  if (dtype == DREAMS_F32) vocab_argmax_kernel<float><<<grid, ARGMAX_THREADS, 0, s>>>(p);
  else vocab_argmax_kernel<__nv_bfloat16><<<grid, ARGMAX_THREADS, 0, s>>>(p);
  return check_launch();
}
