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
// Table 2, Temperature = 1). A row is cut into segments of SEG = 1024
// consecutive values, one warp per segment; a segment is four steps of SUB =
// 256 values, 8 consecutive values per lane in each step.
//   stage 1 (data-parallel over rows x segment ranges): per segment its
//     maximum m (NaN-propagating) and s = sum of 2^((x - m) k), k = log2(e) /
//     tau (lane sums, then a xor-shuffle tree);
//   stage 2 (a second launch, one warp per row): the row maximum M and the
//     total Z over the segments; the segment where the running sum, in
//     segment order, first exceeds u Z; that segment re-read step by step in
//     index order and the value where the running sum crosses.
// Stage 1 keeps each lane's values as raw 16-byte words (the maximum of bf16
// data by packed max instructions) so that it needs few registers and many
// CTAs stream at once.
// Where fp32 rounding leaves the crossing just past a segment's total, the
// draw is the last value of positive weight before it. Rows holding a NaN,
// with maximum +inf, or with every value -inf take their argmax.
constexpr int SUB = 256;
constexpr int SEG = 4 * SUB;
constexpr int SAMPLE_THREADS = 256;  // stage 1: 8 warps, each one segment at a time

struct SampleParams {
  const void *logits;
  int64_t V, row_stride;
  int32_t nseg;         // segments per row
  int32_t seg_per_cta;  // segments per CTA
  int32_t ncta_row;     // CTAs per row
  float k2;             // log2(e) / tau
  bool vec_ok;          // rows start 16-byte aligned
  const float *u;       // [rows]
  float2 *seg;          // [rows][nseg] (m, s)
};

// The 8 values of this lane in step j of the row (elements j * SUB + 8 lane +
// i), as floats; values at or past V read as -inf.
template <typename T>
__device__ __forceinline__ void sub_load(const T *row, int64_t V, bool vec_ok, int64_t j, float (&x)[8]) {
  const int lane = threadIdx.x & 31;
  const int64_t e0 = j * SUB + 8 * lane;
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

// Raw 16-byte words of this lane in step j of the row (elements j * SUB + 8
// lane + i): one word of 8 bf16 values, or two of 4 f32 values; values at or
// past V read as -inf.
template <typename T>
__device__ __forceinline__ void sub_words(const T *row, int64_t V, bool vec_ok, int64_t j, uint4 (&w)[sizeof(T) / 2]) {
  const int lane = threadIdx.x & 31;
  const int64_t e0 = j * SUB + 8 * lane;
  if (vec_ok && e0 + 8 <= V) {
#pragma unroll
    for (int q = 0; q < int(sizeof(T)) / 2; ++q) w[q] = __ldcs(reinterpret_cast<const uint4 *>(row + e0) + q);
  } else {
    uint32_t b[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) b[i] = e0 + i < V ? Elem<T>::bits(row, e0 + i) : 0xff800000u;  // -inf
    if (sizeof(T) == 2) {
      w[0] = make_uint4((b[0] >> 16) | (b[1] & 0xffff0000u), (b[2] >> 16) | (b[3] & 0xffff0000u),
                        (b[4] >> 16) | (b[5] & 0xffff0000u), (b[6] >> 16) | (b[7] & 0xffff0000u));
    } else {
#pragma unroll
      for (int q = 0; q < int(sizeof(T)) / 2; ++q) w[q] = make_uint4(b[4 * q], b[4 * q + 1], b[4 * q + 2], b[4 * q + 3]);
    }
  }
}

// Maximum (NaN-propagating) and the sum of 2^((x - m) k) of raw words.
__device__ __forceinline__ float words_max(const uint4 *w, int n, bool bf16) {
  if (bf16) {
    uint32_t a = bmax2_nan(bmax2_nan(w[0].x, w[0].y), bmax2_nan(w[0].z, w[0].w));
    for (int q = 1; q < n; ++q) a = bmax2_nan(a, bmax2_nan(bmax2_nan(w[q].x, w[q].y), bmax2_nan(w[q].z, w[q].w)));
    a = bmax2_nan(a, __byte_perm(a, 0, 0x1032));
    return __uint_as_float(a << 16);
  }
  float m = fmax_nan(fmax_nan(__uint_as_float(w[0].x), __uint_as_float(w[0].y)),
                     fmax_nan(__uint_as_float(w[0].z), __uint_as_float(w[0].w)));
  for (int q = 1; q < n; ++q)
    m = fmax_nan(m, fmax_nan(fmax_nan(__uint_as_float(w[q].x), __uint_as_float(w[q].y)),
                             fmax_nan(__uint_as_float(w[q].z), __uint_as_float(w[q].w))));
  return m;
}
__device__ __forceinline__ float words_sum(const uint4 *w, int n, bool bf16, float m, float k2) {
  float s = 0.f;
  for (int q = 0; q < n; ++q) {
    const uint32_t v[4] = {w[q].x, w[q].y, w[q].z, w[q].w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (bf16) {
        s += exp2f_approx((__uint_as_float(v[i] << 16) - m) * k2);
        s += exp2f_approx((__uint_as_float(v[i] & 0xffff0000u) - m) * k2);
      } else {
        s += exp2f_approx((__uint_as_float(v[i]) - m) * k2);
      }
    }
  }
  return s;
}

// Stage 1 for segments [g0, g1) of one row: warp w takes g0 + w, g0 + w + 8,
// ..., one segment (4 or 8 words per lane) at a time.
template <typename T>
__device__ void sample_stats(const SampleParams &p, const T *row, float2 *seg_row, int64_t g0, int64_t g1) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int NW = SAMPLE_THREADS / 32;
  constexpr int WPS = 4 * (int(sizeof(T)) / 2);  // words per lane per segment
  constexpr int SPI = 1;                         // segments per iteration
  constexpr bool BF = sizeof(T) == 2;
  for (int64_t g = g0 + warp; g < g1; g += SPI * NW) {
    uint4 w[SPI][WPS];
#pragma unroll
    for (int k = 0; k < SPI; ++k) {
      const int64_t gk = g + k * NW;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        uint4(&wj)[sizeof(T) / 2] = *reinterpret_cast<uint4(*)[sizeof(T) / 2]>(&w[k][j * (sizeof(T) / 2)]);
        if (gk < g1) sub_words<T>(row, p.V, p.vec_ok, 4 * gk + j, wj);
        else
#pragma unroll
          for (int q = 0; q < int(sizeof(T)) / 2; ++q) {
            const uint32_t ninf = BF ? 0xff80ff80u : 0xff800000u;  // -inf
            wj[q] = make_uint4(ninf, ninf, ninf, ninf);
          }
      }
    }
    float m[SPI], sum[SPI];
#pragma unroll
    for (int k = 0; k < SPI; ++k) m[k] = words_max(w[k], WPS, BF);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
#pragma unroll
      for (int k = 0; k < SPI; ++k) m[k] = fmax_nan(m[k], __shfl_xor_sync(0xffffffffu, m[k], off));
#pragma unroll
    for (int k = 0; k < SPI; ++k) sum[k] = words_sum(w[k], WPS, BF, m[k], p.k2);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1)
#pragma unroll
      for (int k = 0; k < SPI; ++k) sum[k] += __shfl_xor_sync(0xffffffffu, sum[k], off);
    if (lane == 0) {
#pragma unroll
      for (int k = 0; k < SPI; ++k)
        if (g + k * NW < g1) seg_row[g + k * NW] = make_float2(m[k], sum[k]);
    }
  }
}

// The 8 segment statistics of this lane in batch `base` (segments base + 8 lane
// .. base + 8 lane + 7), loaded together; past nseg: (-inf, 0).
__device__ __forceinline__ void seg_batch(const float2 *seg_row, int nseg, int base, float2 (&v)[8]) {
  const int g0 = base + 8 * (threadIdx.x & 31);
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = g0 + i < nseg ? __ldcg(seg_row + g0 + i) : make_float2(-INFINITY, 0.f);
}

// Stage 2 for one row (one warp): returns the draw. seg_row was written by
// stage 1 (by other CTAs too: read through L2). The statistics are read in
// batches of 256 segments, 8 consecutive ones per lane: one pass for the row
// maximum M, the total Z (online rescaling per lane, then a shuffle tree) and
// the first NaN or +inf segment; one pass for the running sums in segment
// order (an inclusive warp scan per batch plus the carry of earlier batches)
// up to the crossing; then the crossing segment's values.
template <typename T>
__device__ int sample_select_warp(const SampleParams &p, const T *row, const float2 *seg_row, float u) {
  const int lane = threadIdx.x & 31;
  const int nseg = p.nseg;
  const float k2 = p.k2;
  // ---- pass 1: M, Z, and the first segment whose maximum is NaN / +inf
  float m_l = -INFINITY, z_l = 0.f;
  int first_nan = INT_MAX, first_inf = INT_MAX;
  for (int base = 0; base < nseg; base += 256) {
    float2 v[8];
    seg_batch(seg_row, nseg, base, v);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int g = base + 8 * lane + i;
      if (isnan(v[i].x)) {
        first_nan = min(first_nan, g);
      } else if (v[i].x == INFINITY) {
        first_inf = min(first_inf, g);
      } else if (v[i].x != -INFINITY) {
        if (v[i].x > m_l) {
          z_l = (m_l == -INFINITY ? 0.f : z_l * exp2f_approx((m_l - v[i].x) * k2)) + v[i].y;
          m_l = v[i].x;
        } else {
          z_l += v[i].y * exp2f_approx((v[i].x - m_l) * k2);
        }
      }
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    first_nan = min(first_nan, __shfl_xor_sync(0xffffffffu, first_nan, off));
    first_inf = min(first_inf, __shfl_xor_sync(0xffffffffu, first_inf, off));
  }
  if (first_nan != INT_MAX || first_inf != INT_MAX) {
    // degenerate: the first NaN, else the first +inf (the argmax order)
    const bool want_nan = first_nan != INT_MAX;
    const int g = want_nan ? first_nan : first_inf;
    for (int k = 0; k < 4; ++k) {
      float x[8];
      sub_load<T>(row, p.V, false, 4 * int64_t(g) + k, x);
      int hit = 8;
#pragma unroll
      for (int i = 7; i >= 0; --i)
        if (want_nan ? isnan(x[i]) : x[i] == INFINITY) hit = i;
      const unsigned bal = __ballot_sync(0xffffffffu, hit < 8);
      if (bal) {
        const int l0 = __ffs(bal) - 1;
        return g * SEG + k * SUB + 8 * l0 + __shfl_sync(0xffffffffu, hit, l0);
      }
    }
    return g * SEG;
  }
  float M = m_l;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
  if (M == -INFINITY) return 0;  // every value -inf: the argmax is index 0
  float Z = m_l == -INFINITY ? 0.f : z_l * exp2f_approx((m_l - M) * k2);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) Z += __shfl_xor_sync(0xffffffffu, Z, off);
  const float uc = u > 0.f ? fminf(u, 1.f) : 0.f;  // NaN and negatives count as 0
  const float t = uc * Z;
  // ---- pass 2: running sums in segment order up to the crossing
  int gs = -1;        // segment holding the draw
  float r = 0.f;      // what is left of t at the start of that segment, in its own scale
  bool tail = true;   // no crossing found: take the last value of positive weight
  int last = -1;      // last segment of positive weight seen
  float carry = 0.f;
  for (int base = 0; base < nseg && gs < 0; base += 256) {
    float2 v[8];
    seg_batch(seg_row, nseg, base, v);
    float c[8], ls = 0.f;
    int llast = -1;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      c[i] = v[i].x != -INFINITY ? v[i].y * exp2f_approx((v[i].x - M) * k2) : 0.f;
      ls += c[i];
      if (c[i] > 0.f) llast = base + 8 * lane + i;
    }
    float inc = ls;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float y = __shfl_up_sync(0xffffffffu, inc, off);
      if (lane >= off) inc += y;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) llast = max(llast, __shfl_xor_sync(0xffffffffu, llast, off));
    const int last_before = last;
    if (llast >= 0) last = llast;
    const unsigned cross = __ballot_sync(0xffffffffu, carry + inc > t);
    if (cross) {
      const int L = __ffs(cross) - 1;
      int g_hit = -1, g_prev = -1;
      float r_hit = 0.f;
      if (lane == L) {
        float acc = carry + inc - ls;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (g_hit < 0 && c[i] > 0.f) {
            if (acc + c[i] > t) {
              g_hit = base + 8 * lane + i;
              r_hit = fmaxf(t - acc, 0.f) / exp2f_approx((v[i].x - M) * k2);  // >= 0: positive weight
            } else {
              g_prev = base + 8 * lane + i;
            }
          }
          acc += c[i];
        }
      }
      g_hit = __shfl_sync(0xffffffffu, g_hit, L);
      r_hit = __shfl_sync(0xffffffffu, r_hit, L);
      g_prev = __shfl_sync(0xffffffffu, g_prev, L);
      if (g_hit >= 0) {
        gs = g_hit;
        r = r_hit;
        tail = false;
      } else {
        // rounding left the crossing just past lane L's segments: the last
        // positive one up to there
        int lp = -1;
        for (int i = 0; i < 8; ++i)
          if (c[i] > 0.f && base + 8 * lane + i < base + 8 * L) lp = base + 8 * lane + i;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) lp = max(lp, __shfl_xor_sync(0xffffffffu, lp, off));
        gs = g_prev >= 0 ? g_prev : (lp >= 0 ? lp : last_before);
      }
    }
    carry += __shfl_sync(0xffffffffu, inc, 31);
  }
  if (gs < 0) gs = last;  // t >= every running sum (u = 1, or rounding)
  if (gs < 0) return 0;
  // ---- the crossing segment again, step by step in index order, in its own scale
  const float m = __ldcg(seg_row + gs).x;
  float acc = 0.f;
  int last_i = -1;  // last value of positive weight seen (index)
  for (int k = 0; k < 4; ++k) {
    float x[8];
    sub_load<T>(row, p.V, p.vec_ok, 4 * int64_t(gs) + k, x);
    float w[8], ls = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      w[i] = exp2f_approx((x[i] - m) * k2);
      ls += w[i];
    }
    float linc = ls;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float y = __shfl_up_sync(0xffffffffu, linc, off);
      if (lane >= off) linc += y;
    }
    const int base_e = gs * SEG + k * SUB + 8 * lane;
    const unsigned lc = tail ? 0u : __ballot_sync(0xffffffffu, acc + linc > r);
    if (lc) {
      const int L = __ffs(lc) - 1;
      int pick = -1;
      if (lane == L) {
        float a = acc + linc - ls;
        bool done = false;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          a += w[i];
          if (!done && w[i] > 0.f) {
            pick = base_e + i;
            done = a > r;
          }
        }
      }
      pick = __shfl_sync(0xffffffffu, pick, L);
      if (pick >= 0) return pick;
    }
    int li = -1;
#pragma unroll
    for (int i = 0; i < 8; ++i)
      if (w[i] > 0.f) li = base_e + i;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) li = max(li, __shfl_xor_sync(0xffffffffu, li, off));
    if (li >= 0) last_i = li;
    acc += __shfl_sync(0xffffffffu, linc, 31);
  }
  // no crossing in the segment (t at its very end, or u = 1): its last value
  // of positive weight
  return last_i >= 0 ? last_i : gs * SEG;
}

template <typename T>
__global__ void __launch_bounds__(SAMPLE_THREADS, sizeof(T) == 2 ? 6 : 4) vocab_sample_stats_kernel(const SampleParams p) {
  const int64_t r = blockIdx.x / p.ncta_row;
  const int c = blockIdx.x % p.ncta_row;
  const int64_t g0 = int64_t(c) * p.seg_per_cta, g1 = std::min<int64_t>(p.nseg, g0 + p.seg_per_cta);
  sample_stats<T>(p, static_cast<const T *>(p.logits) + r * p.row_stride, p.seg + r * p.nseg, g0, g1);
  // the selection grid may launch as this one drains
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Stage 2, one warp per row, chained to stage 1 by programmatic dependent
// launch (it waits until stage 1 has completed).
template <typename T>
__global__ void __launch_bounds__(256) vocab_sample_select_kernel(const SampleParams p, int64_t rows, int32_t *out) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int64_t r = int64_t(blockIdx.x) * 8 + (threadIdx.x >> 5);
  if (r >= rows) return;
  const int idx = sample_select_warp<T>(p, static_cast<const T *>(p.logits) + r * p.row_stride, p.seg + r * p.nseg,
                                        __ldg(p.u + r));
  if ((threadIdx.x & 31) == 0) out[r] = idx;
}

// ------------------------------------------------------------------ tree walk
struct WalkOut {
  int n;    // drafts accepted (-1: bad sequence)
  int bad;  // data-error bits
};

// The tree alone, one warp, two nodes per lane (i = lane, lane + 32): each
// node's parent, draft token, depth and ancestor set (itself included), by
// pointer jumping. Needs no prediction, so the verification tail computes it
// before waiting for the argmax grid.
struct TreeShape {
  int par[2], tok[2], dist[2];
  unsigned long long anc[2];
  int bad;  // DREAMS_DATA_BAD_PARENT or 0
};

__device__ TreeShape tree_shape_warp(const int32_t *par_row, const int32_t *tok_row, int T) {
  __shared__ int s_dist[64], s_jump[64];
  __shared__ unsigned long long s_anc[64];
  const int lane = threadIdx.x & 31;
  TreeShape ts;
  int bad = 0, jump[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int i = lane + 32 * h;
    const bool live = i < T;
    ts.par[h] = live ? __ldg(par_row + i) : -1;
    ts.tok[h] = live ? __ldg(tok_row + i) : 0;
    if (i == 0) bad |= (ts.par[h] != -1);
    else if (live) bad |= (ts.par[h] < 0 || ts.par[h] >= i);
  }
  ts.bad = __any_sync(0xffffffffu, bad) ? DREAMS_DATA_BAD_PARENT : 0;
  if (ts.bad) return ts;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int i = lane + 32 * h;
    const bool live = i < T;
    ts.dist[h] = (i == 0 || !live) ? 0 : 1;
    jump[h] = live ? ts.par[h] : -1;
    ts.anc[h] = 1ull << i;
    s_dist[i] = ts.dist[h];
    s_jump[i] = jump[h];
    s_anc[i] = ts.anc[h];
  }
  __syncwarp();
  for (int r = 0; r < 6; ++r) {
    int dd[2], jj[2];
    unsigned long long aa[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int j = jump[h];
      dd[h] = j >= 0 ? s_dist[j] : 0;
      jj[h] = j >= 0 ? s_jump[j] : -1;
      aa[h] = j >= 0 ? s_anc[j] : 0ull;
    }
    __syncwarp();
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int i = lane + 32 * h;
      ts.dist[h] += dd[h];
      jump[h] = jj[h];
      ts.anc[h] |= aa[h];
      s_dist[i] = ts.dist[h];
      s_jump[i] = jump[h];
      s_anc[i] = ts.anc[h];
    }
    __syncwarp();
  }
  return ts;
}

// The walk over a valid tree shape, one warp: a node matches when its draft
// token equals its parent's prediction (the root always matches); a node is
// accepted when every node of its root path matches. Writes the accepted
// path into s_path[0..n] and, when s_out is given, the tokens the step emits
// into s_out[0..n] (the accepted drafts' tokens, from the shape's registers,
// then the bonus prediction). Pred rows may have been written by other CTAs
// of this grid or by the preceding grid, so they are read through L2.
__device__ WalkOut tree_walk_finish(const TreeShape &ts, const int32_t *pred_row, int T, int max_path,
                                    int32_t *s_path, int32_t *s_out = nullptr) {
  __shared__ int s_pred[64];
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int i = lane + 32 * h;
    s_pred[i] = (i < T) ? __ldcg(pred_row + i) : 0;
  }
  __syncwarp();
  bool match[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int i = lane + 32 * h;
    match[h] = (i == 0) || (i < T && ts.tok[h] == s_pred[ts.par[h]]);
  }
  const unsigned long long mm = uint64_t(__ballot_sync(0xffffffffu, match[0])) |
                                (uint64_t(__ballot_sync(0xffffffffu, match[1])) << 32);
  bool good[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) good[h] = lane + 32 * h < T && (ts.anc[h] & ~mm) == 0ull;
  // longest matching depth, cut to max_path - 1 drafts
  int n = 0;
#pragma unroll
  for (int h = 0; h < 2; ++h)
    if (good[h]) n = max(n, ts.dist[h]);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) n = max(n, __shfl_xor_sync(0xffffffffu, n, off));
  n = min(n, max_path - 1);
  // union of the root paths of the candidates (matching nodes at depth >= n)
  unsigned long long mark = 0ull;
#pragma unroll
  for (int h = 0; h < 2; ++h)
    if (good[h] && ts.dist[h] >= n) mark |= ts.anc[h];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mark |= __shfl_xor_sync(0xffffffffu, mark, off);
  // top-down: lowest marked child at each level
  int cur = 0;
  if (lane == 0) s_path[0] = 0;
  for (int k = 1; k <= n; ++k) {
    const unsigned lo = __ballot_sync(0xffffffffu, ts.par[0] == cur && ((mark >> lane) & 1ull));
    const unsigned hi = __ballot_sync(0xffffffffu, ts.par[1] == cur && ((mark >> (lane + 32)) & 1ull));
    cur = lo ? (__ffs(lo) - 1) : (__ffs(hi) + 31);
    // node cur's token sits in lane cur % 32, slot cur / 32
    const int tk = __shfl_sync(0xffffffffu, cur < 32 ? ts.tok[0] : ts.tok[1], cur & 31);
    if (lane == 0) {
      s_path[k] = cur;
      if (s_out != nullptr) s_out[k - 1] = tk;
    }
  }
  if (lane == 0 && s_out != nullptr) s_out[n] = s_pred[cur];
  __syncwarp();
  return {n, 0};
}

// Both phases at once (the stand-alone accept walk).
__device__ WalkOut tree_walk_warp(const int32_t *par_row, const int32_t *tok_row, const int32_t *pred_row, int T,
                                  int max_path, int32_t *s_path) {
  const TreeShape ts = tree_shape_warp(par_row, tok_row, T);
  if (ts.bad) return {-1, ts.bad};
  return tree_walk_finish(ts, pred_row, T, max_path, s_path);
}

// Writes accept_len, path, out_tokens and new_kv_len of sequence b (warp).
// The emitted tokens come from s_out when the walk filled it, else from the
// token and prediction rows in global memory.
__device__ void write_walk(int b, int n, int L, const int32_t *tok_row, const int32_t *pred_row, const int32_t *s_path,
                           int max_path, int32_t *accept_len, int32_t *path, int32_t *out_tokens,
                           int32_t *new_kv_len, const int32_t *s_out = nullptr) {
  const int lane = threadIdx.x & 31;
  for (int k = lane; k < max_path; k += 32) {
    int pv = -1, ov = -1;
    if (n >= 0 && k <= n) {
      pv = s_path[k];
      if (s_out != nullptr) ov = s_out[k];
      else ov = (k < n) ? __ldg(tok_row + s_path[k + 1]) : __ldcg(pred_row + s_path[n]);
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

// The same from a cached page-table entry: pg = the entry of the slot's page.
__device__ __forceinline__ int64_t slot_off16_pg(const KVParams &kv, int pg, int s) {
  if (pg < 0 || pg >= kv.num_pages) return -1;
  return (int64_t(pg) * 64 + (s & 63)) * kv.Hkv * kv.ch;
}

// Slot offsets of the moves of sequence b into s_src / s_dst (x = 1 .. n),
// computed by one warp; returns false (and flags) on a bad page. With a paged
// cache, s_pg (when given) holds the entries of pages L / 64 and L / 64 + 1,
// which cover every slot a move touches (L .. L + T - 1, T <= 64).
__device__ bool move_offsets(const KVParams &kv, int b, int L, int n, const int32_t *s_path, int64_t *s_src,
                             int64_t *s_dst, int32_t *status, const int32_t *s_pg = nullptr) {
  const int lane = threadIdx.x & 31;
  int bad = 0;
  const bool cached = s_pg != nullptr && kv.page_table != nullptr;
  for (int x = 1 + lane; x <= n; x += 32) {
    const int ss = L + s_path[x], sd = L + x;
    const int64_t so = cached ? slot_off16_pg(kv, s_pg[(ss >> 6) - (L >> 6)], ss) : slot_off16(kv, b, ss);
    const int64_t dst = cached ? slot_off16_pg(kv, s_pg[(sd >> 6) - (L >> 6)], sd) : slot_off16(kv, b, sd);
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
  SampleParams sp;  // the draws at temperature tau (sampled step)
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

// Launches 1 and 2 of the sampled verification tail: stage 1 over the rows of
// tree nodes (grid.x = B * T_max * ncta_row; padding nodes return at once),
// then stage 2 (one warp per node row; grid.x = B * T_max / 8 rounded up),
// which writes the draws as the predictions.
template <typename T>
__global__ void __launch_bounds__(SAMPLE_THREADS, sizeof(T) == 2 ? 6 : 4) verify_sample_stats_kernel(const StepParams p) {
  const int ncta = p.sp.ncta_row;
  const int rowg = blockIdx.x / ncta;
  const int b = rowg / p.tr.T_max, i = rowg % p.tr.T_max;
  const int tl = __ldg(p.tr.tree_len + b);
  if (tl >= 1 && tl <= p.tr.T_max && i < tl) {
    const int64_t r = int64_t(b) * p.tr.T_max + i;
    const int64_t g0 = int64_t(blockIdx.x % ncta) * p.sp.seg_per_cta;
    const int64_t g1 = std::min<int64_t>(p.sp.nseg, g0 + p.sp.seg_per_cta);
    sample_stats<T>(p.sp, static_cast<const T *>(p.sp.logits) + r * p.sp.row_stride, p.sp.seg + r * p.sp.nseg,
                    g0, g1);
  }
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename T>
__global__ void __launch_bounds__(256) verify_sample_select_kernel(const StepParams p) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int rowg = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int b = rowg / p.tr.T_max, i = rowg % p.tr.T_max;
  if (b >= p.tr.B) return;
  const int tl = __ldg(p.tr.tree_len + b);
  if (tl < 1 || tl > p.tr.T_max || i >= tl) return;
  const int64_t r = int64_t(b) * p.tr.T_max + i;
  const int idx = sample_select_warp<T>(p.sp, static_cast<const T *>(p.sp.logits) + r * p.sp.row_stride,
                                        p.sp.seg + r * p.sp.nseg, __ldg(p.sp.u + r));
  if ((threadIdx.x & 31) == 0) p.pred[r] = idx;
}

// Launch 2 of the verification tail, one CTA per sequence, chained to launch 1
// by programmatic dependent launch (it may start early and waits until launch
// 1 has completed): the acceptance walk, its outputs, and the KV compaction.
__global__ void __launch_bounds__(TAIL_THREADS) verify_tail_kernel(const StepParams p) {
  __shared__ int32_t s_path[65], s_out[65], s_pg[2];
  __shared__ int64_t s_src[65], s_dst[65];
  __shared__ int s_n;
  const int b = blockIdx.x, Tm = p.tr.T_max;
  const int64_t rb = int64_t(b) * Tm;
  const int T = __ldg(p.tr.tree_len + b);
  const int L = __ldg(p.tr.kv_len + b);
  // Everything that needs no prediction is done while the argmax grid runs:
  // the tree's shape (with its tokens, which the walk then emits from
  // registers) and, for a paged cache, the page-table entries of the tree's
  // slots L .. L + T - 1 (two pages at most), which the compaction needs.
  const bool lens_ok = T >= 1 && T <= Tm && L >= 0 && L <= p.kv.capacity - T;
  TreeShape ts{};
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    int e = -1;
    if (lane < 2 && lens_ok && p.kv.page_table != nullptr && (L >> 6) + lane < p.kv.pages_per_seq)
      e = __ldg(p.kv.page_table + int64_t(b) * p.kv.pages_per_seq + (L >> 6) + lane);
    if (lens_ok) ts = tree_shape_warp(p.tr.parent + rb, p.tr.tokens + rb, T);
    if (lane < 2) s_pg[lane] = e;
  }
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if (threadIdx.x < 32) {
    WalkOut w{-1, 0};
    if (T < 1 || T > Tm) w.bad = DREAMS_DATA_BAD_TREE_LEN;
    else if (L < 0 || L > p.kv.capacity - T) w.bad = DREAMS_DATA_BAD_KV_LEN;
    else if (ts.bad) w.bad = ts.bad;
    else w = tree_walk_finish(ts, p.pred + rb, T, p.max_path, s_path, s_out);
    if (w.bad) {
      w.n = -1;
      if (threadIdx.x == 0) flag(p.status, w.bad);
    }
    write_walk(b, w.n, L, p.tr.tokens + rb, p.pred + rb, s_path, p.max_path, p.accept_len, p.path, p.out_tokens,
               p.new_kv_len, s_out);
    if (p.pred_in_ws && T >= 1 && T <= Tm) {  // leave the workspace zero-filled
      __syncwarp();
      for (int x = threadIdx.x; x < T; x += 32) p.pred[rb + x] = 0;
    }
    bool ok = w.n > 0;
    if (ok) ok = move_offsets(p.kv, b, L, w.n, s_path, s_src, s_dst, p.status, s_pg);
    if (threadIdx.x == 0) s_n = ok ? w.n : 0;
  }
  __syncthreads();
  const int n = s_n;
  if (n > 0) compact_units(p.kv, n, s_src, s_dst, threadIdx.x, blockDim.x);
}

// ------------------------------------------------------------------ speculative sampling
// Verification at temperature tau by speculative sampling (Leviathan et al.,
// cited in the paper's Sec. 1; T = 1 in Table 2), over the draft tree: at node
// cur the target's distribution is p = softmax(target[cur] / tau) and the
// draft's q = softmax(draft[cur] / tau), from which the drafts of cur's
// children were drawn. Children are tried in index order against the residual
// r (p at first): child c with draft x is accepted when u_acc[c] <
// min(1, r(x) / q(x)); a rejection replaces r by max(0, r - q) / Z with
// Z = sum max(0, r - q) (kept when Z = 0). The bonus is drawn from r by
// inverse transform with u_res of the node where the walk stops.
//
// The kernel keeps r in closed form. With r = max(0, p - s q) / P, where
// P = F(s) = sum_v max(0, p_v - s q_v) (s = 0, P = 1: r = p), a rejection gives
// max(0, r - q) = max(0, p - (s + P) q) / P (where p - s q <= 0 the term is 0
// either way), so the next residual is max(0, p - s' q) / F(s') with
// s' = s + P, and Z = F(s') / P. In the unnormalised exponentials
// e_v = 2^((x_v - M) k2) of the two rows (sums Zt, Zd) this reads
//     r ~ max(0, et - c ed),  Pu = sum_v max(0, et_v - c ed_v),
//     c = 0, Pu = Zt at the node;  a rejection: c' = c + Pu / Zd,
//     a child with draft x: accepted when u < Zd max(0, et_x - c ed_x) / (Pu ed_x)
// (c = s Zt / Zd, Pu = Zt P): one sum over the vocabulary per rejection, and
// the bonus is drawn from the weights max(0, et - c ed) (et when c = 0).
//
// One thread-block cluster per sequence; CTA `rank` of the cluster holds the
// vocabulary slice [rank * S, (rank + 1) * S) of the rows of the node being
// visited, as exponentials in shared memory (each thread's relative to its own
// maximum m, with the factor a = 2^((m - M) k2) to the row's maximum M kept in
// a register). Only the rows of visited nodes are read. A sum over the
// vocabulary: warps reduce their threads' values, warp 0 the warps' and stores
// the CTA's value into every CTA's shared memory (distributed shared memory),
// one cluster barrier, then each warp combines the cs values in rank order:
// all CTAs hold bit-identical results, take the same decisions and pass the
// same cluster barriers. The rows' maxima and exponential sums take one such
// exchange of (maximum, sum) pairs.
constexpr int SPEC_THREADS = 512;                    // 16 warps
constexpr int SPEC_CHUNK = 8 * SPEC_THREADS;         // values per chunk: 8 per thread
constexpr int SPEC_MAX_J = 6;                        // chunks per CTA slice (192 KB of f32 pairs)
constexpr int SPEC_MAX_CS = 16;                      // CTAs per cluster

struct SpecParams {
  const void *tgt, *drf;  // [B * T_max] rows of V logits, row_stride apart
  int64_t V, row_stride;
  float k2;               // log2(e) / tau
  int vec_ok;             // rows start on 16 bytes and strides keep them there
  int cs, J;              // CTAs per cluster, chunks per slice
  TreeParams tr;
  KVParams kv;
  int32_t max_path;
  const float *u_acc, *u_res;  // [B, T_max] each
  int32_t *accept_len, *path, *out_tokens, *new_kv_len;
  int32_t *status;
};

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// Every thread of every CTA of the cluster: release this CTA's shared-memory
// writes (local and remote), then wait for all CTAs (a superset of
// __syncthreads).
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_addr(const void *local_ptr, uint32_t rank) {
  const uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(local_ptr));
  uint32_t ra;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(a), "r"(rank));
  return ra;
}
__device__ __forceinline__ void st_cluster_f4(const float4 *local_ptr, uint32_t rank, float4 v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(cluster_addr(local_ptr, rank)), "f"(v.x),
               "f"(v.y), "f"(v.z), "f"(v.w)
               : "memory");
}
__device__ __forceinline__ void st_cluster_s32(const int32_t *local_ptr, uint32_t rank, int32_t v) {
  asm volatile("st.shared::cluster.s32 [%0], %1;" ::"r"(cluster_addr(local_ptr, rank)), "r"(v) : "memory");
}

struct SpecShared {
  float4 slot[2][SPEC_MAX_CS];       // [parity][rank]: every CTA's partial of the current exchange
  float chunk[SPEC_MAX_J][16];       // the bonus draw: per-warp sums of each chunk
  float red[16];                     // the bonus draw: per-warp sums of the slice
  float4 red4[16];                   // per-warp partials of a sum or of (maximum, sum) pairs
  int32_t hit[16], last[16];
  int32_t par[64], tok[64], path[65];
  int64_t src[65], dst[65];
  float cxt[64], cxd[64];  // the target / draft logits at each child's draft token
  float cu[64];            // u_acc of each child
  int32_t pick;            // the draw inside this CTA's slice
  int32_t bonus;           // rank 0: the bonus token, written by the CTA that drew it
  int32_t cmd;
};

// Loads issued where they stand (volatile), so that their latency overlaps the
// work between the load and the first use of its value.
__device__ __forceinline__ int ld_issue_now(const int32_t *ptr) {
  int v;
  asm volatile("ld.global.nc.b32 %0, [%1];" : "=r"(v) : "l"(ptr));
  return v;
}
__device__ __forceinline__ float ld_now_f32(const float *ptr) {
  float v;
  asm volatile("ld.global.nc.f32 %0, [%1];" : "=f"(v) : "l"(ptr));
  return v;
}
template <typename T>
__device__ __forceinline__ float ld_now_val(const T *ptr);
template <>
__device__ __forceinline__ float ld_now_val<float>(const float *ptr) {
  return ld_now_f32(ptr);
}
template <>
__device__ __forceinline__ float ld_now_val<__nv_bfloat16>(const __nv_bfloat16 *ptr) {
  unsigned short v;
  asm volatile("ld.global.nc.u16 %0, [%1];" : "=h"(v) : "l"(ptr));
  return __uint_as_float(uint32_t(v) << 16);
}

__device__ __forceinline__ float warp_sum_bcast(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return __shfl_sync(0xffffffffu, v, 0);  // lane 0's bits on every lane
}

// (maximum, sum of 2^((x - maximum) k2)) of two rows over the warp's lanes,
// from each lane's pair (x, y) and (z, w); lane 0's bits on every lane.
__device__ __forceinline__ float4 ms4_lanes(float4 v, float k2) {
  float Mt = v.x, Md = v.z;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    Mt = fmaxf(Mt, __shfl_xor_sync(0xffffffffu, Mt, off));
    Md = fmaxf(Md, __shfl_xor_sync(0xffffffffu, Md, off));
  }
  const float st = v.x == -INFINITY ? 0.f : v.y * exp2f_approx((v.x - Mt) * k2);
  const float sd = v.z == -INFINITY ? 0.f : v.w * exp2f_approx((v.z - Md) * k2);
  return make_float4(Mt, warp_sum_bcast(st), Md, warp_sum_bcast(sd));
}

// A sum over the cluster: warps, then warp 0 over the warps, then one value
// per CTA into slot [parity][rank] of every CTA; after the cluster barrier
// every warp combines the cs values in lane order (the same bits everywhere).
__device__ __forceinline__ float spec_cluster_sum(SpecShared &sh, float v, int parity, int cs, uint32_t rank) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float wv = warp_sum_bcast(v);
  if (lane == 0) sh.red4[warp] = make_float4(wv, 0.f, 0.f, 0.f);
  __syncthreads();
  if (warp == 0) {
    const float cta = warp_sum_bcast(lane < 16 ? sh.red4[lane].x : 0.f);
    if (lane < cs) st_cluster_f4(&sh.slot[parity][rank], uint32_t(lane), make_float4(cta, 0.f, 0.f, 0.f));
  }
  cluster_sync();
  return warp_sum_bcast(lane < cs ? sh.slot[parity][lane].x : 0.f);
}

// The rows' maxima and exponential sums over the cluster from each thread's
// (m_t, s_t, m_d, s_d), s = sum 2^((x - m) k2): (Mt, Zt, Md, Zd). The same
// three levels as a sum: warps, warp 0 over the warps, the CTAs.
__device__ float4 spec_cluster_ms(SpecShared &sh, float4 v, int parity, int cs, uint32_t rank, float k2) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float4 w = ms4_lanes(v, k2);
  if (lane == 0) sh.red4[warp] = w;
  __syncthreads();
  if (warp == 0) {
    const float4 cta = ms4_lanes(lane < 16 ? sh.red4[lane] : make_float4(-INFINITY, 0.f, -INFINITY, 0.f), k2);
    if (lane < cs) st_cluster_f4(&sh.slot[parity][rank], uint32_t(lane), cta);
  }
  cluster_sync();
  return ms4_lanes(lane < cs ? sh.slot[parity][lane] : make_float4(-INFINITY, 0.f, -INFINITY, 0.f), k2);
}

// Warp 0: the parent and token rows of a sequence into sh (entries past
// tree_len: parent -1, token 0); DREAMS_DATA_BAD_PARENT when parent[0] != -1
// or a parent[i] lies outside [0, i). pre_par / pre_tok: the rows' first Tm
// entries, loaded before tree_len was known.
__device__ int spec_tree_warp(SpecShared &sh, const int (&pre_par)[2], const int (&pre_tok)[2], int T) {
  const int lane = threadIdx.x & 31;
  int bad = 0;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int i = lane + 32 * h;
    const bool live = i < T;
    const int pa = live ? pre_par[h] : -1;
    sh.par[i] = pa;
    sh.tok[i] = live ? pre_tok[h] : 0;
    if (i == 0) bad |= pa != -1;
    else if (live) bad |= pa < 0 || pa >= i;
  }
  return __any_sync(0xffffffffu, bad) ? DREAMS_DATA_BAD_PARENT : 0;
}

// This thread's values of one slice as floats into e (values past V: -inf);
// returns their maximum.
template <typename T>
__device__ __forceinline__ float spec_store_raw(const SpecParams &p, const uint4 (&w)[SPEC_MAX_J][sizeof(T) / 2],
                                                float *e) {
  constexpr int NW = int(sizeof(T)) / 2;  // 16-byte words per 8 values
  const int tid = threadIdx.x;
  float m = -INFINITY;
#pragma unroll
  for (int j = 0; j < SPEC_MAX_J; ++j)
    if (j < p.J) {
      float y[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        y[i] = __uint_as_float(Elem<T>::lane_bits(w[j][NW == 1 ? 0 : i >> 2], NW == 1 ? i : (i & 3)));
        m = fmaxf(m, y[i]);
      }
      float4 *dst = reinterpret_cast<float4 *>(e + j * SPEC_CHUNK + 8 * tid);
      dst[0] = make_float4(y[0], y[1], y[2], y[3]);
      dst[1] = make_float4(y[4], y[5], y[6], y[7]);
    }
  return m;
}

// This CTA's slices of the target row (and of the draft row when `both`) as
// floats into et / ed; this thread's maxima of each. bf16 rows have both
// rows' loads in flight at once; f32 rows are taken one after the other.
template <typename T>
__device__ float2 spec_load_rows(const SpecParams &p, const T *trow, const T *drow, bool both, int64_t v0, float *et,
                                 float *ed) {
  constexpr int NW = int(sizeof(T)) / 2;
  const int warp = threadIdx.x >> 5;
  const int64_t Vs = p.V - v0;  // values of the row from the slice start on
  float2 m = make_float2(-INFINITY, -INFINITY);
  uint4 wt[SPEC_MAX_J][NW];
#pragma unroll
  for (int j = 0; j < SPEC_MAX_J; ++j)
    if (j < p.J) sub_words<T>(trow + v0, Vs, p.vec_ok, int64_t(j) * (SPEC_CHUNK / SUB) + warp, wt[j]);
  if (NW == 1) {
    uint4 wd[SPEC_MAX_J][NW];
#pragma unroll
    for (int j = 0; j < SPEC_MAX_J; ++j)
      if (both && j < p.J) sub_words<T>(drow + v0, Vs, p.vec_ok, int64_t(j) * (SPEC_CHUNK / SUB) + warp, wd[j]);
    m.x = spec_store_raw<T>(p, wt, et);
    if (both) m.y = spec_store_raw<T>(p, wd, ed);
  } else {
    m.x = spec_store_raw<T>(p, wt, et);
    if (both) {
#pragma unroll
      for (int j = 0; j < SPEC_MAX_J; ++j)
        if (j < p.J) sub_words<T>(drow + v0, Vs, p.vec_ok, int64_t(j) * (SPEC_CHUNK / SUB) + warp, wt[j]);
      m.y = spec_store_raw<T>(p, wt, ed);
    }
  }
  return m;
}

// e <- 2^((e - M) k2) in place over this thread's values; returns their sum.
// M = -inf (every value past V): zeros.
__device__ __forceinline__ float spec_exp_inplace(float *e, float M, float k2, int J) {
  const int tid = threadIdx.x;
  if (M == -INFINITY) {
    for (int j = 0; j < J; ++j) {
      float4 *q = reinterpret_cast<float4 *>(e + j * SPEC_CHUNK + 8 * tid);
      q[0] = q[1] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    return 0.f;
  }
  float s0 = 0.f, s1 = 0.f;
  for (int j = 0; j < J; ++j) {
    float4 *q = reinterpret_cast<float4 *>(e + j * SPEC_CHUNK + 8 * tid);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float4 v = q[h];
      v.x = exp2f_approx((v.x - M) * k2);
      v.y = exp2f_approx((v.y - M) * k2);
      v.z = exp2f_approx((v.z - M) * k2);
      v.w = exp2f_approx((v.w - M) * k2);
      q[h] = v;
      s0 += v.x + v.y;
      s1 += v.z + v.w;
    }
  }
  return s0 + s1;
}

// The residual's numerator at one vocabulary entry: max(0, et - c ed).
__device__ __forceinline__ float spec_w(float et, float ed, float c) { return fmaxf(fmaf(-c, ed, et), 0.f); }

// The residual's numerator over this thread's values, a_t max(0, et - ct ed)
// (a_t et alone when use_q is false): its sum, per chunk into wj, and the last
// index of positive weight.
__device__ __forceinline__ float spec_weights(const float *et, const float *ed, float at, float ct, bool use_q, int J,
                                              float (&wj)[SPEC_MAX_J], int &last) {
  const int tid = threadIdx.x;
  float tot = 0.f;
  last = -1;
#pragma unroll
  for (int j = 0; j < SPEC_MAX_J; ++j) {
    wj[j] = 0.f;
    if (j < J) {
      const int e0 = j * SPEC_CHUNK + 8 * tid;
      const float4 *t4 = reinterpret_cast<const float4 *>(et + e0);
      const float4 *d4 = reinterpret_cast<const float4 *>(ed + e0);
      float w[8];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const float4 tv = t4[h];
        if (use_q) {
          const float4 dv = d4[h];
          w[4 * h] = spec_w(tv.x, dv.x, ct), w[4 * h + 1] = spec_w(tv.y, dv.y, ct);
          w[4 * h + 2] = spec_w(tv.z, dv.z, ct), w[4 * h + 3] = spec_w(tv.w, dv.w, ct);
        } else {
          w[4 * h] = tv.x, w[4 * h + 1] = tv.y, w[4 * h + 2] = tv.z, w[4 * h + 3] = tv.w;
        }
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        w[i] *= at;
        wj[j] += w[i];
        if (w[i] > 0.f) last = e0 + i;
      }
      tot += wj[j];
    }
  }
  return tot;
}

// The bonus draw inside this CTA's slice: the entry where the running sum of
// the weights (in vocabulary order) first exceeds rem; tail: the last entry
// of positive weight. Returns the slice-relative index (-1: no positive
// weight) on every thread of the CTA.
__device__ int spec_slice_draw(SpecShared &sh, const float *et, const float *ed, float at, float ct, bool use_q,
                               const float (&wj)[SPEC_MAX_J], int last, int J, float rem, bool tail) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) last = max(last, __shfl_xor_sync(0xffffffffu, last, off));
#pragma unroll
  for (int j = 0; j < SPEC_MAX_J; ++j) {
    float v = j < J ? wj[j] : 0.f;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    if (lane == 0 && j < J) sh.chunk[j][warp] = v;
  }
  if (lane == 0) sh.last[warp] = last;
  __syncthreads();
  // lane w < 16 holds warp w's values: maxima and sums across the lanes (the
  // same bits in every warp)
  int slast = lane < 16 ? sh.last[lane] : -1;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) slast = max(slast, __shfl_xor_sync(0xffffffffu, slast, off));
  if (tail || slast < 0) return slast;
  // the crossing chunk: chunk totals, then their running sum in chunk order
  int jc = -1;
  float before = 0.f, cw = 0.f;  // cw: lane w's sum of chunk jc
#pragma unroll
  for (int j = 0; j < SPEC_MAX_J; ++j) {
    if (j >= J) break;
    const float v = lane < 16 ? sh.chunk[j][lane] : 0.f;
    const float t = warp_sum_bcast(v);
    if (jc < 0) {
      if (t > 0.f && before + t > rem) jc = j, cw = v;
      else before += t;
    }
  }
  if (jc < 0) return slast;  // rounding: no crossing inside the slice
  rem -= before;
  // this warp's offset in chunk jc: the sums of the warps before it
  float wi = cw;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, wi, off);
    if (lane >= off) wi += y;
  }
  const float wbase = __shfl_sync(0xffffffffu, wi - cw, warp);
  // exclusive scan of the threads' sums of chunk jc, in thread order
  float mine = 0.f;
#pragma unroll
  for (int j = 0; j < SPEC_MAX_J; ++j)
    if (j == jc) mine = wj[j];
  float inc = mine;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, inc, off);
    if (lane >= off) inc += y;
  }
  const float excl = wbase + inc - mine;
  const bool cross = mine > 0.f && excl + mine > rem;
  const unsigned bal = __ballot_sync(0xffffffffu, cross);
  if (lane == 0) sh.hit[warp] = bal ? warp * 32 + __ffs(bal) - 1 : INT_MAX;
  __syncthreads();
  int th = lane < 16 ? sh.hit[lane] : INT_MAX;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) th = min(th, __shfl_xor_sync(0xffffffffu, th, off));
  if (th == INT_MAX) return slast;
  if (tid == th) {
    const int e0 = jc * SPEC_CHUNK + 8 * tid;
    float a = excl;
    int hit = -1, lp = -1;
    for (int i = 0; i < 8; ++i) {
      const float w = at * (use_q ? spec_w(et[e0 + i], ed[e0 + i], ct) : et[e0 + i]);
      a += w;
      if (w > 0.f) lp = e0 + i;
      if (hit < 0 && w > 0.f && a > rem) hit = e0 + i;
    }
    sh.pick = hit >= 0 ? hit : lp;
  }
  __syncthreads();
  return sh.pick;
}

// One cluster of p.cs CTAs per sequence (grid.x = B * cs): the walk with its
// decisions, the bonus draw, the outputs and the KV compaction.
template <typename T>
__global__ void __launch_bounds__(SPEC_THREADS) spec_walk_kernel(const SpecParams p) {
  extern __shared__ __align__(16) float spec_dyn[];
  __shared__ SpecShared sh;
  const int cs = p.cs, J = p.J;
  const uint32_t rank = cluster_rank();
  const int b = int(blockIdx.x / cs);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int Tm = p.tr.T_max;
  const int64_t rb = int64_t(b) * Tm;
  const int64_t S = int64_t(J) * SPEC_CHUNK;
  const int64_t v0 = int64_t(rank) * S;
  float *et = spec_dyn, *ed = spec_dyn + S;
  const float k2 = p.k2;
  // the root's rows towards L2 while the tree is checked
  for (int j = 0; j < J; ++j) {
    const int64_t e = v0 + int64_t(j) * SPEC_CHUNK + 8 * tid;
    if (e < p.V) {
      const char *tp = static_cast<const char *>(p.tgt) + (rb * p.row_stride + e) * int64_t(sizeof(T));
      const char *dp = static_cast<const char *>(p.drf) + (rb * p.row_stride + e) * int64_t(sizeof(T));
      asm volatile("prefetch.L2 [%0];" ::"l"(tp));
      asm volatile("prefetch.L2 [%0];" ::"l"(dp));
    }
  }
  // the tree rows go out with the lengths (rows of T_max entries exist)
  int pre_par[2] = {-1, -1}, pre_tok[2] = {0, 0};
  if (warp == 0) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int i = lane + 32 * h;
      if (i < Tm) {
        pre_par[h] = ld_issue_now(p.tr.parent + rb + i);
        pre_tok[h] = ld_issue_now(p.tr.tokens + rb + i);
      }
    }
  }
  const int TL = __ldg(p.tr.tree_len + b), L = __ldg(p.tr.kv_len + b);
  if (warp == 0) {
    int bad = 0;
    if (TL < 1 || TL > Tm) bad = DREAMS_DATA_BAD_TREE_LEN;
    else if (L < 0 || L > p.kv.capacity - TL) bad = DREAMS_DATA_BAD_KV_LEN;
    else bad = spec_tree_warp(sh, pre_par, pre_tok, TL);
    if (lane == 0) {
      sh.cmd = bad;
      if (bad && rank == 0) flag(p.status, bad);
    }
  }
  __syncthreads();
  const bool bad = sh.cmd != 0;
  int n = -1, bonus = 0, parity = 0;
  if (!bad) {
    int cur = 0;
    n = 0;
    if (tid == 0) sh.path[0] = 0;
    for (;;) {
      const int64_t row = rb + cur;
      const T *trow = static_cast<const T *>(p.tgt) + row * p.row_stride;
      const T *drow = static_cast<const T *>(p.drf) + row * p.row_stride;
      // cur's children as a bit mask (nodes past tree_len hold parent -1)
      const uint64_t kids = uint64_t(__ballot_sync(0xffffffffu, sh.par[lane] == cur && lane > cur)) |
                            uint64_t(__ballot_sync(0xffffffffu, sh.par[lane + 32] == cur)) << 32;
      const bool try_kids = kids != 0 && n < p.max_path - 1;
      // each child's logits at its draft token and its uniform, loaded while
      // the rows are (children have larger indices than every node read before)
      const bool my_kid = try_kids && tid < 64 && ((kids >> tid) & 1);
      float kid_t = -INFINITY, kid_d = -INFINITY, kid_u = 0.f;
      if (my_kid) {
        const int x = sh.tok[tid];
        if (x >= 0 && x < p.V) {
          kid_t = ld_now_val<T>(trow + x);
          kid_d = ld_now_val<T>(drow + x);
        }
        kid_u = ld_now_f32(p.u_acc + rb + tid);
      }
      const float u_bonus = ld_now_f32(p.u_res + rb + cur);
      // the rows' maxima and exponential sums: per thread, then over the cluster
      const float2 m = spec_load_rows<T>(p, trow, drow, try_kids, v0, et, ed);
      if (my_kid) {  // stored after the rows' loads are out
        sh.cxt[tid] = kid_t;
        sh.cxd[tid] = kid_d;
        sh.cu[tid] = kid_u;
      }
      const float st = spec_exp_inplace(et, m.x, k2, J);
      const float sd = try_kids ? spec_exp_inplace(ed, m.y, k2, J) : 0.f;
      const float4 g = spec_cluster_ms(sh, make_float4(m.x, st, m.y, sd), parity, cs, rank, k2);
      parity ^= 1;
      const float Mt = g.x, Zd = g.w;
      // this thread's factors to the rows' maxima (its exponentials are
      // relative to its own maxima), and their ratio for the passes
      const float at = m.x == -INFINITY ? 0.f : exp2f_approx((m.x - Mt) * k2);
      const float ad = m.y == -INFINITY ? 0.f : exp2f_approx((m.y - g.z) * k2);
      const float rd = at > 0.f ? ad / at : 0.f;
      float c = 0.f, Pu = g.y;  // the residual ~ max(0, et - c ed), Pu its sum
      int next = -1;
      for (uint64_t rest = try_kids ? kids : 0; rest != 0; rest &= rest - 1) {
        const int ch = __ffsll(static_cast<long long>(rest)) - 1;
        const float et_x = exp2f_approx((sh.cxt[ch] - Mt) * k2), ed_x = exp2f_approx((sh.cxd[ch] - g.z) * k2);
        const float num = fmaxf(fmaf(-c, ed_x, et_x), 0.f);
        float a = 0.f;  // min(1, r(x) / q(x)) = Zd num / (Pu ed_x); q(x) = 0: 1 when r(x) > 0
        if (num > 0.f) a = ed_x > 0.f ? fminf(1.f, (num / ed_x) * (Zd / Pu)) : 1.f;
        if (sh.cu[ch] < a) {
          next = ch;
          break;
        }
        // a rejection: the new residual's sum over the slice, then over the cluster
        const float c2 = c + Pu / Zd, ct = c2 * rd;
        float acc0 = 0.f, acc1 = 0.f;
        for (int j = 0; j < J && at > 0.f; ++j) {
          const float4 *t4 = reinterpret_cast<const float4 *>(et + j * SPEC_CHUNK + 8 * tid);
          const float4 *d4 = reinterpret_cast<const float4 *>(ed + j * SPEC_CHUNK + 8 * tid);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const float4 tv = t4[h], dv = d4[h];
            acc0 += spec_w(tv.x, dv.x, ct) + spec_w(tv.y, dv.y, ct);
            acc1 += spec_w(tv.z, dv.z, ct) + spec_w(tv.w, dv.w, ct);
          }
        }
        const float Pn = spec_cluster_sum(sh, at * (acc0 + acc1), parity, cs, rank);
        parity ^= 1;
        if (Pn > 0.f) c = c2, Pu = Pn;  // a zero sum (r == q) keeps the residual
      }
      if (next >= 0) {
        ++n;
        cur = next;
        if (tid == 0) sh.path[n] = next;
        continue;
      }
      // the bonus: the weights max(0, et - c ed) (et when c = 0) per chunk,
      // per slice and over the cluster; the slice where the running sum
      // crosses u * total draws the entry
      const bool use_q = c > 0.f;
      const float ct = c * rd;
      float wj[SPEC_MAX_J];
      int last;
      const float tot = spec_weights(et, ed, at, ct, use_q, J, wj, last);
      // the slice's total (warps, then warp 0 over them) to slot [parity][rank]
      // of every CTA; lane r then holds slice r's total, the same bits on
      // every warp of every CTA
      {
        const float wt = warp_sum_bcast(tot);
        if (lane == 0) sh.red[warp] = wt;
        __syncthreads();
        if (warp == 0) {
          const float slice = warp_sum_bcast(lane < 16 ? sh.red[lane] : 0.f);
          if (lane < cs) st_cluster_f4(&sh.slot[parity][rank], uint32_t(lane), make_float4(slice, 0.f, 0.f, 0.f));
        }
        cluster_sync();
      }
      const float tr = lane < cs ? sh.slot[parity][lane].x : 0.f;
      parity ^= 1;
      // their running sum across the lanes, then the crossing slice
      float inc = tr;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, inc, off);
        if (lane >= off) inc += y;
      }
      const float total = __shfl_sync(0xffffffffu, inc, 31);
      const float u = u_bonus > 0.f ? fminf(u_bonus, 1.f) : 0.f;
      const float target = u * total;
      const unsigned pos = __ballot_sync(0xffffffffu, tr > 0.f);
      const unsigned crs = __ballot_sync(0xffffffffu, tr > 0.f && inc > target);
      int cr = crs ? __ffs(crs) - 1 : -1;
      const int lastpos = pos ? 31 - __clz(pos) : -1;
      const float before = __shfl_sync(0xffffffffu, inc - tr, cr >= 0 ? cr : 0);
      const bool tail = cr < 0;
      if (tail) cr = lastpos;
      if (cr < 0) {  // no positive weight anywhere (rounding): token 0
        if (rank == 0 && tid == 0) sh.bonus = 0;
      } else if (int(rank) == cr) {
        const int e = spec_slice_draw(sh, et, ed, at, ct, use_q, wj, last, J, target - before, tail);
        if (tid == 0) st_cluster_s32(&sh.bonus, 0, e >= 0 ? int32_t(v0 + e) : 0);
      }
      cluster_sync();
      bonus = int(std::min<int64_t>(std::max(sh.bonus, 0), p.V - 1));  // used by rank 0 only
      break;
    }
  }
  // outputs (rank 0): path, drafts then the bonus, lengths; the compaction is
  // shared by the cluster's CTAs
  if (warp == 0) {
    if (rank == 0) {
      const int mp = p.max_path;
      for (int kk = lane; kk < mp; kk += 32) {
        int pv = -1, ov = -1;
        if (n >= 0 && kk <= n) {
          pv = sh.path[kk];
          ov = kk < n ? sh.tok[sh.path[kk + 1]] : bonus;
        }
        p.path[int64_t(b) * mp + kk] = pv;
        p.out_tokens[int64_t(b) * mp + kk] = ov;
      }
      if (lane == 0) {
        p.accept_len[b] = n >= 0 ? n + 1 : 0;
        p.new_kv_len[b] = n >= 0 ? L + n + 1 : L;
      }
    }
    bool ok = n > 0;
    if (ok) ok = move_offsets(p.kv, b, L, n, sh.path, sh.src, sh.dst, rank == 0 ? p.status : nullptr);
    if (lane == 0) sh.cmd = ok ? n : 0;
  }
  __syncthreads();
  const int nm = sh.cmd;
  if (nm > 0) compact_units(p.kv, nm, sh.src, sh.dst, int64_t(rank) * SPEC_THREADS + tid, int64_t(cs) * SPEC_THREADS);
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

// Launches `kernel` as a programmatic dependent of the previous launch on the stream.
template <typename... Args>
dreams_status_t launch_dependent(void (*kernel)(Args...), dim3 grid, dim3 block, cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, args...);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  return check_launch();
}

// CTAs per sequence of the speculative walk (a power of two): the fewest whose
// slices of at most SPEC_MAX_J chunks cover V, doubled while every CTA keeps a
// chunk of the vocabulary and the batch leaves SMs idle: up to 8, or 16 for
// batches of at most 4 (clusters of 16 take most of a GPC each). cs = 0: V
// too large.
struct SpecPlan {
  int cs, J;
};
inline SpecPlan plan_spec(int64_t B, int64_t V) {
  const int64_t per_cta = int64_t(SPEC_MAX_J) * SPEC_CHUNK;
  int cs = 1;
  while (cs < SPEC_MAX_CS && int64_t(cs) * per_cta < V) cs *= 2;
  if (int64_t(cs) * per_cta < V) return {0, 0};
  const int64_t chunks = (V + SPEC_CHUNK - 1) / SPEC_CHUNK;
  const int cap = B <= 4 ? 16 : 8;
  while (cs < cap && B * cs * 2 <= num_sms() && chunks >= 2 * cs) cs *= 2;
  const int64_t span = int64_t(cs) * SPEC_CHUNK;
  return {cs, int((V + span - 1) / span)};
}

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
  const cudaError_t e = cudaLaunchKernelEx(&cfg, verify_tail_kernel, p);
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
  const dim3 grid(static_cast<unsigned>(ctas)), g2(static_cast<unsigned>((rows + 7) / 8));
  if (dtype == DREAMS_F32) vocab_sample_stats_kernel<float><<<grid, SAMPLE_THREADS, 0, s>>>(p);
  else vocab_sample_stats_kernel<__nv_bfloat16><<<grid, SAMPLE_THREADS, 0, s>>>(p);
  dreams_status_t st = check_launch();
  if (st != DREAMS_OK) return st;
  if (dtype == DREAMS_F32) return launch_dependent(vocab_sample_select_kernel<float>, g2, dim3(256), s, p, rows, out_idx);
  return launch_dependent(vocab_sample_select_kernel<__nv_bfloat16>, g2, dim3(256), s, p, rows, out_idx);
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
  const dim3 grid(static_cast<unsigned>(ctas)), g2(static_cast<unsigned>((rows + 7) / 8));
  if (dtype == DREAMS_F32) verify_sample_stats_kernel<float><<<grid, SAMPLE_THREADS, 0, s>>>(p);
  else verify_sample_stats_kernel<__nv_bfloat16><<<grid, SAMPLE_THREADS, 0, s>>>(p);
  dreams_status_t st = check_launch();
  if (st != DREAMS_OK) return st;
  st = dtype == DREAMS_F32 ? launch_dependent(verify_sample_select_kernel<float>, g2, dim3(256), s, p)
                           : launch_dependent(verify_sample_select_kernel<__nv_bfloat16>, g2, dim3(256), s, p);
  if (st != DREAMS_OK) return st;
  return launch_dependent(verify_tail_kernel, dim3(unsigned(tree->B)), dim3(TAIL_THREADS), s, p);
}

extern "C" dreams_status_t dreams_verify_step_speculative(
    const void *target_logits, const void *draft_logits, dreams_dtype_t dtype, int64_t V, int64_t row_stride,
    const dreams_tree_t *tree, const dreams_kv_cache_t *kv, int32_t max_path, float temperature,
    const float *u_accept, const float *u_resample, int32_t *accept_len, int32_t *path, int32_t *out_tokens,
    int32_t *new_kv_len, int32_t *status_word, dreams_stream_t stream) {
  SpecParams p{};
  if (target_logits == nullptr || draft_logits == nullptr || u_accept == nullptr || u_resample == nullptr || V < 1 ||
      row_stride < V || !tree_params(tree, true, p.tr) || !kv_params(kv, p.kv) || max_path < 1 || max_path > 65 ||
      accept_len == nullptr || path == nullptr || out_tokens == nullptr || new_kv_len == nullptr)
    return DREAMS_ERR_INVALID_ARG;
  if (dtype != DREAMS_F32 && dtype != DREAMS_BF16) return DREAMS_ERR_UNSUPPORTED;
  const size_t esz = dtype == DREAMS_F32 ? 4 : 2;
  if (reinterpret_cast<uintptr_t>(target_logits) % esz || reinterpret_cast<uintptr_t>(draft_logits) % esz ||
      (reinterpret_cast<uintptr_t>(u_accept) & 3) || (reinterpret_cast<uintptr_t>(u_resample) & 3))
    return DREAMS_ERR_INVALID_ARG;
  const float k2 = 1.4426950408889634f / temperature;
  if (!(temperature > 0.f) || !isfinite(temperature) || !isfinite(k2)) return DREAMS_ERR_INVALID_ARG;
  const SpecPlan pl = plan_spec(tree->B, V);
  if (pl.cs == 0) return DREAMS_ERR_UNSUPPORTED;
  if (int64_t(tree->B) * pl.cs > INT_MAX) return DREAMS_ERR_UNSUPPORTED;
  p.tgt = target_logits;
  p.drf = draft_logits;
  p.V = V;
  p.row_stride = row_stride;
  p.k2 = k2;
  p.vec_ok = aligned16(target_logits) && aligned16(draft_logits) && (row_stride * int64_t(esz)) % 16 == 0;
  p.cs = pl.cs;
  p.J = pl.J;
  p.max_path = max_path;
  p.u_acc = u_accept;
  p.u_res = u_resample;
  p.accept_len = accept_len;
  p.path = path;
  p.out_tokens = out_tokens;
  p.new_kv_len = new_kv_len;
  p.status = status_word;
  const int smem = pl.J * SPEC_CHUNK * 2 * int(sizeof(float));
  void (*kernel)(const SpecParams) =
      dtype == DREAMS_F32 ? spec_walk_kernel<float> : spec_walk_kernel<__nv_bfloat16>;
  dreams_status_t st = ensure_max_dynamic_smem(reinterpret_cast<const void *>(kernel), smem);
  if (st != DREAMS_OK) return st;
  if (pl.cs > 8) {
    const cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) {
      set_last_cuda_error(e);
      return DREAMS_ERR_CUDA;
    }
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(int64_t(tree->B) * pl.cs));
  cfg.blockDim = dim3(SPEC_THREADS);
  cfg.dynamicSmemBytes = size_t(smem);
  cfg.stream = reinterpret_cast<cudaStream_t>(stream);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = unsigned(pl.cs);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, p);
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
