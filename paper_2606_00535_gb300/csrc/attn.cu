// attn.cu -- tree-masked verification attention (paper Sec. 2, "Speculative
// decoding": the target scores every draft token in one parallel pass; Sec. 2,
// "Vision-Language Models": every cached visual and text token is attended at
// each decoding step; attention = softmax(Q K^T * scale), Sec. 3.2).
//
// Work decomposition: one CTA per (split of the KV sequence, KV head g,
// sequence b, block of query rows). The query rows of a CTA are all
// (tree node t, query head of group g) pairs, row = t * G + (h - g * G), so
// one pass over a K/V tile serves every query head that shares it (GQA) and
// every tree node. K/V tiles of 64 tokens stream through shared memory with
// cp.async double buffering; QK^T and PV run on tensor cores (bf16 inputs,
// fp32 accumulation) with an online base-2 softmax. The ancestor mask is only
// evaluated on tiles that reach the tree slots [L, L + T). Splits of one
// (b, g, row block) write unnormalised partials (m, l, O) to the workspace,
// and a second kernel, chained by programmatic dependent launch, merges them
// by log-sum-exp. The workspace holds no state between calls.
#include <math.h>
#include <string.h>

#include <cuda.h>

#include <algorithm>

#include "common.cuh"
#include "tc.cuh"

namespace dreams {
namespace {

constexpr int KT = 64;      // KV tokens per shared-memory tile
constexpr int STAGES = 2;   // cp.async pipeline depth
constexpr float LOG2E = 1.4426950408889634f;
constexpr float LN2 = 0.6931471805599453f;

struct AttnParams {
  const __nv_bfloat16 *q;
  __nv_bfloat16 *out;
  float *lse;
  const __nv_bfloat16 *k;
  const __nv_bfloat16 *v;
  const int32_t *page_table;  // nullptr: contiguous cache
  int32_t pages_per_seq;
  int32_t num_pages;
  int32_t capacity;
  const int32_t *parent;
  const int32_t *tree_len;
  const int32_t *kv_len;
  int32_t B, T_max, Hq, Hkv, G;
  int32_t nrb;     // query-row blocks per (b, g)
  int32_t nsplit;  // KV splits in the grid
  int32_t chunk;   // KV tokens per split, a multiple of KT
  float scale_log2;
  float *ws_o;      // [B][Hkv][nrb][nsplit][RPC][D]
  float2 *ws_ml;    // [B][Hkv][nrb][nsplit][RPC]  (m in log2 units, l)
  int32_t *status;
};

// Element offset of (b, slot s, head g, d = 0), or -1 for a bad page id.
__device__ __forceinline__ int64_t kv_row(const AttnParams &p, int b, int s, int g, int D) {
  if (p.page_table == nullptr) return ((int64_t(b) * p.capacity + s) * p.Hkv + g) * D;
  const int pg = __ldg(p.page_table + int64_t(b) * p.pages_per_seq + (s >> 6));
  if (pg < 0 || pg >= p.num_pages) return -1;
  return ((int64_t(pg) * 64 + (s & 63)) * p.Hkv + g) * D;
}

template <int D, int NW>
__global__ void __launch_bounds__(NW * 32, 1) tree_attn_mma_kernel(const AttnParams p) {
  constexpr int NT = NW * 32;
  constexpr int RPC = NW * 16;  // query rows per CTA
  constexpr int CH = D / 8;     // 16-byte chunks per row
  constexpr int KS = D / 16;    // k-steps of QK^T
  constexpr int NTO = D / 8;    // n-tiles of the output
  extern __shared__ __align__(128) uint8_t smem[];
  __nv_bfloat16 *sQ = reinterpret_cast<__nv_bfloat16 *>(smem);
  __nv_bfloat16 *sK = sQ + RPC * D;
  __nv_bfloat16 *sV = sK + STAGES * KT * D;
  __shared__ unsigned long long s_anc[64];
  __shared__ int s_jump[64];
  __shared__ int s_flag;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rb = blockIdx.x % p.nrb, split = blockIdx.x / p.nrb;
  const int g = blockIdx.y, b = blockIdx.z;
  const bool reporter = (rb == 0 && split == 0 && g == 0);

  const int T = __ldg(p.tree_len + b);
  const int L = __ldg(p.kv_len + b);
  if (T < 1 || T > p.T_max) {
    if (reporter && tid == 0) flag(p.status, DREAMS_DATA_BAD_TREE_LEN);
    return;
  }
  if (L < 0 || L > p.capacity - T) {
    if (reporter && tid == 0) flag(p.status, DREAMS_DATA_BAD_KV_LEN);
    return;
  }
  const int total = L + T;
  const int nsplit_b = (total + p.chunk - 1) / p.chunk;
  const int rows_b = T * p.G;
  if (split >= nsplit_b || rb * RPC >= rows_b) return;

  // ---- ancestor-or-self masks of the tree nodes (pointer jumping, warp 0)
  if (warp == 0) {
    int par[2], bad = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int i = lane + 32 * h;
      par[h] = (i < T) ? __ldg(p.parent + int64_t(b) * p.T_max + i) : -1;
      if (i == 0) bad |= (par[h] != -1);
      else if (i < T) bad |= (par[h] < 0 || par[h] >= i);
    }
    bad = __any_sync(0xffffffffu, bad);
    if (bad) {
      if (lane == 0) {
        s_flag = 1;
        if (reporter) flag(p.status, DREAMS_DATA_BAD_PARENT);
      }
    } else {
      if (lane == 0) s_flag = 0;
      unsigned long long m[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int i = lane + 32 * h;
        m[h] = 1ull << i;
        s_anc[i] = m[h];
        s_jump[i] = par[h];
      }
      __syncwarp();
      for (int r = 0; r < 6; ++r) {
        unsigned long long am[2];
        int jj[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int j = par[h];
          am[h] = (j >= 0) ? s_anc[j] : 0ull;
          jj[h] = (j >= 0) ? s_jump[j] : -1;
        }
        __syncwarp();
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          m[h] |= am[h];
          par[h] = jj[h];
          s_anc[lane + 32 * h] = m[h];
          s_jump[lane + 32 * h] = par[h];
        }
        __syncwarp();
      }
    }
  }

  __syncthreads();
  if (s_flag) return;

  // ---- query rows -> shared memory (swizzled 16-byte chunks)
  const int64_t q_base = int64_t(b) * p.T_max * p.Hq;
  for (int idx = tid; idx < RPC * CH; idx += NT) {
    const int r = idx / CH, c = idx % CH;
    const int gr = rb * RPC + r;
    const int t = gr / p.G, hg = gr - t * p.G;
    const bool ok = gr < rows_b;
    const __nv_bfloat16 *src = ok ? p.q + ((q_base + int64_t(t) * p.Hq + g * p.G + hg) * D + c * 8) : p.q;
    cp_async_16(smem_u32(sQ + r * D + ((c ^ (r & 7)) * 8)), src, ok ? 16u : 0u);
  }
  cp_async_commit();

  const int c0 = split * p.chunk;
  const int c1 = min(c0 + p.chunk, total);
  const int ntiles = (c1 - c0 + KT - 1) / KT;

  int bad_page = 0;
  auto load_tile = [&](int stage, int tile) {
    const int s0 = c0 + tile * KT;
    __nv_bfloat16 *dk = sK + stage * KT * D;
    __nv_bfloat16 *dv = sV + stage * KT * D;
    for (int idx = tid; idx < KT * CH; idx += NT) {
      const int r = idx / CH, c = idx % CH;
      const int s = s0 + r;
      int64_t off = -1;
      if (s < c1) {
        off = kv_row(p, b, s, g, D);
        if (off < 0) bad_page = 1;
      }
      const uint32_t n = off >= 0 ? 16u : 0u;
      const int64_t o = off >= 0 ? off + c * 8 : 0;
      const int sw = (c ^ (r & 7)) * 8;
      cp_async_16(smem_u32(dk + r * D + sw), p.k + o, n);
      cp_async_16(smem_u32(dv + r * D + sw), p.v + o, n);
    }
  };

  // thread's two accumulator rows
  const int r0 = warp * 16 + (lane >> 2);
  const int gr0 = rb * RPC + r0, gr1 = gr0 + 8;
  const int t0 = gr0 / p.G, t1 = gr1 / p.G;
  const unsigned long long anc0 = (t0 < T) ? s_anc[t0] : 0ull;
  const unsigned long long anc1 = (t1 < T) ? s_anc[t1] : 0ull;

  uint32_t qf[KS][4];
  float o[NTO][4];
#pragma unroll
  for (int j = 0; j < NTO; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

  load_tile(0, 0);
  cp_async_commit();

  for (int tile = 0; tile < ntiles; ++tile) {
    if (tile + 1 < ntiles) {
      load_tile((tile + 1) % STAGES, tile + 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (tile == 0) {
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        const int r = warp * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int c = ks * 2 + (lane >> 4);
        ldmatrix_x4(smem_u32(sQ + r * D + ((c ^ (r & 7)) * 8)), qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3]);
      }
    }
    const __nv_bfloat16 *tk = sK + (tile % STAGES) * KT * D;
    const __nv_bfloat16 *tv = sV + (tile % STAGES) * KT * D;

    // S = Q K^T  (16 rows x 64 tokens per warp)
    float sc[KT / 8][4];
#pragma unroll
    for (int j = 0; j < KT / 8; ++j) sc[j][0] = sc[j][1] = sc[j][2] = sc[j][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
#pragma unroll
      for (int np = 0; np < KT / 16; ++np) {
        const int tok = np * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int c = ks * 2 + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldmatrix_x4(smem_u32(tk + tok * D + ((c ^ (tok & 7)) * 8)), b0, b1, b2, b3);
        mma_bf16_16816(sc[2 * np], qf[ks], b0, b1);
        mma_bf16_16816(sc[2 * np + 1], qf[ks], b2, b3);
      }
    }

    // scale, tree mask, online softmax (base 2)
    const int s0 = c0 + tile * KT;
    const bool need_mask = (s0 + KT > L) || (s0 + KT > c1);
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int j = 0; j < KT / 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float x = sc[j][e] * p.scale_log2;
        if (need_mask) {
          const int col = s0 + j * 8 + 2 * (lane & 3) + (e & 1);
          const unsigned long long an = (e < 2) ? anc0 : anc1;
          const bool ok = col < c1 && (col < L || ((an >> (col - L)) & 1ull));
          if (!ok) x = -INFINITY;
        }
        sc[j][e] = x;
      }
      mx0 = fmaxf(mx0, fmaxf(sc[j][0], sc[j][1]));
      mx1 = fmaxf(mx1, fmaxf(sc[j][2], sc[j][3]));
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    const float mu0 = (mn0 == -INFINITY) ? 0.f : mn0;
    const float mu1 = (mn1 == -INFINITY) ? 0.f : mn1;
    const float cr0 = exp2f(m0 - mu0), cr1 = exp2f(m1 - mu1);
    m0 = mn0;
    m1 = mn1;
    float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
    for (int j = 0; j < KT / 8; ++j) {
      sc[j][0] = exp2f(sc[j][0] - mu0);
      sc[j][1] = exp2f(sc[j][1] - mu0);
      sc[j][2] = exp2f(sc[j][2] - mu1);
      sc[j][3] = exp2f(sc[j][3] - mu1);
      ps0 += sc[j][0] + sc[j][1];
      ps1 += sc[j][2] + sc[j][3];
    }
    l0 = l0 * cr0 + ps0;
    l1 = l1 * cr1 + ps1;
#pragma unroll
    for (int j = 0; j < NTO; ++j) {
      o[j][0] *= cr0;
      o[j][1] *= cr0;
      o[j][2] *= cr1;
      o[j][3] *= cr1;
    }

    // O += P V
#pragma unroll
    for (int ks = 0; ks < KT / 16; ++ks) {
      uint32_t a[4];
      a[0] = pack_bf16x2(sc[2 * ks][0], sc[2 * ks][1]);
      a[1] = pack_bf16x2(sc[2 * ks][2], sc[2 * ks][3]);
      a[2] = pack_bf16x2(sc[2 * ks + 1][0], sc[2 * ks + 1][1]);
      a[3] = pack_bf16x2(sc[2 * ks + 1][2], sc[2 * ks + 1][3]);
#pragma unroll
      for (int dp = 0; dp < NTO / 2; ++dp) {
        const int kv = ks * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int c = dp * 2 + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldmatrix_x4_trans(smem_u32(tv + kv * D + ((c ^ (kv & 7)) * 8)), b0, b1, b2, b3);
        mma_bf16_16816(o[2 * dp], a, b0, b1);
        mma_bf16_16816(o[2 * dp + 1], a, b2, b3);
      }
    }
    __syncthreads();
  }
  if (bad_page) flag(p.status, DREAMS_DATA_BAD_PAGE);

  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);

  const int cq = 2 * (lane & 3);
  if (nsplit_b == 1) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int gr = half ? gr1 : gr0;
      if (gr >= rows_b) continue;
      const int t = gr / p.G, h = g * p.G + (gr - t * p.G);
      const float inv = 1.f / (half ? l1 : l0);
      __nv_bfloat16 *dst = p.out + ((q_base + int64_t(t) * p.Hq + h) * D);
#pragma unroll
      for (int j = 0; j < NTO; ++j) {
        const uint32_t v2 = pack_bf16x2(o[j][2 * half] * inv, o[j][2 * half + 1] * inv);
        *reinterpret_cast<uint32_t *>(dst + j * 8 + cq) = v2;
      }
      if (p.lse != nullptr && (lane & 3) == 0) {
        const float mm = half ? m1 : m0, ll = half ? l1 : l0;
        p.lse[(q_base + int64_t(t) * p.Hq + h)] = (mm + log2f(ll)) * LN2;
      }
    }
    return;
  }

  // ---- split partials; the merge kernel combines them
  const int64_t pair = (int64_t(b) * p.Hkv + g) * p.nrb + rb;
  const int64_t pbase = (pair * p.nsplit + split) * RPC;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int r = r0 + 8 * half;
    float *dst = p.ws_o + (pbase + r) * D;
#pragma unroll
    for (int j = 0; j < NTO; ++j)
      *reinterpret_cast<float2 *>(dst + j * 8 + cq) = make_float2(o[j][2 * half], o[j][2 * half + 1]);
    if ((lane & 3) == 0) p.ws_ml[pbase + r] = make_float2(half ? m1 : m0, half ? l1 : l0);
  }
  __syncthreads();
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}


// ============================================================================
// tcgen05 path (sm_103a): one CTA per (KV split, KV head, sequence, block of
// 128 query rows). Warp 0 streams 64-token K/V tiles with TMA into a
// two-stage shared-memory ring; one thread of warp 1 issues the tensor-core
// MMAs (S = Q K^T into TMEM, O += P V with P read from TMEM); warps 2-5 own
// one query row per thread, turn S into P with an online base-2 softmax and
// write P back over S in TMEM. S/P are double-buffered in TMEM so the
// QK^T of tile j+1 overlaps the softmax of tile j. The running maximum used
// for the exponentials is raised only when a tile's maximum exceeds it by
// more than 2^8, and only then is O (in TMEM) rescaled; results do not depend
// on the reference value, only the fp32 range does. Every mbarrier wait is
// bounded (2 s); on a timeout the CTA flags DREAMS_DATA_TIMEOUT, drains its
// copies and MMAs, frees its TMEM and exits.
// ============================================================================
constexpr int TC_KT = 64;
constexpr int TC_ROWS = 128;
constexpr int TC_STAGES = 2;
constexpr int TC_THREADS = 192;
constexpr float TC_RESCALE = 8.f;
constexpr uint32_t TC_TMEM_COLS = 256;

struct TcParams {
  CUtensorMap tmap_k;
  CUtensorMap tmap_v;
  AttnParams a;
  int32_t paged;
};

template <int D>
__global__ void __launch_bounds__(TC_THREADS, 2) tree_attn_tc_kernel(const __grid_constant__ TcParams P) {
  const AttnParams &p = P.a;
  constexpr int NR = D / 64;                       // 128-byte column regions of a row
  constexpr uint32_t Q_REGION = TC_ROWS * 128;     // 16 KB
  constexpr uint32_t KV_REGION = TC_KT * 128;      // 8 KB
  constexpr uint32_t Q_BYTES = NR * Q_REGION;
  constexpr uint32_t STAGE_BYTES = 2 * NR * KV_REGION;
  constexpr uint32_t S_COL0 = 0, S_COL1 = 64, O_COL = 128;
  constexpr uint32_t IDESC_QK = tc::idesc_bf16_f32(TC_ROWS, TC_KT, false);
  constexpr uint32_t IDESC_PV = tc::idesc_bf16_f32(TC_ROWS, D, true);

  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar_full[TC_STAGES], bar_empty[TC_STAGES], bar_s[2], bar_p[2], bar_o, bar_drain;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;
  __shared__ int s_zero;
  __shared__ int s_flag;
  __shared__ unsigned long long s_anc[64];
  __shared__ int s_jump[64];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rb = blockIdx.x % p.nrb, split = blockIdx.x / p.nrb;
  const int g = blockIdx.y, b = blockIdx.z;
  const bool reporter = (rb == 0 && split == 0 && g == 0);
  const int T = __ldg(p.tree_len + b);
  const int L = __ldg(p.kv_len + b);
  if (T < 1 || T > p.T_max) {
    if (reporter && tid == 0) flag(p.status, DREAMS_DATA_BAD_TREE_LEN);
    return;
  }
  if (L < 0 || L > p.capacity - T) {
    if (reporter && tid == 0) flag(p.status, DREAMS_DATA_BAD_KV_LEN);
    return;
  }
  const int total = L + T;
  const int nsplit_b = (total + p.chunk - 1) / p.chunk;
  const int rows_b = T * p.G;
  if (split >= nsplit_b || rb * TC_ROWS >= rows_b) return;

  // ---- tree check and ancestor masks (warp 2, pointer jumping)
  if (warp == 2) {
    int par[2], bad = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int i = lane + 32 * h;
      par[h] = (i < T) ? __ldg(p.parent + int64_t(b) * p.T_max + i) : -1;
      if (i == 0) bad |= (par[h] != -1);
      else if (i < T) bad |= (par[h] < 0 || par[h] >= i);
    }
    bad = __any_sync(0xffffffffu, bad);
    if (lane == 0) s_flag = bad;
    if (bad) {
      if (lane == 0 && reporter) flag(p.status, DREAMS_DATA_BAD_PARENT);
    } else {
      unsigned long long m[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        m[h] = 1ull << (lane + 32 * h);
        s_anc[lane + 32 * h] = m[h];
        s_jump[lane + 32 * h] = par[h];
      }
      __syncwarp();
      for (int r = 0; r < 6; ++r) {
        unsigned long long am[2];
        int jj[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          am[h] = par[h] >= 0 ? s_anc[par[h]] : 0ull;
          jj[h] = par[h] >= 0 ? s_jump[par[h]] : -1;
        }
        __syncwarp();
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          m[h] |= am[h];
          par[h] = jj[h];
          s_anc[lane + 32 * h] = m[h];
          s_jump[lane + 32 * h] = par[h];
        }
        __syncwarp();
      }
    }
  }
  __syncthreads();
  if (s_flag) return;

  const uint32_t smem_base = smem_u32(smem);
  const uint32_t q_s = smem_base;
  auto k_s = [&](int st) { return smem_base + Q_BYTES + st * STAGE_BYTES; };
  auto v_s = [&](int st) { return smem_base + Q_BYTES + st * STAGE_BYTES + NR * KV_REGION; };
  const uint32_t full0 = smem_u32(&bar_full[0]), empty0 = smem_u32(&bar_empty[0]);
  const uint32_t bs0 = smem_u32(&bar_s[0]), bp0 = smem_u32(&bar_p[0]);
  const uint32_t bo = smem_u32(&bar_o), bdrain = smem_u32(&bar_drain);

  if (tid == 0) {
    for (int i = 0; i < TC_STAGES; ++i) {
      tc::mbar_init(full0 + 8 * i, 1);
      tc::mbar_init(empty0 + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(bs0 + 8 * i, 1);
      tc::mbar_init(bp0 + 8 * i, 128);
    }
    tc::mbar_init(bo, 1);
    tc::mbar_init(bdrain, 1);
    s_abort = 0;
    s_zero = 0;
    tc::fence_barrier_init();
  }
  if (warp == 1) {
    tc::tmem_alloc(smem_u32(&s_tmem), TC_TMEM_COLS);
    tc::tmem_relinquish();
  }
  // ---- query rows -> shared memory in the 128-byte-swizzled K-major layout
  const int row = 32 * (warp & 3) + lane;  // softmax warps: TMEM lane quadrant = warp % 4
  const int grow = rb * TC_ROWS + row;
  const int t_row = grow / p.G;
  if (warp >= 2) {
    const bool ok = grow < rows_b;
    const int hg = grow - t_row * p.G;
    const uint4 *src = reinterpret_cast<const uint4 *>(
        p.q + ((int64_t(b) * p.T_max + (ok ? t_row : 0)) * p.Hq + g * p.G + hg) * D);
#pragma unroll
    for (int c = 0; c < D / 8; ++c) {
      const uint4 v = ok ? __ldg(src + c) : make_uint4(0u, 0u, 0u, 0u);
      const uint32_t dst = q_s + (c >> 3) * Q_REGION + row * 128 + (((c & 7) ^ (row & 7)) << 4);
      asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(dst), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                   : "memory");
    }
    tc::fence_proxy_async_smem();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = s_tmem;

  const int c0 = split * p.chunk;
  const int c1 = min(c0 + p.chunk, total);
  const int ntiles = (c1 - c0 + TC_KT - 1) / TC_KT;
  volatile int *abort_flag = &s_abort;
  auto give_up = [&]() {
    *abort_flag = 1;
    flag(p.status, DREAMS_DATA_TIMEOUT);
  };

  if (warp == 0) {
    // ---------------- TMA producer
    if (lane == 0) {
      tc::prefetch_tmap(&P.tmap_k);
      tc::prefetch_tmap(&P.tmap_v);
      int issued = 0;
      for (int j = 0; j < ntiles; ++j) {
        const int st = j % TC_STAGES;
        if (j >= TC_STAGES && !tc::mbar_wait(empty0 + 8 * st, ((j / TC_STAGES) - 1) & 1, abort_flag)) {
          give_up();
          break;
        }
        const int s0 = c0 + j * TC_KT;
        int c2, c3;
        if (P.paged) {
          int pg = __ldg(p.page_table + int64_t(b) * p.pages_per_seq + (s0 >> 6));
          if (pg < 0 || pg >= p.num_pages) {
            flag(p.status, DREAMS_DATA_BAD_PAGE);
            pg = p.num_pages;  // out of range for the tensor map: the copy fills zeros
          }
          c2 = 0;
          c3 = pg;
        } else {
          c2 = s0;
          c3 = b;
        }
        tc::mbar_arrive_expect_tx(full0 + 8 * st, STAGE_BYTES);
#pragma unroll
        for (int r = 0; r < NR; ++r) {
          tc::tma_load_4d(k_s(st) + r * KV_REGION, &P.tmap_k, full0 + 8 * st, r * 64, g, c2, c3);
          tc::tma_load_4d(v_s(st) + r * KV_REGION, &P.tmap_v, full0 + 8 * st, r * 64, g, c2, c3);
        }
        issued = j + 1;
      }
      // no copy may still be landing in shared memory when the CTA ends
      for (int j = max(0, issued - TC_STAGES); j < issued; ++j)
        tc::mbar_wait(full0 + 8 * (j % TC_STAGES), (j / TC_STAGES) & 1, &s_zero);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      bool ok = true;
      auto pv = [&](int i) {
        if (!tc::mbar_wait(bp0 + 8 * (i & 1), (i >> 1) & 1, abort_flag)) {
          give_up();
          return false;
        }
        tc::fence_after_sync();
        const int st = i % TC_STAGES;
        const uint32_t scol = (i & 1) ? S_COL1 : S_COL0;
#pragma unroll
        for (int ks = 0; ks < TC_KT / 16; ++ks) {
          const uint64_t bd = tc::smem_desc_sw128(v_s(st) + ks * 2048, KV_REGION, 1024);
          tc::mma_ts(tmem + O_COL, tmem + scol + ks * 8, bd, IDESC_PV, (i > 0 || ks > 0) ? 1u : 0u);
        }
        tc::mma_commit(bo);
        tc::mma_commit(empty0 + 8 * st);
        return true;
      };
      for (int j = 0; j < ntiles && ok; ++j) {
        const int st = j % TC_STAGES;
        if (!tc::mbar_wait(full0 + 8 * st, (j / TC_STAGES) & 1, abort_flag)) {
          give_up();
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const uint32_t scol = (j & 1) ? S_COL1 : S_COL0;
#pragma unroll
        for (int k = 0; k < D / 16; ++k) {
          const uint32_t off = (k & 3) << 5;  // 32 bytes per 16-element K step
          const uint64_t ad = tc::smem_desc_sw128(q_s + (k >> 2) * Q_REGION + off, 16, 1024);
          const uint64_t bd = tc::smem_desc_sw128(k_s(st) + (k >> 2) * KV_REGION + off, 16, 1024);
          tc::mma_ss(tmem + scol, ad, bd, IDESC_QK, k > 0 ? 1u : 0u);
        }
        tc::mma_commit(bs0 + 8 * (j & 1));
        if (j >= 1) ok = pv(j - 1);
      }
      if (ok && ntiles > 0) pv(ntiles - 1);
      tc::mma_commit(bdrain);
      tc::mbar_wait(bdrain, 0, &s_zero);
    }
  } else {
    // ---------------- softmax: one query row per thread
    const uint32_t tl = tmem + (uint32_t(32 * (warp & 3)) << 16);
    const unsigned long long anc = (t_row < T) ? s_anc[t_row] : 0ull;
    float m_ref = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < ntiles; ++j) {
      const uint32_t scol = (j & 1) ? S_COL1 : S_COL0;
      if (!__all_sync(0xffffffffu, tc::mbar_wait(bs0 + 8 * (j & 1), (j >> 1) & 1, abort_flag))) {
        give_up();
        ok = false;
        break;
      }
      tc::fence_after_sync();
      uint32_t sv[64];
      tc::tmem_ld32(tl + scol, *reinterpret_cast<uint32_t(*)[32]>(&sv[0]));
      tc::tmem_ld32(tl + scol + 32, *reinterpret_cast<uint32_t(*)[32]>(&sv[32]));
      tc::tmem_wait_ld();
      const int s0 = c0 + j * TC_KT;
      const bool need_mask = (s0 + TC_KT > L) || (s0 + TC_KT > c1);
      float x[64];
      float mx = -INFINITY;
#pragma unroll
      for (int c = 0; c < 64; ++c) {
        float v = __uint_as_float(sv[c]) * p.scale_log2;
        if (need_mask) {
          const int col = s0 + c;
          const bool allowed = col < c1 && (col < L || ((anc >> (col - L)) & 1ull));
          if (!allowed) v = -INFINITY;
        }
        x[c] = v;
        mx = fmaxf(mx, v);
      }
      const bool resc = mx > m_ref + TC_RESCALE;
      float corr = 1.f;
      if (resc) {
        corr = (m_ref == -INFINITY) ? 0.f : tc::ex2(m_ref - mx);
        m_ref = mx;
        l *= corr;
      }
      const float mu = (m_ref == -INFINITY) ? 0.f : m_ref;
      uint32_t pk[32];
      float ps = 0.f;
#pragma unroll
      for (int c = 0; c < 32; ++c) {
        const float p0 = tc::ex2(x[2 * c] - mu), p1 = tc::ex2(x[2 * c + 1] - mu);
        ps += p0 + p1;
        pk[c] = pack_bf16x2(p0, p1);
      }
      l += ps;
      if (c1 - s0 < TC_KT) {
        // slots past the sequence end may hold any bits (0 * NaN = NaN in
        // the PV product): zero those V rows before the MMA reads them
        const int first = c1 - s0, nz = (TC_KT - first) * NR * 8;
        const int st = j % TC_STAGES;
        for (int i = tid - 64; i < nz; i += 128) {
          const int r = first + i / (NR * 8), rc = i % (NR * 8);
          const uint32_t dst = v_s(st) + (rc >> 3) * KV_REGION + r * 128 + ((rc & 7) << 4);
          asm volatile("st.shared.v4.b32 [%0], {%1,%1,%1,%1};" ::"r"(dst), "r"(0u) : "memory");
        }
        tc::fence_proxy_async_smem();
      }
      if (j > 0 && __any_sync(0xffffffffu, resc)) {
        // O must not change under a running PV: wait for the previous one
        if (!__all_sync(0xffffffffu, tc::mbar_wait(bo, (j - 1) & 1, abort_flag))) {
          give_up();
          ok = false;
          break;
        }
        tc::fence_after_sync();
#pragma unroll
        for (int c4 = 0; c4 < D / 32; ++c4) {
          uint32_t ov[32];
          tc::tmem_ld32(tl + O_COL + c4 * 32, ov);
          tc::tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * corr);
          tc::tmem_st32(tl + O_COL + c4 * 32, ov);
        }
      }
      tc::tmem_st32(tl + scol, pk);
      tc::tmem_wait_st();
      tc::fence_before_sync();
      tc::mbar_arrive(bp0 + 8 * (j & 1));
    }
    // ---- epilogue: O row from TMEM to the output (or to the split partials)
    if (ok && __all_sync(0xffffffffu, tc::mbar_wait(bo, (ntiles - 1) & 1, abort_flag))) {
      tc::fence_after_sync();
      const bool valid = grow < rows_b;
      const int hg = grow - t_row * p.G;
      const int64_t orow = (int64_t(b) * p.T_max + t_row) * p.Hq + g * p.G + hg;
      if (nsplit_b == 1) {
        const float inv = 1.f / l;
#pragma unroll
        for (int c4 = 0; c4 < D / 32; ++c4) {
          uint32_t ov[32];
          tc::tmem_ld32(tl + O_COL + c4 * 32, ov);
          tc::tmem_wait_ld();
          if (valid) {
            uint4 *dst = reinterpret_cast<uint4 *>(p.out + orow * D + c4 * 32);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              uint4 w;
              w.x = pack_bf16x2(__uint_as_float(ov[8 * e + 0]) * inv, __uint_as_float(ov[8 * e + 1]) * inv);
              w.y = pack_bf16x2(__uint_as_float(ov[8 * e + 2]) * inv, __uint_as_float(ov[8 * e + 3]) * inv);
              w.z = pack_bf16x2(__uint_as_float(ov[8 * e + 4]) * inv, __uint_as_float(ov[8 * e + 5]) * inv);
              w.w = pack_bf16x2(__uint_as_float(ov[8 * e + 6]) * inv, __uint_as_float(ov[8 * e + 7]) * inv);
              dst[e] = w;
            }
          }
        }
        if (valid && p.lse != nullptr) p.lse[orow] = (m_ref + log2f(l)) * LN2;
      } else {
        const int64_t pair = (int64_t(b) * p.Hkv + g) * p.nrb + rb;
        const int64_t prow = (pair * p.nsplit + split) * TC_ROWS + row;
#pragma unroll
        for (int c4 = 0; c4 < D / 32; ++c4) {
          uint32_t ov[32];
          tc::tmem_ld32(tl + O_COL + c4 * 32, ov);
          tc::tmem_wait_ld();
          uint4 *dst = reinterpret_cast<uint4 *>(p.ws_o + prow * D + c4 * 32);
#pragma unroll
          for (int e = 0; e < 8; ++e) dst[e] = make_uint4(ov[4 * e], ov[4 * e + 1], ov[4 * e + 2], ov[4 * e + 3]);
        }
        p.ws_ml[prow] = make_float2(m_ref, l);
      }
    } else if (ok) {
      give_up();
    }
  }

  // ---- teardown: every copy and MMA has completed (or timed out) by now
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, TC_TMEM_COLS);
  }
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Log-sum-exp merge of the split partials: one warp per query row of a
// (b, g, row block); rows of sequences that needed a single split were
// written by the partial kernel and are skipped. Launched as a programmatic
// dependent of the partial kernel: griddepcontrol.wait returns once that grid
// has completed and its writes are visible.
template <int D, int NW>
__global__ void __launch_bounds__(256) tree_attn_merge_kernel(const AttnParams p) {
  constexpr int RPC = NW * 16;
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t row = int64_t(blockIdx.x) * 8 + warp;
  const int64_t pair = row / RPC;
  const int r = int(row - pair * RPC);
  const int rb = int(pair % p.nrb);
  const int64_t bg = pair / p.nrb;
  const int g = int(bg % p.Hkv);
  const int b = int(bg / p.Hkv);
  if (b >= p.B) return;
  const int T = __ldg(p.tree_len + b);
  const int L = __ldg(p.kv_len + b);
  if (T < 1 || T > p.T_max || L < 0 || L > p.capacity - T) return;
  const int nsplit_b = (L + T + p.chunk - 1) / p.chunk;
  const int gr = rb * RPC + r;
  if (nsplit_b == 1 || gr >= T * p.G) return;
  int bad = 0;  // the partial kernel skipped malformed trees; so does the merge
  for (int i = lane; i < T; i += 32) {
    const int par = __ldg(p.parent + int64_t(b) * p.T_max + i);
    bad |= (i == 0) ? (par != -1) : (par < 0 || par >= i);
  }
  if (__any_sync(0xffffffffu, bad)) return;

  const int64_t sbase = pair * p.nsplit * RPC;
  float M = -INFINITY;
  for (int s = 0; s < nsplit_b; ++s) M = fmaxf(M, __ldcg(p.ws_ml + sbase + int64_t(s) * RPC + r).x);
  const float Mu = (M == -INFINITY) ? 0.f : M;
  if (lane >= D / 4) return;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float Ls = 0.f;
  for (int s = 0; s < nsplit_b; ++s) {
    const float2 ml = __ldcg(p.ws_ml + sbase + int64_t(s) * RPC + r);
    const float w = exp2f(ml.x - Mu);
    const float4 x = __ldcg(reinterpret_cast<const float4 *>(p.ws_o + (sbase + int64_t(s) * RPC + r) * D) + lane);
    Ls += w * ml.y;
    acc.x += w * x.x;
    acc.y += w * x.y;
    acc.z += w * x.z;
    acc.w += w * x.w;
  }
  const float inv = 1.f / Ls;
  const int t = gr / p.G, h = g * p.G + (gr - t * p.G);
  const int64_t orow = (int64_t(b) * p.T_max + t) * p.Hq + h;
  uint2 pk;
  pk.x = pack_bf16x2(acc.x * inv, acc.y * inv);
  pk.y = pack_bf16x2(acc.z * inv, acc.w * inv);
  *reinterpret_cast<uint2 *>(p.out + orow * D + lane * 4) = pk;
  if (p.lse != nullptr && lane == 0) p.lse[orow] = (M + log2f(Ls)) * LN2;
}

struct AttnPlan {
  int nw;
  int rpc;
  int nrb;
  int nsplit;
  int chunk;
  size_t ws_o_bytes, ws_ml_bytes;
  size_t ws_bytes;
};

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

AttnPlan plan(const dreams_kv_cache_t *kv, const dreams_tree_t *tree, int Hq) {
  AttnPlan pl{};
  const int G = Hq / kv->Hkv;
  const int rows = tree->T_max * G;
  pl.nw = TC_ROWS / 16;
  pl.rpc = TC_ROWS;
  pl.nrb = (rows + pl.rpc - 1) / pl.rpc;
  // about two waves of two CTAs per SM, splits of at least 256 tokens
  const int64_t base = int64_t(tree->B) * kv->Hkv * pl.nrb;
  const int64_t target = int64_t(num_sms()) * 2 * 2;
  int64_t ns = (target + base - 1) / base;
  const int64_t max_ns = std::max<int64_t>(1, (kv->capacity + 255) / 256);
  ns = std::min(std::max<int64_t>(ns, 1), max_ns);
  int64_t chunk = (kv->capacity + ns - 1) / ns;
  chunk = (chunk + TC_KT - 1) / TC_KT * TC_KT;
  pl.chunk = int(chunk);
  pl.nsplit = int((kv->capacity + chunk - 1) / chunk);
  if (pl.nsplit > 1) {
    const size_t slots = size_t(base) * pl.nsplit * pl.rpc;
    pl.ws_o_bytes = align_up(slots * kv->D * sizeof(float), 256);
    pl.ws_ml_bytes = align_up(slots * sizeof(float2), 256);
  }
  pl.ws_bytes = pl.ws_o_bytes + pl.ws_ml_bytes;
  return pl;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

// 4-D view of one layer's K or V cache with a (64 columns, 1 head, 64 slots,
// 1) box, 128-byte swizzle; out-of-range boxes read as zeros.
//   contiguous: (D, Hkv, capacity, B);  paged: (D, Hkv, 64, num_pages).
bool make_kv_map(CUtensorMap *m, const void *base, const dreams_kv_cache_t *kv, int B) {
  EncodeTiledFn enc = encode_tiled();
  if (enc == nullptr) return false;
  const cuuint64_t D = cuuint64_t(kv->D), H = cuuint64_t(kv->Hkv);
  cuuint64_t dims[4] = {D, H, 0, 0};
  cuuint64_t strides[3] = {D * 2, H * D * 2, 0};
  if (kv->page_table != nullptr) {
    dims[2] = 64;
    dims[3] = cuuint64_t(kv->num_pages);
    strides[2] = 64 * H * D * 2;
  } else {
    dims[2] = cuuint64_t(kv->capacity);
    dims[3] = cuuint64_t(B);
    strides[2] = cuuint64_t(kv->capacity) * H * D * 2;
  }
  const cuuint32_t box[4] = {64, 1, 64, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D>
dreams_status_t launch_attn_tc(const AttnParams &a, const AttnPlan &pl, const dreams_kv_cache_t *kv, int B,
                               cudaStream_t stream) {
  constexpr size_t smem = size_t(D / 64) * TC_ROWS * 128 + size_t(TC_STAGES) * 2 * (D / 64) * TC_KT * 128 + 1024;
  static int configured_mask = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 31 && !(configured_mask & (1 << dev))) {
    cudaError_t e =
        cudaFuncSetAttribute(tree_attn_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e != cudaSuccess) {
      set_last_cuda_error(e);
      return DREAMS_ERR_CUDA;
    }
    configured_mask |= (1 << dev);
  }
  TcParams P;
  memset(&P, 0, sizeof(P));
  P.a = a;
  P.paged = kv->page_table != nullptr;
  if (!make_kv_map(&P.tmap_k, a.k, kv, B) || !make_kv_map(&P.tmap_v, a.v, kv, B)) return DREAMS_ERR_UNSUPPORTED;
  dim3 grid(pl.nrb * pl.nsplit, a.Hkv, B);
  tree_attn_tc_kernel<D><<<grid, TC_THREADS, smem, stream>>>(P);
  dreams_status_t st = check_launch();
  if (st != DREAMS_OK || pl.nsplit == 1) return st;
  const int64_t rows = int64_t(B) * a.Hkv * pl.nrb * TC_ROWS;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned((rows + 7) / 8));
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, tree_attn_merge_kernel<D, TC_ROWS / 16>, a);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  return check_launch();
}

bool valid_shapes(const dreams_kv_cache_t *kv, const dreams_tree_t *tree, int Hq) {
  return kv != nullptr && tree != nullptr && tree->B >= 1 && tree->B <= 65535 && tree->T_max >= 1 &&
         tree->T_max <= 64 && kv->Hkv >= 1 && kv->Hkv <= 65535 && Hq >= kv->Hkv && Hq % kv->Hkv == 0 &&
         kv->capacity >= 1 && kv->n_layers >= 1;
}

template <int D, int NW>
dreams_status_t launch_attn(const AttnParams &p, const AttnPlan &pl, int B, cudaStream_t stream) {
  const size_t smem = size_t(NW * 16 + STAGES * 2 * KT) * D * sizeof(__nv_bfloat16);
  static int configured_mask = 0;  // per device bit
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 31 && !(configured_mask & (1 << dev))) {
    cudaError_t e = cudaFuncSetAttribute(tree_attn_mma_kernel<D, NW>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e != cudaSuccess) {
      set_last_cuda_error(e);
      return DREAMS_ERR_CUDA;
    }
    configured_mask |= (1 << dev);
  }
  dim3 grid(pl.nrb * pl.nsplit, p.Hkv, B);
  tree_attn_mma_kernel<D, NW><<<grid, NW * 32, smem, stream>>>(p);
  dreams_status_t st = check_launch();
  if (st != DREAMS_OK || pl.nsplit == 1) return st;
  const int64_t rows = int64_t(B) * p.Hkv * pl.nrb * (NW * 16);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned((rows + 7) / 8));
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, tree_attn_merge_kernel<D, NW>, p);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  return check_launch();
}

}  // namespace
}  // namespace dreams

using namespace dreams;

extern "C" size_t dreams_tree_verify_attn_workspace_size(const dreams_kv_cache_t *kv,
                                                         const dreams_tree_t *tree, int32_t Hq) {
  if (!valid_shapes(kv, tree, Hq)) return 0;
  return plan(kv, tree, Hq).ws_bytes;
}

extern "C" dreams_status_t dreams_tree_verify_attn(const void *q, const dreams_kv_cache_t *kv, int32_t layer,
                                                   const dreams_tree_t *tree, int32_t Hq, float scale,
                                                   void *out, float *lse, void *workspace,
                                                   size_t workspace_bytes, int32_t *status_word,
                                                   dreams_stream_t stream) {
  if (q == nullptr || out == nullptr || kv == nullptr || tree == nullptr) return DREAMS_ERR_INVALID_ARG;
  if (kv->k == nullptr || kv->v == nullptr || tree->parent == nullptr || tree->tree_len == nullptr ||
      tree->kv_len == nullptr)
    return DREAMS_ERR_INVALID_ARG;
  if (!valid_shapes(kv, tree, Hq)) return DREAMS_ERR_INVALID_ARG;
  if (kv->D != 64 && kv->D != 128) return DREAMS_ERR_UNSUPPORTED;
  if (layer < 0 || layer >= kv->n_layers || kv->layer_stride < 0) return DREAMS_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out) || !aligned16(kv->k) || !aligned16(kv->v) ||
      (kv->layer_stride * 2) % 16 != 0 || (lse != nullptr && (reinterpret_cast<uintptr_t>(lse) & 3)))
    return DREAMS_ERR_INVALID_ARG;
  if (!isfinite(scale)) return DREAMS_ERR_INVALID_ARG;
  if (kv->page_table != nullptr) {
    if (kv->page_size != 64) return DREAMS_ERR_UNSUPPORTED;
    if (kv->pages_per_seq < 1 || kv->num_pages < 1 || int64_t(kv->pages_per_seq) * 64 != kv->capacity)
      return DREAMS_ERR_INVALID_ARG;
  }
  const AttnPlan pl = plan(kv, tree, Hq);
  if (pl.ws_bytes > 0 && (workspace == nullptr || workspace_bytes < pl.ws_bytes || !aligned16(workspace)))
    return DREAMS_ERR_WORKSPACE;
  if (int64_t(pl.nrb) * pl.nsplit > 0x7fffffff) return DREAMS_ERR_UNSUPPORTED;

  AttnParams p{};
  p.q = static_cast<const __nv_bfloat16 *>(q);
  p.out = static_cast<__nv_bfloat16 *>(out);
  p.lse = lse;
  p.k = static_cast<const __nv_bfloat16 *>(kv->k) + int64_t(layer) * kv->layer_stride;
  p.v = static_cast<const __nv_bfloat16 *>(kv->v) + int64_t(layer) * kv->layer_stride;
  p.page_table = kv->page_table;
  p.pages_per_seq = kv->pages_per_seq;
  p.num_pages = kv->num_pages;
  p.capacity = kv->capacity;
  p.parent = tree->parent;
  p.tree_len = tree->tree_len;
  p.kv_len = tree->kv_len;
  p.B = tree->B;
  p.T_max = tree->T_max;
  p.Hq = Hq;
  p.Hkv = kv->Hkv;
  p.G = Hq / kv->Hkv;
  p.nrb = pl.nrb;
  p.nsplit = pl.nsplit;
  p.chunk = pl.chunk;
  p.scale_log2 = scale * LOG2E;
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  if (pl.ws_bytes > 0) {
    p.ws_o = reinterpret_cast<float *>(ws);
    p.ws_ml = reinterpret_cast<float2 *>(ws + pl.ws_o_bytes);
  }
  p.status = status_word;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return kv->D == 128 ? launch_attn_tc<128>(p, pl, kv, tree->B, s) : launch_attn_tc<64>(p, pl, kv, tree->B, s);
}
