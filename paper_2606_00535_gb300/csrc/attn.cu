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
// (b, g, row block) write unnormalised partials (m, l, O) to the workspace;
// the last split to finish (ticket counter, no waiting) merges them by
// log-sum-exp and resets its counter.
#include <math.h>

#include <algorithm>

#include "common.cuh"

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
  int32_t T_max, Hq, Hkv, G;
  int32_t nrb;     // query-row blocks per (b, g)
  int32_t nsplit;  // KV splits in the grid
  int32_t chunk;   // KV tokens per split, a multiple of KT
  float scale_log2;
  float *ws_o;      // [B][Hkv][nrb][nsplit][RPC][D]
  float2 *ws_ml;    // [B][Hkv][nrb][nsplit][RPC]  (m in log2 units, l)
  int32_t *ws_cnt;  // [B][Hkv][nrb]
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

  // ---- split partials, then the last split of (b, g, rb) merges
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
  __threadfence();
  __syncthreads();
  if (tid == 0) s_flag = (atomicAdd(p.ws_cnt + pair, 1) == nsplit_b - 1);
  __syncthreads();
  if (!s_flag) return;
  __threadfence();

  const int64_t sbase = pair * p.nsplit * RPC;
  for (int idx = tid; idx < RPC * (D / 4); idx += NT) {
    const int r = idx / (D / 4), d4 = idx % (D / 4);
    const int gr = rb * RPC + r;
    if (gr >= rows_b) continue;
    float M = -INFINITY;
    for (int s = 0; s < nsplit_b; ++s) M = fmaxf(M, __ldcg(p.ws_ml + sbase + int64_t(s) * RPC + r).x);
    const float Mu = (M == -INFINITY) ? 0.f : M;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    float Ls = 0.f;
    for (int s = 0; s < nsplit_b; ++s) {
      const float2 ml = __ldcg(p.ws_ml + sbase + int64_t(s) * RPC + r);
      const float w = exp2f(ml.x - Mu);
      const float4 x = __ldcg(reinterpret_cast<const float4 *>(p.ws_o + (sbase + int64_t(s) * RPC + r) * D) + d4);
      Ls += w * ml.y;
      acc.x += w * x.x;
      acc.y += w * x.y;
      acc.z += w * x.z;
      acc.w += w * x.w;
    }
    const float inv = 1.f / Ls;
    const int t = gr / p.G, h = g * p.G + (gr - t * p.G);
    __nv_bfloat16 *dst = p.out + ((q_base + int64_t(t) * p.Hq + h) * D) + d4 * 4;
    uint2 pk;
    pk.x = pack_bf16x2(acc.x * inv, acc.y * inv);
    pk.y = pack_bf16x2(acc.z * inv, acc.w * inv);
    *reinterpret_cast<uint2 *>(dst) = pk;
    if (p.lse != nullptr && d4 == 0) p.lse[q_base + int64_t(t) * p.Hq + h] = (M + log2f(Ls)) * LN2;
  }
  if (tid == 0) p.ws_cnt[pair] = 0;
}

struct AttnPlan {
  int nw;
  int rpc;
  int nrb;
  int nsplit;
  int chunk;
  size_t ws_o_bytes, ws_ml_bytes, ws_cnt_bytes;
  size_t ws_bytes;
};

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

AttnPlan plan(const dreams_kv_cache_t *kv, const dreams_tree_t *tree, int Hq) {
  AttnPlan pl{};
  const int G = Hq / kv->Hkv;
  const int rows = tree->T_max * G;
  pl.nw = rows <= 64 ? 4 : 8;
  pl.rpc = pl.nw * 16;
  pl.nrb = (rows + pl.rpc - 1) / pl.rpc;
  const int64_t base = int64_t(tree->B) * kv->Hkv * pl.nrb;
  const int64_t target = int64_t(num_sms()) * (pl.nw == 4 ? 2 : 1) * 2;
  int64_t ns = (target + base - 1) / base;
  const int64_t max_ns = std::max<int64_t>(1, (kv->capacity + 255) / 256);
  ns = std::min(std::max<int64_t>(ns, 1), max_ns);
  int64_t chunk = (kv->capacity + ns - 1) / ns;
  chunk = (chunk + KT - 1) / KT * KT;
  pl.chunk = int(chunk);
  pl.nsplit = int((kv->capacity + chunk - 1) / chunk);
  if (pl.nsplit > 1) {
    const size_t slots = size_t(base) * pl.nsplit * pl.rpc;
    pl.ws_o_bytes = align_up(slots * kv->D * sizeof(float), 256);
    pl.ws_ml_bytes = align_up(slots * sizeof(float2), 256);
    pl.ws_cnt_bytes = align_up(size_t(base) * sizeof(int32_t), 256);
  }
  pl.ws_bytes = pl.ws_o_bytes + pl.ws_ml_bytes + pl.ws_cnt_bytes;
  return pl;
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
    p.ws_cnt = reinterpret_cast<int32_t *>(ws + pl.ws_o_bytes + pl.ws_ml_bytes);
  }
  p.status = status_word;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (kv->D == 128) {
    return pl.nw == 4 ? launch_attn<128, 4>(p, pl, tree->B, s) : launch_attn<128, 8>(p, pl, tree->B, s);
  }
  return pl.nw == 4 ? launch_attn<64, 4>(p, pl, tree->B, s) : launch_attn<64, 8>(p, pl, tree->B, s);
}
