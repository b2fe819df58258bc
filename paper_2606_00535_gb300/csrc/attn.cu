// attn.cu -- tree-masked verification attention on tcgen05 tensor cores.
//
// What it computes (paper Sec. 2, "Speculative decoding": the target scores
// every draft token in one parallel pass; Sec. 2, "Vision-Language Models":
// every cached visual and text token is attended at each decoding step;
// attention = softmax(Q K^T * scale), Sec. 3.2): for tree node t of sequence b
// and query head h, softmax attention over the prefix slots 0..L-1 and the
// slots L + a of t and its ancestors a, with KV head g = h / G.
//
// Work decomposition: one CTA per work item (sequence b, KV split, KV head g,
// row block rb), one CTA per SM. A row block holds TB = 128 / G tree nodes
// times the G query heads of the group, row = (t - rb*TB) * G + (h - gG), so
// one pass over a K/V tile serves every query head of the GQA group and every
// tree node of the block. With more than one sequence the CTAs take the
// (sequence, split) pairs longest first, so that the hardware, which hands out
// CTAs in index order as SMs free up, schedules the items longest-processing-
// time first: with up to 64 pairs each CTA ranks the pairs itself, with more a
// one-CTA kernel orders them first.
//
// Roles (320 threads):
//   warp 8, one thread  TMA producer: the Q block first (one 5-D box per
//                       64-column region), then 128-token K tiles into a
//                       3-stage ring and V tiles into a 3-stage ring (4-D
//                       boxes of 64 slots x 64 head columns, 128-byte
//                       swizzle). It polls both rings without blocking and
//                       keeps V a tile behind K (QK^T of tile j + 1 runs
//                       before PV of tile j); page-table entries are loaded
//                       one tile ahead.
//   warp 9, one thread  MMA issuer: S = Q K^T (M128 N128, K-major operands) into
//                       TMEM, O += P V (M128 N=D, P read from TMEM, V as an
//                       MN-major operand). Tile j goes to warpgroup j % 2, and
//                       the QK^T of tile j + 2 follows the PV of tile j (they
//                       share that warpgroup's S/P columns). The tensor pipe
//                       queues about one MMA, so the thread must not stall
//                       between MMAs: per tile it waits once (for P_j), then
//                       issues PV_j and QK_{j+2} (16 MMAs) under one commit.
//                       Tree and cross-attention rows hand P_j over in two
//                       halves of 64 keys, so the first half of PV_j runs
//                       while the softmax finishes the tile; on a paged cache
//                       the thread also commits V_j's stage free right after
//                       PV_j.
//   warps 0-3, 4-7      two softmax warpgroups, one query row per thread. A
//                       warpgroup owns one S/P buffer and its own O in TMEM
//                       (256 columns each), so the two alternate over the
//                       tiles. A thread loads its 128 scores, applies the
//                       ancestor mask on tiles that reach the tree slots,
//                       exponentiates with ex2.approx against a reference
//                       maximum that is raised only when a tile's maximum
//                       exceeds it by 2^8 (and only then rescales its O), and
//                       writes P as bf16 over S. Woken by the commit after
//                       QK_j (which also covers PV_{j-2}), one thread
//                       releases the K stage of tile j and (unless the MMA
//                       thread did) the V stage of tile j - 2 to the
//                       producer; before the warpgroup signals P_j (or its
//                       first half) it waits for V_j and K_{j+2} (or V_j) to
//                       land, so that the MMA thread needs no other wait.
//                       Warps whose rows are all padding sit out.
// At the end the two warpgroups combine their (m, l, O) by log-sum-exp. A
// block whose rows all lie inside the tensor leaves through TMA stores of the
// output staged in shared memory; other blocks write each row's half of the
// columns with 16-byte stores: the output, or the split partials that a merge
// kernel (chained by programmatic dependent launch) combines. Every mbarrier wait is bounded (2 s); on a
// timeout the CTA flags DREAMS_DATA_TIMEOUT, drains its copies and MMAs, frees
// its TMEM and exits. The workspace holds no state between calls.
#include <cuda.h>
#include <limits.h>
#include <math.h>
#include <string.h>

#include <algorithm>

#include "common.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace dreams {
namespace {

constexpr float LOG2E = 1.4426950408889634f;
constexpr float LN2 = 0.6931471805599453f;

constexpr int KT = 128;        // KV tokens per tile (UMMA N of QK^T)
constexpr int ROWS = 128;      // query rows per CTA (UMMA M)
constexpr int NK = 3;          // K ring stages
constexpr int NV = 3;          // V ring stages
constexpr int CRD = 8;         // producer's ring of tile coordinates (V trails K by < CRD tiles)
constexpr int THREADS = 320;   // 8 softmax warps, TMA warp, MMA warp
constexpr int TMA_WARP = 8, MMA_WARP = 9;
constexpr float RESCALE = 8.f; // log2 headroom of the reference maximum
constexpr uint32_t TMEM_COLS = 512;
constexpr int MAX_SPLITS = 32; // KV splits per sequence (one merge lane each)
constexpr int ORDER_THREADS = 1024;
constexpr int RANK_PAIRS = 64;     // up to this many (sequence, split) pairs each CTA ranks them itself
constexpr int ORDER_KEYS = 4096;  // item sizes (tiles) above this share the top bucket
constexpr int PAST_TABLE = INT_MIN;  // page-table slot past the table: reads as zeros

struct AttnParams {
  const __nv_bfloat16 *q;
  __nv_bfloat16 *out;
  float *lse;
  const int32_t *page_table;  // nullptr: contiguous cache
  int32_t pages_per_seq;
  int32_t num_pages;
  int32_t capacity;
  const int32_t *parent;
  const int32_t *tree_len;
  const int32_t *kv_len;
  int32_t B, T_max, Hq, Hkv, G;
  int32_t TB;      // tree nodes per row block (ROWS / G)
  int32_t nrb;     // row blocks per (b, g)
  int32_t nsplit;  // KV splits per sequence in the grid
  int32_t chunk;   // KV tokens per split, a multiple of KT
  float scale_log2;
  float *ws_o;     // [B][Hkv][nrb][nsplit][ROWS][D] unnormalised partial O
  float2 *ws_ml;   // [B][Hkv][nrb][nsplit][ROWS] (max in log2 units, sum)
  int32_t *order;  // [B * nsplit] pair index b * nsplit + split, longest first; nullptr: see rank
  int32_t rank;    // with no order: 1 = each CTA ranks the pairs itself (B * nsplit <= RANK_PAIRS), 0 = natural order
  int32_t *status;
  int32_t mode;    // ATTN_TREE, ATTN_FULL or ATTN_CAUSAL: which slots a query row attends
  float *ent;      // [B, T_max, Hq] attention entropy of each query row (nats), with the entropy kernels
  float *ws_w;     // [B][Hkv][nrb][nsplit][ROWS] sum_j P_j (x_j - m) of the split partials (entropy)
  uint64_t wait_ns;  // limit of every pipeline wait (2 s unless a test shortens it)
  int32_t stall_at;  // test hook: K tiles from this index on are never issued (-1: off)
};

constexpr int ATTN_TREE = 0;    // prefix slots plus the node's own ancestors among the tree slots
constexpr int ATTN_FULL = 1;    // slots 0 .. kv_len - 1 (cross-attention: no mask)
constexpr int ATTN_CAUSAL = 2;  // slots 0 .. kv_len + t for query t (prefill self-attention)

// Keys of sequence b: the prefix plus the query rows' own slots (tree,
// causal), or the prefix alone (full).
__device__ __forceinline__ int key_total(const AttnParams &p, int L, int T) { return p.mode == ATTN_FULL ? L : L + T; }

// A read-only global load issued where it stands (the compiler may not sink it
// to the value's first use).
__device__ __forceinline__ int ld_issue_now(const int32_t *ptr) {
  int v;
  asm volatile("ld.global.nc.b32 %0, [%1];" : "=r"(v) : "l"(ptr));
  return v;
}

struct TcParams {
  CUtensorMap tmap_q;
  CUtensorMap tmap_k;
  CUtensorMap tmap_v;
  CUtensorMap tmap_o;  // the output, with the query block's box
  AttnParams a;
  int32_t paged;
};

__device__ __forceinline__ void named_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// Three-input maximum, and f32 pairs for the packed (f32x2) FMA and add.
__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
__device__ __forceinline__ uint64_t f32x2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f32x2_split(uint64_t v, float &lo, float &hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// KV tiles of split s of sequence b (0 for an empty split or bad lengths).
__device__ __forceinline__ int split_tiles(const AttnParams &p, int b, int s) {
  const int T = __ldg(p.tree_len + b);
  const int L = __ldg(p.kv_len + b);
  const int total = key_total(p, L, T);
  if (T < 1 || T > p.T_max || L < 0 || total > p.capacity || total < 1) return 0;
  const int tiles = (total + KT - 1) / KT;
  const int ct = p.chunk / KT;
  return ::max(0, ::min(ct, tiles - s * ct));
}

// Orders the (sequence, split) pairs by their number of KV tiles, largest
// first (a counting sort; pairs of equal size may come in any order, which
// changes only which SM computes them, not the result).
__global__ void __launch_bounds__(ORDER_THREADS) tree_attn_order_kernel(const AttnParams p) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  __shared__ int bucket[ORDER_KEYS];
  __shared__ int warp_sum[ORDER_THREADS / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int P = p.B * p.nsplit;
  for (int k = tid; k < ORDER_KEYS; k += ORDER_THREADS) bucket[k] = 0;
  __syncthreads();
  for (int e = tid; e < P; e += ORDER_THREADS) {
    const int b = e / p.nsplit;
    atomicAdd(&bucket[::min(split_tiles(p, b, e - b * p.nsplit), ORDER_KEYS - 1)], 1);
  }
  __syncthreads();
  // start of key k = number of pairs with a larger key; thread t owns keys
  // ORDER_KEYS-1-4t down to ORDER_KEYS-4-4t
  int v[4], sum = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    v[i] = bucket[ORDER_KEYS - 1 - 4 * tid - i];
    sum += v[i];
  }
  int x = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sum[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = warp_sum[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    warp_sum[lane] = w;
  }
  __syncthreads();
  int run = x - sum + (warp > 0 ? warp_sum[warp - 1] : 0);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    bucket[ORDER_KEYS - 1 - 4 * tid - i] = run;
    run += v[i];
  }
  __syncthreads();
  for (int e = tid; e < P; e += ORDER_THREADS) {
    const int b = e / p.nsplit;
    const int pos = atomicAdd(&bucket[::min(split_tiles(p, b, e - b * p.nsplit), ORDER_KEYS - 1)], 1);
    p.order[pos] = e;
  }
}

// SPLIT: P is handed to the MMA thread in two halves, so that the first half
// of PV_j runs while the softmax warps finish the tile (tree and
// cross-attention rows, bound by the softmax-MMA chain), or whole (causal
// rows, bound by the tensor pipe, where the extra wait between the PV halves
// costs more than it saves). VREL (with SPLIT): a V stage goes back to the
// producer as soon as its PV has completed (one more commit per tile) rather
// than at the next wake-up of the softmax warps: worth it where the copies
// land late, on paged caches. The host picks both by mode and cache layout.
template <int D, bool ENT, bool SPLIT, bool VREL>
__global__ void __launch_bounds__(THREADS, 1) tree_attn_tc_kernel(const __grid_constant__ TcParams P) {
  static_assert(SPLIT || !VREL, "the early V release goes with the two-half hand-off");
  const AttnParams &p = P.a;
  constexpr int NR = D / 64;                     // 128-byte column regions of a row
  constexpr uint32_t Q_REGION = ROWS * 128;      // 16 KB
  constexpr uint32_t KV_REGION = KT * 128;       // 16 KB: 128 slots x 64 columns
  constexpr uint32_t Q_BYTES = NR * Q_REGION;
  constexpr uint32_t KV_TILE = NR * KV_REGION;   // one K or V tile
  constexpr uint32_t IDESC_QK = tc::idesc_bf16_f32(ROWS, KT, false);
  constexpr uint32_t IDESC_PV = tc::idesc_bf16_f32(ROWS, D, true);

  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar_kf[NK], bar_ke[NK], bar_vf[NV], bar_ve[NV];
  __shared__ __align__(8) uint64_t bar_s[2], bar_p[2], bar_ph[2], bar_q, bar_drain, bar_never;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_zero, s_flag, s_tma;
  __shared__ unsigned long long s_anc[64];
  __shared__ int s_jump[64];
  __shared__ int s_key[RANK_PAIRS];
  __shared__ int s_pair;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int per_pair = p.Hkv * p.nrb;
  const int pair_pos = blockIdx.x / per_pair;
  const int gr = blockIdx.x - pair_pos * per_pair;
  // Tree and cross-attention rows: KV head, then row block (the row blocks of
  // a head, adjacent, share its K/V tiles through L2). Causal rows: the last
  // row blocks have the most keys, so the order is row block (last first),
  // then KV head: the hardware, handing out CTAs in index order, then
  // schedules longest first.
  const bool causal = p.mode == ATTN_CAUSAL;
  const int g = causal ? gr % p.Hkv : gr / p.nrb;
  const int rb = causal ? p.nrb - 1 - gr / p.Hkv : gr - g * p.nrb;
  int pair = pair_pos;
  if (p.order != nullptr) {
    // the order comes from the preceding kernel (programmatic dependent launch)
    asm volatile("griddepcontrol.wait;" ::: "memory");
    pair = __ldcg(p.order + pair_pos);
  } else if (p.rank) {
    // few pairs: the CTA takes the pair of rank pair_pos in the order by KV
    // tiles, largest first, ties by pair index (every CTA computes the same
    // order, one pair per thread)
    const int np = p.B * p.nsplit;
    int key = 0;
    if (tid < np) {
      key = split_tiles(p, tid / p.nsplit, tid % p.nsplit);
      s_key[tid] = key;
    }
    __syncthreads();
    if (tid < np) {
      int r = 0;
      for (int f = 0; f < np; ++f) {
        const int kf = s_key[f];
        r += (kf > key) || (kf == key && f < tid);
      }
      if (r == pair_pos) s_pair = tid;
    }
    __syncthreads();
    pair = s_pair;
  }
  const int b = pair / p.nsplit, split = pair - b * p.nsplit;
  // The loads the prologue depends on go out together: the tree row (softmax
  // warp 0, which builds the masks) and the first page-table entries
  // (producer), next to the lengths. Volatile, so that they are issued here
  // and not where their values are first used.
  int par_pre[2] = {-1, -1};
  if (warp == 0 && p.mode == ATTN_TREE) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int i = lane + 32 * h;
      if (i < p.T_max) par_pre[h] = ld_issue_now(p.parent + int64_t(b) * p.T_max + i);
    }
  }
  int pn_pre[2] = {PAST_TABLE, PAST_TABLE};
  if (tid == TMA_WARP * 32 && P.paged) {
    const int pi = (split * p.chunk) >> 6;
    const int32_t *prow = p.page_table + int64_t(b) * p.pages_per_seq;
    if (pi < p.pages_per_seq) pn_pre[0] = __ldg(prow + pi);
    if (pi + 1 < p.pages_per_seq) pn_pre[1] = __ldg(prow + pi + 1);
  }
  const uint32_t smem_base = smem_u32(smem);
  const uint32_t q_s = smem_base;
  auto k_s = [&](int st) { return smem_base + Q_BYTES + uint32_t(st) * KV_TILE; };
  auto v_s = [&](int st) { return smem_base + Q_BYTES + uint32_t(NK + st) * KV_TILE; };
  const uint32_t kf0 = smem_u32(&bar_kf[0]), ke0 = smem_u32(&bar_ke[0]);
  const uint32_t vf0 = smem_u32(&bar_vf[0]), ve0 = smem_u32(&bar_ve[0]);
  const uint32_t bs0 = smem_u32(&bar_s[0]), bp0 = smem_u32(&bar_p[0]), bph0 = smem_u32(&bar_ph[0]);
  const uint32_t bq = smem_u32(&bar_q), bdrain = smem_u32(&bar_drain), bnever = smem_u32(&bar_never);
  const int t0 = rb * p.TB;  // first tree node of the row block
  const int c0 = split * p.chunk;

  // With a contiguous cache and the pair known from the grid index, the Q
  // block and the first K tile have known coordinates before the lengths
  // arrive: the producer sets up the copy barriers and issues both at once.
  // A CTA that then turns out to have nothing to do waits for them to land
  // before it exits.
  const bool early = !P.paged && p.order == nullptr && !p.rank && p.stall_at < 0;
  auto init_copy_barriers = [&]() {
    for (int i = 0; i < NK; ++i) {
      tc::mbar_init(kf0 + 8 * i, 1);
      tc::mbar_init(ke0 + 8 * i, 1);
    }
    for (int i = 0; i < NV; ++i) {
      tc::mbar_init(vf0 + 8 * i, 1);
      tc::mbar_init(ve0 + 8 * i, 1);
    }
    tc::mbar_init(bq, 1);
    s_zero = 0;
  };
  auto issue_q = [&]() {
    tc::prefetch_tmap(&P.tmap_q);
    tc::prefetch_tmap(&P.tmap_k);
    tc::prefetch_tmap(&P.tmap_v);
    // the Q rows of the block: G heads x TB nodes per 64-column region
    // (nodes past T_max read as zeros; the transaction counts the full box)
    tc::mbar_arrive_expect_tx(bq, uint32_t(NR * p.G * p.TB * 128));
#pragma unroll
    for (int r = 0; r < NR; ++r) tc::tma_load_5d(q_s + r * Q_REGION, &P.tmap_q, bq, r * 64, 0, g, t0, b);
  };
  if (early && tid == TMA_WARP * 32) {
    init_copy_barriers();
    tc::fence_barrier_init();
    issue_q();
    tc::mbar_arrive_expect_tx(kf0, KV_TILE);
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      tc::tma_load_4d(k_s(0) + r * KV_REGION, &P.tmap_k, kf0, r * 64, g, c0, b);
      tc::tma_load_4d(k_s(0) + r * KV_REGION + 8192, &P.tmap_k, kf0, r * 64, g, c0 + 64, b);
    }
  }
  auto leave = [&]() {
    if (early && tid == TMA_WARP * 32) {
      tc::mbar_wait(bq, 0, &s_zero);
      tc::mbar_wait(kf0, 0, &s_zero);
    }
  };

  const bool reporter = (rb == 0 && split == 0 && g == 0);
  const int T = __ldg(p.tree_len + b);
  const int L = __ldg(p.kv_len + b);
  if (T < 1 || T > p.T_max) {
    if (reporter && tid == 0) flag(p.status, DREAMS_DATA_BAD_TREE_LEN);
    leave();
    return;
  }
  const int total = key_total(p, L, T);
  if (L < 0 || total > p.capacity || total < 1) {
    if (reporter && tid == 0) flag(p.status, DREAMS_DATA_BAD_KV_LEN);
    leave();
    return;
  }
  const int nsplit_b = (total + p.chunk - 1) / p.chunk;
  // keys any row of the block may attend: a causal block stops after its last row's own slot
  const int kend = p.mode == ATTN_CAUSAL ? L + ::min(T, t0 + p.TB) : total;
  if (split >= nsplit_b || t0 >= T || c0 >= kend) {
    leave();
    return;
  }
  const int rows_blk = ::min(p.TB, T - t0) * p.G;  // real query rows of this CTA
  // softmax warps whose 32 rows hold at least one real query row
  const int n_act = ::min(4, (rows_blk + 31) / 32);

  if (tid == TMA_WARP * 32) {
    if (!early) init_copy_barriers();
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(bs0 + 8 * i, 1);
      tc::mbar_init(bp0 + 8 * i, 32 * n_act);
      tc::mbar_init(bph0 + 8 * i, 32 * n_act);
    }
    tc::mbar_init(bdrain, 1);
    tc::mbar_init(bnever, 1);  // nothing arrives on it (the stall test hook waits on it)
    s_abort = 0;
    s_flag = 0;
    tc::fence_barrier_init();
  }
  if (warp == MMA_WARP) {
    tc::tmem_alloc(smem_u32(&s_tmem), TMEM_COLS);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = s_tmem;

  const int c1 = ::min(c0 + p.chunk, kend);
  const int ntiles = (c1 - c0 + KT - 1) / KT;
  volatile int *abort_flag = &s_abort;
  const uint64_t wait_ns = p.wait_ns;
  // abort codes: 1 = a wait timed out, 2 = malformed tree (nothing to compute)
  auto give_up = [&]() {
    if (*abort_flag == 0) {
      *abort_flag = 1;
      flag(p.status, DREAMS_DATA_TIMEOUT);
    }
  };

  // While the producer streams Q, K and V and the MMA thread starts on them,
  // softmax warp 0 checks the tree and builds the ancestor masks; named
  // barrier 2 (the softmax warps) publishes them before the first tile. A
  // malformed tree stops the producer and the MMA thread through the abort
  // flag.
  const int wg = warp >> 2;                  // softmax warpgroup (warps 0-7)
  const int row = 32 * (warp & 3) + lane;    // TMEM lane = query row
  const bool real_row = row < rows_blk;
  const int t_row = t0 + row / p.G;
  if (warp == 0 && p.mode == ATTN_TREE) {
    int par[2], bad = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int i = lane + 32 * h;
      par[h] = (i < T) ? par_pre[h] : -1;
      if (i == 0) bad |= (par[h] != -1);
      else if (i < T) bad |= (par[h] < 0 || par[h] >= i);
    }
    bad = __any_sync(0xffffffffu, bad);
    if (lane == 0) s_flag = bad;
    if (bad) {
      if (lane == 0) {
        *abort_flag = 2;  // stops the producer; nothing is computed
        if (reporter) flag(p.status, DREAMS_DATA_BAD_PARENT);
      }
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
  if (warp < 8) named_sync(2, 256);
  // the producer and the MMA thread learn of a malformed tree from the abort flag
  const bool tree_ok = warp >= 8 || !s_flag;

  float m_ref = -INFINITY, l = 0.f;  // this thread's row state (softmax warps)
  float wsum = 0.f;                  // entropy: sum_j P_j (x_j - m_ref), x = scaled score in log2 units
  bool sm_ok = false;                // the softmax loop ran to completion

  if (warp == TMA_WARP) {
    // ---------------- TMA producer
    if (lane == 0) {
      if (!early) issue_q();  // (else already issued, with K_0)
      // raw page-table entries of the two 64-slot halves of tile j
      const int32_t *prow = P.paged ? p.page_table + int64_t(b) * p.pages_per_seq : nullptr;
      auto fetch = [&](int j, int &e0, int &e1) {
        if (P.paged && j < ntiles) {
          const int pi = (c0 + j * KT) >> 6;
          e0 = pi < p.pages_per_seq ? __ldg(prow + pi) : PAST_TABLE;
          e1 = pi + 1 < p.pages_per_seq ? __ldg(prow + pi + 1) : PAST_TABLE;
        }
      };
      // tensor-map coordinate (dim 3) of half h of tile j
      auto page_coord = [&](int j, int h, int e) {
        if (!P.paged) return b;
        if (e == PAST_TABLE) return p.num_pages;  // past the table: the copy fills zeros
        if (e < 0 || e >= p.num_pages) {
          if (c0 + j * KT + 64 * h < c1) flag(p.status, DREAMS_DATA_BAD_PAGE);
          return p.num_pages;  // outside the tensor map: the copy fills zeros
        }
        return e;
      };
      int ring[CRD][2];
      int pn0 = pn_pre[0], pn1 = pn_pre[1];  // tile 0 (loaded at the start)
      int nk = 0, nv = 0;  // tiles issued into each ring
      if (early) {  // K_0 went out at the start
        ring[0][0] = ring[0][1] = b;
        nk = 1;
      }
      uint32_t idle = 0;
      uint64_t t_idle = 0;
      while (nv < ntiles && !*abort_flag) {
        bool progress = false;
        if (nk < ntiles && nk - nv < CRD &&
            (nk < NK || tc::mbar_test_wait(ke0 + 8 * (nk % NK), ((nk / NK) - 1) & 1))) {
          if (p.stall_at >= 0 && nk >= p.stall_at) {
            // test hook: this copy is never issued; its consumers' waits run
            // out, like this one on a barrier that nothing arrives on
            tc::mbar_wait(bnever, 0, abort_flag, wait_ns);
            give_up();
            break;
          }
          const int c3a = page_coord(nk, 0, pn0), c3b = page_coord(nk, 1, pn1);
          ring[nk % CRD][0] = c3a;
          ring[nk % CRD][1] = c3b;
          fetch(nk + 1, pn0, pn1);
          const int ks = nk % NK, s0 = c0 + nk * KT;
          tc::mbar_arrive_expect_tx(kf0 + 8 * ks, KV_TILE);
#pragma unroll
          for (int r = 0; r < NR; ++r) {
            tc::tma_load_4d(k_s(ks) + r * KV_REGION, &P.tmap_k, kf0 + 8 * ks, r * 64, g, P.paged ? 0 : s0, c3a);
            tc::tma_load_4d(k_s(ks) + r * KV_REGION + 8192, &P.tmap_k, kf0 + 8 * ks, r * 64, g,
                            P.paged ? 0 : s0 + 64, c3b);
          }
          ++nk;
          progress = true;
        }
        // V_j once K_{j+1} is out (or K is done): QK^T needs K a tile before PV needs V
        if ((nv + 1 < nk || nk == ntiles) &&
            (nv < NV || tc::mbar_test_wait(ve0 + 8 * (nv % NV), ((nv / NV) - 1) & 1))) {
          const int vs = nv % NV, s0 = c0 + nv * KT;
          const int c3a = ring[nv % CRD][0], c3b = ring[nv % CRD][1];
          tc::mbar_arrive_expect_tx(vf0 + 8 * vs, KV_TILE);
#pragma unroll
          for (int r = 0; r < NR; ++r) {
            tc::tma_load_4d(v_s(vs) + r * KV_REGION, &P.tmap_v, vf0 + 8 * vs, r * 64, g, P.paged ? 0 : s0, c3a);
            tc::tma_load_4d(v_s(vs) + r * KV_REGION + 8192, &P.tmap_v, vf0 + 8 * vs, r * 64, g,
                            P.paged ? 0 : s0 + 64, c3b);
          }
          ++nv;
          progress = true;
        }
        if (progress) {
          idle = 0;
        } else if ((++idle & 255u) == 0) {
          const uint64_t now = tc::global_ns();
          if (idle == 256u) {
            t_idle = now;
          } else if (now - t_idle > wait_ns) {
            give_up();
            break;
          }
        }
      }
      // no copy may still be landing in shared memory when the CTA ends
      tc::mbar_wait(bq, 0, &s_zero);
      for (int j = ::max(0, nk - NK); j < nk; ++j) tc::mbar_wait(kf0 + 8 * (j % NK), (j / NK) & 1, &s_zero);
      for (int j = ::max(0, nv - NV); j < nv; ++j) tc::mbar_wait(vf0 + 8 * (j % NV), (j / NV) & 1, &s_zero);
    }
  } else if (warp == MMA_WARP) {
    // ---------------- MMA issuer
    if (lane == 0) {  // a malformed tree stops it through the abort flag
      // Base descriptors: an operand's descriptor is its base plus its byte
      // offset / 16 (the address field holds bits 4-17 of a shared-memory
      // address below 256 KB, so the addition never carries out of it); each
      // MMA then costs one add.
      const uint64_t qd0 = tc::smem_desc_sw128(q_s, 16, 1024);
      const uint64_t kd0 = tc::smem_desc_sw128(k_s(0), 16, 1024);
      const uint64_t vd0 = tc::smem_desc_sw128(v_s(0), KV_REGION, 1024);
      // The tensor pipe queues only about one MMA, so any latency in the
      // issuing thread between MMAs idles it: per tile the thread takes one
      // wait, then issues PV_j and QK_{j+2} (16 MMAs) under one commit (with
      // SPLIT, one wait before each half of PV_j).
      // S_j = Q K_j^T into warpgroup (j % 2)'s S buffer
      auto qk = [&](int j) {
        const int ks = j % NK;
        const uint32_t scol = 256u * (j & 1);
#pragma unroll
        for (int k = 0; k < D / 16; ++k) {
          const uint32_t off = (k & 3) << 5;  // 32 bytes per 16-element K step
          const uint64_t ad = qd0 + (((k >> 2) * Q_REGION + off) >> 4);
          const uint64_t bd = kd0 + ((uint32_t(ks) * KV_TILE + (k >> 2) * KV_REGION + off) >> 4);
          tc::mma_ss(tmem + scol, ad, bd, IDESC_QK, k > 0 ? 1u : 0u);
        }
      };
      // O_w += P_j V_j, w = j % 2, over the tile's first (h = 0) or last 64 keys
      auto pv = [&](int j, int h) {
        const int w = j & 1, ii = j >> 1, vs = j % NV;
        const uint32_t scol = 256u * w, ocol = 256u * w + 128u;
#pragma unroll
        for (int kk = 0; kk < KT / 32; ++kk) {
          const int ks = h * (KT / 32) + kk;
          const uint64_t bd = vd0 + ((uint32_t(vs) * KV_TILE + ks * 2048) >> 4);
          tc::mma_ts(tmem + ocol, tmem + scol + ks * 8, bd, IDESC_PV, (ii > 0 || ks > 0) ? 1u : 0u);
        }
      };
      auto kwait = [&](int j) { return tc::mbar_wait(kf0 + 8 * (j % NK), (j / NK) & 1, abort_flag, wait_ns); };
      bool ok = tc::mbar_wait(bq, 0, abort_flag, wait_ns) && kwait(0);
      if (ok) {
        tc::fence_after_sync();
        qk(0);
        tc::mma_commit(bs0);
      }
      if (ok && ntiles > 1) {
        ok = kwait(1);
        if (ok) {
          tc::fence_after_sync();
          qk(1);
          tc::mma_commit(bs0 + 8);
        }
      }
      // The commit after QK_{j+2} also covers PV_j (the pipe completes in
      // order): the softmax warps, woken by it, release the stages of K_{j+2}
      // and (without VREL) V_j to the producer.
      for (int j = 0; j < ntiles && ok; ++j) {
        const int w = j & 1;
        // P_j over the first 64 keys (the softmax warps arrive once one of
        // them has also seen V_j land): its PV half runs while they finish
        // the tile; then the rest of P_j (K_{j+2} landed as well). Without
        // SPLIT, P_j whole.
        if constexpr (SPLIT) {
          ok = tc::mbar_wait(bph0 + 8 * w, (j >> 1) & 1, abort_flag, wait_ns);
          if (!ok) break;
          tc::fence_after_sync();
          pv(j, 0);
        }
        ok = tc::mbar_wait(bp0 + 8 * w, (j >> 1) & 1, abort_flag, wait_ns);
        if (!ok) break;
        tc::fence_after_sync();
        if constexpr (!SPLIT) pv(j, 0);
        pv(j, 1);
        // with VREL, V_j's stage goes back to the producer as soon as PV_j
        // has completed, ahead of QK_{j+2} (an arrival on its empty barrier)
        if constexpr (VREL) tc::mma_commit(ve0 + 8 * (j % NV));
        if (j + 2 < ntiles) {
          qk(j + 2);
          tc::mma_commit(bs0 + 8 * w);
        }
      }
      if (!ok) give_up();
      tc::mma_commit(bdrain);
      tc::mbar_wait(bdrain, 0, &s_zero);
    }
  } else if ((warp & 3) < n_act && tree_ok) {
    // ---------------- softmax warpgroup wg: tiles wg, wg + 2, ...
    const uint32_t tl = tmem + (uint32_t(32 * (warp & 3)) << 16) + 256u * wg;
    const unsigned long long anc = (real_row && p.mode == ATTN_TREE) ? s_anc[t_row] : 0ull;
    // slots below lim are allowed besides the ancestors: the prefix, or for a
    // causal row the prefix and the rows up to its own
    const int lim = p.mode == ATTN_CAUSAL ? L + t_row + 1 : L;
    const int nw = (ntiles - wg + 1) / 2;
    bool ok = true;
    for (int ii = 0; ii < nw; ++ii) {
      const int j = 2 * ii + wg;
      if (!__all_sync(0xffffffffu, tc::mbar_wait(bs0 + 8 * wg, ii & 1, abort_flag, wait_ns))) {
        give_up();
        ok = false;
        break;
      }
      // S_j is complete, and so (issued earlier) is this warpgroup's previous
      // PV, so O may be rescaled below. The K stage of tile j and (unless the
      // MMA thread's commit already did, VREL) the V stage of tile j - 2, read
      // by that PV, go back to the producer.
      tc::fence_after_sync();
      if (warp == 4 * wg && lane == 0) {
        tc::mbar_arrive(ke0 + 8 * (j % NK));
        if (!VREL && j >= 2) tc::mbar_arrive(ve0 + 8 * ((j - 2) % NV));  // (with VREL: the MMA thread's commit)
      }
      uint32_t sv[KT];
#pragma unroll
      for (int q4 = 0; q4 < KT / 32; ++q4)
        tc::tmem_ld32(tl + 32 * q4, *reinterpret_cast<uint32_t(*)[32]>(&sv[32 * q4]));
      tc::tmem_wait_ld();
      const int s0 = c0 + j * KT;
      if ((s0 + KT > lim) || (s0 + KT > c1)) {
        // tree columns outside the row's ancestors, and columns past this
        // split: -inf. The allowed columns as four 32-bit words: prefix
        // slots (< L), the row's ancestors among the tree slots (bit a of
        // anc is slot L + a), nothing at or past c1. Kept compact: this runs
        // on one or two tiles of a CTA, so its code is rarely in the
        // instruction cache.
        uint32_t w[KT / 32];
#pragma unroll
        for (int q = 0; q < KT / 32; ++q) {
          const int cb = s0 + 32 * q;  // slot of bit 0 of this word
          const int np = lim - cb, ne = c1 - cb, sh = cb - L;
          const uint32_t pre = np >= 32 ? 0xffffffffu : (np <= 0 ? 0u : (1u << np) - 1u);
          const uint32_t end = ne >= 32 ? 0xffffffffu : (ne <= 0 ? 0u : (1u << ne) - 1u);
          const uint32_t tr = (sh >= 64 || sh <= -32) ? 0u
                              : (sh >= 0 ? uint32_t(anc >> sh) : uint32_t(anc << (-sh)));
          w[q] = (pre | tr) & end;
        }
#pragma unroll
        for (int c = 0; c < KT; ++c)
          if (!((w[c >> 5] >> (c & 31)) & 1u)) sv[c] = 0xff800000u;
      }
      // row maximum of the raw scores as a tree of three-input maxima (scale
      // > 0, so it commutes with the scaling)
      float mt[43];
#pragma unroll
      for (int i = 0; i < 42; ++i)
        mt[i] = max3f(__uint_as_float(sv[3 * i]), __uint_as_float(sv[3 * i + 1]), __uint_as_float(sv[3 * i + 2]));
      mt[42] = fmaxf(__uint_as_float(sv[126]), __uint_as_float(sv[127]));
#pragma unroll
      for (int i = 0; i < 14; ++i) mt[i] = max3f(mt[3 * i], mt[3 * i + 1], mt[3 * i + 2]);
      mt[14] = mt[42];  // 15 left
#pragma unroll
      for (int i = 0; i < 5; ++i) mt[i] = max3f(mt[3 * i], mt[3 * i + 1], mt[3 * i + 2]);
      const float mx = max3f(max3f(mt[0], mt[1], mt[2]), mt[3], mt[4]) * p.scale_log2;
      const bool resc = mx > m_ref + RESCALE;
      float corr = 1.f;
      if (resc) {
        const float m_old = m_ref;
        corr = (m_old == -INFINITY) ? 0.f : tc::ex2(m_old - mx);
        // the entropy sum sum_j P_j (x_j - m) follows the new reference
        if (ENT) wsum = (m_old == -INFINITY) ? 0.f : corr * (wsum - (mx - m_old) * l);
        m_ref = mx;
        l *= corr;
      }
      if constexpr (SPLIT) {
        // P in two halves of 64 keys: exponents scale * s - m two at a time
        // (f32x2 FMA), their sum two at a time (f32x2 add), P as bf16 pairs
        // over the first 64 columns of S, 32 keys per step
        const float nmu = (m_ref == -INFINITY) ? 0.f : -m_ref;
        const uint64_t scale2 = f32x2(p.scale_log2, p.scale_log2), nmu2 = f32x2(nmu, nmu);
        uint64_t acc2[2] = {f32x2(0.f, 0.f), f32x2(0.f, 0.f)};
        uint64_t wacc2 = f32x2(0.f, 0.f);  // entropy: sum of P e over the tile
        auto p_step = [&](int q4) {
          uint32_t pk[16];
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            float e0, e1;
            f32x2_split(ffma2(f32x2(__uint_as_float(sv[32 * q4 + 2 * c]), __uint_as_float(sv[32 * q4 + 2 * c + 1])),
                              scale2, nmu2),
                        e0, e1);
            const float p0 = tc::ex2(e0), p1 = tc::ex2(e1);
            acc2[c & 1] = fadd2(acc2[c & 1], f32x2(p0, p1));
            // masked slots have e = -inf and P = 0: clamp e so that P e is 0, not NaN
            if (ENT) wacc2 = ffma2(f32x2(p0, p1), f32x2(fmaxf(e0, -200.f), fmaxf(e1, -200.f)), wacc2);
            pk[c] = pack_bf16x2(p0, p1);
          }
          tc::tmem_st16(tl + 16 * q4, pk);
        };
        p_step(0);
        p_step(1);
        // Before the first half goes to the MMA thread (with half the scores
        // consumed, so that the registers allow it): slots past the sequence
        // end may hold any bits (0 * NaN = NaN in the PV product), so their V
        // rows are zeroed once the tile's copy has landed (a later landing
        // would undo the zeros); and O follows a raised reference before
        // PV_j's first half adds to it.
        if (c1 - s0 < KT) {
          const int st = j % NV;
          if (!__all_sync(0xffffffffu, tc::mbar_wait(vf0 + 8 * st, (j / NV) & 1, abort_flag, wait_ns))) {
            give_up();
            ok = false;
            break;
          }
          const int first = c1 - s0, nz = (KT - first) * NR * 8;
          for (int i = 32 * (warp & 3) + lane; i < nz; i += 32 * n_act) {
            const int r = first + i / (NR * 8), rc = i % (NR * 8);
            const uint32_t dst = v_s(st) + (rc >> 3) * KV_REGION + r * 128 + ((rc & 7) << 4);
            asm volatile("st.shared.v4.b32 [%0], {%1,%1,%1,%1};" ::"r"(dst), "r"(0u) : "memory");
          }
          tc::fence_proxy_async_smem();
        }
        if (ii > 0 && __any_sync(0xffffffffu, resc)) {
#pragma unroll
          for (int c4 = 0; c4 < D / 32; ++c4) {
            uint32_t ov[32];
            tc::tmem_ld32(tl + 128 + c4 * 32, ov);
            tc::tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * corr);
            tc::tmem_st32(tl + 128 + c4 * 32, ov);
          }
        }
        // One thread also waits for the copies the MMA thread needs next, V_j
        // for the first half of PV_j, then K_{j+2} for QK_{j+2} (usually
        // landed by now; the waits overlap the TMEM stores): the MMA thread
        // then waits for P alone.
        bool kv_ok = true;
        if (warp == 4 * wg && lane == 0)
          kv_ok = tc::mbar_wait(vf0 + 8 * (j % NV), (j / NV) & 1, abort_flag, wait_ns);
        if (!__all_sync(0xffffffffu, kv_ok)) {
          give_up();
          ok = false;
          break;
        }
        tc::tmem_wait_st();
        tc::fence_before_sync();
        tc::mbar_arrive(bph0 + 8 * wg);
        p_step(2);
        p_step(3);
        {
          float a0, a1, b0, b1;
          f32x2_split(acc2[0], a0, a1);
          f32x2_split(acc2[1], b0, b1);
          l += (a0 + a1) + (b0 + b1);
          if (ENT) {
            f32x2_split(wacc2, a0, a1);
            wsum += a0 + a1;
          }
        }
        if (warp == 4 * wg && lane == 0)
          kv_ok = j + 2 >= ntiles ||
                  tc::mbar_wait(kf0 + 8 * ((j + 2) % NK), ((j + 2) / NK) & 1, abort_flag, wait_ns);
        if (!__all_sync(0xffffffffu, kv_ok)) {
          give_up();
          ok = false;
          break;
        }
      } else {
        const float nmu = (m_ref == -INFINITY) ? 0.f : -m_ref;
        // exponents scale * s - m two at a time (f32x2 FMA), their sum two at a
        // time (f32x2 add), P as bf16 pairs
        const uint64_t scale2 = f32x2(p.scale_log2, p.scale_log2), nmu2 = f32x2(nmu, nmu);
        uint64_t acc2[2] = {f32x2(0.f, 0.f), f32x2(0.f, 0.f)};
        uint64_t wacc2 = f32x2(0.f, 0.f);  // entropy: sum of P e over the tile
#pragma unroll
        for (int q4 = 0; q4 < KT / 32; ++q4) {
          uint32_t pk[16];
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            float e0, e1;
            f32x2_split(ffma2(f32x2(__uint_as_float(sv[32 * q4 + 2 * c]), __uint_as_float(sv[32 * q4 + 2 * c + 1])),
                              scale2, nmu2),
                        e0, e1);
            const float p0 = tc::ex2(e0), p1 = tc::ex2(e1);
            acc2[c & 1] = fadd2(acc2[c & 1], f32x2(p0, p1));
            // masked slots have e = -inf and P = 0: clamp e so that P e is 0, not NaN
            if (ENT) wacc2 = ffma2(f32x2(p0, p1), f32x2(fmaxf(e0, -200.f), fmaxf(e1, -200.f)), wacc2);
            pk[c] = pack_bf16x2(p0, p1);
          }
          tc::tmem_st16(tl + 16 * q4, pk);  // P (bf16 pairs) over the first 64 columns of S
        }
        {
          float a0, a1, b0, b1;
          f32x2_split(acc2[0], a0, a1);
          f32x2_split(acc2[1], b0, b1);
          l += (a0 + a1) + (b0 + b1);
          if (ENT) {
            f32x2_split(wacc2, a0, a1);
            wsum += a0 + a1;
          }
        }
        if (c1 - s0 < KT) {
          // slots past the sequence end may hold any bits (0 * NaN = NaN in the
          // PV product): zero those V rows before the MMA reads them, once the
          // tile's copy has landed (a later landing would undo the zeros)
          const int st = j % NV;
          if (!__all_sync(0xffffffffu, tc::mbar_wait(vf0 + 8 * st, (j / NV) & 1, abort_flag, wait_ns))) {
            give_up();
            ok = false;
            break;
          }
          const int first = c1 - s0, nz = (KT - first) * NR * 8;
          for (int i = 32 * (warp & 3) + lane; i < nz; i += 32 * n_act) {
            const int r = first + i / (NR * 8), rc = i % (NR * 8);
            const uint32_t dst = v_s(st) + (rc >> 3) * KV_REGION + r * 128 + ((rc & 7) << 4);
            asm volatile("st.shared.v4.b32 [%0], {%1,%1,%1,%1};" ::"r"(dst), "r"(0u) : "memory");
          }
          tc::fence_proxy_async_smem();
        }
        if (ii > 0 && __any_sync(0xffffffffu, resc)) {
#pragma unroll
          for (int c4 = 0; c4 < D / 32; ++c4) {
            uint32_t ov[32];
            tc::tmem_ld32(tl + 128 + c4 * 32, ov);
            tc::tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * corr);
            tc::tmem_st32(tl + 128 + c4 * 32, ov);
          }
        }
        // One thread also waits for the copies the MMA thread needs next, V_j
        // and K_{j+2} (usually landed by now; the wait overlaps the TMEM
        // stores): the MMA thread then waits for P_j alone.
        bool kv_ok = true;
        if (warp == 4 * wg && lane == 0)
          kv_ok = tc::mbar_wait(vf0 + 8 * (j % NV), (j / NV) & 1, abort_flag, wait_ns) &&
                  (j + 2 >= ntiles ||
                   tc::mbar_wait(kf0 + 8 * ((j + 2) % NK), ((j + 2) / NK) & 1, abort_flag, wait_ns));
        if (!__all_sync(0xffffffffu, kv_ok)) {
          give_up();
          ok = false;
          break;
        }
      }
      tc::tmem_wait_st();
      tc::fence_before_sync();
      tc::mbar_arrive(bp0 + 8 * wg);
    }
    // all MMAs done (the issuer commits this single-use barrier after its last PV)
    if (ok && nw > 0 && !__all_sync(0xffffffffu, tc::mbar_wait(bdrain, 0, abort_flag, wait_ns))) {
      give_up();
      ok = false;
    }
    sm_ok = ok;
  }

  // ---- epilogue: the two warpgroups combine their (m, l, O) by log-sum-exp
  // ((m, l) pass through the last V stage, idle once every MMA has completed);
  // each thread then writes its row's half of the columns straight to global
  // memory in 16-byte stores: the output, or the split partials.
  if (warp < 8) {
    const bool act = (warp & 3) < n_act && tree_ok;
    // the output directly, unless the block's keys span several splits
    const bool direct = (kend + p.chunk - 1) / p.chunk == 1;
    float2 *s_ml = reinterpret_cast<float2 *>(smem + Q_BYTES + (NK + NV - 1) * KV_TILE);
    float *s_w = reinterpret_cast<float *>(s_ml + 2 * ROWS);  // entropy sums of both warpgroups
    if (act && sm_ok) {
      s_ml[wg * ROWS + row] = make_float2(m_ref, l);
      if (ENT) s_w[wg * ROWS + row] = wsum;
    }
    // A block whose every row inside the tensor is a real query row leaves
    // through one TMA store per 64-column region (the box of the Q map, over
    // the output): the rows are staged in shared memory in the box's 128-byte
    // swizzled layout (the first K stage, idle once every MMA has completed).
    // Other blocks store row by row (rows past tree_len / q_len stay untouched).
    if (tid == 0) s_tma = direct && ::min(t0 + p.TB, p.T_max) <= T && !*abort_flag;
    tc::fence_before_sync();
    named_sync(1, 256);
    tc::fence_after_sync();
    const bool tma_out = s_tma != 0;
    const int64_t slot = (((int64_t(b) * p.Hkv + g) * p.nrb + rb) * p.nsplit + split) * ROWS;
    if (act && !*abort_flag) {
      const float2 a = s_ml[row], c = s_ml[ROWS + row];
      const float M = fmaxf(a.x, c.x);
      const float ca = (a.y > 0.f) ? tc::ex2(a.x - M) : 0.f;
      const float cb = (c.y > 0.f) ? tc::ex2(c.x - M) : 0.f;
      const float Ls = ca * a.y + cb * c.y;
      const uint32_t lanes = tmem + (uint32_t(32 * (warp & 3)) << 16);
      const float inv = direct ? 1.f / Ls : 1.f;
      const int64_t orow = (int64_t(b) * p.T_max + t_row) * p.Hq + g * p.G + (row - (t_row - t0) * p.G);
#pragma unroll 1
      for (int c4 = 0; c4 < D / 64; ++c4) {
        const int col = wg * (D / 2) + c4 * 32;
        uint32_t oa[32], ob[32];
        tc::tmem_ld32(lanes + 128 + col, oa);
        tc::tmem_ld32(lanes + 256 + 128 + col, ob);
        tc::tmem_wait_ld();
        float o[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const float va = ca != 0.f ? ca * __uint_as_float(oa[e]) : 0.f;
          const float vb = cb != 0.f ? cb * __uint_as_float(ob[e]) : 0.f;
          o[e] = (va + vb) * inv;
        }
        if (tma_out) {
          // region col / 64, 16-byte chunk (col % 64) / 8 + e of row `row`
          const uint32_t rbase = k_s(0) + uint32_t((col >> 6) * Q_REGION + row * 128);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int c = ((col & 63) >> 3) + e;
            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(rbase + uint32_t((c ^ (row & 7)) << 4)),
                         "r"(pack_bf16x2(o[8 * e], o[8 * e + 1])), "r"(pack_bf16x2(o[8 * e + 2], o[8 * e + 3])),
                         "r"(pack_bf16x2(o[8 * e + 4], o[8 * e + 5])), "r"(pack_bf16x2(o[8 * e + 6], o[8 * e + 7]))
                         : "memory");
          }
          continue;
        }
        if (!real_row) continue;
        if (direct) {
          uint4 *dst = reinterpret_cast<uint4 *>(p.out + orow * D + col);
#pragma unroll
          for (int e = 0; e < 4; ++e)
            dst[e] = make_uint4(pack_bf16x2(o[8 * e + 0], o[8 * e + 1]), pack_bf16x2(o[8 * e + 2], o[8 * e + 3]),
                                pack_bf16x2(o[8 * e + 4], o[8 * e + 5]), pack_bf16x2(o[8 * e + 6], o[8 * e + 7]));
        } else {
          float4 *dst = reinterpret_cast<float4 *>(p.ws_o + (slot + row) * D + col);
#pragma unroll
          for (int e = 0; e < 8; ++e) dst[e] = make_float4(o[4 * e], o[4 * e + 1], o[4 * e + 2], o[4 * e + 3]);
        }
      }
      if (wg == 0 && real_row) {
        // entropy of the row: with P_j = 2^(x_j - M) and Z = sum_j P_j,
        // H = ln Z - ln 2 * sum_j P_j (x_j - M) / Z; each warpgroup's sum moves
        // from its own reference m to M as c * (W + (m - M) l)
        float Wt = 0.f;
        if (ENT) {
          if (ca != 0.f) Wt += ca * (s_w[row] + (a.x - M) * a.y);
          if (cb != 0.f) Wt += cb * (s_w[ROWS + row] + (c.x - M) * c.y);
        }
        if (direct) {
          if (p.lse != nullptr) p.lse[orow] = (M + log2f(Ls)) * LN2;
          if (ENT && p.ent != nullptr) p.ent[orow] = logf(Ls) - LN2 * Wt / Ls;
        } else {
          p.ws_ml[slot + row] = make_float2(Ls > 0.f ? M : -INFINITY, Ls);
          if (ENT) p.ws_w[slot + row] = Ls > 0.f ? Wt : 0.f;
        }
      }
    } else if (act && *abort_flag == 1 && !direct && wg == 0 && real_row) {
      // a wait gave up: the negative sum tells the merge to leave the row alone
      p.ws_ml[slot + row] = make_float2(-INFINITY, -1.f);
    }
    if (tma_out) {
      tc::fence_proxy_async_smem();  // the staged rows, to the TMA engine
      named_sync(1, 256);
      if (tid == 0) {
#pragma unroll
        for (int r = 0; r < NR; ++r) tc::tma_store_5d(&P.tmap_o, k_s(0) + r * Q_REGION, r * 64, 0, g, t0, b);
        tc::bulk_commit_group();
        tc::bulk_wait_group_read0();  // shared memory stays until the copy engine has read it
      }
    }
  }

  // ---- teardown: every copy and MMA has completed (or timed out) by now
  tc::fence_before_sync();
  __syncthreads();
  if (warp == MMA_WARP) {
    __syncwarp();
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, TMEM_COLS);
  }
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Log-sum-exp merge of the split partials: one warp per query row of a
// (b, g, row block); rows of sequences that needed a single split were
// written by the attention kernel and are skipped. The partial O rows of all
// splits are loaded together with their (m, l) (a split that saw no allowed
// key wrote zeros), so a row costs about one memory latency. Launched as a
// programmatic dependent of the attention kernel: griddepcontrol.wait returns
// once that grid has completed and its writes are visible.
template <int D, bool ENT>
__global__ void __launch_bounds__(256) tree_attn_merge_kernel(const AttnParams p) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  constexpr int NL = D / 4;  // lanes holding 4 columns each
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t row = int64_t(blockIdx.x) * 8 + warp;
  const int64_t item = row / ROWS;
  const int r = int(row - item * ROWS);
  const int rb = int(item % p.nrb);
  const int64_t bg = item / p.nrb;
  const int g = int(bg % p.Hkv);
  const int b = int(bg / p.Hkv);
  if (b >= p.B) return;
  const int T = __ldg(p.tree_len + b);
  const int L = __ldg(p.kv_len + b);
  const int total = key_total(p, L, T);
  if (T < 1 || T > p.T_max || L < 0 || total > p.capacity || total < 1) return;
  const int t0 = rb * p.TB;
  if (t0 >= T || r >= ::min(p.TB, T - t0) * p.G) return;
  // splits of the row block (it was written directly when there is one) and
  // of this row (a causal row's keys end at its own slot)
  const int kend = p.mode == ATTN_CAUSAL ? L + ::min(T, t0 + p.TB) : total;
  const int nsplit_blk = (kend + p.chunk - 1) / p.chunk;
  if (nsplit_blk == 1) return;
  const int tn = r / p.G;
  const int nsplit_b = p.mode == ATTN_CAUSAL ? (L + t0 + tn + 1 + p.chunk - 1) / p.chunk : nsplit_blk;

  const int64_t sbase = item * p.nsplit * ROWS + r;
  float4 x[8];
#pragma unroll
  for (int k = 0; k < 8; ++k)
    x[k] = (k < nsplit_b && lane < NL)
               ? __ldcg(reinterpret_cast<const float4 *>(p.ws_o + (sbase + int64_t(k) * ROWS) * D) + lane)
               : make_float4(0.f, 0.f, 0.f, 0.f);
  const float2 ml = lane < nsplit_b ? __ldcg(p.ws_ml + sbase + int64_t(lane) * ROWS) : make_float2(-INFINITY, 0.f);
  const float wl = (ENT && lane < nsplit_b) ? __ldcg(p.ws_w + sbase + int64_t(lane) * ROWS) : 0.f;
  int bad = 0;  // the attention kernel skipped malformed trees; so does the merge
  if (p.mode == ATTN_TREE) {
    for (int i = lane; i < T; i += 32) {
      const int par = __ldg(p.parent + int64_t(b) * p.T_max + i);
      bad |= (i == 0) ? (par != -1) : (par < 0 || par >= i);
    }
  }
  // a split that gave up waiting left a negative sum: the row stays untouched
  bad |= ml.y < 0.f;
  if (__any_sync(0xffffffffu, bad)) return;

  float M = ml.y > 0.f ? ml.x : -INFINITY;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
  const float w = ml.y > 0.f ? tc::ex2(ml.x - M) : 0.f;
  float Ls = w * ml.y;
  float Wt = (ENT && ml.y > 0.f) ? w * (wl + (ml.x - M) * ml.y) : 0.f;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    Ls += __shfl_xor_sync(0xffffffffu, Ls, off);
    if (ENT) Wt += __shfl_xor_sync(0xffffffffu, Wt, off);
  }
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const float wk = __shfl_sync(0xffffffffu, w, k);
    acc.x += wk * x[k].x;
    acc.y += wk * x[k].y;
    acc.z += wk * x[k].z;
    acc.w += wk * x[k].w;
  }
  for (int k = 8; k < nsplit_b; ++k) {
    const float wk = __shfl_sync(0xffffffffu, w, k);
    if (lane < NL) {
      const float4 y = __ldcg(reinterpret_cast<const float4 *>(p.ws_o + (sbase + int64_t(k) * ROWS) * D) + lane);
      acc.x += wk * y.x;
      acc.y += wk * y.y;
      acc.z += wk * y.z;
      acc.w += wk * y.w;
    }
  }
  if (lane >= NL) return;
  const float inv = 1.f / Ls;
  const int64_t orow = (int64_t(b) * p.T_max + t0 + tn) * p.Hq + g * p.G + (r - tn * p.G);
  uint2 pk;
  pk.x = pack_bf16x2(acc.x * inv, acc.y * inv);
  pk.y = pack_bf16x2(acc.z * inv, acc.w * inv);
  *reinterpret_cast<uint2 *>(p.out + orow * D + lane * 4) = pk;
  if (lane == 0) {
    if (p.lse != nullptr) p.lse[orow] = (M + log2f(Ls)) * LN2;
    if (ENT && p.ent != nullptr) p.ent[orow] = logf(Ls) - LN2 * Wt / Ls;
  }
}

// ------------------------------------------------------------------ host side
struct AttnPlan {
  int TB;
  int nrb;
  int nsplit;
  int chunk;
  bool ordered;  // a separate kernel orders the pairs
  bool ranked;   // each CTA ranks the pairs itself
  size_t ws_o_bytes, ws_ml_bytes, ws_w_bytes, order_bytes;
  size_t ws_bytes;
};

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// KV splits: one CTA per SM, so pick the split count whose grid, in whole
// waves of num_sms CTAs, gives the shortest estimated time (a wave costs its
// chunk plus a fixed start-up and write-out of about four tiles: the first
// tiles of all SMs arrive together; a merge pass about two more); splits of
// >= 256 tokens, at most MAX_SPLITS.
AttnPlan plan(const dreams_kv_cache_t *kv, int B, int T_max, int Hq, bool ent) {
  AttnPlan pl{};
  const int G = Hq / kv->Hkv;
  pl.TB = std::max(1, ROWS / G);
  pl.nrb = (T_max + pl.TB - 1) / pl.TB;
  const int64_t base = int64_t(B) * kv->Hkv * pl.nrb;
  const int64_t sms = num_sms();
  const int64_t max_ns = std::max<int64_t>(1, (kv->capacity + 255) / 256);
  int64_t best_ns = 1;
  double best_cost = 1e300;
  for (int64_t ns = 1; ns <= std::min<int64_t>(max_ns, MAX_SPLITS); ++ns) {
    int64_t chunk = (kv->capacity + ns - 1) / ns;
    chunk = (chunk + KT - 1) / KT * KT;
    const int64_t n = (kv->capacity + chunk - 1) / chunk;
    const int64_t waves = (base * n + sms - 1) / sms;
    const double cost = double(waves) * double(chunk + 4 * KT) + (n > 1 ? 2.0 * KT : 0.0);
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best_ns = ns;
    }
  }
  int64_t chunk = (kv->capacity + best_ns - 1) / best_ns;
  chunk = (chunk + KT - 1) / KT * KT;
  pl.chunk = int(chunk);
  pl.nsplit = int((kv->capacity + chunk - 1) / chunk);
  if (pl.nsplit > 1) {
    const size_t slots = size_t(base) * pl.nsplit * ROWS;
    pl.ws_o_bytes = align_up(slots * kv->D * sizeof(float), 256);
    pl.ws_ml_bytes = align_up(slots * sizeof(float2), 256);
    if (ent) pl.ws_w_bytes = align_up(slots * sizeof(float), 256);
  }
  pl.ranked = B > 1 && int64_t(B) * pl.nsplit <= RANK_PAIRS;
  pl.ordered = B > 1 && !pl.ranked;
  if (pl.ordered) pl.order_bytes = align_up(size_t(B) * pl.nsplit * sizeof(int32_t), 256);
  pl.ws_bytes = pl.ws_o_bytes + pl.ws_ml_bytes + pl.ws_w_bytes + pl.order_bytes;
  return pl;
}

bool valid_shapes(const dreams_kv_cache_t *kv, int B, int T_max, int Hq, int mode) {
  const int tmax_limit = mode == ATTN_TREE ? 64 : (1 << 20);
  return kv != nullptr && B >= 1 && B <= 65535 && T_max >= 1 && T_max <= tmax_limit && kv->Hkv >= 1 &&
         kv->Hkv <= 65535 && Hq >= kv->Hkv && Hq % kv->Hkv == 0 && Hq / kv->Hkv <= ROWS && kv->capacity >= 1 &&
         kv->n_layers >= 1;
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

// 5-D view of the queries, (D, G, Hkv, T_max, B), with a (64 columns, G
// heads, 1 KV head, TB nodes, 1) box: the query rows of one row block in
// (node, head) order, 128-byte swizzle. A token's Hq head rows are dense;
// tokens and sequences are q_stride_t and q_stride_b elements apart.
bool make_q_map(CUtensorMap *m, const void *q, int B, int T_max, int Hq, int Hkv, int D, int TB, int64_t q_stride_b,
                int64_t q_stride_t) {
  EncodeTiledFn enc = encode_tiled();
  if (enc == nullptr) return false;
  const int G = Hq / Hkv;
  const cuuint64_t dims[5] = {cuuint64_t(D), cuuint64_t(G), cuuint64_t(Hkv), cuuint64_t(T_max), cuuint64_t(B)};
  const cuuint64_t strides[4] = {cuuint64_t(D) * 2, cuuint64_t(G) * D * 2, cuuint64_t(q_stride_t) * 2,
                                 cuuint64_t(q_stride_b) * 2};
  const cuuint32_t box[5] = {64, cuuint32_t(G), 1, cuuint32_t(TB), 1};
  const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void *>(q), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Dynamic shared memory; at least 120 KB so that one CTA runs per SM (the
// CTA takes all 512 TMEM columns).
template <int D>
constexpr size_t smem_bytes() {
  return std::max<size_t>(size_t(D / 64) * ROWS * 128 + size_t(NK + NV) * (D / 64) * KT * 128 + 1024, 120 * 1024);
}

cudaError_t launch_pdl(const void *func, dim3 grid, dim3 block, size_t smem, cudaStream_t stream, bool pdl,
                       void **args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelExC(&cfg, func, args);
}

template <int D, bool ENT>
dreams_status_t launch(const AttnParams &a, const AttnPlan &pl, const dreams_kv_cache_t *kv, const void *k,
                       const void *v, int B, int64_t q_stride_b, int64_t q_stride_t, cudaStream_t stream) {
  constexpr size_t smem = smem_bytes<D>();
  const void *kernel =
      a.mode == ATTN_CAUSAL
          ? reinterpret_cast<const void *>(tree_attn_tc_kernel<D, ENT, false, false>)
          : (kv->page_table != nullptr ? reinterpret_cast<const void *>(tree_attn_tc_kernel<D, ENT, true, true>)
                                       : reinterpret_cast<const void *>(tree_attn_tc_kernel<D, ENT, true, false>));
  {
    const dreams_status_t st = ensure_max_dynamic_smem(kernel, int(smem));
    if (st != DREAMS_OK) return st;
  }
  TcParams P;
  memset(&P, 0, sizeof(P));
  P.a = a;
  P.paged = kv->page_table != nullptr;
  if (!make_kv_map(&P.tmap_k, k, kv, B) || !make_kv_map(&P.tmap_v, v, kv, B) ||
      !make_q_map(&P.tmap_q, a.q, B, a.T_max, a.Hq, a.Hkv, D, a.TB, q_stride_b, q_stride_t) ||
      !make_q_map(&P.tmap_o, a.out, B, a.T_max, a.Hq, a.Hkv, D, a.TB, int64_t(a.T_max) * a.Hq * D,
                  int64_t(a.Hq) * D))
    return DREAMS_ERR_UNSUPPORTED;
  if (pl.ordered) {
    tree_attn_order_kernel<<<1, ORDER_THREADS, 0, stream>>>(a);
    dreams_status_t st = check_launch();
    if (st != DREAMS_OK) return st;
  }
  const int64_t ctas = int64_t(B) * pl.nsplit * a.Hkv * pl.nrb;
  void *args_attn[] = {&P};
  cudaError_t e = launch_pdl(kernel, dim3(unsigned(ctas)), dim3(THREADS), smem, stream, pl.ordered, args_attn);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  dreams_status_t st = check_launch();
  if (st != DREAMS_OK || pl.nsplit == 1) return st;
  const int64_t rows = int64_t(B) * a.Hkv * pl.nrb * ROWS;
  AttnParams am = a;
  void *args_merge[] = {&am};
  e = launch_pdl(reinterpret_cast<const void *>(tree_attn_merge_kernel<D, ENT>), dim3(unsigned((rows + 7) / 8)),
                 dim3(256), 0, stream, true, args_merge);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  return check_launch();
}

}  // namespace
}  // namespace dreams

using namespace dreams;

namespace {

// The shared body of the two attention entry points.
dreams_status_t attention_impl(const void *q, int64_t q_stride_b, int64_t q_stride_t, const dreams_kv_cache_t *kv,
                               int32_t layer, const int32_t *parent,
                               const int32_t *q_len, const int32_t *kv_len, int32_t B, int32_t T_max, int32_t Hq,
                               float scale, int32_t mode, void *out, float *lse, float *ent, void *workspace,
                               size_t workspace_bytes, int32_t *status_word, dreams_stream_t stream) {
  if (q == nullptr || out == nullptr || kv == nullptr || q_len == nullptr || kv_len == nullptr)
    return DREAMS_ERR_INVALID_ARG;
  if (kv->k == nullptr || kv->v == nullptr || (mode == ATTN_TREE && parent == nullptr)) return DREAMS_ERR_INVALID_ARG;
  if (!valid_shapes(kv, B, T_max, Hq, mode)) return DREAMS_ERR_INVALID_ARG;
  if (kv->D != 64 && kv->D != 128) return DREAMS_ERR_UNSUPPORTED;
  if (layer < 0 || layer >= kv->n_layers || kv->layer_stride < 0) return DREAMS_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out) || !aligned16(kv->k) || !aligned16(kv->v) ||
      (kv->layer_stride * 2) % 16 != 0 || (lse != nullptr && (reinterpret_cast<uintptr_t>(lse) & 3)) ||
      (ent != nullptr && (reinterpret_cast<uintptr_t>(ent) & 3)))
    return DREAMS_ERR_INVALID_ARG;
  if (!isfinite(scale) || !(scale > 0.f)) return DREAMS_ERR_INVALID_ARG;
  // Q rows: a token's head rows are dense, tokens and sequences are strided
  // (16-byte multiples, as the tensor-map copy requires); with one sequence
  // the sequence stride is not used
  if (B == 1) q_stride_b = int64_t(T_max) * q_stride_t;
  if (q_stride_t < int64_t(Hq) * kv->D || q_stride_b < int64_t(Hq) * kv->D || q_stride_t % 8 != 0 ||
      q_stride_b % 8 != 0 || q_stride_t >= (int64_t(1) << 38) || q_stride_b >= (int64_t(1) << 38))
    return DREAMS_ERR_INVALID_ARG;
  if (kv->page_table != nullptr) {
    if (kv->page_size != 64) return DREAMS_ERR_UNSUPPORTED;
    if (kv->pages_per_seq < 1 || kv->num_pages < 1 || int64_t(kv->pages_per_seq) * 64 != kv->capacity)
      return DREAMS_ERR_INVALID_ARG;
  }
  const bool want_ent = ent != nullptr;
  const AttnPlan pl = plan(kv, B, T_max, Hq, want_ent);
  if (pl.ws_bytes > 0 && (workspace == nullptr || workspace_bytes < pl.ws_bytes || !aligned16(workspace)))
    return DREAMS_ERR_WORKSPACE;
  if (int64_t(B) * pl.nsplit * kv->Hkv * pl.nrb > 0x7fffffff ||
      int64_t(B) * kv->Hkv * pl.nrb * ROWS / 8 > 0x7fffffff)
    return DREAMS_ERR_UNSUPPORTED;

  AttnParams p{};
  p.q = static_cast<const __nv_bfloat16 *>(q);
  p.out = static_cast<__nv_bfloat16 *>(out);
  p.lse = lse;
  p.page_table = kv->page_table;
  p.pages_per_seq = kv->pages_per_seq;
  p.num_pages = kv->num_pages;
  p.capacity = kv->capacity;
  p.parent = parent;
  p.tree_len = q_len;
  p.kv_len = kv_len;
  p.B = B;
  p.T_max = T_max;
  p.Hq = Hq;
  p.Hkv = kv->Hkv;
  p.G = Hq / kv->Hkv;
  p.TB = pl.TB;
  p.nrb = pl.nrb;
  p.nsplit = pl.nsplit;
  p.chunk = pl.chunk;
  p.scale_log2 = scale * LOG2E;
  p.mode = mode;
  p.ent = ent;
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  if (pl.nsplit > 1) {
    p.ws_o = reinterpret_cast<float *>(ws);
    p.ws_ml = reinterpret_cast<float2 *>(ws + pl.ws_o_bytes);
    if (want_ent) p.ws_w = reinterpret_cast<float *>(ws + pl.ws_o_bytes + pl.ws_ml_bytes);
  }
  if (pl.ordered) p.order = reinterpret_cast<int32_t *>(ws + pl.ws_o_bytes + pl.ws_ml_bytes + pl.ws_w_bytes);
  p.rank = pl.ranked ? 1 : 0;
  p.status = status_word;
  test_stall(DREAMS_TEST_ATTENTION, &p.stall_at, &p.wait_ns);
  const void *k = static_cast<const __nv_bfloat16 *>(kv->k) + int64_t(layer) * kv->layer_stride;
  const void *v = static_cast<const __nv_bfloat16 *>(kv->v) + int64_t(layer) * kv->layer_stride;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int64_t sb = q_stride_b, st = q_stride_t;
  if (want_ent)
    return kv->D == 128 ? launch<128, true>(p, pl, kv, k, v, B, sb, st, s) : launch<64, true>(p, pl, kv, k, v, B, sb, st, s);
  return kv->D == 128 ? launch<128, false>(p, pl, kv, k, v, B, sb, st, s)
                      : launch<64, false>(p, pl, kv, k, v, B, sb, st, s);
}

}  // namespace

extern "C" size_t dreams_tree_verify_attn_workspace_size(const dreams_kv_cache_t *kv,
                                                         const dreams_tree_t *tree, int32_t Hq) {
  if (tree == nullptr || !valid_shapes(kv, tree->B, tree->T_max, Hq, ATTN_TREE)) return 0;
  return plan(kv, tree->B, tree->T_max, Hq, false).ws_bytes;
}

extern "C" int32_t dreams_tree_verify_attn_launches(const dreams_kv_cache_t *kv, const dreams_tree_t *tree,
                                                    int32_t Hq) {
  if (tree == nullptr || !valid_shapes(kv, tree->B, tree->T_max, Hq, ATTN_TREE) || (kv->D != 64 && kv->D != 128))
    return 0;
  const AttnPlan pl = plan(kv, tree->B, tree->T_max, Hq, false);
  return 1 + (pl.ordered ? 1 : 0) + (pl.nsplit > 1 ? 1 : 0);
}

extern "C" dreams_status_t dreams_tree_verify_attn(const void *q, int64_t q_stride_b, int64_t q_stride_t,
                                                   const dreams_kv_cache_t *kv, int32_t layer,
                                                   const dreams_tree_t *tree, int32_t Hq, float scale,
                                                   void *out, float *lse, void *workspace,
                                                   size_t workspace_bytes, int32_t *status_word,
                                                   dreams_stream_t stream) {
  if (tree == nullptr) return DREAMS_ERR_INVALID_ARG;
  return attention_impl(q, q_stride_b, q_stride_t, kv, layer, tree->parent, tree->tree_len, tree->kv_len, tree->B, tree->T_max, Hq, scale,
                        ATTN_TREE, out, lse, nullptr, workspace, workspace_bytes, status_word, stream);
}

extern "C" size_t dreams_attention_workspace_size(const dreams_kv_cache_t *kv, int32_t B, int32_t T_max, int32_t Hq,
                                                  int32_t mode, int32_t want_entropy) {
  if ((mode != DREAMS_ATTN_FULL && mode != DREAMS_ATTN_CAUSAL) || !valid_shapes(kv, B, T_max, Hq, mode)) return 0;
  return plan(kv, B, T_max, Hq, want_entropy != 0).ws_bytes;
}

extern "C" dreams_status_t dreams_attention(const void *q, int64_t q_stride_b, int64_t q_stride_t,
                                            const dreams_kv_cache_t *kv, int32_t layer,
                                            const int32_t *q_len, const int32_t *kv_len, int32_t B, int32_t T_max,
                                            int32_t Hq, float scale, int32_t mode, void *out, float *lse,
                                            float *entropy, void *workspace, size_t workspace_bytes,
                                            int32_t *status_word, dreams_stream_t stream) {
  if (mode != DREAMS_ATTN_FULL && mode != DREAMS_ATTN_CAUSAL) return DREAMS_ERR_INVALID_ARG;
  return attention_impl(q, q_stride_b, q_stride_t, kv, layer, nullptr, q_len, kv_len, B, T_max, Hq, scale, mode, out, lse, entropy,
                        workspace, workspace_bytes, status_word, stream);
}
