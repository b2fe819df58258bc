// lmhead.cu -- the target's greedy prediction per node straight from its final
// hidden states: logits = H W^T (the LM head), reduced to their argmax inside
// the GEMM's epilogue, so the logits never reach HBM (paper Sec. 2
// "Speculative decoding" at temperature 0; the logits are the target's
// per-node distribution that the acceptance reads).
//
// tcgen05 GEMM, persistent, one CTA per SM, 192 threads:
//   warp 0, one thread  TMA producer: per k-block a 128 x 64 tile of H and a
//                       256 x 64 tile of W (128-byte swizzle) into a 4-stage ring
//   warp 1, one thread  MMA issuer (M128 N256 K16, bf16 -> f32) into one of two
//                       TMEM accumulators of 256 columns; allocates TMEM
//   warps 2-5           epilogue: each thread owns one row of the 128 x 256
//                       accumulator, reads it from TMEM 32 columns at a time,
//                       keeps the row's best (value, first index) and merges
//                       it into the row's 64-bit slot with atomicMax; the
//                       accumulator is released right after the loads, so the
//                       next tile's MMAs overlap the reduction
// Tiles (m, n) are visited n-major (tile t: m = t % nm, n = t / nm), so the
// CTAs working at one time share weight tiles through L2. A second kernel,
// chained by programmatic dependent launch, turns each slot into the index
// (and the maximum value) and resets it. Every wait is bounded (2 s); on a
// timeout the CTA flags DREAMS_DATA_TIMEOUT in the status word, merges no
// further tile, waits for the copies and MMAs it issued, frees its TMEM and
// exits.
#include <cuda.h>
#include <limits.h>
#include <string.h>

#include <algorithm>

#include "common.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace dreams {
namespace {

constexpr int BM = 128, BN = 256, BK = 64;  // BK: one 128-byte swizzle row of bf16
constexpr int STAGES = 4;
constexpr int LM_THREADS = 192;
constexpr uint32_t A_STAGE = BM * BK * 2;  // 16 KB
constexpr uint32_t B_STAGE = BN * BK * 2;  // 32 KB

struct LmParams {
  CUtensorMap tmap_h;
  CUtensorMap tmap_w;
  int64_t rows, V;
  int32_t nm, nn, nk;  // tiles along rows and vocabulary; k-blocks
  unsigned long long *slot;
  int32_t *status;
  uint64_t wait_ns;  // limit of every pipeline wait (2 s unless a test shortens it)
  int32_t stall_at;  // test hook: k-blocks from this index on (counted per CTA) are never issued (-1: off)
};

template <int dummy = 0>
__global__ void __launch_bounds__(LM_THREADS, 1) lm_head_argmax_kernel(const __grid_constant__ LmParams P) {
  constexpr uint32_t IDESC = tc::idesc_bf16_f32(BM, BN, false);
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar_full[STAGES], bar_empty[STAGES], bar_tf[2], bar_te[2], bar_never;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_zero;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  auto a_s = [&](int st) { return sbase + uint32_t(st) * A_STAGE; };
  auto b_s = [&](int st) { return sbase + STAGES * A_STAGE + uint32_t(st) * B_STAGE; };
  const uint32_t full0 = smem_u32(&bar_full[0]), empty0 = smem_u32(&bar_empty[0]);
  const uint32_t tf0 = smem_u32(&bar_tf[0]), te0 = smem_u32(&bar_te[0]);
  if (tid == 0) {
    for (int i = 0; i < STAGES; ++i) {
      tc::mbar_init(full0 + 8 * i, 1);
      tc::mbar_init(empty0 + 8 * i, 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(tf0 + 8 * i, 1);
      tc::mbar_init(te0 + 8 * i, 4);  // one arrival per epilogue warp
    }
    tc::mbar_init(smem_u32(&bar_never), 1);  // nothing arrives on it (the stall test hook waits on it)
    s_abort = 0;
    s_zero = 0;
    tc::fence_barrier_init();
  }
  if (warp == 1) {
    tc::tmem_alloc(smem_u32(&s_tmem), 512);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = s_tmem;
  volatile int *abort_flag = &s_abort;
  const uint64_t wait_ns = P.wait_ns;
  auto give_up = [&]() {
    if (*abort_flag == 0) {
      *abort_flag = 1;
      flag(P.status, DREAMS_DATA_TIMEOUT);
    }
  };
  const int64_t ntiles = int64_t(P.nm) * P.nn;
  const int nk = P.nk;

  if (warp == 0) {
    // ---------------- TMA producer
    if (lane == 0) {
      tc::prefetch_tmap(&P.tmap_h);
      tc::prefetch_tmap(&P.tmap_w);
      int64_t g = 0;  // k-blocks issued
      for (int64_t t = blockIdx.x; t < ntiles && !*abort_flag; t += gridDim.x) {
        const int m = int(t % P.nm), n = int(t / P.nm);
        for (int kb = 0; kb < nk; ++kb, ++g) {
          const int st = int(g % STAGES);
          if (g >= STAGES && !tc::mbar_wait(empty0 + 8 * st, ((g / STAGES) - 1) & 1, abort_flag, wait_ns)) {
            give_up();
            break;
          }
          if (P.stall_at >= 0 && g >= P.stall_at) {
            // test hook: this copy is never issued; its consumers' waits run
            // out, like this one on a barrier that nothing arrives on
            tc::mbar_wait(smem_u32(&bar_never), 0, abort_flag, wait_ns);
            give_up();
            break;
          }
          tc::mbar_arrive_expect_tx(full0 + 8 * st, A_STAGE + B_STAGE);
          tc::tma_load_2d(a_s(st), &P.tmap_h, full0 + 8 * st, kb * BK, m * BM);
          tc::tma_load_2d(b_s(st), &P.tmap_w, full0 + 8 * st, kb * BK, n * BN);
        }
      }
      // no copy may still be landing in shared memory when the CTA ends
      for (int64_t j = std::max<int64_t>(0, g - STAGES); j < g; ++j)
        tc::mbar_wait(full0 + 8 * int(j % STAGES), (j / STAGES) & 1, &s_zero);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      const uint64_t ad0 = tc::smem_desc_sw128(a_s(0), 16, 1024);
      const uint64_t bd0 = tc::smem_desc_sw128(b_s(0), 16, 1024);
      int64_t g = 0;
      int it = 0;  // tiles of this CTA
      int nd = 0;  // commits that a final wait covers
      bool ok = true;
      for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++it) {
        const int ab = it & 1;
        // the epilogue has read this accumulator's previous tile
        if (it >= 2 && !tc::mbar_wait(te0 + 8 * ab, ((it >> 1) - 1) & 1, abort_flag, wait_ns)) {
          give_up();
          break;
        }
        tc::fence_after_sync();
        for (int kb = 0; kb < nk; ++kb, ++g) {
          const int st = int(g % STAGES);
          if (!tc::mbar_wait(full0 + 8 * st, (g / STAGES) & 1, abort_flag, wait_ns)) {
            give_up();
            ok = false;
            break;
          }
          tc::fence_after_sync();
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint32_t off = k * 32;  // 16 bf16 along K
            tc::mma_ss(tmem + 256u * ab, ad0 + ((uint32_t(st) * A_STAGE + off) >> 4),
                       bd0 + ((uint32_t(st) * B_STAGE + off) >> 4), IDESC, (kb > 0 || k > 0) ? 1u : 0u);
          }
          tc::mma_commit(empty0 + 8 * st);
        }
        tc::mma_commit(tf0 + 8 * ab);
        ++nd;
      }
      // every MMA has completed before TMEM is freed
      if (nd > 0) tc::mbar_wait(tf0 + 8 * ((nd - 1) & 1), ((nd - 1) >> 1) & 1, &s_zero);
    }
  } else {
    // ---------------- epilogue warps 2-5: TMEM lane quarter = warp % 4
    const int q = warp & 3;
    const int r_in = 32 * q + lane;
    int it = 0;
    for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x, ++it) {
      const int ab = it & 1;
      const int m = int(t % P.nm), n = int(t / P.nm);
      if (!__all_sync(0xffffffffu, tc::mbar_wait(tf0 + 8 * ab, (it >> 1) & 1, abort_flag, wait_ns))) {
        give_up();
        break;
      }
      // after a give-up the MMA thread commits what it issued, so this
      // accumulator may be unfinished: nothing more is merged
      if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
      tc::fence_after_sync();
      const uint32_t taddr = tmem + (uint32_t(32 * q) << 16) + 256u * ab;
      const int64_t v0 = int64_t(n) * BN;
      const int nvalid = int(std::min<int64_t>(BN, P.V - v0));
      int bk = INT_MIN, bi = 0;
#pragma unroll 1
      for (int c = 0; c < BN; c += 64) {
        uint32_t x0[32], x1[32];
        tc::tmem_ld32(taddr + c, x0);
        tc::tmem_ld32(taddr + c + 32, x1);
        tc::tmem_wait_ld();
        if (c + 64 >= BN) {
          // all of this accumulator is in registers: release it
          tc::fence_before_sync();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive(te0 + 8 * ab);
        }
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const int k0 = order_key(x0[e]);
          if (c + e < nvalid && k0 > bk) {
            bk = k0;
            bi = c + e;
          }
        }
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const int k1 = order_key(x1[e]);
          if (c + 32 + e < nvalid && k1 > bk) {
            bk = k1;
            bi = c + 32 + e;
          }
        }
      }
      const int64_t row = int64_t(m) * BM + r_in;
      if (row < P.rows && bk != INT_MIN) atomicMax(P.slot + row, pack_key_idx(bk, int(v0) + bi));
    }
  }

  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// The row's index (and its maximum value) from its slot; resets the slot. A
// slot that no tile reached (only when a wait gave up: every tile merges a
// candidate, and no (key, index) pair packs to 0) leaves the row untouched.
__global__ void __launch_bounds__(256) lm_head_finish_kernel(unsigned long long *slot, int64_t rows, int32_t *out_idx,
                                                             float *out_max) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int64_t r = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (r >= rows) return;
  const unsigned long long v = slot[r];
  if (v == 0ull) return;
  slot[r] = 0ull;
  out_idx[r] = int32_t(~uint32_t(v & 0xffffffffull));
  if (out_max != nullptr) {
    const int key = int(uint32_t(v >> 32) ^ 0x80000000u);
    uint32_t u;
    if (key == INT_MAX) u = 0x7fc00000u;  // NaN
    else if (key >= 0) u = uint32_t(key);
    else u = uint32_t(key ^ 0x7fffffff);
    out_max[r] = __uint_as_float(u);
  }
}

// 2-D view (K innermost, rows) of a row-major bf16 matrix, box (BK, box_rows),
// 128-byte swizzle; rows past the end read as zeros.
bool make_2d_map(CUtensorMap *m, const void *base, int64_t K, int64_t rows, int64_t ld, int box_rows) {
  EncodeTiledFn enc = encode_tiled();
  if (enc == nullptr) return false;
  const cuuint64_t dims[2] = {cuuint64_t(K), cuuint64_t(rows)};
  const cuuint64_t strides[1] = {cuuint64_t(ld) * 2};
  const cuuint32_t box[2] = {cuuint32_t(BK), cuuint32_t(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

constexpr size_t LM_SMEM = size_t(STAGES) * (A_STAGE + B_STAGE) + 1024;

}  // namespace
}  // namespace dreams

using namespace dreams;

extern "C" size_t dreams_lm_head_argmax_workspace_size(int64_t rows) {
  if (rows < 1) return 0;
  return (size_t(rows) * 8 + 255) / 256 * 256;
}

extern "C" dreams_status_t dreams_lm_head_argmax(const void *hidden, int64_t rows, int64_t hidden_dim,
                                                 int64_t ld_hidden, const void *weight, int64_t V, int64_t ld_weight,
                                                 int32_t *out_idx, float *out_max, void *workspace,
                                                 size_t workspace_bytes, int32_t *status_word,
                                                 dreams_stream_t stream) {
  if (hidden == nullptr || weight == nullptr || out_idx == nullptr || rows < 1 || V < 1 || hidden_dim < BK)
    return DREAMS_ERR_INVALID_ARG;
  if (hidden_dim % BK != 0 || ld_hidden < hidden_dim || ld_weight < hidden_dim || ld_hidden % 8 != 0 ||
      ld_weight % 8 != 0 || !aligned16(hidden) || !aligned16(weight) ||
      (out_max != nullptr && (reinterpret_cast<uintptr_t>(out_max) & 3)))
    return DREAMS_ERR_INVALID_ARG;
  if (V > INT_MAX - BN || rows > (int64_t(1) << 31) || hidden_dim / BK > INT_MAX) return DREAMS_ERR_UNSUPPORTED;
  if (workspace == nullptr || workspace_bytes < dreams_lm_head_argmax_workspace_size(rows) || !aligned16(workspace))
    return DREAMS_ERR_WORKSPACE;
  LmParams P;
  memset(&P, 0, sizeof(P));
  if (!make_2d_map(&P.tmap_h, hidden, hidden_dim, rows, ld_hidden, BM) ||
      !make_2d_map(&P.tmap_w, weight, hidden_dim, V, ld_weight, BN))
    return DREAMS_ERR_UNSUPPORTED;
  P.rows = rows;
  P.V = V;
  P.nm = int32_t((rows + BM - 1) / BM);
  P.nn = int32_t((V + BN - 1) / BN);
  P.nk = int32_t(hidden_dim / BK);
  P.slot = static_cast<unsigned long long *>(workspace);
  P.status = status_word;
  test_stall(DREAMS_TEST_LM_HEAD, &P.stall_at, &P.wait_ns);
  {
    const dreams_status_t st =
        ensure_max_dynamic_smem(reinterpret_cast<const void *>(lm_head_argmax_kernel<0>), int(LM_SMEM));
    if (st != DREAMS_OK) return st;
  }
  const int64_t ntiles = int64_t(P.nm) * P.nn;
  const unsigned grid = unsigned(std::min<int64_t>(ntiles, num_sms()));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  lm_head_argmax_kernel<0><<<grid, LM_THREADS, LM_SMEM, s>>>(P);
  dreams_status_t st = check_launch();
  if (st != DREAMS_OK) return st;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned((rows + 255) / 256));
  cfg.blockDim = dim3(256);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, lm_head_finish_kernel, P.slot, rows, out_idx, out_max);
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return DREAMS_ERR_CUDA;
  }
  return check_launch();
}
