// LM head with a fused top-k epilogue: the per-node logits h_v W^T (the model's next-token
// scores P(y_T | ...) of Alg. 1 step 2) and their top-k (Sec. 3.1 drafts d_v, Sec. 3.2
// verification tokens V_n), without writing the logits anywhere.
//
// HBM-bound: W (vocab x d_model bf16, 1.05 GB for 128256 x 4096) is streamed once; the
// node rows H (at most 128) are the tcgen05 A operand, re-read from L2.  Persistent: one
// CTA per SM walks the vocabulary in tiles of 128 tokens (tile t, t + grid, ...).
//   warp 0     TMA producer: per 64-column chunk of d_model, H rows 0..127 (rows past
//              `rows` read as zero) and the tile's 128 W rows, 16 KB each, 128-byte
//              swizzle, into a 7-stage ring (112 KB of W in flight per SM);
//   warp 1     allocates TMEM, one thread issues 4 MMAs (M 128, N 128, K 16, bf16 -> fp32)
//              per chunk into one of two accumulators (tiles alternate), commits;
//   warps 2-5  epilogue: TMEM lane r holds node r's 128 logits of the tile; thread r reads
//              them 16 columns at a time and keeps its running top-k in registers as
//              64-bit keys (order-preserving value bits << 32 | ~token), so ties keep the
//              lower token first.
// After the last tile every CTA leaves its per-node lists in the workspace; a second small
// kernel (one CTA per node row) merges them and writes the outputs.  (Merging them in the
// CTA that finished last cost about 40 us of dependent loads on one SM.)
#include <cuda_runtime.h>

#include <cstdint>

#include "lm_head.cuh"
#include "ptd_device.cuh"

namespace ptd {
namespace lm {

constexpr int kThreads = 192;
constexpr int kStages = 7;
constexpr uint32_t kChunkBytes = 128 * 128;             // 128 rows x 64 bf16
constexpr uint32_t kStageBytes = 2 * kChunkBytes;       // H chunk, then W chunk
constexpr uint32_t kOffBar = kStages * kStageBytes;
constexpr int kNumBars = 2 * kStages + 5;               // full, empty, acc_full[2], acc_empty[2], drain
constexpr uint32_t kOffTmemPtr = kOffBar + kNumBars * 8;
constexpr uint32_t kOffAbort = kOffTmemPtr + 4;
constexpr uint32_t kSmemBytes = kOffAbort + 16 + 1024;  // slack to align the base to 1024 B
constexpr uint32_t kTmemCols = 256;                     // two 128-column accumulators
constexpr uint32_t kIdesc = idesc_bf16_f32(128, 128, 0, 0);
static_assert(kSmemBytes <= 232448, "shared memory budget");

__device__ __forceinline__ uint64_t make_key(float v, int token) {
  uint32_t u = __float_as_uint(v);
  if (u == 0x80000000u) u = 0u;   // -0.0 == +0.0
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((uint64_t)u << 32) | (uint32_t)(~(uint32_t)token);
}
__device__ __forceinline__ float key_value(uint64_t key) {
  const uint32_t o = (uint32_t)(key >> 32);
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}
__device__ __forceinline__ int key_token(uint64_t key) { return (int)(~(uint32_t)key); }

// Insert key into a descending list of KM keys (0 = empty: below every real key).
template <int KM>
__device__ __forceinline__ void insert(uint64_t (&top)[KM], uint64_t key) {
  if (key <= top[KM - 1]) return;
  top[KM - 1] = key;
#pragma unroll
  for (int j = KM - 1; j > 0; --j) {
    if (top[j] > top[j - 1]) {
      const uint64_t x = top[j];
      top[j] = top[j - 1];
      top[j - 1] = x;
    }
  }
}

template <int KM>
__global__ void __launch_bounds__(kThreads, 1)
    lm_head_topk_kernel(const __grid_constant__ CUtensorMap map_h, const __grid_constant__ CUtensorMap map_w,
                        int rows, int d_model, int vocab, int k, int32_t* __restrict__ out_idx,
                        float* __restrict__ out_val, uint64_t* __restrict__ partial, int32_t* __restrict__ dev_status) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint32_t base = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (base & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  base += pad;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  auto bar = [&](int i) { return base + kOffBar + 8u * (uint32_t)i; };
  auto full_bar = [&](int s) { return bar(s); };
  auto empty_bar = [&](int s) { return bar(kStages + s); };
  auto accf_bar = [&](int b) { return bar(2 * kStages + b); };
  auto acce_bar = [&](int b) { return bar(2 * kStages + 2 + b); };
  const uint32_t drain_bar = bar(2 * kStages + 4);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffAbort);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accf_bar(b), 1);
      mbar_init(acce_bar(b), 4);   // one arrival per epilogue warp
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(base + kOffTmemPtr, kTmemCols);
    tmem_relinquish();
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + kOffTmemPtr);
  const int n_tiles = (vocab + 127) / 128;
  const int n_chunks = d_model / 64;

  if (warp == 0) {
    // ================================================================ TMA producer
    if (lane == 0) {
      prefetch_tensormap(&map_h);
      prefetch_tensormap(&map_w);
      bool ok = true;
      int g = 0;   // chunks issued by this CTA (ring position)
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
        for (int c = 0; c < n_chunks && ok; ++c, ++g) {
          const int s = g % kStages;
          ok = mbar_wait(empty_bar(s), (uint32_t)(((g / kStages) & 1) ^ 1), abort_flag, dev_status);
          if (!ok) break;
          const uint32_t dst = base + (uint32_t)s * kStageBytes;
          mbar_arrive_expect_tx(full_bar(s), kStageBytes);
          tma_load_2d(dst, &map_h, full_bar(s), c * 64, 0);
          tma_load_2d(dst + kChunkBytes, &map_w, full_bar(s), c * 64, tile * 128);
        }
      }
      if (!ok) {   // let the copies already issued land before the CTA can exit
        for (int back = 1; back <= kStages && g - back >= 0; ++back)
          mbar_drain(full_bar((g - back) % kStages), (uint32_t)(((g - back) / kStages) & 1), 100000000ull);
      }
    }
  } else if (warp == 1) {
    // ================================================================ MMA issuer
    if (lane == 0) {
      bool ok = true;
      int g = 0, it = 0;
      for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x, ++it) {
        const int buf = it & 1;
        ok = mbar_wait(acce_bar(buf), (uint32_t)(((it >> 1) & 1) ^ 1), abort_flag, dev_status);
        if (!ok) break;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)buf * 128u;
        for (int c = 0; c < n_chunks && ok; ++c, ++g) {
          const int s = g % kStages;
          ok = mbar_wait(full_bar(s), (uint32_t)((g / kStages) & 1), abort_flag, dev_status);
          if (!ok) break;
          tc_fence_after();
          const uint32_t a0 = base + (uint32_t)s * kStageBytes, b0 = a0 + kChunkBytes;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint64_t ad = smem_desc_sw128(a0 + (uint32_t)kk * 32u, 16, 1024);
            const uint64_t bd = smem_desc_sw128(b0 + (uint32_t)kk * 32u, 16, 1024);
            mma_bf16_ss(d, ad, bd, kIdesc, (c > 0 || kk > 0) ? 1u : 0u);
          }
          mma_commit(empty_bar(s));   // the stage is free once these MMAs have read it
        }
        if (ok) mma_commit(accf_bar(buf));
      }
      if (!ok) {   // let the tensor core finish what was issued before TMEM is freed
        mma_commit(drain_bar);
        mbar_drain(drain_bar, 0, 100000000ull);
      }
    }
  } else {
    // ================================================================ epilogue
    const int wq = warp & 3;                     // TMEM lane quarter of this warp
    const int r = wq * 32 + lane;                // node row
    const uint32_t lane_base = (uint32_t)(wq * 32) << 16;
    uint64_t top[KM];
#pragma unroll
    for (int j = 0; j < KM; ++j) top[j] = 0ull;
    bool ok = true;
    int it = 0;
    for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x, ++it) {
      const int buf = it & 1;
      if (!(ok = mbar_wait_warp(accf_bar(buf), (uint32_t)((it >> 1) & 1), abort_flag, dev_status))) break;
      tc_fence_after();
      const int t0 = tile * 128;
#pragma unroll 1
      for (int c8 = 0; c8 < 8; ++c8) {
        uint32_t v[16];
        tmem_ld16(tmem + lane_base + (uint32_t)buf * 128u + (uint32_t)c8 * 16u, v);
        tmem_ld_wait();
        const int tb = t0 + c8 * 16;
        if (tb + 16 <= vocab) {
#pragma unroll
          for (int e = 0; e < 16; ++e) insert<KM>(top, make_key(__uint_as_float(v[e]), tb + e));
        } else {
#pragma unroll
          for (int e = 0; e < 16; ++e)
            if (tb + e < vocab) insert<KM>(top, make_key(__uint_as_float(v[e]), tb + e));
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acce_bar(buf));
    }
    if (ok && r < rows) {
      uint64_t* mine = partial + ((size_t)blockIdx.x * rows + r) * KM;
#pragma unroll
      for (int j = 0; j < KM; ++j) mine[j] = top[j];
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Per-row merge of the CTAs' candidate lists: one CTA per node row, each thread folds a few
// lists into its own, then KM rounds of a warp-wide maximum (the owning lane pops its head)
// per warp and once more across the warps.
constexpr int kMergeThreads = 128;

// Largest key of the warp: the largest high word (one warp reduction), then the largest low
// word among the lanes that hold it (a second one).
template <int KM>
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t x) {
  const uint32_t hi = (uint32_t)(x >> 32);
  const uint32_t mhi = __reduce_max_sync(0xffffffffu, hi);
  const uint32_t mlo = __reduce_max_sync(0xffffffffu, hi == mhi ? (uint32_t)x : 0u);
  return ((uint64_t)mhi << 32) | mlo;
}

template <int KM>
__device__ __forceinline__ void warp_top(uint64_t (&top)[KM], uint64_t (&out)[KM]) {
  // top: this lane's descending list; out (every lane): the warp's KM largest keys
#pragma unroll
  for (int j = 0; j < KM; ++j) {
    const uint64_t m = warp_max_u64<KM>(top[0]);
    out[j] = m;
    if (m != 0ull && top[0] == m) {   // keys are distinct (each token lives in one tile)
#pragma unroll
      for (int q = 0; q < KM - 1; ++q) top[q] = top[q + 1];
      top[KM - 1] = 0ull;
    }
  }
}

template <int KM>
__global__ void __launch_bounds__(kMergeThreads)
    lm_merge_kernel(const uint64_t* __restrict__ partial, int ctas, int rows, int k, int32_t* __restrict__ out_idx,
                    float* __restrict__ out_val) {
  __shared__ uint64_t warp_s[kMergeThreads / 32][KM];
  const int r = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint64_t top[KM];
#pragma unroll
  for (int j = 0; j < KM; ++j) top[j] = 0ull;
  for (int c = threadIdx.x; c < ctas; c += kMergeThreads) {
    const uint64_t* lst = partial + ((size_t)c * rows + r) * KM;
#pragma unroll
    for (int j = 0; j < KM; ++j) insert<KM>(top, lst[j]);
  }
  uint64_t best[KM];
  warp_top<KM>(top, best);
  if (lane == 0) {
#pragma unroll
    for (int j = 0; j < KM; ++j) warp_s[warp][j] = best[j];
  }
  __syncthreads();
  if (warp == 0) {
#pragma unroll
    for (int j = 0; j < KM; ++j) top[j] = lane < kMergeThreads / 32 ? warp_s[lane][j] : 0ull;
    warp_top<KM>(top, best);
    if (lane == 0) {
#pragma unroll
      for (int j = 0; j < KM; ++j) {
        if (j < k) {
          out_idx[(size_t)r * k + j] = best[j] ? key_token(best[j]) : -1;
          out_val[(size_t)r * k + j] = best[j] ? key_value(best[j]) : 0.f;
        }
      }
    }
  }
}

}  // namespace lm

size_t lm_head_workspace_bytes(int ctas, int rows) {
  return 256 + (size_t)ctas * rows * kLmMaxK * sizeof(uint64_t);
}

int lm_head_ctas(int num_sms, int vocab) {
  const int tiles = (vocab + 127) / 128;
  return tiles < num_sms ? tiles : num_sms;
}

cudaError_t launch_lm_head_topk(const CUtensorMap& map_h, const CUtensorMap& map_w, int rows, int d_model, int vocab,
                                int k, int32_t* out_idx, float* out_val, void* workspace, int ctas,
                                int32_t* dev_status, cudaStream_t stream) {
  uint64_t* partial = reinterpret_cast<uint64_t*>(static_cast<char*>(workspace) + 256);
  cudaError_t e = cudaSuccess;
#define PTD_LM_LAUNCH(KMV)                                                                                        \
  do {                                                                                                            \
    e = cudaFuncSetAttribute(lm::lm_head_topk_kernel<KMV>, cudaFuncAttributeMaxDynamicSharedMemorySize,          \
                             (int)lm::kSmemBytes);                                                                \
    if (e != cudaSuccess) return e;                                                                               \
    lm::lm_head_topk_kernel<KMV><<<ctas, lm::kThreads, lm::kSmemBytes, stream>>>(                                 \
        map_h, map_w, rows, d_model, vocab, k, out_idx, out_val, partial, dev_status);                            \
    e = cudaGetLastError();                                                                                       \
    if (e != cudaSuccess) return e;                                                                               \
    lm::lm_merge_kernel<KMV><<<rows, lm::kMergeThreads, 0, stream>>>(partial, ctas, rows, k, out_idx, out_val);   \
  } while (0)
  if (k <= 4)
    PTD_LM_LAUNCH(4);
  else if (k <= 8)
    PTD_LM_LAUNCH(8);
  else
    PTD_LM_LAUNCH(16);
#undef PTD_LM_LAUNCH
  return cudaGetLastError();
}

}  // namespace ptd
