// Per-node top-k of the logits (Sec. 3.1 "Progressive Expansion" and "Width Control":
// each node's draft token d_v and at most k children; Sec. 3.2: the greedy verification
// token V_n is entry 0).  Pure HBM streaming.
//
// One thread-block cluster per logit row.  Every CTA of the cluster scans a contiguous
// slice of the row with 16-byte vector loads; each thread keeps a sorted list of its KM
// best (value, index) pairs in registers.  The lists are merged by warp shuffles, then
// across the 8 warps of the CTA in shared memory, then across the CTAs of the cluster
// through distributed shared memory (no global scratch, one launch).
//
// Order: a 64-bit key (order-preserving bits of the fp32 value) << 32 | ~index, so a
// larger key is a larger value or, on equal values, a lower index.  -0.0 is folded into
// +0.0 before the key is formed.
#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "ptd_device.cuh"
#include "topk.cuh"

namespace cg = cooperative_groups;

namespace ptd {
namespace topk {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxCluster = 8;

__device__ __forceinline__ uint32_t ordered_bits(float f) {
  uint32_t u = __float_as_uint(f);
  if (u == 0x80000000u) u = 0u;   // -0.0 == +0.0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float from_ordered(uint32_t o) {
  const uint32_t u = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
  return __uint_as_float(u);
}

__device__ __forceinline__ uint64_t make_key(uint32_t ord, uint32_t idx) {
  return ((uint64_t)ord << 32) | (uint64_t)(~idx);
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t w = __shfl_xor_sync(0xffffffffu, v, o);
    v = w > v ? w : v;
  }
  return v;
}

// Sorted (descending) per-thread list of the KM best elements seen by this thread.
// Elements arrive in increasing index order, so a strict ">" keeps the lower index first.
template <int KM>
struct ThreadList {
  uint32_t ord[KM];
  uint32_t idx[KM];
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int s = 0; s < KM; ++s) {
      ord[s] = 0u;
      idx[s] = 0xFFFFFFFFu;
    }
  }
  __device__ __forceinline__ void push(uint32_t o, uint32_t i) {
    if (o <= ord[KM - 1]) return;
    ord[KM - 1] = o;
    idx[KM - 1] = i;
#pragma unroll
    for (int s = KM - 1; s > 0; --s) {
      if (ord[s] > ord[s - 1]) {
        const uint32_t to = ord[s], ti = idx[s];
        ord[s] = ord[s - 1];
        idx[s] = idx[s - 1];
        ord[s - 1] = to;
        idx[s - 1] = ti;
      }
    }
  }
  __device__ __forceinline__ uint64_t head() const { return make_key(ord[0], idx[0]); }
  __device__ __forceinline__ void pop() {
#pragma unroll
    for (int s = 0; s < KM - 1; ++s) {
      ord[s] = ord[s + 1];
      idx[s] = idx[s + 1];
    }
    ord[KM - 1] = 0u;
    idx[KM - 1] = 0xFFFFFFFFu;
  }
};

template <typename T>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int kN = 8;
  __device__ __forceinline__ static void unpack(const uint4& v, float (&f)[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      f[2 * j] = __uint_as_float(w[j] << 16);
      f[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
    }
  }
  __device__ __forceinline__ static float scalar(const __nv_bfloat16* p) {
    return __uint_as_float((uint32_t)(*reinterpret_cast<const uint16_t*>(p)) << 16);
  }
};
template <>
struct Vec<float> {
  static constexpr int kN = 4;
  __device__ __forceinline__ static void unpack(const uint4& v, float (&f)[8]) {
    f[0] = __uint_as_float(v.x);
    f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z);
    f[3] = __uint_as_float(v.w);
  }
  __device__ __forceinline__ static float scalar(const float* p) { return *p; }
};

template <int KM, typename T>
__global__ void __launch_bounds__(kThreads) topk_cluster_kernel(const T* __restrict__ logits, int64_t rows,
                                                                int vocab, int64_t row_stride, int k,
                                                                int32_t* __restrict__ out_idx,
                                                                float* __restrict__ out_val) {
  constexpr int VN = Vec<T>::kN;
  __shared__ uint64_t warp_keys[kWarps][KM];
  __shared__ uint64_t cta_keys[KM];

  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int csize = (int)cluster.num_blocks();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  for (int64_t r = blockIdx.y; r < rows; r += gridDim.y) {
    const T* row = logits + r * row_stride;
    // vector body [a0, a1): 16-byte aligned; head [0, a0) and tail [a1, vocab) scalar
    const uintptr_t addr = reinterpret_cast<uintptr_t>(row);
    int a0 = (int)(((16 - (addr & 15)) & 15) / sizeof(T));
    if (a0 > vocab) a0 = vocab;
    const int nvec = (vocab - a0) / VN;
    const int a1 = a0 + nvec * VN;
    const int per = (nvec + csize - 1) / csize;
    const int v_begin = min(nvec, rank * per), v_end = min(nvec, v_begin + per);

    ThreadList<KM> list;
    list.init();
    if (rank == 0 && threadIdx.x == 0)
      for (int i = 0; i < a0; ++i) list.push(ordered_bits(Vec<T>::scalar(row + i)), (uint32_t)i);

    const uint4* vrow = reinterpret_cast<const uint4*>(row + a0);
    constexpr int U = 4;
    int v = v_begin + threadIdx.x;
    for (; v + (U - 1) * kThreads < v_end; v += U * kThreads) {
      uint4 x[U];
#pragma unroll
      for (int q = 0; q < U; ++q) x[q] = __ldg(vrow + v + q * kThreads);
#pragma unroll
      for (int q = 0; q < U; ++q) {
        float f[8];
        Vec<T>::unpack(x[q], f);
        const uint32_t i0 = (uint32_t)(a0 + (v + q * kThreads) * VN);
#pragma unroll
        for (int e = 0; e < VN; ++e) list.push(ordered_bits(f[e]), i0 + e);
      }
    }
    for (; v < v_end; v += kThreads) {
      float f[8];
      Vec<T>::unpack(__ldg(vrow + v), f);
      const uint32_t i0 = (uint32_t)(a0 + v * VN);
#pragma unroll
      for (int e = 0; e < VN; ++e) list.push(ordered_bits(f[e]), i0 + e);
    }
    if (rank == csize - 1 && threadIdx.x == kThreads - 1)
      for (int i = a1; i < vocab; ++i) list.push(ordered_bits(Vec<T>::scalar(row + i)), (uint32_t)i);

    // warp merge: k rounds of "largest head wins"
    for (int s = 0; s < k; ++s) {
      const uint64_t mine = list.head();
      const uint64_t best = warp_max_u64(mine);
      if (mine == best) list.pop();
      if (lane == 0) warp_keys[warp][s] = best;
    }
    __syncthreads();
    // CTA merge across warps (warp 0, lane w owns warp w's list)
    if (warp == 0) {
      int cur = 0;
      for (int s = 0; s < k; ++s) {
        const uint64_t mine = (lane < kWarps && cur < k) ? warp_keys[lane][cur] : 0ull;
        const uint64_t best = warp_max_u64(mine);
        if (lane < kWarps && mine == best && best != 0ull) ++cur;
        if (lane == 0) cta_keys[s] = best;
      }
    }
    cluster.sync();
    // cluster merge through distributed shared memory (rank 0, lane c owns CTA c's list)
    if (rank == 0 && warp == 0) {
      const uint64_t* remote = lane < csize ? cluster.map_shared_rank(cta_keys, lane) : nullptr;
      int cur = 0;
      for (int s = 0; s < k; ++s) {
        const uint64_t mine = (lane < csize && cur < k) ? remote[cur] : 0ull;
        const uint64_t best = warp_max_u64(mine);
        if (lane < csize && mine == best && best != 0ull) ++cur;
        if (lane == 0) {
          out_idx[r * k + s] = (int32_t)(~(uint32_t)(best & 0xFFFFFFFFull));
          out_val[r * k + s] = from_ordered((uint32_t)(best >> 32));
        }
      }
    }
    cluster.sync();   // keep every CTA's shared memory alive until rank 0 has read it
  }
}

template <int KM, typename T>
cudaError_t launch_km(const T* logits, int64_t rows, int vocab, int64_t row_stride, int k, int32_t* out_idx,
                      float* out_val, int cluster, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  const int64_t gy = rows < 65535 ? rows : 65535;
  cfg.gridDim = dim3((unsigned)cluster, (unsigned)gy, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, topk_cluster_kernel<KM, T>, logits, rows, vocab, row_stride, k, out_idx,
                            out_val);
}

template <typename T>
cudaError_t launch_t(const T* logits, int64_t rows, int vocab, int64_t row_stride, int k, int32_t* out_idx,
                     float* out_val, cudaStream_t stream) {
  // enough CTAs per row to keep HBM busy, at most one portable cluster (8 CTAs)
  const int per_cta = (int)(16384 / sizeof(T)) * 2;   // ~32 KB of logits per CTA
  int cluster = (vocab + per_cta - 1) / per_cta;
  cluster = cluster < 1 ? 1 : (cluster > kMaxCluster ? kMaxCluster : cluster);
  if (k <= 1) return launch_km<1>(logits, rows, vocab, row_stride, k, out_idx, out_val, cluster, stream);
  if (k <= 2) return launch_km<2>(logits, rows, vocab, row_stride, k, out_idx, out_val, cluster, stream);
  if (k <= 4) return launch_km<4>(logits, rows, vocab, row_stride, k, out_idx, out_val, cluster, stream);
  if (k <= 8) return launch_km<8>(logits, rows, vocab, row_stride, k, out_idx, out_val, cluster, stream);
  return launch_km<16>(logits, rows, vocab, row_stride, k, out_idx, out_val, cluster, stream);
}

}  // namespace topk

cudaError_t launch_topk(const void* logits, bool bf16, int64_t rows, int vocab, int64_t row_stride, int k,
                        int32_t* out_idx, float* out_val, cudaStream_t stream) {
  if (bf16)
    return topk::launch_t(static_cast<const __nv_bfloat16*>(logits), rows, vocab, row_stride, k, out_idx,
                          out_val, stream);
  return topk::launch_t(static_cast<const float*>(logits), rows, vocab, row_stride, k, out_idx, out_val, stream);
}

}  // namespace ptd
