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
#include "verify_tree.cuh"

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

// Largest key of the warp: the largest high word (one warp reduction), then the largest low
// word among the lanes that hold it (a second one).
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
  const uint32_t hi = (uint32_t)(v >> 32);
  const uint32_t mhi = __reduce_max_sync(0xffffffffu, hi);
  const uint32_t mlo = __reduce_max_sync(0xffffffffu, hi == mhi ? (uint32_t)v : 0u);
  return ((uint64_t)mhi << 32) | mlo;
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
  // Insert a full key (any index order): larger key first, ties impossible (distinct indices).
  __device__ __forceinline__ void push_key(uint64_t key) {
    const uint32_t o = (uint32_t)(key >> 32), i = ~(uint32_t)key;
    if (key <= make_key(ord[KM - 1], idx[KM - 1])) return;
    ord[KM - 1] = o;
    idx[KM - 1] = i;
#pragma unroll
    for (int s = KM - 1; s > 0; --s) {
      if (make_key(ord[s], idx[s]) > make_key(ord[s - 1], idx[s - 1])) {
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

  if (threadIdx.x == 0) grid_launch_dependents();   // the next grid may be placed now; it waits for this one
  grid_dependency_wait();   // the logits and outputs belong to the stream's previous work
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

// ------------------------------------------------------------------ the step's verification
// Trees that no row can complete (an empty or out-of-range node range, or offsets that do not
// run from 0 to n_total): their outputs and the status are written at once (one warp).
__device__ __forceinline__ void flag_bad_trees_warp(const VerifyArgs& va) {
  const int lane = threadIdx.x & 31;
  for (int b = lane; b < va.batch; b += 32) {
    const int n0 = va.node_offsets[b], n1 = va.node_offsets[b + 1];
    const bool bad = n1 - n0 < 1 || n1 - n0 > va.max_nodes || n0 < 0 || n1 > va.n_total ||
                     (b == 0 && n0 != 0) || (b == va.batch - 1 && n1 != va.n_total);
    if (bad) {
      for (int j = 0; j < va.max_nodes; ++j) va.accepted[(size_t)b * va.max_nodes + j] = -1;
      va.accept_len[b] = 0;
      va.bonus[b] = -1;
      atomicMax(va.dev_status, (int)PTD_ERR_INVALID_TREE);
    }
  }
}

// Greedy verification of tree b on the calling warp, on column 0 of the top-k rows already
// written (and made visible to this warp), and the tree's outputs.
__device__ __forceinline__ void verify_and_write_warp(const VerifyArgs& va, int b, const vt::TreeInputs& tin,
                                                      const int32_t* out_idx, int k, vt::VerifyScratch& sc,
                                                      vt::TreeVerdict& vd) {
  const int lane = threadIdx.x & 31;
  vt::verify_tree_warp(tin, out_idx, k, sc, &vd);
  __syncwarp();
  int len = vd.len;
  if (len > va.max_nodes) len = va.max_nodes;
  int32_t* acc_row = va.accepted + (size_t)b * va.max_nodes;
  for (int j = lane; j < va.max_nodes; j += 32) acc_row[j] = j < len ? vd.path[j] : -1;
  if (lane == 0) {
    va.accept_len[b] = len;
    va.bonus[b] = vd.bonus;
    if (vd.invalid) atomicMax(va.dev_status, (int)PTD_ERR_INVALID_TREE);
  }
}

// ------------------------------------------------------------------ bf16 fast path
// Each CTA stages its contiguous slice of the row (up to kSliceVec 16-byte vectors) into
// shared memory with bulk asynchronous copies, so the row is read from HBM exactly once.
// Then every warp works on its own share of the slice (vectors lane + 32 w + 256 j) without
// waiting for the others:
//   1. every lane's maximum;
//   2. T_w = the k-th largest lane maximum of the warp (k rounds of "largest wins"): the k
//      lanes holding those maxima own k distinct elements >= T_w, so the warp's top-k is
//      among its elements >= T_w;
//   3. each lane keeps its elements >= T_w in an exact sorted list of KM (value, index)
//      pairs (elements arrive in increasing index order, so ties keep the lower index), and
//      the warp selects its top-k from the lists' heads.
// One CTA barrier, then warp 0 merges the 8 warps' lists and the CTAs of the cluster merge
// theirs over distributed shared memory.  With verification (the step's tail), the cluster
// that writes the last row of a tree then verifies that tree (greedy, on one warp), so no
// separate verification launch follows.
constexpr int kSliceVec = 4096;            // 64 KB of bf16 logits per CTA
constexpr uint32_t kChunkBytes = 16384;    // bytes per bulk copy

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
// Lane-wise maximum of two bf16 pairs in one instruction (exact: a maximum only compares)
__device__ __forceinline__ uint32_t bf16x2_max(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
constexpr uint32_t kBf16x2NegInf = 0xFF80FF80u;

template <int KM, bool kVerify>
__global__ void __launch_bounds__(kThreads) topk_bf16_kernel(const __nv_bfloat16* __restrict__ logits,
                                                             int64_t rows, int vocab, int64_t row_stride, int k,
                                                             int32_t* __restrict__ out_idx,
                                                             float* __restrict__ out_val, int32_t* dev_status,
                                                             const VerifyArgs va) {
  extern __shared__ __align__(128) uint4 slice[];
  __shared__ uint64_t warp_keys[kWarps][KM];
  __shared__ uint64_t cta_keys[KM];
  __shared__ __align__(8) uint64_t bar_s;
  __shared__ int abort_s;

  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int csize = (int)cluster.num_blocks();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tid = threadIdx.x;
  const uint32_t bar = smem_u32(&bar_s);
  if (tid == 0) {
    mbar_init(bar, 1);
    abort_s = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (tid == 0) grid_launch_dependents();   // the next grid may be placed now; it waits for this one
  // the tree of a row (rank 0's thread 0 looks it up while the row's copy is in flight)
  auto tree_of = [&](int64_t r) {
    int lo = 0, hi = va.batch;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (va.node_offsets[mid] <= r) lo = mid; else hi = mid;
    }
    return lo;
  };
  int row_tree = 0;
  grid_dependency_wait();   // the logits, the trees and the outputs belong to the stream's previous work
  if constexpr (kVerify) {
    // Trees that no row completes (an empty or out-of-range node range, or offsets that do not
    // run from 0 to n_total): their outputs and the status are written here, by warp 1 of the
    // first CTA, while its copy is in flight; a tree whose rows all arrive is verified below.
    if (blockIdx.x == 0 && blockIdx.y == 0 && warp == 1) flag_bad_trees_warp(va);
  }
  uint32_t phase = 0;

  for (int64_t r = blockIdx.y; r < rows; r += gridDim.y, phase ^= 1u) {
    const __nv_bfloat16* row = logits + r * row_stride;
    const uintptr_t addr = reinterpret_cast<uintptr_t>(row);
    int a0 = (int)(((16 - (addr & 15)) & 15) / 2);
    if (a0 > vocab) a0 = vocab;
    const int nvec = (vocab - a0) / 8;
    const int a1 = a0 + nvec * 8;
    const int per = (nvec + csize - 1) / csize;
    const int v_begin = min(nvec, rank * per), v_end = min(nvec, v_begin + per);
    const int nv = v_end - v_begin;
    const uint4* vrow = reinterpret_cast<const uint4*>(row + a0) + v_begin;
    const bool own_head = rank == 0 && tid == 0;
    const bool own_tail = rank == csize - 1 && tid == kThreads - 1;

    if (tid == 0) {
      fence_proxy_async_smem();   // the previous row's reads of the slice precede this copy
      const uint32_t total = (uint32_t)nv * 16u;
      mbar_arrive_expect_tx(bar, total);
      for (uint32_t off = 0; off < total; off += kChunkBytes) {
        const uint32_t n = total - off < kChunkBytes ? total - off : kChunkBytes;
        bulk_load(smem_u32(slice) + off, reinterpret_cast<const uint8_t*>(vrow) + off, n, bar);
      }
      if constexpr (kVerify) {
        if (rank == 0) row_tree = tree_of(r);
      }
    }
    // with verification: warp 0 of rank 0 loads its row's tree (parents, tokens) while the copy is
    // in flight, for the case that this cluster turns out to complete the tree
    vt::TreeInputs tin;
    if constexpr (kVerify) {
      if (rank == 0 && warp == 0) {
        const int b = __shfl_sync(0xffffffffu, row_tree, 0);
        vt::load_tree_warp(va.node_offsets, va.parents, va.tokens, va.n_total, va.max_nodes, b, tin);
      }
    }
    // head / tail scalars while the copy is in flight
    float tmax = -INFINITY;
    if (own_head)
      for (int i = 0; i < a0; ++i) tmax = fmaxf(tmax, Vec<__nv_bfloat16>::scalar(row + i));
    if (own_tail)
      for (int i = a1; i < vocab; ++i) tmax = fmaxf(tmax, Vec<__nv_bfloat16>::scalar(row + i));
    mbar_wait(bar, phase, &abort_s, dev_status);   // bounded: a lost copy only flags PTD_ERR_TIMEOUT

    // 1. lane maximum (four vectors in flight, two chains of packed pair maxima)
    {
      uint32_t h0 = kBf16x2NegInf, h1 = kBf16x2NegInf;
      int v = tid;
      for (; v + 3 * kThreads < nv; v += 4 * kThreads) {
        uint4 x[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) x[u] = slice[v + u * kThreads];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          h0 = bf16x2_max(h0, bf16x2_max(x[u].x, x[u].y));
          h1 = bf16x2_max(h1, bf16x2_max(x[u].z, x[u].w));
        }
      }
      for (; v < nv; v += kThreads) {
        const uint4 x = slice[v];
        h0 = bf16x2_max(h0, bf16x2_max(x.x, x.y));
        h1 = bf16x2_max(h1, bf16x2_max(x.z, x.w));
      }
      h0 = bf16x2_max(h0, h1);
      tmax = fmax3(tmax, bf16_lo(h0), bf16_hi(h0));
    }
    const bool has_elems = tid < nv || (own_head && a0 > 0) || (own_tail && a1 < vocab);

    // 2. T_w: the k-th largest lane maximum of this warp (-inf when fewer lanes hold elements)
    float thr;
    {
      uint64_t mine = has_elems ? make_key(ordered_bits(tmax), (uint32_t)lane) : 0ull;
      uint64_t kth = 0ull;
      for (int s = 0; s < k; ++s) {
        const uint64_t best = warp_max_u64(mine);
        if (mine == best) mine = 0ull;
        kth = best;
      }
      thr = kth != 0ull ? from_ordered((uint32_t)(kth >> 32)) : -INFINITY;
    }

    // 3. every lane's exact list of its elements >= T_w, then the warp's top-k
    ThreadList<KM> list;
    list.init();
    if (own_head)
      for (int i = 0; i < a0; ++i) {
        const float f = Vec<__nv_bfloat16>::scalar(row + i);
        if (f >= thr) list.push(ordered_bits(f), (uint32_t)i);
      }
    {
      auto vec_max = [](const uint4& x) {
        const uint32_t h = bf16x2_max(bf16x2_max(x.x, x.y), bf16x2_max(x.z, x.w));
        return fmaxf(bf16_lo(h), bf16_hi(h));
      };
      auto push_vec = [&](const uint4& x, int v) {
        const uint32_t gi = (uint32_t)(a0 + (v_begin + v) * 8);
        const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float f0 = bf16_lo(w[q]), f1 = bf16_hi(w[q]);
          if (f0 >= thr) list.push(ordered_bits(f0), gi + 2 * q);
          if (f1 >= thr) list.push(ordered_bits(f1), gi + 2 * q + 1);
        }
      };
      // four vectors in flight; the few that reach T_w are read again and pushed, in index order
      int v = tid;
      for (; v + 3 * kThreads < nv; v += 4 * kThreads) {
        uint4 x[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) x[u] = slice[v + u * kThreads];
        uint32_t hits = 0u;
#pragma unroll
        for (int u = 0; u < 4; ++u) hits |= (vec_max(x[u]) >= thr ? 1u : 0u) << u;
#pragma unroll 1
        for (; hits != 0u; hits &= hits - 1u) {   // rare: read the vector again
          const int vu = v + (__ffs(hits) - 1) * kThreads;
          push_vec(slice[vu], vu);
        }
      }
      for (; v < nv; v += kThreads) {
        const uint4 x = slice[v];
        if (vec_max(x) >= thr) push_vec(x, v);
      }
    }
    if (own_tail)
      for (int i = a1; i < vocab; ++i) {
        const float f = Vec<__nv_bfloat16>::scalar(row + i);
        if (f >= thr) list.push(ordered_bits(f), (uint32_t)i);
      }
    for (int s = 0; s < k; ++s) {
      const uint64_t mine = list.head();
      const uint64_t best = warp_max_u64(mine);
      if (mine == best) list.pop();
      if (lane == 0) warp_keys[warp][s] = best;
    }
    __syncthreads();   // also: every thread is done reading the slice
    if (warp == 0) {   // CTA merge across warps (lane w owns warp w's list)
      int cur = 0;
      for (int s = 0; s < k; ++s) {
        const uint64_t mine = (lane < kWarps && cur < k) ? warp_keys[lane][cur] : 0ull;
        const uint64_t best = warp_max_u64(mine);
        if (lane < kWarps && mine == best && best != 0ull) ++cur;
        if (lane == 0) cta_keys[s] = best;
      }
    }
    cluster.sync();
    // cluster merge: lane c of rank 0's warp 0 reads CTA c's sorted list at once, then k rounds
    // of "largest head wins"; lane s writes entry s
    if (rank == 0 && warp == 0) {
      ThreadList<KM> ml;
      ml.init();
      if (lane < csize) {
        const uint64_t* remote = cluster.map_shared_rank(cta_keys, lane);
        uint64_t got[KM];
#pragma unroll
        for (int s = 0; s < KM; ++s) got[s] = s < k ? remote[s] : 0ull;
#pragma unroll
        for (int s = 0; s < KM; ++s)
          if (got[s] != 0ull) ml.push_key(got[s]);
      }
      uint64_t out = 0ull;
      for (int s = 0; s < k; ++s) {
        const uint64_t mine = ml.head();
        const uint64_t best = warp_max_u64(mine);
        if (mine == best && best != 0ull) ml.pop();
        if (lane == s) out = best;
      }
      if (lane < k) {
        out_idx[r * k + lane] = (int32_t)(~(uint32_t)(out & 0xFFFFFFFFull));
        out_val[r * k + lane] = from_ordered((uint32_t)(out >> 32));
      }
      if constexpr (kVerify) {
        // the last row of a tree to be written: this cluster verifies the tree
        int vb = -1;
        __syncwarp();   // every lane's entries of this row are written before lane 0 counts the row
        if (lane == 0) {
          const int b = row_tree;
          const int T = tin.T;
          // release: this row's top-k before its count; acquire: the other rows' top-k (each
          // written before its own count) before this cluster reads them
          const int done = (int)atom_add_acq_rel_gpu(va.counters + b, 1u) + 1;
          if (done == T) vb = b;
        }
        vb = __shfl_sync(0xffffffffu, vb, 0);
        if (vb >= 0) {
          __shared__ vt::VerifyScratch vsc[1];
          __shared__ vt::TreeVerdict verdict[1];
          __syncwarp();   // lane 0's acquire precedes every lane's reads of the tree's rows
          verify_and_write_warp(va, vb, tin, out_idx, k, vsc[0], verdict[0]);
        }
      }
    }
    cluster.sync();   // keep every CTA's shared memory alive until rank 0 has read it
  }
}

// ------------------------------------------------------------------ streaming top-k of the step
// The step's rows (its trees' nodes) lie back to back in memory: as one sequence of 16-byte
// vectors (8 logits), CTA c of a persistent grid takes vectors [c L, (c + 1) L) of it, so every
// CTA moves the same number of bytes however many rows there are.  One producer warp streams
// the CTA's range through a ring of shared-memory chunks (bulk copies, one mbarrier pair per
// stage); copy and selection overlap across row boundaries and the grid never waits between
// waves.  The piece of a row that falls in one CTA's range (a row part) is selected by the 8
// selection warps much as in the clustered kernel: a threshold T is taken on the part's first
// chunk (the k-th largest of the CTA's 256 lane maxima over that chunk: the lanes holding the
// k largest own k elements >= T, so no element below T is among the CTA's top-k of the part),
// each warp raises its own threshold as its lanes' candidates grow, each lane keeps its
// elements at or above the threshold in an exact sorted list, and at the part's end the warps'
// lists are merged into the part's top-k, which goes to a global slot.  The part that
// completes its row (a per-row counter) merges the row's slots
// and writes the row; the row that completes its tree (a per-tree counter) has the tree
// verified on the same warp.  The part ends (the CTA merge, the global slot, the counters, a
// row's merge and a tree's verification: a chain of L2 round trips) run on a merge warp of
// their own, fed through a double buffer of the selection warps' keys, so that the stream
// never waits for them.  Counters are cleared by the launch before this one (the step's
// attention); slots are written before they are read within the launch.

// The k-th largest of the warp's 32 order-preserving values (0 = a lane without one), or 0 when
// fewer than k lanes hold one: one warp maximum and one ballot per distinct value, equal values
// counted together.  Any x with k elements >= x bounds the warp's top-k from below.
__device__ __forceinline__ uint32_t kth_largest_ord(uint32_t v, int k) {
  int count = 0;
  for (int s = 0; s < k; ++s) {
    const uint32_t m = __reduce_max_sync(0xffffffffu, v);
    if (m == 0u) return 0u;
    count += __popc(__ballot_sync(0xffffffffu, v == m));
    if (count >= k) return m;
    if (v == m) v = 0u;
  }
  return 0u;
}

// The k-th largest of the 256 values v[0..7] of the warp's lanes (0 = none), or 0 when fewer
// than k are nonzero: per distinct value one warp maximum and one warp sum of its copies.
__device__ __forceinline__ uint32_t kth_largest_ord8(uint32_t (&v)[8], int k) {
  int count = 0;
  for (int s = 0; s < k; ++s) {
    uint32_t lmax = 0u;
#pragma unroll
    for (int i = 0; i < 8; ++i) lmax = v[i] > lmax ? v[i] : lmax;
    const uint32_t m = __reduce_max_sync(0xffffffffu, lmax);
    if (m == 0u) return 0u;
    int c = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) c += v[i] == m ? 1 : 0;
    count += (int)__reduce_add_sync(0xffffffffu, (unsigned)c);
    if (count >= k) return m;
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = v[i] == m ? 0u : v[i];
  }
  return 0u;
}

constexpr int kSelWarps = 8;
constexpr int kSelThreads = kSelWarps * 32;
constexpr int kProducerWarp = kSelWarps;
constexpr int kMergeWarp = kSelWarps + 1;
constexpr int kStreamThreads = kSelThreads + 64;   // + the producer and merge warps
constexpr int kStreamStages = 6;
constexpr int kStreamChunkVec = 1024;              // 16 KB of logits per chunk
constexpr int kStreamMinVec = 2048;                // at least 32 KB per CTA
constexpr int kPartSlot = 16;                      // keys per part slot (the largest k)
constexpr int kCachedOffsets = 257;                // trees whose node offsets sit in shared memory
constexpr int kRaiseAfter = 8;                     // new candidate lanes before a warp's threshold is raised

struct StreamArgs {
  const __nv_bfloat16* logits;      // [rows][nvec_row * 8], back to back, 16-byte aligned
  int64_t rows;
  int nvec_row;
  int k;
  int64_t total_vec, per_cta;       // rows * nvec_row; vectors per CTA (the last may have fewer)
  int32_t* out_idx;                 // [rows][k]
  float* out_val;                   // [rows][k]
  unsigned int* row_counters;       // [rows], zero before the launch
  unsigned long long* part_keys;    // [(rows + gridDim.x) * kPartSlot]: slot of row r in CTA c = r + c
  int32_t* dev_status;
};

template <int KM>
__global__ void __launch_bounds__(kStreamThreads, 2) topk_stream_kernel(const StreamArgs a, const VerifyArgs va) {
  extern __shared__ __align__(128) uint4 ring[];
  __shared__ __align__(8) uint64_t bars_s[2 * kStreamStages + 4];
  __shared__ uint64_t warp_keys[2][kSelWarps][KM];
  __shared__ uint32_t lane_max_s[2][kSelThreads];   // a row part's first-chunk lane maxima
  __shared__ int offsets_s[kCachedOffsets];
  __shared__ int abort_s;
  __shared__ vt::VerifyScratch vsc;
  __shared__ vt::TreeVerdict verdict;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t full0 = smem_u32(&bars_s[0]), empty0 = smem_u32(&bars_s[kStreamStages]);
  auto full_bar = [&](int st) { return full0 + 8u * (uint32_t)st; };
  auto empty_bar = [&](int st) { return empty0 + 8u * (uint32_t)st; };
  // the selection warps' keys of a part: buffer pb full (8 warps) / empty (the merge warp)
  auto kfull_bar = [&](int pb) { return smem_u32(&bars_s[2 * kStreamStages + pb]); };
  auto kempty_bar = [&](int pb) { return smem_u32(&bars_s[2 * kStreamStages + 2 + pb]); };
  if (threadIdx.x == 0) {
    for (int st = 0; st < kStreamStages; ++st) {
      mbar_init(full_bar(st), 1);
      mbar_init(empty_bar(st), kSelWarps);
    }
    for (int pb = 0; pb < 2; ++pb) {
      mbar_init(kfull_bar(pb), kSelWarps);
      mbar_init(kempty_bar(pb), 1);
    }
    abort_s = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) grid_launch_dependents();   // the next grid may be placed now; it waits for this one
  const int64_t vbeg = (int64_t)blockIdx.x * a.per_cta;
  const int64_t vend = vbeg + a.per_cta < a.total_vec ? vbeg + a.per_cta : a.total_vec;
  const int nvr = a.nvec_row;
  // the chunk at vector position pos: its row, offset in the row and length (never across a row)
  auto chunk_at = [&](int64_t pos, int64_t& row, int& off, int& n) {
    row = pos / nvr;
    off = (int)(pos - row * nvr);
    int64_t m = vend - pos;
    if (m > kStreamChunkVec) m = kStreamChunkVec;
    if (m > nvr - off) m = nvr - off;
    n = (int)m;
  };
  grid_dependency_wait();   // the logits, the trees and the outputs belong to the stream's previous work

  if (warp == kProducerWarp) {
    // ================================================================ producer (one lane)
    if (lane == 0) {
      bool ok = true;
      int j = 0;
      for (int64_t pos = vbeg; pos < vend; ++j) {
        int64_t row;
        int off, n;
        chunk_at(pos, row, off, n);
        const int st = j % kStreamStages;
        ok = mbar_wait(empty_bar(st), (uint32_t)(((j / kStreamStages) & 1) ^ 1), &abort_s, a.dev_status);
        if (!ok) break;
        // (the selection warps only read the stage: their arrivals on its empty barrier order
        // those reads before this copy; no proxy fence, which would also wait for the copies
        // still in flight)
        mbar_arrive_expect_tx(full_bar(st), (uint32_t)n * 16u);
        bulk_load(smem_u32(ring) + (uint32_t)st * (kStreamChunkVec * 16u),
                  reinterpret_cast<const uint4*>(a.logits) + pos, (uint32_t)n * 16u, full_bar(st));
        pos += n;
      }
      if (!ok) {
        // drain the copies already issued (bounded) before the CTA can exit
        for (int back = 1; back <= kStreamStages && j - back >= 0; ++back) {
          const int j2 = j - back;
          mbar_drain(full_bar(j2 % kStreamStages), (uint32_t)((j2 / kStreamStages) & 1), 100000000ull);
        }
      }
    }
    return;
  }

  const int k = a.k;
  if (warp == kMergeWarp) {
    // ================================================================ merge warp
    const bool cached = va.batch + 1 <= kCachedOffsets;
    if (cached)
      for (int i = lane; i <= va.batch; i += 32) offsets_s[i] = va.node_offsets[i];
    if (blockIdx.x == 0) flag_bad_trees_warp(va);
    __syncwarp();
    auto tree_of = [&](int64_t r) {
      int lo = 0, hi = va.batch;
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if ((cached ? offsets_s[mid] : va.node_offsets[mid]) <= r) lo = mid; else hi = mid;
      }
      return lo;
    };
    int part = 0;
    for (int64_t pos = vbeg; pos < vend;) {
      int64_t row;
      int off, n;
      chunk_at(pos, row, off, n);
      pos += n;
      if (!(pos == vend || off + n == nvr)) continue;   // not the end of a row part
      const int pb = part & 1;
      if (!mbar_wait_warp(kfull_bar(pb), (uint32_t)((part >> 1) & 1), &abort_s, a.dev_status)) break;
      // the CTA's top-k of the part: lane w (< 8) owns warp w's sorted keys
      int cur = 0;
      uint64_t pk = 0ull;
      for (int s = 0; s < k; ++s) {
        const uint64_t mine = (lane < kSelWarps && cur < k) ? warp_keys[pb][lane][cur] : 0ull;
        const uint64_t best = warp_max_u64(mine);
        if (lane < kSelWarps && mine == best && best != 0ull) ++cur;
        if (lane == s) pk = best;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(kempty_bar(pb));   // the buffer is read (the keys are in registers)
      ++part;
      const int64_t c_first = row * nvr / a.per_cta;
      int64_t c_last = ((row + 1) * nvr - 1) / a.per_cta;
      if (c_last > (int64_t)gridDim.x - 1) c_last = gridDim.x - 1;
      const int nparts = (int)(c_last - c_first + 1);
      int last_part = 1;   // a row that lies in this CTA alone has the part's top-k
      if (nparts > 1) {
        if (lane < k) a.part_keys[(size_t)(row + blockIdx.x) * kPartSlot + lane] = pk;
        __syncwarp();   // every lane's key of this part is written before lane 0 counts the part
        if (lane == 0) last_part = (int)atom_add_acq_rel_gpu(a.row_counters + row, 1u) + 1 == nparts;
        last_part = __shfl_sync(0xffffffffu, last_part, 0);
      }
      if (!last_part) continue;
      if (nparts > 1) {
        // the row's top-k from its parts' slots (each written before its part was counted)
        ThreadList<KM> ml;
        ml.init();
        __syncwarp();   // lane 0's acquire precedes every lane's reads of the slots
        for (int q = lane; q < nparts * k; q += 32) {
          const uint64_t key = __ldcg(a.part_keys + (size_t)(row + c_first + q / k) * kPartSlot + q % k);
          if (key != 0ull) ml.push_key(key);
        }
        pk = 0ull;
        for (int s = 0; s < k; ++s) {
          const uint64_t mine = ml.head();
          const uint64_t best = warp_max_u64(mine);
          if (mine == best && best != 0ull) ml.pop();
          if (lane == s) pk = best;
        }
      }
      if (lane < k) {
        a.out_idx[row * k + lane] = (int32_t)(~(uint32_t)(pk & 0xFFFFFFFFull));
        a.out_val[row * k + lane] = from_ordered((uint32_t)(pk >> 32));
      }
      // count the row for its tree; the tree's last row verifies it (its parents and tokens
      // are loaded while the count is in flight)
      const int b = tree_of(row);
      vt::TreeInputs tin;
      vt::load_tree_warp(va.node_offsets, va.parents, va.tokens, va.n_total, va.max_nodes, b, tin);
      int vb = -1;
      __syncwarp();   // every lane's entries of this row are written before lane 0 counts the row
      if (lane == 0) {
        // release: this row's top-k before its count; acquire: the other rows' top-k (each
        // written before its own count) before this warp reads them
        if ((int)atom_add_acq_rel_gpu(va.counters + b, 1u) + 1 == tin.T) vb = b;
      }
      vb = __shfl_sync(0xffffffffu, vb, 0);
      if (vb >= 0) {
        __syncwarp();   // lane 0's acquire precedes every lane's reads of the tree's rows
        verify_and_write_warp(va, vb, tin, a.out_idx, k, vsc, verdict);
      }
    }
    return;
  }

  // ================================================================ selection warps
  const int tid = threadIdx.x;
  ThreadList<KM> list;
  list.init();
  float thr = -INFINITY;
  int fresh = 0;   // lanes that pushed since T_w was last set (summed over chunks)
  int part = 0;
  // After a failed wait (timeout, or another warp's) a warp keeps walking the schedule without
  // data, so that every selection warp meets every part's barrier; the merge warp sees the
  // abort flag within its own bounded waits.
  bool ok = true;
  int j = 0;
  for (int64_t pos = vbeg; pos < vend; ++j) {
    int64_t row;
    int off, n;
    chunk_at(pos, row, off, n);
    const bool first = pos == vbeg || off == 0;
    const bool last = pos + n == vend || off + n == nvr;
    const int st = j % kStreamStages;
    if (ok) ok = mbar_wait_warp(full_bar(st), (uint32_t)((j / kStreamStages) & 1), &abort_s, a.dev_status);
    const uint4* chunk = ring + (size_t)st * kStreamChunkVec;
    uint32_t hv[4];   // per vector: the packed maximum of its four pairs
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int vi = tid + u * kSelThreads;
      const uint4 x =
          ok && vi < n ? chunk[vi] : make_uint4(kBf16x2NegInf, kBf16x2NegInf, kBf16x2NegInf, kBf16x2NegInf);
      hv[u] = bf16x2_max(bf16x2_max(x.x, x.y), bf16x2_max(x.z, x.w));
    }
    if (first) {
      // a new row part: T from this chunk, the k-th largest of the CTA's 256 lane maxima
      // (lanes without a vector here hold none): k elements of the part are >= T, so no
      // element below T is among the CTA's top-k of the part (a warp's own T_w is never above)
      list.init();
      fresh = 0;
      const uint32_t h = bf16x2_max(bf16x2_max(hv[0], hv[1]), bf16x2_max(hv[2], hv[3]));
      lane_max_s[part & 1][tid] = ok && tid < n ? ordered_bits(fmaxf(bf16_lo(h), bf16_hi(h))) : 0u;
      asm volatile("bar.sync 1, %0;" ::"n"(kSelThreads) : "memory");   // the 8 selection warps only
      uint32_t v[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = lane_max_s[part & 1][lane * 8 + i];
      const uint32_t kth = kth_largest_ord8(v, k);
      thr = kth != 0u ? from_ordered(kth) : -INFINITY;
    }
    uint32_t hits = 0u;
#pragma unroll
    for (int u = 0; u < 4; ++u)
      hits |= (ok && tid + u * kSelThreads < n && fmaxf(bf16_lo(hv[u]), bf16_hi(hv[u])) >= thr ? 1u : 0u) << u;
    // the few vectors that reach the threshold: read again and pushed, in index order
    fresh += __popc(__ballot_sync(0xffffffffu, hits != 0u));
#pragma unroll 1
    for (; hits != 0u; hits &= hits - 1u) {
      const int vi = tid + (__ffs(hits) - 1) * kSelThreads;
      const uint4 x = chunk[vi];
      const uint32_t gi = (uint32_t)(off + vi) * 8u;
      const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float f0 = bf16_lo(w[q]), f1 = bf16_hi(w[q]);
        if (f0 >= thr) list.push(ordered_bits(f0), gi + 2 * q);
        if (f1 >= thr) list.push(ordered_bits(f1), gi + 2 * q + 1);
      }
    }
    __syncwarp();
    if (ok && lane == 0) mbar_arrive(empty_bar(st));   // this warp is done with the stage
    if (!last && fresh >= kRaiseAfter) {
      // raise the threshold once enough new candidates came in: if k lanes hold candidates >= x, no
      // element below x is among the warp's top-k; x = the k-th largest of the lanes' largest
      fresh = 0;
      const uint32_t kth = kth_largest_ord(list.ord[0], k);
      if (kth != 0u) thr = fmaxf(thr, from_ordered(kth));
    }
    pos += n;
    if (!last) continue;
    // ---- the end of a row part: the warp's top-k into buffer part % 2 (free once the merge
    // warp has read the part two before this one)
    const int pb = part & 1;
    if (ok) ok = mbar_wait_warp(kempty_bar(pb), (uint32_t)(((part >> 1) & 1) ^ 1), &abort_s, a.dev_status);
    if (ok) {
      for (int s = 0; s < k; ++s) {
        const uint64_t mine = list.head();
        const uint64_t best = warp_max_u64(mine);
        if (mine == best) list.pop();
        if (lane == 0) warp_keys[pb][warp][s] = best;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(kfull_bar(pb));
    }
    ++part;
  }
}

template <int KM>
cudaError_t launch_stream_km(const StreamArgs& a, int grid, const VerifyArgs& va, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid, 1, 1);
  cfg.blockDim = dim3(kStreamThreads, 1, 1);
  cfg.dynamicSmemBytes = (size_t)kStreamStages * kStreamChunkVec * 16;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // set-up overlaps the previous kernel
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaFuncSetAttribute(topk_stream_kernel<KM>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)cfg.dynamicSmemBytes);
  if (e != cudaSuccess) return e;
  return cudaLaunchKernelEx(&cfg, topk_stream_kernel<KM>, a, va);
}

template <int KM, typename T, bool kFast, bool kVerify>
cudaError_t launch_km(const T* logits, int64_t rows, int vocab, int64_t row_stride, int k, int32_t* out_idx,
                      float* out_val, int cluster, int32_t* dev_status, const VerifyArgs& va, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  const int64_t gy = rows < 65535 ? rows : 65535;
  cfg.gridDim = dim3((unsigned)cluster, (unsigned)gy, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // set-up overlaps the previous kernel
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if constexpr (kFast) {
    const int nvec = vocab / 8 + 1;
    const int per = (nvec + cluster - 1) / cluster;
    cfg.dynamicSmemBytes = (size_t)per * 16;
    cudaError_t e = cudaFuncSetAttribute(topk_bf16_kernel<KM, kVerify>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSliceVec * 16);
    if (e != cudaSuccess) return e;
    return cudaLaunchKernelEx(&cfg, topk_bf16_kernel<KM, kVerify>, logits, rows, vocab, row_stride, k, out_idx,
                              out_val, dev_status, va);
  } else {
    cfg.dynamicSmemBytes = 0;
    return cudaLaunchKernelEx(&cfg, topk_cluster_kernel<KM, T>, logits, rows, vocab, row_stride, k, out_idx,
                              out_val);
  }
}

template <typename T, bool kFast, bool kVerify>
cudaError_t launch_t(const T* logits, int64_t rows, int vocab, int64_t row_stride, int k, int32_t* out_idx,
                     float* out_val, int32_t* dev_status, const VerifyArgs& va, cudaStream_t stream) {
  int cluster;
  if (kFast) {
    const int nvec = vocab / 8 + 1;
    cluster = (nvec + kSliceVec - 1) / kSliceVec;   // slices of at most 64 KB
  } else {
    const int per_cta = (int)(16384 / sizeof(T)) * 2;   // ~32 KB of logits per CTA
    cluster = (vocab + per_cta - 1) / per_cta;
  }
  cluster = cluster < 1 ? 1 : (cluster > kMaxCluster ? kMaxCluster : cluster);
#define PTD_TOPK_LAUNCH(KMV) \
  return launch_km<KMV, T, kFast, kVerify>(logits, rows, vocab, row_stride, k, out_idx, out_val, cluster, dev_status, \
                                           va, stream)
  if (k <= 1) PTD_TOPK_LAUNCH(1);
  if (k <= 2) PTD_TOPK_LAUNCH(2);
  if (k <= 4) PTD_TOPK_LAUNCH(4);
  if (k <= 8) PTD_TOPK_LAUNCH(8);
  PTD_TOPK_LAUNCH(16);
#undef PTD_TOPK_LAUNCH
}

}  // namespace topk

bool topk_stream_ok(const void* logits, int vocab) {
  return vocab >= 8 && vocab % 8 == 0 && (reinterpret_cast<uintptr_t>(logits) & 15u) == 0;
}

size_t topk_stream_slot_bytes(int64_t rows, int sms) {
  return (size_t)(rows + 2 * (int64_t)sms) * topk::kPartSlot * sizeof(unsigned long long);
}

cudaError_t launch_topk_stream(const void* logits, int64_t rows, int vocab, int k, int32_t* out_idx, float* out_val,
                               int32_t* dev_status, const VerifyArgs& va, unsigned int* row_counters,
                               unsigned long long* part_keys, int sms, cudaStream_t stream) {
  if (!topk_stream_ok(logits, vocab) || rows < 1 || k < 1 || k > topk::kPartSlot || sms < 1)
    return cudaErrorInvalidValue;
  topk::StreamArgs a = {};
  a.logits = static_cast<const __nv_bfloat16*>(logits);
  a.rows = rows;
  a.nvec_row = vocab / 8;
  a.k = k;
  a.total_vec = rows * (int64_t)a.nvec_row;
  // two CTAs per SM, each with at least kStreamMinVec vectors; equal ranges
  int64_t grid = (a.total_vec + topk::kStreamMinVec - 1) / topk::kStreamMinVec;
  if (grid > 2 * (int64_t)sms) grid = 2 * (int64_t)sms;
  if (grid < 1) grid = 1;
  a.per_cta = (a.total_vec + grid - 1) / grid;
  grid = (a.total_vec + a.per_cta - 1) / a.per_cta;
  a.out_idx = out_idx;
  a.out_val = out_val;
  a.row_counters = row_counters;
  a.part_keys = part_keys;
  a.dev_status = dev_status;
  if (k <= 1) return topk::launch_stream_km<1>(a, (int)grid, va, stream);
  if (k <= 2) return topk::launch_stream_km<2>(a, (int)grid, va, stream);
  if (k <= 4) return topk::launch_stream_km<4>(a, (int)grid, va, stream);
  if (k <= 8) return topk::launch_stream_km<8>(a, (int)grid, va, stream);
  return topk::launch_stream_km<16>(a, (int)grid, va, stream);
}

int topk_cluster_size(int vocab) {
  const int nvec = vocab / 8 + 1;
  int cluster = (nvec + topk::kSliceVec - 1) / topk::kSliceVec;
  return cluster < 1 ? 1 : (cluster > topk::kMaxCluster ? topk::kMaxCluster : cluster);
}

bool topk_can_verify(bool bf16, int vocab) {
  return bf16 && (int64_t)vocab / 8 + 1 <= (int64_t)topk::kMaxCluster * topk::kSliceVec;
}

cudaError_t launch_topk(const void* logits, bool bf16, int64_t rows, int vocab, int64_t row_stride, int k,
                        int32_t* out_idx, float* out_val, int32_t* dev_status, const VerifyArgs* va,
                        cudaStream_t stream) {
  const VerifyArgs none = {};
  if (bf16) {
    // the shared-memory path covers rows up to kMaxCluster slices of kSliceVec vectors
    if (topk_can_verify(true, vocab)) {
      if (va != nullptr)
        return topk::launch_t<__nv_bfloat16, true, true>(static_cast<const __nv_bfloat16*>(logits), rows, vocab,
                                                         row_stride, k, out_idx, out_val, dev_status, *va, stream);
      return topk::launch_t<__nv_bfloat16, true, false>(static_cast<const __nv_bfloat16*>(logits), rows, vocab,
                                                        row_stride, k, out_idx, out_val, dev_status, none, stream);
    }
    if (va != nullptr) return cudaErrorInvalidValue;
    return topk::launch_t<__nv_bfloat16, false, false>(static_cast<const __nv_bfloat16*>(logits), rows, vocab,
                                                       row_stride, k, out_idx, out_val, dev_status, none, stream);
  }
  if (va != nullptr) return cudaErrorInvalidValue;
  return topk::launch_t<float, false, false>(static_cast<const float*>(logits), rows, vocab, row_stride, k, out_idx,
                                             out_val, dev_status, none, stream);
}

}  // namespace ptd
