// Greedy verification (Sec. 3.2: eligible edges I = {(n, V_n) | V_n in sigma(n)} and the
// accepted sequence X' = (n_0, ..., n_k, V_{n_k})) and KV-cache compaction (Alg. 1 step 6:
// X' joins the committed prefix).
//
// verify: one CTA of 128 threads per tree, thread i = node i.  Pointer jumping over the
// parent array gives every node its depth and whether all edges on its root path are
// eligible (token of the child == greedy token of the parent) in log2(T) rounds.  The
// longest reachable depth is a block max; the lexicographically smallest longest path is
// then walked top down one level per step (smallest child index that still leads to a
// node of that depth).
//
// compact: one CTA per (layer, tree, K or V); thread = 16-byte column chunk of a slot.
// Rows are copied in ascending path order in groups of 8 (all loads of a group before its
// stores).  This equals a copy from a snapshot because the path node at position j has
// index >= j (a node of depth j has j smaller-indexed ancestors in a topological order):
// destination slot C+j can only be the source of an EARLIER position j' < j, whose load
// happened in an earlier group or earlier in the same group.
#include <cuda_runtime.h>

#include <cstdint>

#include "ptd_device.cuh"
#include "verify_compact.cuh"
#include "verify_tree.cuh"

namespace ptd {
namespace vc {

constexpr int kVerifyThreads = 128;

__global__ void __launch_bounds__(kVerifyThreads)
    verify_greedy_kernel(const int32_t* __restrict__ node_offsets, const int32_t* __restrict__ parents,
                         const int32_t* __restrict__ tokens, const int32_t* __restrict__ target, int target_stride,
                         int n_total, int max_nodes, int32_t* __restrict__ accepted, int32_t* __restrict__ accept_len,
                         int32_t* __restrict__ bonus, int32_t* __restrict__ dev_status) {
  __shared__ int jump_s[kVerifyThreads];
  __shared__ int reach_s[kVerifyThreads];
  __shared__ int depth_s[kVerifyThreads];
  __shared__ int par_s[kVerifyThreads];
  __shared__ int onpath_s[kVerifyThreads];
  __shared__ int maxdepth_s;
  __shared__ int next_s;

  const int b = blockIdx.x;
  const int i = threadIdx.x;
  const int node0 = node_offsets[b];
  const int T = node_offsets[b + 1] - node0;
  int32_t* acc_row = accepted + (size_t)b * max_nodes;

  const bool bad_shape = T < 1 || T > max_nodes || T > kVerifyThreads || node0 < 0 || node0 + T > n_total;
  bool bad = false;
  int p = -1;
  if (!bad_shape && i < T) {
    p = parents[node0 + i];
    bad = i == 0 ? (p != -1) : (p < 0 || p >= i);
  }
  if (__syncthreads_or(bad) || bad_shape) {
    if (i == 0) {
      atomicMax(dev_status, (int)PTD_ERR_INVALID_TREE);
      accept_len[b] = 0;
      bonus[b] = -1;
    }
    for (int j = i; j < max_nodes; j += kVerifyThreads) acc_row[j] = -1;
    return;
  }

  // eligible edge into node i: tokens[i] == V_{parent}
  int elig = 1;
  if (i < T && i > 0) elig = tokens[node0 + i] == target[(size_t)(node0 + p) * target_stride];
  if (i < T) {
    par_s[i] = p;
    jump_s[i] = i == 0 ? 0 : p;
    reach_s[i] = elig;
    depth_s[i] = i == 0 ? 0 : 1;
    onpath_s[i] = 0;
  }
  if (i == 0) maxdepth_s = 0;
  __syncthreads();
  // pointer jumping: after round r, jump[i] is the 2^r-th ancestor (clamped at the root)
  for (int r = 0; (1 << r) < T; ++r) {
    int j = 0, rj = 1, dj = 0, jj = 0;
    if (i < T) {
      j = jump_s[i];
      rj = reach_s[j];
      dj = depth_s[j];
      jj = jump_s[j];
    }
    __syncthreads();
    if (i < T && j != 0) {
      reach_s[i] &= rj;
      depth_s[i] += dj;
      jump_s[i] = jj;
    }
    __syncthreads();
  }
  if (i < T && reach_s[i]) atomicMax(&maxdepth_s, depth_s[i]);
  __syncthreads();
  const int D = maxdepth_s;
  // mark every node on a root path that reaches depth D through eligible edges
  if (i < T && reach_s[i] && depth_s[i] == D)
    for (int a = i; a >= 0 && !onpath_s[a]; a = par_s[a]) onpath_s[a] = 1;
  __syncthreads();
  int cur = 0;
  if (i == 0) acc_row[0] = 0;
  for (int d = 1; d <= D; ++d) {
    if (i == 0) next_s = 0x7FFFFFFF;
    __syncthreads();
    if (i < T && par_s[i] == cur && onpath_s[i]) atomicMin(&next_s, i);
    __syncthreads();
    cur = next_s;
    if (i == 0) acc_row[d] = cur;
    __syncthreads();
  }
  for (int j = D + 1 + i; j < max_nodes; j += kVerifyThreads) acc_row[j] = -1;
  if (i == 0) {
    accept_len[b] = D + 1;
    bonus[b] = target[(size_t)(node0 + cur) * target_stride];
  }
}

constexpr int kCompactThreads = 256;
constexpr int kGroup = 8;

__global__ void __launch_bounds__(kCompactThreads)
    kv_compact_kernel(uint8_t* __restrict__ k_cache, uint8_t* __restrict__ v_cache, int row_bytes, int batch,
                      int page_size, int seq_capacity, int num_pages, const int32_t* __restrict__ block_table,
                      int max_pages, const int32_t* __restrict__ ctx_lens, const int32_t* __restrict__ accepted,
                      const int32_t* __restrict__ accept_len, int max_nodes, int32_t* __restrict__ new_ctx) {
  const int layer = blockIdx.x, b = blockIdx.y;
  uint8_t* base = blockIdx.z == 0 ? k_cache : v_cache;
  grid_dependency_wait();   // the path, its length and the cache belong to the stream's previous work
  const int32_t* path = accepted + (size_t)b * max_nodes;
  // the path's first entries are read together with its length and the context (one round
  // trip for the common short path)
  int head[kGroup];
#pragma unroll
  for (int q = 0; q < kGroup; ++q) head[q] = 1 + q < max_nodes ? path[1 + q] : 0;
  const int C = ctx_lens[b];
  int len = accept_len[b];
  if (len < 0) len = 0;
  if (len > max_nodes) len = max_nodes;
  if (layer == 0 && blockIdx.z == 0 && threadIdx.x == 0) new_ctx[b] = C + len;
  if (len <= 1 || C < 0) return;   // the root already sits at slot C
  const int cap = page_size > 0 ? max_pages * page_size : seq_capacity;

  auto row_ptr = [&](int slot) -> uint8_t* {
    size_t r;
    if (page_size > 0) {
      const int pg = block_table[(size_t)b * max_pages + slot / page_size];
      if (pg < 0 || pg >= num_pages) return nullptr;
      r = ((size_t)layer * num_pages + pg) * page_size + slot % page_size;
    } else {
      r = ((size_t)layer * batch + b) * seq_capacity + slot;
    }
    return base + r * (size_t)row_bytes;
  };

  const int nchunk = row_bytes / 16;
  for (int c = threadIdx.x; c < nchunk; c += kCompactThreads) {
    for (int j0 = 1; j0 < len; j0 += kGroup) {
      uint4 v[kGroup];
      bool ok[kGroup];
#pragma unroll
      for (int q = 0; q < kGroup; ++q) {
        const int j = j0 + q;
        v[q] = make_uint4(0, 0, 0, 0);
        ok[q] = false;
        if (j < len) {
          const int pj = j0 == 1 ? head[q] : path[j];
          const int src = C + pj;
          const uint8_t* sp = (pj > j && src < cap) ? row_ptr(src) : nullptr;
          if (sp) {
            v[q] = reinterpret_cast<const uint4*>(sp)[c];
            ok[q] = true;
          }
        }
      }
#pragma unroll
      for (int q = 0; q < kGroup; ++q) {
        uint8_t* dp = ok[q] ? row_ptr(C + j0 + q) : nullptr;
        if (dp) reinterpret_cast<uint4*>(dp)[c] = v[q];
      }
    }
  }
}

// ------------------------------------------------------------------ fused (whole step)
// Verification and compaction in one launch for the whole step: every CTA of the compaction
// grid (layer, tree, K or V) verifies its tree on warp 0 (a tree is at most 128 nodes: 4 per
// lane, pointer jumping with warp barriers only), so the path is in shared memory before
// the copy; CTA (0, b, K) writes the verification outputs.  The computation is that of
// verify_greedy_kernel followed by kv_compact_kernel.
__global__ void __launch_bounds__(kCompactThreads)
    verify_compact_kernel(const int32_t* __restrict__ node_offsets, const int32_t* __restrict__ parents,
                          const int32_t* __restrict__ tokens, const int32_t* __restrict__ target, int target_stride,
                          int n_total, int max_nodes, int32_t* __restrict__ accepted, int32_t* __restrict__ accept_len,
                          int32_t* __restrict__ bonus, int32_t* __restrict__ dev_status, uint8_t* __restrict__ k_cache,
                          uint8_t* __restrict__ v_cache, int row_bytes, int batch, int page_size, int seq_capacity,
                          int num_pages, const int32_t* __restrict__ block_table, int max_pages,
                          const int32_t* __restrict__ ctx_lens, int32_t* __restrict__ new_ctx) {
  __shared__ vt::VerifyScratch vsc;
  __shared__ vt::TreeVerdict verdict;
  const int layer = blockIdx.x, b = blockIdx.y;
  grid_dependency_wait();   // the targets, the trees and the cache belong to the stream's previous work
  vt::TreeInputs in;
  if (threadIdx.x < 32) vt::load_tree_warp(node_offsets, parents, tokens, n_total, max_nodes, b, in);
  const int C = ctx_lens[b];
  if (threadIdx.x < 32)
    vt::verify_tree_warp(in, target, target_stride, vsc, &verdict);
  __syncthreads();
  int len = verdict.len;
  if (len > max_nodes) len = max_nodes;
  if (layer == 0 && blockIdx.z == 0) {
    int32_t* acc_row = accepted + (size_t)b * max_nodes;
    for (int j = threadIdx.x; j < max_nodes; j += kCompactThreads) acc_row[j] = j < len ? verdict.path[j] : -1;
    if (threadIdx.x == 0) {
      accept_len[b] = len;
      bonus[b] = verdict.bonus;
      if (verdict.invalid) atomicMax(dev_status, (int)PTD_ERR_INVALID_TREE);
      new_ctx[b] = C + len;
    }
  }
  if (len <= 1 || C < 0) return;   // the root already sits at slot C
  uint8_t* base = blockIdx.z == 0 ? k_cache : v_cache;
  const int cap = page_size > 0 ? max_pages * page_size : seq_capacity;
  auto row_ptr = [&](int slot) -> uint8_t* {
    size_t r;
    if (page_size > 0) {
      const int pg = block_table[(size_t)b * max_pages + slot / page_size];
      if (pg < 0 || pg >= num_pages) return nullptr;
      r = ((size_t)layer * num_pages + pg) * page_size + slot % page_size;
    } else {
      r = ((size_t)layer * batch + b) * seq_capacity + slot;
    }
    return base + r * (size_t)row_bytes;
  };
  const int nchunk = row_bytes / 16;
  for (int c = threadIdx.x; c < nchunk; c += kCompactThreads) {
    for (int j0 = 1; j0 < len; j0 += kGroup) {
      uint4 v[kGroup];
      bool ok[kGroup];
#pragma unroll
      for (int q = 0; q < kGroup; ++q) {
        const int j = j0 + q;
        v[q] = make_uint4(0, 0, 0, 0);
        ok[q] = false;
        if (j < len) {
          const int pj = verdict.path[j];
          const int src = C + pj;
          const uint8_t* sp = (pj > j && src < cap) ? row_ptr(src) : nullptr;
          if (sp) {
            v[q] = reinterpret_cast<const uint4*>(sp)[c];
            ok[q] = true;
          }
        }
      }
#pragma unroll
      for (int q = 0; q < kGroup; ++q) {
        uint8_t* dp = ok[q] ? row_ptr(C + j0 + q) : nullptr;
        if (dp) reinterpret_cast<uint4*>(dp)[c] = v[q];
      }
    }
  }
}

}  // namespace vc

cudaError_t launch_verify(const int32_t* node_offsets, const int32_t* parents, const int32_t* tokens,
                          const int32_t* target, int target_stride, int batch, int n_total, int max_nodes,
                          int32_t* accepted, int32_t* accept_len, int32_t* bonus, int32_t* dev_status,
                          cudaStream_t stream) {
  vc::verify_greedy_kernel<<<batch, vc::kVerifyThreads, 0, stream>>>(node_offsets, parents, tokens, target,
                                                                     target_stride, n_total, max_nodes, accepted,
                                                                     accept_len, bonus, dev_status);
  return cudaGetLastError();
}

cudaError_t launch_verify_compact(const int32_t* node_offsets, const int32_t* parents, const int32_t* tokens,
                                  const int32_t* target, int target_stride, int n_total, int max_nodes,
                                  int32_t* accepted, int32_t* accept_len, int32_t* bonus, int32_t* dev_status, void* k,
                                  void* v, int row_bytes, int layers, int batch, int page_size, int seq_capacity,
                                  int num_pages, const int32_t* block_table, int max_pages, const int32_t* ctx_lens,
                                  int32_t* new_ctx, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(layers, batch, 2);
  cfg.blockDim = dim3(vc::kCompactThreads, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // set-up overlaps the previous kernel
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, vc::verify_compact_kernel, node_offsets, parents, tokens, target, target_stride,
                            n_total, max_nodes, accepted, accept_len, bonus, dev_status, static_cast<uint8_t*>(k),
                            static_cast<uint8_t*>(v), row_bytes, batch, page_size, seq_capacity, num_pages,
                            block_table, max_pages, ctx_lens, new_ctx);
}

cudaError_t launch_compact(void* k, void* v, int row_bytes, int layers, int batch, int page_size, int seq_capacity,
                           int num_pages, const int32_t* block_table, int max_pages, const int32_t* ctx_lens,
                           const int32_t* accepted, const int32_t* accept_len, int max_nodes, int32_t* new_ctx,
                           cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(layers, batch, 2);
  cfg.blockDim = dim3(vc::kCompactThreads, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // placed while the previous kernel drains
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, vc::kv_compact_kernel, static_cast<uint8_t*>(k), static_cast<uint8_t*>(v), row_bytes,
                            batch, page_size, seq_capacity, num_pages, block_table, max_pages, ctx_lens, accepted,
                            accept_len, max_nodes, new_ctx);
}

}  // namespace ptd
