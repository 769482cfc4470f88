// Draft tree update: one step of the draft forest's evolution (Sec. 3.1 "Progressive
// Expansion", "Width Control", "Stepping Mechanism (Depth Control)"; Alg. 1 step 3).
//
// One CTA of 128 threads per forest, thread i owning node i (forests hold at most 128
// nodes, in creation order, a seed's parent being -1).  Every global read (the count and
// each node's parent, token and draft row) is issued at once; the rest works in shared
// memory.
//   1. Expansion.  Node v tries its first `expand` draft tokens in rank order; a token
//      equal to the token of an existing child of v (found by the children themselves,
//      each comparing its token with its parent's draft row) or to an earlier rank's
//      token is that child, not a new node; otherwise it is added while v has fewer than
//      `width` children.  The additions, in (node, rank) order, take indices T, T+1, ...
//      from an exclusive scan of the per-node counts, and those at or past `capacity`
//      are dropped.
//   2. Depth, seed and the seed's child on the path of every node of the expanded
//      forest, by pointer jumping (7 rounds for 128 nodes).
//   3. Stepping: a seed subtree deeper than `max_depth` keeps only the subtree of the
//      seed's lowest-index child (the earliest added), which becomes a seed.
//   4. Stable compaction of the survivors by a block scan; parents renumbered, depths
//      (the nodes' position offsets |pi(v)|) less one in a stepped subtree.
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>

#include "draft_update.cuh"
#include "ptd_device.cuh"

namespace ptd {
namespace du {

constexpr int kThreads = 128;   // = PTD_MAX_TREE_NODES
constexpr int kWarps = kThreads / 32;

// Exclusive scan of x over the block; *total receives the sum.  Every thread calls it.
__device__ __forceinline__ int block_exclusive_scan(int x, int* warp_s, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  __syncthreads();   // warp_s may still be read by a previous scan
  if (lane == 31) warp_s[warp] = incl;
  __syncthreads();
  int base = 0, sum = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    base += w < warp ? warp_s[w] : 0;
    sum += warp_s[w];
  }
  *total = sum;
  return base + incl - x;
}

__global__ void __launch_bounds__(kThreads)
    draft_update_kernel(int in_stride, const int32_t* __restrict__ in_count, const int32_t* __restrict__ in_parents,
                        const int32_t* __restrict__ in_tokens, const int32_t* __restrict__ drafts, int draft_stride,
                        int expand, int width, int max_depth, int capacity, int32_t* __restrict__ out_count,
                        int32_t* __restrict__ out_parents, int32_t* __restrict__ out_tokens,
                        int32_t* __restrict__ out_depths, int32_t* __restrict__ old_to_new,
                        int32_t* __restrict__ dev_status) {
  __shared__ int par_s[kThreads], tok_s[kThreads];
  __shared__ int draft_s[kThreads][kMaxExpand];   // each input node's first `expand` draft tokens
  __shared__ int nkids_s[kThreads];               // existing children of each node
  __shared__ uint32_t have_s[kThreads];           // bit r: rank r's token is an existing child
  __shared__ int jmp_s[2][kThreads], dep_s[2][kThreads], sd_s[2][kThreads], top_s[2][kThreads];
  __shared__ int sub_depth_s[kThreads], first_kid_s[kThreads], newidx_s[kThreads];
  __shared__ int warp_s[kWarps];

  const int b = blockIdx.x, i = threadIdx.x;
  const size_t in0 = (size_t)b * in_stride, out0 = (size_t)b * capacity;

  // ---- every global read at once: the count, and node i's parent, token and draft row
  // (rows below in_stride exist whatever the count)
  int par = -1, tok = 0;
  int my_draft[kMaxExpand];
  if (i < in_stride && i < kThreads) {
    par = in_parents[in0 + i];
    tok = in_tokens[in0 + i];
    const int32_t* row = drafts + (in0 + i) * (size_t)draft_stride;
#pragma unroll
    for (int r = 0; r < kMaxExpand; ++r) my_draft[r] = r < expand ? row[r] : 0;
  }
  const int T = in_count[b];
  bool bad = T < 0 || T > in_stride || T > capacity;
  if (!bad && i < T) bad = !(par == -1 || (par >= 0 && par < i));
  nkids_s[i] = 0;
  have_s[i] = 0u;
  sub_depth_s[i] = 0;
  first_kid_s[i] = INT_MAX;
  if (i < T) {
    par_s[i] = par;
    tok_s[i] = tok;
#pragma unroll
    for (int r = 0; r < kMaxExpand; ++r) draft_s[i][r] = my_draft[r];
  }
  if (__syncthreads_or(bad)) {
    if (i == 0) {
      atomicMax(dev_status, (int)PTD_ERR_INVALID_TREE);
      out_count[b] = 0;
    }
    for (int j = i; j < capacity; j += kThreads) {
      out_parents[out0 + j] = -1;
      out_tokens[out0 + j] = -1;
      out_depths[out0 + j] = -1;
    }
    for (int j = i; j < in_stride; j += kThreads) old_to_new[in0 + j] = -1;
    return;
  }
  if (i < T && par >= 0) {
    atomicAdd(&nkids_s[par], 1);
    // does this node carry one of its parent's draft tokens?
    uint32_t bits = 0u;
    for (int r = 0; r < expand; ++r) bits |= (draft_s[par][r] == tok ? 1u : 0u) << r;
    if (bits) atomicOr(&have_s[par], bits);
  }
  __syncthreads();

  // ---- 1. expansion: which ranks node i adds (width control), then their indices
  uint32_t add = 0u;
  int n_add = 0;
  if (i < T) {
    int kids = nkids_s[i];
    const uint32_t have = have_s[i];
#pragma unroll
    for (int r = 0; r < kMaxExpand; ++r) {
      if (r < expand) {
        const int d = my_draft[r];
        bool dup = (have >> r) & 1u;   // already a child
#pragma unroll
        for (int r2 = 0; r2 < kMaxExpand; ++r2)
          if (r2 < r) dup |= my_draft[r2] == d;   // an earlier rank: that child, or dropped alike
        if (!dup && kids < width) {
          add |= 1u << r;
          ++kids;
          ++n_add;
        }
      }
    }
  }
  int total_add;
  const int first_new = T + block_exclusive_scan(n_add, warp_s, &total_add);
  const int Te = min(capacity, T + total_add);   // nodes of the expanded forest
  {
    int k = first_new;
#pragma unroll
    for (int r = 0; r < kMaxExpand; ++r) {
      if ((add >> r) & 1u) {
        if (k < capacity) {
          par_s[k] = i;
          tok_s[k] = my_draft[r];
        }
        ++k;
      }
    }
  }
  __syncthreads();

  // ---- 2. depth, seed and level-2 ancestor by pointer jumping (list ranking; parents
  // precede children, depths are at most 128, so 7 rounds suffice).  jmp: the first node
  // above i not yet counted (-1 past the seed); dep: nodes counted from i up to jmp;
  // sd: converges to the seed; top: converges to the ancestor whose parent is a seed (a
  // node of level 2 points at itself; a seed has -1).
  const int p = i < Te ? par_s[i] : -1;
  if (i < Te) {
    jmp_s[0][i] = p;
    dep_s[0][i] = 1;
    sd_s[0][i] = p == -1 ? i : p;
    top_s[0][i] = p == -1 ? -1 : (par_s[p] == -1 ? i : p);
  }
  __syncthreads();
  int cur = 0;
#pragma unroll 1
  for (int round = 0; round < 7; ++round) {
    if (i < Te) {
      const int j = jmp_s[cur][i];
      dep_s[cur ^ 1][i] = j < 0 ? dep_s[cur][i] : dep_s[cur][i] + dep_s[cur][j];
      jmp_s[cur ^ 1][i] = j < 0 ? -1 : jmp_s[cur][j];
      sd_s[cur ^ 1][i] = sd_s[cur][sd_s[cur][i]];
      const int t = top_s[cur][i];
      top_s[cur ^ 1][i] = t < 0 ? -1 : top_s[cur][t];
    }
    __syncthreads();
    cur ^= 1;
  }
  int seed = 0, depth = 0, top = -1;
  if (i < Te) {
    seed = sd_s[cur][i];
    depth = dep_s[cur][i];
    top = top_s[cur][i];
    atomicMax(&sub_depth_s[seed], depth);
    if (p >= 0 && par_s[p] == -1) atomicMin(&first_kid_s[p], i);
  }
  __syncthreads();

  // ---- 3. stepping, 4. stable compaction
  const bool stepped = i < Te && sub_depth_s[seed] > max_depth;
  const bool keep = i < Te && (!stepped || top == first_kid_s[seed]);
  int n_keep;
  const int ni = block_exclusive_scan(keep ? 1 : 0, warp_s, &n_keep);
  newidx_s[i] = keep ? ni : -1;
  __syncthreads();
  if (keep) {
    out_parents[out0 + ni] = (p == -1 || newidx_s[p] < 0) ? -1 : newidx_s[p];
    out_tokens[out0 + ni] = tok_s[i];
    out_depths[out0 + ni] = stepped ? depth - 1 : depth;
  }
  for (int j = n_keep + i; j < capacity; j += kThreads) {
    out_parents[out0 + j] = -1;
    out_tokens[out0 + j] = -1;
    out_depths[out0 + j] = -1;
  }
  for (int j = i; j < in_stride; j += kThreads) old_to_new[in0 + j] = j < T ? newidx_s[j] : -1;
  if (i == 0) out_count[b] = n_keep;
}

}  // namespace du

cudaError_t launch_draft_update(int batch, int in_stride, const int32_t* in_count, const int32_t* in_parents,
                                const int32_t* in_tokens, const int32_t* drafts, int draft_stride, int expand,
                                int width, int max_depth, int capacity, int32_t* out_count, int32_t* out_parents,
                                int32_t* out_tokens, int32_t* out_depths, int32_t* old_to_new, int32_t* dev_status,
                                cudaStream_t stream) {
  du::draft_update_kernel<<<batch, du::kThreads, 0, stream>>>(in_stride, in_count, in_parents, in_tokens, drafts,
                                                             draft_stride, expand, width, max_depth, capacity,
                                                             out_count, out_parents, out_tokens, out_depths,
                                                             old_to_new, dev_status);
  return cudaGetLastError();
}

}  // namespace ptd
