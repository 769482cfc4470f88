// Greedy verification of one tree on one warp (Sec. 3.2: eligible edges
// I = {(n, V_n) | V_n in sigma(n)}, the longest eligible root path, ties to the
// lexicographically smallest node sequence, X' = (n_0, ..., n_k, V_{n_k})).  Internal device
// code shared by the kernels that verify (not part of the C ABI).
//
// A tree is at most 128 nodes: each lane holds nodes lane + 32 q, q < 4.  Pointer jumping over
// the parent array (log2 T rounds, warp barriers only) gives every node its depth and whether
// every edge on its root path is eligible; the deepest such node fixes the accepted length;
// the nodes on root paths that reach it are marked, and the lexicographically smallest path
// is walked top down one level at a time (smallest marked child).
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

namespace ptd {
namespace vt {

constexpr int kMaxTreeNodes = 128;

struct TreeVerdict {
  int path[kMaxTreeNodes];
  int len;      // accepted length (0: the tree failed the checks)
  int bonus;
  int invalid;
};

// Shared-memory scratch of one verification.
struct VerifyScratch {
  int par[kMaxTreeNodes], jump[kMaxTreeNodes], reach[kMaxTreeNodes];
  int depth[kMaxTreeNodes], onpath[kMaxTreeNodes], tgt[kMaxTreeNodes];
};

// The tree inputs of one verification (warp-collective): first node, size, and the parent
// and token of nodes lane + 32 q.
struct TreeInputs {
  int node0, T, bad_shape;
  int par[4], tok[4];
};

static __device__ __forceinline__ void load_tree_warp(const int32_t* __restrict__ node_offsets,
                                               const int32_t* __restrict__ parents,
                                               const int32_t* __restrict__ tokens, int n_total, int max_nodes, int b,
                                               TreeInputs& in) {
  const int lane = threadIdx.x & 31;
  in.node0 = node_offsets[b];
  in.T = node_offsets[b + 1] - in.node0;
  in.bad_shape = in.T < 1 || in.T > max_nodes || in.T > kMaxTreeNodes || in.node0 < 0 || in.node0 + in.T > n_total;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int i = lane + 32 * q;
    in.par[q] = -1;
    in.tok[q] = 0;
    if (!in.bad_shape && i < in.T) {
      in.par[q] = parents[in.node0 + i];
      in.tok[q] = tokens[in.node0 + i];
    }
  }
}

static __device__ __noinline__ void verify_tree_warp(const TreeInputs& in, const int32_t* __restrict__ target,
                                                     int target_stride, VerifyScratch& sc, TreeVerdict* out) {
  int* const par_s = sc.par;
  int* const jump_s = sc.jump;
  int* const reach_s = sc.reach;
  int* const depth_s = sc.depth;
  int* const onpath_s = sc.onpath;
  int* const tgt_s = sc.tgt;
  const int lane = threadIdx.x & 31;
  const int node0 = in.node0, T = in.T;
  const bool bad_shape = in.bad_shape != 0;
  bool bad = false;
  int par[4], tok[4];
  // every node's own greedy token V_i (the parents and tokens are already in registers)
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int i = lane + 32 * q;
    par[q] = in.par[q];
    tok[q] = in.tok[q];
    if (!bad_shape && i < T) tgt_s[i] = target[(size_t)(node0 + i) * target_stride];
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int i = lane + 32 * q;
    if (!bad_shape && i < T) bad = bad || (i == 0 ? (par[q] != -1) : (par[q] < 0 || par[q] >= i));
  }
  if (__any_sync(0xffffffffu, bad) || bad_shape) {
    if (lane == 0) {
      out->len = 0;
      out->bonus = -1;
      out->invalid = 1;
    }
    return;
  }
  __syncwarp();   // tgt_s complete
  // eligible edge into node i: tokens[i] == V_{parent}
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int i = lane + 32 * q;
    if (i < T) {
      const int elig = i == 0 ? 1 : (tok[q] == tgt_s[par[q]]);
      par_s[i] = par[q];
      jump_s[i] = i == 0 ? 0 : par[q];
      reach_s[i] = elig;
      depth_s[i] = i == 0 ? 0 : 1;
      onpath_s[i] = 0;
    }
  }
  __syncwarp();
  // pointer jumping: after round r, jump[i] is the 2^r-th ancestor (clamped at the root)
  for (int r = 0; (1 << r) < T; ++r) {
    int j[4], rj[4], dj[4], jj[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = lane + 32 * q;
      j[q] = 0;
      if (i < T) {
        j[q] = jump_s[i];
        rj[q] = reach_s[j[q]];
        dj[q] = depth_s[j[q]];
        jj[q] = jump_s[j[q]];
      }
    }
    __syncwarp();
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = lane + 32 * q;
      if (i < T && j[q] != 0) {
        reach_s[i] &= rj[q];
        depth_s[i] += dj[q];
        jump_s[i] = jj[q];
      }
    }
    __syncwarp();
  }
  int dmax = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int i = lane + 32 * q;
    if (i < T && reach_s[i]) dmax = max(dmax, depth_s[i]);
  }
  const int D = __reduce_max_sync(0xffffffffu, dmax);
  // mark every node on a root path that reaches depth D through eligible edges
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int i = lane + 32 * q;
    if (i < T && reach_s[i] && depth_s[i] == D)
      for (int a = i; a >= 0 && !onpath_s[a]; a = par_s[a]) onpath_s[a] = 1;
  }
  __syncwarp();
  // the lexicographically smallest longest path, one level per step
  int cur = 0;
  if (lane == 0) out->path[0] = 0;
  for (int d = 1; d <= D; ++d) {
    int best = 0x7FFFFFFF;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = lane + 32 * q;
      if (i < T && par_s[i] == cur && onpath_s[i]) best = min(best, i);
    }
    cur = __reduce_min_sync(0xffffffffu, best);
    if (lane == 0) out->path[d] = cur;
  }
  if (lane == 0) {
    out->len = D + 1;
    out->bonus = tgt_s[cur];
    out->invalid = 0;
  }
}

}  // namespace vt
}  // namespace ptd
