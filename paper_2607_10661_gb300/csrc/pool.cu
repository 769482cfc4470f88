// Candidate pool on the GPU (Sec. 3.1 "Draft Extraction via Merging": the merge M of trees
// with the same root value; Sec. 3.2 and Alg. 1 steps 1 and 4: retrieval of C_X and the
// pool update).
//
// The pool is a hash table of trie nodes in caller memory.  A node is the slot holding its
// key (parent slot + 1) << 32 | token (parent slot -1 for an entry's root); its slot index
// is its identity.  Next to the keys: each node's order key, the (step, v, u) of the first
// merge pair that inserted it (the sequential merge's insertion order), and the slots of
// its earliest kPoolKids children, sorted by order key (retrieval never takes more).
//
// Merge of a draft forest (one CTA, thread u = node u): every node's subtree joins the
// entry of its token, i.e. every pair (v, u) with v an ancestor of u (or u) inserts the
// token path v .. u.  Level L handles the pairs whose u lies L below v: thread u inserts
// token(u) under the slot its parent's pair got at level L - 1 (level 0: the entry root of
// token(u)), so one level is one hash operation per node.  A new node's order key is the
// minimum (step, v, u) over the pairs that reach it; the children created at a level are
// ranked among their siblings by that key and appended to the parent's array, which stays
// sorted because nodes from earlier steps (and earlier levels never share a parent with
// this one) have smaller keys.  A merge that could push the occupied slots past max_load
// is refused as a whole (a deterministic rule; the status word says so).
//
// Retrieval (one CTA): the entry of the root token, then breadth first, each frontier node
// taking its first `width` children from its sorted array; a block scan places them.
#include <cuda_runtime.h>

#include <cstdint>

#include "pool.cuh"
#include "ptd_device.cuh"

namespace ptd {
namespace pl {

constexpr int kThreads = 128;   // = PTD_MAX_TREE_NODES
constexpr int kWarps = kThreads / 32;
constexpr uint64_t kEmpty = ~0ull;
constexpr int kHeaderBytes = 256;

struct View {
  int32_t* used;        // occupied slots
  uint64_t* keys;       // [cap]
  uint64_t* order;      // [cap]
  int32_t* nkids;       // [cap]
  int32_t* kids;        // [cap][kPoolKids]
};

__host__ __device__ inline View view(void* pool, int cap) {
  char* p = static_cast<char*>(pool);
  View v;
  v.used = reinterpret_cast<int32_t*>(p);
  p += kHeaderBytes;
  v.keys = reinterpret_cast<uint64_t*>(p);
  p += (size_t)cap * 8;
  v.order = reinterpret_cast<uint64_t*>(p);
  p += (size_t)cap * 8;
  v.nkids = reinterpret_cast<int32_t*>(p);
  p += (size_t)cap * 4;
  v.kids = reinterpret_cast<int32_t*>(p);
  return v;
}

__device__ __forceinline__ uint64_t node_key(int parent_slot, int token) {
  return ((uint64_t)(uint32_t)(parent_slot + 1) << 32) | (uint32_t)token;
}

// 64-bit finaliser of SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom number
// generators", OOPSLA 2014), used as the hash.
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
  z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
  return z ^ (z >> 31);
}

// Slot of key (linear probing), inserting it when absent: returns the slot and whether
// this call created it, or -1 when every slot is taken by other keys.
__device__ int find_or_insert(const View& pv, int cap, uint64_t key, bool* created) {
  const uint32_t mask = (uint32_t)cap - 1u;
  uint32_t s = (uint32_t)mix64(key) & mask;
  *created = false;
  for (int probe = 0; probe < cap; ++probe, s = (s + 1u) & mask) {
    const uint64_t k = *reinterpret_cast<volatile uint64_t*>(&pv.keys[s]);
    if (k == key) return (int)s;
    if (k != kEmpty) continue;
    const unsigned long long old = atomicCAS(reinterpret_cast<unsigned long long*>(&pv.keys[s]),
                                             (unsigned long long)kEmpty, (unsigned long long)key);
    if (old == kEmpty) {
      *created = true;
      return (int)s;
    }
    if (old == key) return (int)s;
  }
  return -1;
}

__device__ int find(const View& pv, int cap, uint64_t key) {
  const uint32_t mask = (uint32_t)cap - 1u;
  uint32_t s = (uint32_t)mix64(key) & mask;
  for (int probe = 0; probe < cap; ++probe, s = (s + 1u) & mask) {
    const uint64_t k = pv.keys[s];
    if (k == key) return (int)s;
    if (k == kEmpty) return -1;
  }
  return -1;
}

__device__ __forceinline__ int block_exclusive_scan(int x, int* warp_s, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  __syncthreads();
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
    pool_merge_kernel(void* pool, int cap, int max_load, int step, const int32_t* __restrict__ count,
                      const int32_t* __restrict__ parents, const int32_t* __restrict__ tokens,
                      int32_t* __restrict__ dev_status) {
  __shared__ int par_s[kThreads], slot_s[2][kThreads];
  __shared__ int new_parent_s[kThreads], new_slot_s[kThreads];
  __shared__ uint64_t new_key_s[kThreads];
  __shared__ int warp_s[kWarps];
  __shared__ int used_s, fail_s;
  const View pv = view(pool, cap);
  const int u = threadIdx.x;
  const int T = *count;
  bool bad = T < 0 || T > kThreads;
  int par = -1, tok = 0;
  if (!bad && u < T) {
    par = parents[u];
    tok = tokens[u];
    bad = !(par == -1 || (par >= 0 && par < u));
  }
  if (u == 0) {
    used_s = *pv.used;   // read once, before any insertion
    fail_s = 0;
  }
  if (__syncthreads_or(bad)) {
    if (u == 0) atomicMax(dev_status, (int)PTD_ERR_INVALID_TREE);
    return;
  }
  par_s[u] = u < T ? par : -1;
  __syncthreads();
  // depth of every node: a walk up the chain (at most 128 shared-memory reads)
  int depth = 0;
  if (u < T)
    for (int a = u; a != -1; a = par_s[a]) ++depth;
  int pairs;
  block_exclusive_scan(depth, warp_s, &pairs);   // pairs (v, u), an upper bound on new nodes
  int max_depth = depth;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) max_depth = max(max_depth, __shfl_xor_sync(0xffffffffu, max_depth, o));
  __syncthreads();
  if ((u & 31) == 0) warp_s[u >> 5] = max_depth;
  __syncthreads();
#pragma unroll
  for (int w = 0; w < kWarps; ++w) max_depth = max(max_depth, warp_s[w]);
  // refuse, as a whole, a merge that could take the table past max_load (uniform decision)
  if (used_s + pairs > max_load) {
    if (u == 0) atomicMax(dev_status, (int)PTD_ERR_POOL_FULL);
    return;
  }
  int anc = u;   // the v of this level's pair (v, u): the ancestor L levels above u
#pragma unroll 1
  for (int L = 0; L < max_depth; ++L) {
    const int wr = L & 1, rd = wr ^ 1;
    // ---- A: insert token(u) under the slot of the pair (v, parent(u)) of level L - 1
    new_parent_s[u] = -2;
    int rank = 0, n_same = 0, base = 0, ps = -1;
    if (u < T && depth > L) {
      const int pslot = L == 0 ? -1 : slot_s[rd][par_s[u]];
      bool created = false;
      const int slot = pslot < -1 ? -1 : find_or_insert(pv, cap, node_key(pslot, tok), &created);
      slot_s[wr][u] = slot < 0 ? -2 : slot;
      if (slot < 0) {
        fail_s = 1;
      } else {
        const uint64_t key = ((uint64_t)(uint32_t)step << 32) | ((uint64_t)anc << 16) | (uint64_t)u;
        atomicMin(reinterpret_cast<unsigned long long*>(&pv.order[slot]), (unsigned long long)key);
        if (created) {
          atomicAdd(pv.used, 1);
          if (pslot >= 0) {            // an entry's root has no parent array to join
            new_parent_s[u] = pslot;
            new_slot_s[u] = slot;
          }
        }
      }
      anc = par_s[anc];
    }
    __syncthreads();   // every insertion and order key of this level is in place
    // ---- B: the final order keys of this level's new nodes
    if (new_parent_s[u] >= 0) new_key_s[u] = pv.order[new_slot_s[u]];
    __syncthreads();
    // ---- C: rank among the new siblings, placed after the parent's existing children
    if (new_parent_s[u] >= 0) {
      ps = new_parent_s[u];
      const uint64_t key = new_key_s[u];
      for (int j = 0; j < kThreads; ++j) {
        if (new_parent_s[j] != ps) continue;
        ++n_same;
        rank += new_key_s[j] < key ? 1 : 0;
      }
      base = pv.nkids[ps];
      if (base + rank < kPoolKids) pv.kids[(size_t)ps * kPoolKids + base + rank] = new_slot_s[u];
    }
    __syncthreads();
    // ---- D: the parent's child count
    if (ps >= 0 && rank == 0) pv.nkids[ps] = min(kPoolKids, base + n_same);
    __syncthreads();
  }
  if (u == 0 && fail_s) atomicMax(dev_status, (int)PTD_ERR_POOL_FULL);
}

__global__ void __launch_bounds__(kThreads)
    pool_retrieve_kernel(const void* pool, int cap, const int32_t* __restrict__ root_token, int width,
                         int max_depth, int max_nodes, int32_t* __restrict__ out_count,
                         int32_t* __restrict__ out_parents, int32_t* __restrict__ out_tokens) {
  __shared__ int slot_s[kThreads], par_s[kThreads], tok_s[kThreads];
  __shared__ int warp_s[kWarps];
  const View pv = view(const_cast<void*>(pool), cap);
  const int t = threadIdx.x;
  const int x = *root_token;
  if (t == 0) {
    slot_s[0] = find(pv, cap, node_key(-1, x));
    par_s[0] = -1;
    tok_s[0] = x;
  }
  __syncthreads();
  int n = 1, lvl_begin = 0, lvl_end = slot_s[0] >= 0 ? 1 : 0;
#pragma unroll 1
  for (int depth = 1; depth < max_depth && lvl_begin < lvl_end && n < max_nodes; ++depth) {
    const int f = lvl_begin + t;
    int c = 0, fs = -1;
    if (f < lvl_end) {
      fs = slot_s[f];
      c = min(width, pv.nkids[fs]);
    }
    int total;
    const int pos = n + block_exclusive_scan(c, warp_s, &total);
    for (int j = 0; j < c && pos + j < max_nodes; ++j) {
      const int s = pv.kids[(size_t)fs * kPoolKids + j];
      slot_s[pos + j] = s;
      par_s[pos + j] = f;
      tok_s[pos + j] = (int)(uint32_t)pv.keys[s];
    }
    __syncthreads();
    lvl_begin = lvl_end;
    lvl_end = min(max_nodes, n + total);
    n = lvl_end;
  }
  for (int i = t; i < max_nodes; i += kThreads) {
    out_parents[i] = i < n ? par_s[i] : -1;
    out_tokens[i] = i < n ? tok_s[i] : -1;
  }
  if (t == 0) *out_count = n;
}

}  // namespace pl

size_t pool_bytes(int capacity) {
  return (size_t)pl::kHeaderBytes + (size_t)capacity * (8 + 8 + 4 + 4 * kPoolKids);
}

cudaError_t pool_init(void* pool, int capacity, cudaStream_t stream) {
  const pl::View v = pl::view(pool, capacity);
  cudaError_t e = cudaMemsetAsync(pool, 0, pl::kHeaderBytes, stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(v.keys, 0xFF, (size_t)capacity * 16, stream);   // keys, order
  if (e == cudaSuccess) e = cudaMemsetAsync(v.nkids, 0, (size_t)capacity * 4, stream);
  return e;
}

cudaError_t launch_pool_merge(void* pool, int capacity, int max_load, int step, const int32_t* count,
                              const int32_t* parents, const int32_t* tokens, int32_t* dev_status, cudaStream_t stream) {
  pl::pool_merge_kernel<<<1, pl::kThreads, 0, stream>>>(pool, capacity, max_load, step, count, parents, tokens,
                                                        dev_status);
  return cudaGetLastError();
}

cudaError_t launch_pool_retrieve(const void* pool, int capacity, const int32_t* root_token, int width, int max_depth,
                                 int max_nodes, int32_t* out_count, int32_t* out_parents, int32_t* out_tokens,
                                 cudaStream_t stream) {
  pl::pool_retrieve_kernel<<<1, pl::kThreads, 0, stream>>>(pool, capacity, root_token, width, max_depth, max_nodes,
                                                           out_count, out_parents, out_tokens);
  return cudaGetLastError();
}

}  // namespace ptd
