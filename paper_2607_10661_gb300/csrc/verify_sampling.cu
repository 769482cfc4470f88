// Sampling verification (Sec. 3.2, "sampling decoding strategy"; Alg. 2, Candidate Tree
// Recursive Sampling; App. E proves the emitted token follows P).
//
// One thread-block cluster per tree; every CTA owns a contiguous slice of the vocabulary
// and every thread a contiguous chunk of it (16-byte vector loads where rows allow).
// Weights are w_t = 2^(x_t * c - M), c = log2(e) / temperature and M the row maximum of
// x * c, so P_v(t) = w_t / Z with Z = sum_t w_t.
//
// Visit of node v (the root first): each thread keeps a running maximum and a float-float
// sum of its chunk's weights relative to it; warps reduce them (maximum first, then the
// rescaled sums) and publish one pair each in shared memory; after a cluster barrier warp
// 0 of EVERY CTA reads all the cluster's pairs through distributed shared memory and
// reduces them in the same order, so every CTA holds the same M and Z with no second
// barrier.  The lanes weigh the children of v in parallel (a token repeated among the
// siblings weighs 0 after its first occurrence), then lane 0 tries them in node order:
// child n is accepted when u_accept[n] * S < w_n, S being the weight not yet rejected
// (S = Z at first; this is u < P_v(token) / S of Alg. 2 with both sides times Z); a
// rejected child's weight leaves S.  An accepted child becomes v.
//
// Bonus, when no child is accepted (or v is a leaf): the inverse CDF of the residual at
// u_bonus[b], i.e. the first token whose running residual weight exceeds u_bonus times
// the residual total.  Each thread's residual weight is its sum from the last visit
// rescaled to M, less the weights of the rejected tokens in its chunk; a scan within the
// warp, one over the CTA's warps and one over the cluster's CTAs give each chunk the
// interval [start, end) of running weight it covers, consecutive chunks sharing their
// end points bit for bit.  The chunk whose interval holds the target (the last chunk of
// positive weight also takes any target past the total) is walked by its warp, 32 tokens
// at a time with a scan, and the token is written with an atomicMax (a target on a shared
// end point, by rounding, may be claimed twice).  Where chunks are at most 32 logits and
// rows allow vector loads, each thread keeps its chunk of the visited row in registers
// and the bonus reads no logits again.
//
// Arithmetic: fp32 per element; sums in float-float pairs (an unevaluated hi + lo built
// from error-free fp32 sums, Knuth's TwoSum and Dekker's Fast2Sum, and an FMA-exact
// product), about 44 significant bits, so that removing a rejected dominant token from
// Z leaves an accurate residual.  The row maximum's own weight is 2^0 in both the sum and
// the test, so it cancels exactly.  This GPU's fp64 rate is a small fraction of its fp32
// rate, and the work here is latency bound.
#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cfloat>
#include <climits>
#include <cmath>
#include <cstdint>

#include "ptd_device.cuh"
#include "verify_sampling.cuh"

namespace cg = cooperative_groups;

namespace ptd {
namespace vs {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxNodes = 128;
constexpr int kMaxCluster = 8;
constexpr int kPerThread = 32;   // target chunk length: the cluster grows until chunks are this short
constexpr int kMaxWarpsCluster = kMaxCluster * kWarps;   // 128: four entries per lane in one warp
static_assert(kMaxWarpsCluster == 128, "the cluster scans assume four warp entries per lane");

// ---- float-float: hi + lo with |lo| <= ulp(hi) / 2.  The _rn intrinsics are never
// contracted into FMAs, which the error-free transformations rely on.
struct ff {
  float hi, lo;
};
__device__ __forceinline__ ff two_sum(float a, float b) {   // exact: a + b = s + e
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  return {s, __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb))};
}
__device__ __forceinline__ ff fast_two_sum(float a, float b) {   // exact when |a| >= |b|
  const float s = __fadd_rn(a, b);
  return {s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ ff ff_add(ff a, ff b) {
  const ff s = two_sum(a.hi, b.hi);
  const ff t = two_sum(a.lo, b.lo);
  const ff u = fast_two_sum(s.hi, __fadd_rn(s.lo, t.hi));
  return fast_two_sum(u.hi, __fadd_rn(u.lo, t.lo));
}
// a + b for a, b >= 0 (Dekker's add; same-sign operands need no second error term)
__device__ __forceinline__ ff ff_add_pos(ff a, ff b) {
  const ff s = two_sum(a.hi, b.hi);
  return fast_two_sum(s.hi, __fadd_rn(s.lo, __fadd_rn(a.lo, b.lo)));
}
__device__ __forceinline__ ff ff_add_f(ff a, float b) {
  const ff t = two_sum(a.hi, b);
  return fast_two_sum(t.hi, __fadd_rn(t.lo, a.lo));
}
__device__ __forceinline__ ff ff_mul(ff a, float b) {
  const float p = __fmul_rn(a.hi, b);
  const float e = fmaf(a.hi, b, -p);   // exact low part of a.hi * b
  return fast_two_sum(p, fmaf(a.lo, b, e));
}
__device__ __forceinline__ bool ff_less(ff a, ff b) { return a.hi < b.hi || (a.hi == b.hi && a.lo < b.lo); }
__device__ __forceinline__ ff shfl_xor(ff a, int o) {
  return {__shfl_xor_sync(0xffffffffu, a.hi, o), __shfl_xor_sync(0xffffffffu, a.lo, o)};
}
__device__ __forceinline__ ff shfl_up(ff a, int o) {
  return {__shfl_up_sync(0xffffffffu, a.hi, o), __shfl_up_sync(0xffffffffu, a.lo, o)};
}
__device__ __forceinline__ ff shfl_idx(ff a, int l) {
  return {__shfl_sync(0xffffffffu, a.hi, l), __shfl_sync(0xffffffffu, a.lo, l)};
}

template <typename T>
__device__ __forceinline__ float load_logit(const T* row, int t);
template <>
__device__ __forceinline__ float load_logit<__nv_bfloat16>(const __nv_bfloat16* row, int t) {
  return __uint_as_float((uint32_t)(*reinterpret_cast<const uint16_t*>(row + t)) << 16);
}
template <>
__device__ __forceinline__ float load_logit<float>(const float* row, int t) {
  return row[t];
}

// Eight consecutive logits from a 16-byte aligned address.
__device__ __forceinline__ void load8(const __nv_bfloat16* row, int t, float (&x)[8]) {
  const uint4 u = __ldg(reinterpret_cast<const uint4*>(row + t));
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    x[2 * i] = __uint_as_float(w[i] << 16);
    x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}
__device__ __forceinline__ void load8(const float* row, int t, float (&x)[8]) {
  const float4 a = __ldg(reinterpret_cast<const float4*>(row + t));
  const float4 b = __ldg(reinterpret_cast<const float4*>(row + t + 4));
  x[0] = a.x, x[1] = a.y, x[2] = a.z, x[3] = a.w, x[4] = b.x, x[5] = b.y, x[6] = b.z, x[7] = b.w;
}

// Calls f(t0, x) over [c0, c1) in order, x holding logits t0.. (8 at a time where the
// row allows vector loads, 32 loads in flight per thread; then one at a time).
template <typename LT, typename F>
__device__ __forceinline__ void for_chunk(const LT* row, int c0, int c1, bool vec_ok, F&& f) {
  int t = c0;
  if (vec_ok) {
    for (; t + 32 <= c1; t += 32) {
      float x[4][8];
#pragma unroll
      for (int q = 0; q < 4; ++q) load8(row, t + 8 * q, x[q]);
#pragma unroll
      for (int q = 0; q < 4; ++q) f(t + 8 * q, x[q]);
    }
    for (; t + 8 <= c1; t += 8) {
      float x[8];
      load8(row, t, x);
      f(t, x);
    }
  }
  for (; t < c1; ++t) {
    float x[1] = {load_logit(row, t)};
    f(t, x);
  }
}

// A thread's chunk held in registers (chunks of at most 32 logits from 16-byte aligned
// rows): logits past the chunk's end read as -inf, which weighs 0.
template <typename LT>
__device__ __forceinline__ void load_chunk32(const LT* row, int c0, int c1, float (&x)[32]) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int t = c0 + 8 * q;
    if (t + 8 <= c1) {
      float y[8];
      load8(row, t, y);
#pragma unroll
      for (int i = 0; i < 8; ++i) x[8 * q + i] = y[i];
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) x[8 * q + i] = t + i < c1 ? load_logit(row, t + i) : -INFINITY;
    }
  }
}

// kRegs: every chunk is at most 32 logits and rows allow vector loads, so a thread keeps
// its chunk of the visited row in registers (the bonus reads no logits again).
template <typename LT, bool kRegs>
__global__ void __launch_bounds__(kThreads)
    verify_sampling_kernel(const int32_t* __restrict__ node_offsets, const int32_t* __restrict__ parents,
                           const int32_t* __restrict__ tokens, const LT* __restrict__ logits, int vocab,
                           int64_t row_stride, int vec_ok, float inv_temp, const float* __restrict__ u_accept,
                           const float* __restrict__ u_bonus, int n_total, int max_nodes,
                           int32_t* __restrict__ accepted, int32_t* __restrict__ accept_len,
                           int32_t* __restrict__ bonus, int32_t* __restrict__ dev_status) {
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank(), csize = (int)cluster.num_blocks();
  __shared__ int par_s[kMaxNodes], tok_s[kMaxNodes], path_s[kMaxNodes];
  __shared__ float clogit_s[kMaxNodes], cu_s[kMaxNodes], cw_s[kMaxNodes];   // children of v: logit, u, weight
  __shared__ unsigned char cdup_s[kMaxNodes];                                // child repeats an earlier sibling
  __shared__ int rej_s[kMaxNodes];     // tokens rejected at the last visit
  __shared__ float rejw_s[kMaxNodes];  //   and their weights
  __shared__ float wm_s[2][kWarps];    // per warp (max, sum) of the visit's row, by visit parity
  __shared__ ff ws_s[2][kWarps];       //   (read by the whole cluster)
  __shared__ ff wt_s[kWarps], wpre_s[kWarps];   // bonus: per warp residual total, exclusive prefix
  __shared__ int wlast_s[kWarps];               // bonus: per warp last chunk of positive weight
  __shared__ ff ct_s;                           // bonus: this CTA's residual total (read by the cluster)
  __shared__ int clast_s;                       // bonus: this CTA's last chunk of positive weight
  __shared__ float m_s;
  __shared__ int chosen_s, nrej_s, len_s;

  const int b = blockIdx.y, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int node0 = node_offsets[b];
  const int T = node_offsets[b + 1] - node0;
  int32_t* acc_row = accepted + (size_t)b * max_nodes;
  const bool bad_shape = T < 1 || T > max_nodes || T > kMaxNodes || node0 < 0 || node0 + T > n_total;

  // this thread's chunk: a multiple of 8 logits, so vector loads stay 16-byte aligned
  const int G = csize * kThreads;
  const int chunk = (((vocab + G - 1) / G) + 7) & ~7;
  const int gidx = rank * kThreads + tid;
  const int c0 = min(vocab, gidx * chunk), c1 = min(vocab, c0 + chunk);
  const int nent = csize * kWarps;   // warp entries in the cluster
  const float c = inv_temp * 1.4426950408889634f;   // log2(e) / temperature
  const float ub = u_bonus[b];                       // read early: it is needed last

  float xr[kRegs ? 32 : 1];
  if constexpr (kRegs) {   // the root's row is loaded while the tree is read
    if (!bad_shape) load_chunk32(logits + (size_t)node0 * row_stride, c0, c1, xr);
  }

  // every CTA checks the tree the same way, so all of them leave here or none does
  bool bad = bad_shape;
  if (!bad_shape && tid < T) {
    const int p = parents[node0 + tid];
    par_s[tid] = p;
    tok_s[tid] = tokens[node0 + tid];
    bad = tid == 0 ? (p != -1) : (p < 0 || p >= tid);
  }
  if (tid == 0) {
    path_s[0] = 0;
    len_s = 1;
    // the claim of the bonus (an atomicMax from any CTA) follows at least one cluster barrier
    if (rank == 0 && !bad_shape) bonus[b] = -1;
  }
  if (__syncthreads_or(bad)) {
    if (rank == 0) {
      if (tid == 0) {
        atomicMax(dev_status, (int)PTD_ERR_INVALID_TREE);
        accept_len[b] = 0;
        bonus[b] = -1;
      }
      for (int j = tid; j < max_nodes; j += kThreads) acc_row[j] = -1;
    }
    return;
  }

  int v = 0;
  float m = -FLT_MAX;    // this thread's maximum of x * c over its chunk (last visit)
  ff s = {0.f, 0.f};     // and the sum of 2^(x * c - m)
  for (int it = 0;; ++it) {
    const LT* row = logits + (size_t)(node0 + v) * row_stride;
    // the children's logits and uniforms, fetched in parallel (read after the barrier below)
    if (tid > v && tid < T && par_s[tid] == v) {
      const int t = tok_s[tid];
      clogit_s[tid] = (t >= 0 && t < vocab) ? load_logit(row, t) : 0.f;
      cu_s[tid] = u_accept[node0 + tid];
    }
    // ---- this thread's (max, sum of weights relative to it) over its chunk
    if constexpr (kRegs) {
      if (it > 0) load_chunk32(row, c0, c1, xr);
      m = -FLT_MAX;
#pragma unroll
      for (int i = 0; i < 32; ++i) m = fmaxf(m, xr[i] * c);
      ff s2 = {0.f, 0.f};   // two accumulators: independent dependency chains
      s = ff{0.f, 0.f};
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        s = ff_add_f(s, exp2f(fmaf(xr[i], c, -m)));
        s2 = ff_add_f(s2, exp2f(fmaf(xr[i + 1], c, -m)));
      }
      s = ff_add_pos(s, s2);
    } else {
      m = -FLT_MAX;
      s = ff{0.f, 0.f};
      for_chunk(row, c0, c1, vec_ok != 0, [&](int, const auto& x) {
        constexpr int n = sizeof(x) / sizeof(float);
        float gm = -FLT_MAX;
#pragma unroll
        for (int i = 0; i < n; ++i) gm = fmaxf(gm, x[i] * c);
        if (gm > m) {   // new running maximum: rescale what has been summed
          s = ff_mul(s, exp2f(m - gm));
          m = gm;
        }
#pragma unroll
        for (int i = 0; i < n; ++i) s = ff_add_f(s, exp2f(fmaf(x[i], c, -m)));
      });
    }
    {
      float mw = m;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mw = fmaxf(mw, __shfl_xor_sync(0xffffffffu, mw, o));
      ff sw = ff_mul(s, exp2f(m - mw));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) sw = ff_add_pos(sw, shfl_xor(sw, o));
      if (lane == 0) {
        wm_s[it & 1][warp] = mw;
        ws_s[it & 1][warp] = sw;
      }
    }
    // the children of v (bit masks over node ids), and which repeat an earlier sibling's token
    uint32_t kids[kMaxNodes / 32];
    if (warp == 0) {
#pragma unroll
      for (int q = 0; q < kMaxNodes / 32; ++q) {
        const int n = lane + 32 * q;
        kids[q] = __ballot_sync(0xffffffffu, n > v && n < T && par_s[n] == v);
      }
#pragma unroll
      for (int q = 0; q < kMaxNodes / 32; ++q) {
        if ((kids[q] >> lane) & 1u) {
          const int n = lane + 32 * q;
          const int t = tok_s[n];
          bool dup = t < 0 || t >= vocab;   // a token outside the vocabulary has probability 0
#pragma unroll
          for (int q2 = 0; q2 <= q; ++q2) {
            uint32_t bits = q2 < q ? kids[q2] : (kids[q2] & ((1u << lane) - 1u));
            while (bits != 0u && !dup) {
              dup = tok_s[32 * q2 + __ffs(bits) - 1] == t;
              bits &= bits - 1u;
            }
          }
          cdup_s[n] = dup ? 1 : 0;
        }
      }
    }
    // A visit's pairs are read after this barrier; the next visit writes the other parity,
    // and the one after that only follows the next visit's barrier, which every CTA passes
    // after its reads here.
    cluster.sync();
    if (warp == 0) {
      // ---- the row's M and Z: lane l reduces entries l, l+32, l+64, l+96 (CTA e / 16,
      // warp e % 16), then the warp; every CTA does this in the same order, same bits
      float em[4];
      ff es[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int e = lane + 32 * q;
        em[q] = -FLT_MAX;
        es[q] = ff{0.f, 0.f};
        if (e < nent) {
          em[q] = *cluster.map_shared_rank(&wm_s[it & 1][e % kWarps], e / kWarps);
          es[q] = *cluster.map_shared_rank(&ws_s[it & 1][e % kWarps], e / kWarps);
        }
      }
      float M = fmaxf(fmaxf(em[0], em[1]), fmaxf(em[2], em[3]));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
      ff Z = ff_mul(es[0], exp2f(em[0] - M));
#pragma unroll
      for (int q = 1; q < 4; ++q) Z = ff_add_pos(Z, ff_mul(es[q], exp2f(em[q] - M)));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) Z = ff_add_pos(Z, shfl_xor(Z, o));
      // the children's weights, by their lanes
#pragma unroll
      for (int q = 0; q < kMaxNodes / 32; ++q) {
        const int n = lane + 32 * q;
        if ((kids[q] >> lane) & 1u) cw_s[n] = cdup_s[n] ? 0.f : exp2f(fmaf(clogit_s[n], c, -M));
      }
      __syncwarp();
      if (lane == 0) {
        // ---- try the children of v in node order
        ff S = Z;
        int nrej = 0, chosen = -1;
#pragma unroll
        for (int q = 0; q < kMaxNodes / 32; ++q) {
          uint32_t bits = kids[q];
          while (bits != 0u && chosen < 0) {
            const int n = 32 * q + __ffs(bits) - 1;
            bits &= bits - 1u;
            const float w = cw_s[n];
            // u < P(t) / S  <=>  u * S < w  (S > 0; with S exhausted nothing is accepted)
            if (S.hi > 0.f && ff_less(ff_mul(S, cu_s[n]), ff{w, 0.f})) {
              chosen = n;
            } else {
              S = ff_add(S, ff{-w, 0.f});
              if (!cdup_s[n]) {
                rej_s[nrej] = tok_s[n];
                rejw_s[nrej] = w;
                ++nrej;
              }
            }
          }
        }
        chosen_s = chosen;
        nrej_s = nrej;
        m_s = M;
        if (chosen >= 0) path_s[len_s++] = chosen;
      }
    }
    // chosen_s is rewritten only after the next cluster barrier, which every thread reaches
    // after reading it here
    __syncthreads();
    if (chosen_s < 0) break;
    v = chosen_s;
  }
  if (rank == 0) {
    const int len = len_s;
    for (int j = tid; j < max_nodes; j += kThreads) acc_row[j] = j < len ? path_s[j] : -1;
    if (tid == 0) accept_len[b] = len;
  }

  // ---- bonus: inverse CDF of the residual (rejected tokens weigh 0)
  {
    const LT* row = logits + (size_t)(node0 + v) * row_stride;
    const float M = m_s;
    const int nrej = nrej_s;
    // this chunk's residual weight: its sum rescaled to M, less its rejected tokens' weights
    // (the row maximum's own weight is 2^0 on both sides, so a dominant token cancels exactly)
    ff local = ff_mul(s, exp2f(m - M));
    bool has_rej = false;
    for (int j = 0; j < nrej; ++j) {
      const int t = rej_s[j];
      if (t >= c0 && t < c1) {
        local = ff_add(local, ff{-rejw_s[j], 0.f});
        has_rej = true;
      }
    }
    if (!(local.hi > 0.f)) local = ff{0.f, 0.f};
    // scan within the warp; per warp total and last chunk of positive weight
    ff incl = local;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const ff y = shfl_up(incl, o);
      if (lane >= o) incl = ff_add_pos(incl, y);
    }
    const uint32_t pos = __ballot_sync(0xffffffffu, local.hi > 0.f);
    if (lane == 31) wt_s[warp] = incl;
    if (lane == 0) wlast_s[warp] = pos ? rank * kThreads + warp * 32 + (31 - __clz(pos)) : -1;
    __syncthreads();
    if (warp == 0) {   // scan over the CTA's warps
      ff x = lane < kWarps ? wt_s[lane] : ff{0.f, 0.f};
#pragma unroll
      for (int o = 1; o < kWarps; o <<= 1) {
        const ff y = shfl_up(x, o);
        if (lane >= o) x = ff_add_pos(x, y);
      }
      ff ex = shfl_up(x, 1);
      if (lane == 0) ex = ff{0.f, 0.f};
      if (lane < kWarps) wpre_s[lane] = ex;
      if (lane == kWarps - 1) ct_s = x;
      int cl = lane < kWarps ? wlast_s[lane] : -1;
#pragma unroll
      for (int o = kWarps / 2; o > 0; o >>= 1) cl = max(cl, __shfl_xor_sync(0xffffffffu, cl, o));
      if (lane == 0) clast_s = cl;
    }
    cluster.sync();   // every CTA's total and last positive chunk are published
    // scan over the cluster's CTAs, the same in every warp
    ff B = lane < csize ? *cluster.map_shared_rank(&ct_s, lane) : ff{0.f, 0.f};
    int glast = lane < csize ? *cluster.map_shared_rank(&clast_s, lane) : -1;
    // no shared memory of another CTA is read after this: arrive now, wait before leaving
    asm volatile("barrier.cluster.arrive.release;" ::: "memory");
#pragma unroll
    for (int o = 1; o < kMaxCluster; o <<= 1) {
      const ff y = shfl_up(B, o);
      if (lane >= o) B = ff_add_pos(B, y);
    }
#pragma unroll
    for (int o = kMaxCluster / 2; o > 0; o >>= 1) glast = max(glast, __shfl_xor_sync(0xffffffffu, glast, o));
    glast = __shfl_sync(0xffffffffu, glast, 0);
    ff Bex = shfl_up(B, 1);
    if (lane == 0) Bex = ff{0.f, 0.f};
    const ff base_cta = shfl_idx(Bex, rank), next_cta = shfl_idx(B, rank);
    const ff total = shfl_idx(B, csize - 1);
    const ff base = warp == 0 ? base_cta : ff_add_pos(base_cta, wpre_s[warp]);
    const ff base_next = warp == kWarps - 1 ? next_cta : ff_add_pos(base_cta, wpre_s[warp + 1]);
    const ff prev = shfl_up(incl, 1);
    const ff start = lane == 0 ? base : ff_add_pos(base, prev);
    const ff end = lane == 31 ? base_next : ff_add_pos(base, incl);
    const ff target = ff_mul(total, ub);
    // The chunk whose [start, end) holds the target claims it (the last chunk of positive
    // weight also any target past the total); its warp walks it, 32 tokens at a time.
    const bool claim = local.hi > 0.f && !ff_less(target, start) && (ff_less(target, end) || gidx == glast);
    uint32_t claims = __ballot_sync(0xffffffffu, claim);
    while (claims != 0u) {
      const int cl = __ffs(claims) - 1;
      claims &= claims - 1u;
      const int k0 = __shfl_sync(0xffffffffu, c0, cl), k1 = __shfl_sync(0xffffffffu, c1, cl);
      const bool krej = __shfl_sync(0xffffffffu, has_rej, cl);
      ff acc = shfl_idx(start, cl);
      int pick = -1, last = -1;
      for (int p0 = k0; p0 < k1; p0 += 32) {   // one pass when chunks are at most 32 logits
        const int t = p0 + lane;
        float x;
        if constexpr (kRegs) {
          x = -INFINITY;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float y = __shfl_sync(0xffffffffu, xr[i], cl);
            if (i == lane) x = y;
          }
        } else {
          x = t < k1 ? load_logit(row, t) : -INFINITY;
        }
        bool rejected = false;
        if (krej)
          for (int j = 0; j < nrej; ++j) rejected |= rej_s[j] == t;
        const float w = (t < k1 && !rejected) ? exp2f(fmaf(x, c, -M)) : 0.f;
        ff run = ff{w, 0.f};   // inclusive scan of the weights over the lanes
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const ff y = shfl_up(run, o);
          if (lane >= o) run = ff_add_pos(run, y);
        }
        run = ff_add_pos(acc, run);
        const uint32_t hit = __ballot_sync(0xffffffffu, w > 0.f && ff_less(target, run));
        const uint32_t wpos = __ballot_sync(0xffffffffu, w > 0.f);
        if (pick < 0 && hit) pick = p0 + __ffs(hit) - 1;
        if (wpos) last = p0 + 31 - __clz(wpos);
        acc = shfl_idx(run, 31);
      }
      // (rounding can let two neighbouring chunks claim a target on their common end point:
      // the larger token wins)
      if (lane == 0) atomicMax(bonus + b, pick >= 0 ? pick : last);
    }
    asm volatile("barrier.cluster.wait.acquire;" ::: "memory");   // keep this CTA's shared memory alive
  }
}

template <typename LT>
cudaError_t launch(const int32_t* node_offsets, const int32_t* parents, const int32_t* tokens, const LT* logits,
                   int vocab, int64_t row_stride, float inv_temp, const float* u_accept, const float* u_bonus,
                   int batch, int n_total, int max_nodes, int32_t* accepted, int32_t* accept_len, int32_t* bonus,
                   int32_t* dev_status, cudaStream_t stream) {
  int csize = (vocab + kThreads * kPerThread - 1) / (kThreads * kPerThread);
  csize = csize < 1 ? 1 : (csize > kMaxCluster ? kMaxCluster : csize);
  const bool vec_ok = (reinterpret_cast<uintptr_t>(logits) % 16 == 0) &&
                      ((uint64_t)row_stride * sizeof(LT)) % 16 == 0;
  const int G = csize * kThreads;
  const int chunk = (((vocab + G - 1) / G) + 7) & ~7;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)csize, (unsigned)batch, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)csize;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (vec_ok && chunk <= 32)
    return cudaLaunchKernelEx(&cfg, verify_sampling_kernel<LT, true>, node_offsets, parents, tokens, logits, vocab,
                              row_stride, 1, inv_temp, u_accept, u_bonus, n_total, max_nodes, accepted,
                              accept_len, bonus, dev_status);
  return cudaLaunchKernelEx(&cfg, verify_sampling_kernel<LT, false>, node_offsets, parents, tokens, logits, vocab,
                            row_stride, vec_ok ? 1 : 0, inv_temp, u_accept, u_bonus, n_total, max_nodes, accepted,
                            accept_len, bonus, dev_status);
}

}  // namespace vs

cudaError_t launch_verify_sampling(const int32_t* node_offsets, const int32_t* parents, const int32_t* tokens,
                                   const void* logits, bool bf16, int vocab, int64_t row_stride, float inv_temp,
                                   const float* u_accept, const float* u_bonus, int batch, int n_total, int max_nodes,
                                   int32_t* accepted, int32_t* accept_len, int32_t* bonus, int32_t* dev_status,
                                   cudaStream_t stream) {
  if (batch > 65535) return cudaErrorInvalidValue;
  if (bf16)
    return vs::launch(node_offsets, parents, tokens, static_cast<const __nv_bfloat16*>(logits), vocab, row_stride,
                      inv_temp, u_accept, u_bonus, batch, n_total, max_nodes, accepted, accept_len, bonus,
                      dev_status, stream);
  return vs::launch(node_offsets, parents, tokens, static_cast<const float*>(logits), vocab, row_stride, inv_temp,
                    u_accept, u_bonus, batch, n_total, max_nodes, accepted, accept_len, bonus, dev_status, stream);
}

}  // namespace ptd
