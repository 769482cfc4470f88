// Sampling verification (Sec. 3.2, "sampling decoding strategy"; Alg. 2, Candidate Tree
// Recursive Sampling; App. E proves the emitted token follows P).
//
// One CTA per tree.  From the root, for the current node v the block computes the row
// statistics of P_v = softmax(logits_v / temperature) in one pass (each thread keeps a
// running maximum and an fp64 sum of exponentials, combined across the block); thread 0
// then tries the children of v in node order: child n is accepted when u_accept[n] <
// P_v(token_n) / S, S being the mass of P_v not yet rejected, and a rejected token gets
// probability 0.  An accepted child becomes v.  When no child is accepted (or v is a leaf)
// the bonus token is the inverse CDF of the residual P_v / S at u_bonus[b]: every thread
// sums a contiguous chunk of the vocabulary in fp64, a block scan finds the chunk holding
// the target, and that thread walks its chunk.  Exponentials are fp32, sums fp64.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "ptd_device.cuh"
#include "verify_sampling.cuh"

namespace ptd {
namespace vs {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxNodes = 128;

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

template <typename LT>
__global__ void __launch_bounds__(kThreads)
    verify_sampling_kernel(const int32_t* __restrict__ node_offsets, const int32_t* __restrict__ parents,
                           const int32_t* __restrict__ tokens, const LT* __restrict__ logits, int vocab,
                           int64_t row_stride, float inv_temp, const float* __restrict__ u_accept,
                           const float* __restrict__ u_bonus, int n_total, int max_nodes,
                           int32_t* __restrict__ accepted, int32_t* __restrict__ accept_len,
                           int32_t* __restrict__ bonus, int32_t* __restrict__ dev_status) {
  __shared__ int par_s[kMaxNodes], tok_s[kMaxNodes], rej_s[kMaxNodes], path_s[kMaxNodes];
  __shared__ float wmax_s[kWarps];
  __shared__ double wsum_s[kWarps];
  __shared__ float m_s;
  __shared__ double z_s, S_s, scan_s[kWarps];
  __shared__ int chosen_s, nrej_s, len_s, bonus_s, fallback_s, bad_s;

  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int node0 = node_offsets[b];
  const int T = node_offsets[b + 1] - node0;
  int32_t* acc_row = accepted + (size_t)b * max_nodes;

  const bool bad_shape = T < 1 || T > max_nodes || T > kMaxNodes || node0 < 0 || node0 + T > n_total;
  if (tid == 0) bad_s = bad_shape ? 1 : 0;
  __syncthreads();
  if (!bad_shape && tid < T) {
    const int p = parents[node0 + tid];
    par_s[tid] = p;
    tok_s[tid] = tokens[node0 + tid];
    if (tid == 0 ? (p != -1) : (p < 0 || p >= tid)) bad_s = 1;
  }
  __syncthreads();
  if (bad_s) {
    if (tid == 0) {
      atomicMax(dev_status, (int)PTD_ERR_INVALID_TREE);
      accept_len[b] = 0;
      bonus[b] = -1;
    }
    for (int j = tid; j < max_nodes; j += kThreads) acc_row[j] = -1;
    return;
  }

  int v = 0;
  if (tid == 0) {
    path_s[0] = 0;
    len_s = 1;
  }
  for (;;) {
    const LT* row = logits + (size_t)(node0 + v) * row_stride;
    // ---- row statistics of P_v: m = max x, Z = sum exp(x - m), x = logit / temperature
    float m = -INFINITY;
    double s = 0.0;
    for (int t = tid; t < vocab; t += kThreads) {
      const float x = load_logit(row, t) * inv_temp;
      if (x > m) {
        s = s * (double)expf(m - x) + 1.0;   // m = -inf at first: expf(-inf) = 0
        m = x;
      } else {
        s += (double)expf(x - m);
      }
    }
    float wm = m;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) wm = fmaxf(wm, __shfl_xor_sync(0xffffffffu, wm, o));
    if (lane == 0) wmax_s[warp] = wm;
    __syncthreads();
    if (tid < 32) {
      float bm = tid < kWarps ? wmax_s[tid] : -INFINITY;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, o));
      if (tid == 0) m_s = bm;
    }
    __syncthreads();
    const float M = m_s;
    double ws = m == -INFINITY ? 0.0 : s * (double)expf(m - M);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ws += __shfl_xor_sync(0xffffffffu, ws, o);
    if (lane == 0) wsum_s[warp] = ws;
    __syncthreads();
    if (tid < 32) {
      double bs = tid < kWarps ? wsum_s[tid] : 0.0;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) bs += __shfl_xor_sync(0xffffffffu, bs, o);
      if (tid == 0) z_s = bs;
    }
    __syncthreads();
    // ---- try the children of v in node order (thread 0)
    if (tid == 0) {
      const double Z = z_s;
      double S = 1.0;
      int nrej = 0, chosen = -1;
      for (int n = v + 1; n < T; ++n) {
        if (par_s[n] != v) continue;
        const int t = tok_s[n];
        bool before = t < 0 || t >= vocab;   // a token outside the vocabulary has probability 0
        for (int j = 0; j < nrej && !before; ++j) before = rej_s[j] == t;
        const double p = before ? 0.0 : (double)expf(load_logit(row, t) * inv_temp - M) / Z;
        const double p_hat = S > 0.0 ? p / S : 0.0;
        if ((double)u_accept[node0 + n] < p_hat) {
          chosen = n;
          break;
        }
        S -= p;
        if (!before) rej_s[nrej++] = t;
      }
      chosen_s = chosen;
      nrej_s = nrej;
      S_s = S;
      if (chosen >= 0) path_s[len_s++] = chosen;
    }
    __syncthreads();
    if (chosen_s < 0) break;
    v = chosen_s;
    __syncthreads();   // everyone has read chosen_s before thread 0 rewrites it
  }

  // ---- bonus: inverse CDF of the residual P_v / S (rejected tokens have probability 0)
  {
    const LT* row = logits + (size_t)(node0 + v) * row_stride;
    const float M = m_s;
    const double Z = z_s;
    const int nrej = nrej_s;
    const double target = (double)u_bonus[b] * S_s;
    const int chunk = (vocab + kThreads - 1) / kThreads;
    const int c0 = min(vocab, tid * chunk), c1 = min(vocab, c0 + chunk);
    auto prob = [&](int t) -> double {
      for (int j = 0; j < nrej; ++j)
        if (rej_s[j] == t) return 0.0;
      return (double)expf(load_logit(row, t) * inv_temp - M) / Z;
    };
    double local = 0.0;
    for (int t = c0; t < c1; ++t) local += prob(t);
    // exclusive prefix of `local` over the block
    double incl = local;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const double y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) scan_s[warp] = incl;
    if (tid == 0) {
      bonus_s = 0x7FFFFFFF;
      fallback_s = -1;
    }
    __syncthreads();
    if (tid < 32) {
      double w = tid < kWarps ? scan_s[tid] : 0.0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const double y = __shfl_up_sync(0xffffffffu, w, o);
        if (tid >= o) w += y;
      }
      if (tid < kWarps) scan_s[tid] = w;   // inclusive prefix over warps
    }
    __syncthreads();
    const double before = (warp > 0 ? scan_s[warp - 1] : 0.0) + (incl - local);
    // The chunk holding the target walks it.  (Rounding can let two neighbouring chunks
    // both claim a target on their common boundary, or none claim one past the total: the
    // lower claim wins, and with no claim the last token of positive probability is taken.)
    int last = -1;
    if (local > 0.0) {
      for (int t = c0; t < c1; ++t)
        if (prob(t) > 0.0) last = t;
      atomicMax(&fallback_s, last);
    }
    if (local > 0.0 && before <= target && target < before + local) {
      double acc = before;
      int pick = -1;
      for (int t = c0; t < c1; ++t) {
        const double pt = prob(t);
        acc += pt;
        if (acc > target && pt > 0.0) {
          pick = t;
          break;
        }
      }
      atomicMin(&bonus_s, pick >= 0 ? pick : last);
    }
    __syncthreads();
    if (tid == 0 && bonus_s == 0x7FFFFFFF) bonus_s = fallback_s;
    __syncthreads();
  }
  const int len = len_s;
  for (int j = tid; j < max_nodes; j += kThreads) acc_row[j] = j < len ? path_s[j] : -1;
  if (tid == 0) {
    accept_len[b] = len;
    bonus[b] = bonus_s;
  }
}

}  // namespace vs

cudaError_t launch_verify_sampling(const int32_t* node_offsets, const int32_t* parents, const int32_t* tokens,
                                   const void* logits, bool bf16, int vocab, int64_t row_stride, float inv_temp,
                                   const float* u_accept, const float* u_bonus, int batch, int n_total, int max_nodes,
                                   int32_t* accepted, int32_t* accept_len, int32_t* bonus, int32_t* dev_status,
                                   cudaStream_t stream) {
  if (bf16)
    vs::verify_sampling_kernel<__nv_bfloat16><<<batch, vs::kThreads, 0, stream>>>(
        node_offsets, parents, tokens, static_cast<const __nv_bfloat16*>(logits), vocab, row_stride, inv_temp, u_accept,
        u_bonus, n_total, max_nodes, accepted, accept_len, bonus, dev_status);
  else
    vs::verify_sampling_kernel<float><<<batch, vs::kThreads, 0, stream>>>(
        node_offsets, parents, tokens, static_cast<const float*>(logits), vocab, row_stride, inv_temp, u_accept,
        u_bonus, n_total, max_nodes, accepted, accept_len, bonus, dev_status);
  return cudaGetLastError();
}

}  // namespace ptd
