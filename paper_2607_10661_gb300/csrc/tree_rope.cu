// Tree positions, the rotary encoding and the tree's K/V append (Sec. 3.1 "Tree
// Construction": a node's position is set by |pi(v)|).
//
// Node i of tree b sits at position p = C_b + |pi(i)| - 1.  One CTA per (node, group of
// four layers): it stages its tree's parent array in shared memory (one load per thread),
// counts |pi(i)| by walking up (<= 128 shared-memory reads), builds the node's D/2
// (cos, sin) pairs once, then, with 16-byte vectors where rows allow, turns every pair
// (x_j, x_{j+D/2}) of the node's query heads (in place) and key heads by p * base^(-2j/D)
// (RoFormer's rotation, rotate-half layout; the angle p * f is carried as an fp32 pair
// from a float-float f computed in double on the host, so that its rounding error is
// corrected to first order after sincosf) and writes the rotated keys and the values into
// cache slot C_b + i of each layer (contiguous or paged); a slot outside the cache (or a
// page number outside the pool) writes nothing and sets the status.  Pure streaming:
// about 1.5 MB per layer for the Llama-3-8B-shaped 63-node tree.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "ptd_device.cuh"
#include "tree_rope.cuh"

namespace ptd {
namespace tr {

constexpr int kThreads = 256;

template <typename T>
__device__ __forceinline__ float ld(const T* p);
template <>
__device__ __forceinline__ float ld<float>(const float* p) { return *p; }
template <>
__device__ __forceinline__ float ld<__nv_bfloat16>(const __nv_bfloat16* p) { return __bfloat162float(*p); }
template <typename T>
__device__ __forceinline__ void st(T* p, float x);
template <>
__device__ __forceinline__ void st<float>(float* p, float x) { *p = x; }
template <>
__device__ __forceinline__ void st<__nv_bfloat16>(__nv_bfloat16* p, float x) { *p = __float2bfloat16_rn(x); }

constexpr int kLayersPerCta = 4;

// One 16-byte vector of T: 16 / sizeof(T) elements, widened to fp32.
template <typename T>
struct Vec {
  static constexpr int N = 16 / sizeof(T);
  float x[N];
};
template <typename T>
__device__ __forceinline__ Vec<T> ld16(const T* p) {   // a plain load: q is also written
  Vec<T> r;
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  if constexpr (sizeof(T) == 2) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      r.x[2 * i] = __uint_as_float(w[i] << 16);
      r.x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  } else {
    r.x[0] = __uint_as_float(u.x), r.x[1] = __uint_as_float(u.y), r.x[2] = __uint_as_float(u.z),
    r.x[3] = __uint_as_float(u.w);
  }
  return r;
}
template <typename T>
__device__ __forceinline__ void st16(T* p, const Vec<T>& r) {
  uint4 u;
  if constexpr (sizeof(T) == 2) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 h = __floats2bfloat162_rn(r.x[2 * i], r.x[2 * i + 1]);
      w[i] = *reinterpret_cast<const uint32_t*>(&h);
    }
    u = make_uint4(w[0], w[1], w[2], w[3]);
  } else {
    u = make_uint4(__float_as_uint(r.x[0]), __float_as_uint(r.x[1]), __float_as_uint(r.x[2]),
                   __float_as_uint(r.x[3]));
  }
  *reinterpret_cast<uint4*>(p) = u;
}

// One CTA per (node, group of kLayersPerCta layers).  kVec: rows are 16-byte aligned and
// D/2 is a multiple of the vector width, so every access is a 16-byte vector.
template <typename T, bool kVec>
__global__ void __launch_bounds__(kThreads)
    tree_rope_kernel(const int32_t* __restrict__ node_offsets, const int32_t* __restrict__ parents,
                     const int32_t* __restrict__ ctx_lens, int batch, int n_total, int num_layers, int D, int hq,
                     int hkv, T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
                     T* __restrict__ k_cache, T* __restrict__ v_cache, int layer_begin, int page_size,
                     int seq_capacity, int num_pages, const int32_t* __restrict__ block_table, int max_pages,
                     const RopeFreqs freqs, int32_t* __restrict__ positions_out, int32_t* __restrict__ dev_status) {
  __shared__ int par_s[kThreads];
  __shared__ float cos_s[kMaxRopeHalf], sin_s[kMaxRopeHalf];
  __shared__ int pos_s, slot_s, b_s;
  const int n = blockIdx.x, t = threadIdx.x;
  const int l0 = blockIdx.y * kLayersPerCta;   // first layer of this CTA, relative to layer_begin
  if (t == 0) {   // the tree holding node n (B is small: a linear search)
    int b = 0;
    while (b + 1 < batch && node_offsets[b + 1] <= n) ++b;
    b_s = b;
  }
  __syncthreads();
  const int b = b_s;
  const int node0 = node_offsets[b];
  const int T_b = node_offsets[b + 1] - node0;
  const int i = n - node0;
  bool bad = T_b < 1 || T_b > kThreads || i < 0 || i >= T_b;
  if (!bad && t < T_b) {
    const int p = parents[node0 + t];
    par_s[t] = p;
    bad = t == 0 ? p != -1 : (p < 0 || p >= t);
  }
  if (__syncthreads_or(bad)) {
    if (t == 0) atomicMax(dev_status, (int)PTD_ERR_INVALID_TREE);
    return;
  }
  if (t == 0) {
    int depth = 0;
    for (int a = i; a != -1; a = par_s[a]) ++depth;
    const int C = ctx_lens[b];
    const int slot = C + i;
    const int cap = page_size > 0 ? max_pages * page_size : seq_capacity;
    int pg = 0;
    if (C >= 0 && slot < cap && page_size > 0) pg = block_table[(size_t)b * max_pages + slot / page_size];
    const bool fits = C >= 0 && slot < cap && pg >= 0 && pg < (page_size > 0 ? num_pages : 1);
    pos_s = C + depth - 1;
    slot_s = fits ? slot : -1;
    if (positions_out && l0 == 0) positions_out[n] = C + depth - 1;
    if (!fits && l0 == 0) atomicMax(dev_status, (int)PTD_ERR_INVALID_TREE);
  }
  __syncthreads();
  const int half = D / 2;
  if (t < half) {
    // angle = pos * (hi + lo) = a_hi + a_err (a_err exact up to pos * lo's rounding); sin
    // and cos of a_hi, corrected to first order in a_err (|a_err| < 1e-3)
    const float pos = (float)pos_s, fh = freqs.hi[t];
    const float a_hi = __fmul_rn(pos, fh);
    const float a_err = fmaf(pos, fh, -a_hi) + pos * freqs.lo[t];
    float s0, c0;
    sincosf(a_hi, &s0, &c0);
    sin_s[t] = fmaf(a_err, c0, s0);
    cos_s[t] = fmaf(-a_err, s0, c0);
  }
  __syncthreads();
  const int slot = slot_s;
  if (slot < 0) return;   // the node's slot is outside the cache: nothing is written
  size_t row;
  if (page_size > 0) {
    const int pg = block_table[(size_t)b * max_pages + slot / page_size];
    row = ((size_t)page_size * pg + slot % page_size);
  } else {
    row = (size_t)b * seq_capacity + slot;
  }
  const size_t layer_rows = page_size > 0 ? (size_t)num_pages * page_size : (size_t)batch * seq_capacity;
  const int l1 = min(num_layers, l0 + kLayersPerCta);
  if constexpr (kVec) {
    constexpr int V = Vec<T>::N;
    const int chunks = half / V;                       // vectors per half row
    const int qwork = hq * chunks, kwork = hkv * chunks, vwork = hkv * (D / V);
    for (int lq = l0; lq < l1; ++lq) {
      T* qn = q + ((size_t)lq * n_total + n) * hq * D;
      const T* kn = k + ((size_t)lq * n_total + n) * hkv * D;
      const T* vn = v + ((size_t)lq * n_total + n) * hkv * D;
      const size_t crow = ((size_t)(layer_begin + lq) * layer_rows + row) * hkv * D;
      for (int e = t; e < qwork + kwork + vwork; e += kThreads) {
        if (e < qwork + kwork) {
          const bool isq = e < qwork;
          const int e2 = isq ? e : e - qwork;
          const int h = e2 / chunks, j0 = (e2 - h * chunks) * V;
          const T* src = (isq ? (const T*)qn : kn) + (size_t)h * D;
          T* dst = isq ? qn + (size_t)h * D : k_cache + crow + (size_t)h * D;
          const Vec<T> a = ld16(src + j0), bb = ld16(src + j0 + half);
          Vec<T> ra, rb;
#pragma unroll
          for (int x = 0; x < V; ++x) {
            const float c = cos_s[j0 + x], s = sin_s[j0 + x];
            ra.x[x] = a.x[x] * c - bb.x[x] * s;
            rb.x[x] = a.x[x] * s + bb.x[x] * c;
          }
          st16(dst + j0, ra);
          st16(dst + j0 + half, rb);
        } else {
          const int e2 = e - qwork - kwork;
          *reinterpret_cast<uint4*>(v_cache + crow + (size_t)e2 * V) =
              __ldg(reinterpret_cast<const uint4*>(vn + (size_t)e2 * V));
        }
      }
    }
  } else {
    for (int lq = l0; lq < l1; ++lq) {
      T* qn = q + ((size_t)lq * n_total + n) * hq * D;
      const T* kn = k + ((size_t)lq * n_total + n) * hkv * D;
      const T* vn = v + ((size_t)lq * n_total + n) * hkv * D;
      const size_t crow = ((size_t)(layer_begin + lq) * layer_rows + row) * hkv * D;
      for (int e = t; e < (hq + hkv) * half; e += kThreads) {
        const bool isq = e < hq * half;
        const int e2 = isq ? e : e - hq * half;
        const int h = e2 / half, j = e2 - h * half;
        const T* src = (isq ? (const T*)qn : kn) + (size_t)h * D;
        T* dst = isq ? qn + (size_t)h * D : k_cache + crow + (size_t)h * D;
        const float a = ld(src + j), bb = ld(src + j + half);
        const float c = cos_s[j], s = sin_s[j];
        st(dst + j, a * c - bb * s);
        st(dst + j + half, a * s + bb * c);
      }
      for (int e = t; e < hkv * D; e += kThreads) v_cache[crow + e] = vn[e];
    }
  }
}

}  // namespace tr

cudaError_t launch_tree_rope(const int32_t* node_offsets, const int32_t* parents, const int32_t* ctx_lens,
                             int batch, int n_total, bool bf16, int head_dim, int hq, int hkv, void* q, const void* k,
                             const void* v, void* k_cache, void* v_cache, int layer_begin, int num_layers,
                             int page_size, int seq_capacity, int num_pages, const int32_t* block_table, int max_pages,
                             const RopeFreqs& freqs, int32_t* positions_out, int32_t* dev_status,
                             cudaStream_t stream) {
  const dim3 grid(n_total, (num_layers + tr::kLayersPerCta - 1) / tr::kLayersPerCta);
  const auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  const bool aligned = al16(q) && al16(k) && al16(v) && al16(k_cache) && al16(v_cache);
#define PTD_ROPE_LAUNCH(T, VEC)                                                                                    \
  tr::tree_rope_kernel<T, VEC><<<grid, tr::kThreads, 0, stream>>>(                                                \
      node_offsets, parents, ctx_lens, batch, n_total, num_layers, head_dim, hq, hkv, static_cast<T*>(q),        \
      static_cast<const T*>(k), static_cast<const T*>(v), static_cast<T*>(k_cache), static_cast<T*>(v_cache),    \
      layer_begin, page_size, seq_capacity, num_pages, block_table, max_pages, freqs, positions_out, dev_status)
  if (bf16) {
    if (aligned && (head_dim / 2) % 8 == 0)
      PTD_ROPE_LAUNCH(__nv_bfloat16, true);
    else
      PTD_ROPE_LAUNCH(__nv_bfloat16, false);
  } else {
    if (aligned && (head_dim / 2) % 4 == 0)
      PTD_ROPE_LAUNCH(float, true);
    else
      PTD_ROPE_LAUNCH(float, false);
  }
#undef PTD_ROPE_LAUNCH
  return cudaGetLastError();
}

}  // namespace ptd
