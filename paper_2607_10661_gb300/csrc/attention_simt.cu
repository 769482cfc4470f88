// Tree-masked attention in fp32 on the CUDA cores (the fp32 path; no tensor cores, so
// the result keeps full fp32 accuracy).
//
// Same operation as the tensor-core kernel (Sec. 3.1 ancestor-only visibility over the
// committed prefix plus the tree, Sec. 3.2): one CTA per (layer, tree, query head), one
// warp per tree node at a time.  For each chunk of 32 keys a lane scores one key, the
// warp keeps an online softmax (running max m, sum l) and every lane accumulates D/32
// output columns.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "attention.cuh"
#include "ptd_device.cuh"

namespace ptd {
namespace simt {

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <int D>
__global__ void __launch_bounds__(128) tree_attn_simt_kernel(const AttnParams p) {
  constexpr int DPL = D / 32;   // output columns per lane
  __shared__ int par_s[128];
  __shared__ uint32_t anc_s[128][4];
  __shared__ __align__(16) float q_s[4][D];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int u = blockIdx.x;
  const int h = u % p.hq;
  u /= p.hq;
  const int b = u % p.batch;
  const int lq = u / p.batch;
  const int layer = p.layer_begin + lq;
  const int hkv = h / p.group;

  const int node0 = p.node_offsets[b];
  const int T = p.node_offsets[b + 1] - node0;
  const int C = p.ctx_lens[b];
  const int N = C + T;
  bool bad_shape = T < 1 || T > p.max_nodes || node0 < 0 || node0 + T > p.n_total || C < 0;
  if (!bad_shape) bad_shape = p.page_size > 0 ? N > p.max_pages * p.page_size : N > p.seq_capacity;
  if (bad_shape) {
    if (threadIdx.x == 0) atomicMax(p.dev_status, (int)PTD_ERR_INVALID_TREE);
    return;
  }

  bool bad = false;
  if (threadIdx.x < T) {
    const int pp = p.parents[node0 + threadIdx.x];
    par_s[threadIdx.x] = pp;
    bad = threadIdx.x == 0 ? (pp != -1) : (pp < 0 || pp >= (int)threadIdx.x);
  }
  const int invalid = __syncthreads_or(bad);
  const float* Q = static_cast<const float*>(p.q);
  float* O = static_cast<float*>(p.out);
  if (invalid) {
    if (threadIdx.x == 0) atomicMax(p.dev_status, (int)PTD_ERR_INVALID_TREE);
    for (int i = warp; i < T; i += 4)
      for (int d = lane; d < D; d += 32) O[(((size_t)lq * p.n_total + node0 + i) * p.hq + h) * D + d] = 0.f;
    return;
  }
  if (threadIdx.x < T) {
    uint32_t m[4] = {0, 0, 0, 0};
    for (int a = threadIdx.x; a >= 0; a = par_s[a]) m[a >> 5] |= 1u << (a & 31);
    for (int w = 0; w < 4; ++w) anc_s[threadIdx.x][w] = m[w];
  }
  __syncthreads();

  const float* Kc = static_cast<const float*>(p.k);
  const float* Vc = static_cast<const float*>(p.v);
  const size_t slot_elems = (size_t)p.hkv * D;
  auto slot_row = [&](int slot) -> size_t {
    size_t r;
    if (p.page_size > 0) {
      const int pg = p.block_table[(size_t)b * p.max_pages + slot / p.page_size];
      r = ((size_t)layer * p.num_pages + pg) * p.page_size + slot % p.page_size;
    } else {
      r = ((size_t)layer * p.batch + b) * p.seq_capacity + slot;
    }
    return r * slot_elems + (size_t)hkv * D;
  };

  for (int i = warp; i < T; i += 4) {
    const size_t qrow = (((size_t)lq * p.n_total + node0 + i) * p.hq + h) * D;
    for (int d = lane; d < D; d += 32) q_s[warp][d] = Q[qrow + d];
    __syncwarp();
    const uint32_t a0 = anc_s[i][0], a1 = anc_s[i][1], a2 = anc_s[i][2], a3 = anc_s[i][3];
    float m = -INFINITY, l = 0.f;
    float acc[DPL];
#pragma unroll
    for (int c = 0; c < DPL; ++c) acc[c] = 0.f;

    for (int k0 = 0; k0 < N; k0 += 32) {
      const int key = k0 + lane;
      bool vis = key < C;
      if (!vis && key < N) {
        const int a = key - C;
        const uint32_t w = a < 32 ? a0 : a < 64 ? a1 : a < 96 ? a2 : a3;
        vis = (w >> (a & 31)) & 1u;
      }
      float s = -INFINITY;
      if (vis) {
        const float4* kr = reinterpret_cast<const float4*>(Kc + slot_row(key));
        const float4* qr = reinterpret_cast<const float4*>(q_s[warp]);
        float dot = 0.f;
#pragma unroll 8
        for (int c = 0; c < D / 4; ++c) {
          const float4 kv = __ldg(kr + c), qv = qr[c];
          dot = fmaf(qv.x, kv.x, dot);
          dot = fmaf(qv.y, kv.y, dot);
          dot = fmaf(qv.z, kv.z, dot);
          dot = fmaf(qv.w, kv.w, dot);
        }
        s = dot * p.scale;
      }
      const float m_new = fmaxf(m, warp_max(s));
      if (m_new == -INFINITY) continue;   // nothing visible yet
      const float alpha = m == -INFINITY ? 0.f : expf(m - m_new);
      const float pj = vis ? expf(s - m_new) : 0.f;
      l = l * alpha + warp_sum(pj);
#pragma unroll
      for (int c = 0; c < DPL; ++c) acc[c] *= alpha;
      for (int j = 0; j < 32; ++j) {
        const float pjj = __shfl_sync(0xffffffffu, pj, j);
        if (pjj == 0.f) continue;   // warp-uniform: the value is broadcast
        const float* vr = Vc + slot_row(k0 + j);
#pragma unroll
        for (int c = 0; c < DPL; ++c) acc[c] = fmaf(pjj, __ldg(vr + c * 32 + lane), acc[c]);
      }
      m = m_new;
    }
    const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
    for (int c = 0; c < DPL; ++c) O[qrow + c * 32 + lane] = acc[c] * inv;
    __syncwarp();
  }
}

}  // namespace simt

cudaError_t launch_tree_attn_simt(const AttnParams& p, cudaStream_t stream) {
  const unsigned grid = (unsigned)(p.layers * p.batch * p.hq);
  switch (p.head_dim) {
    case 32:
      simt::tree_attn_simt_kernel<32><<<grid, 128, 0, stream>>>(p);
      break;
    case 64:
      simt::tree_attn_simt_kernel<64><<<grid, 128, 0, stream>>>(p);
      break;
    case 128:
      simt::tree_attn_simt_kernel<128><<<grid, 128, 0, stream>>>(p);
      break;
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace ptd
