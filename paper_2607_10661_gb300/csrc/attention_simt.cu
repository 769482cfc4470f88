// Tree-masked attention in fp32 on the CUDA cores (the fp32 path; no tensor cores, so
// the result keeps full fp32 accuracy).
//
// Same operation as the tensor-core kernel (Sec. 3.1 ancestor-only visibility over the
// committed prefix plus the tree, Sec. 3.2): one CTA of 4 warps per (layer, node, query
// head).  The keys are cut into chunks of 32 and warp w takes chunks w, w + 4, ...: in a
// chunk lane j scores key j (its K row read with independent 16-byte loads), the warp keeps
// an online softmax (running max m, sum l), and every lane accumulates D/32 output columns
// from the chunk's 32 V rows, all of whose loads are issued before the first multiply.  The
// four warps' (m, l, O) are combined in shared memory at the end.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "attention.cuh"
#include "ptd_device.cuh"

namespace ptd {
namespace simt {

constexpr int kWarps = 4;

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
__global__ void __launch_bounds__(kWarps * 32) tree_attn_simt_kernel(const AttnParams p) {
  constexpr int DPL = D / 32;   // output columns per lane
  __shared__ int par_s[128];
  __shared__ __align__(16) float q_s[D];
  __shared__ uint32_t anc_s[4];
  __shared__ float m_s[kWarps], l_s[kWarps];
  __shared__ float o_s[kWarps][D];
  __shared__ int meta_s[3];     // tree b, node within the tree, invalid

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x, n = blockIdx.y, lq = blockIdx.z;
  const int layer = p.layer_begin + lq;
  const int hkv = h / p.group;
  float* O = static_cast<float*>(p.out);
  const size_t qrow = (((size_t)lq * p.n_total + n) * p.hq + h) * D;

  if (threadIdx.x == 0) {
    int lo = 0, hi = p.batch;   // tree b with node_offsets[b] <= n < node_offsets[b + 1]
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (p.node_offsets[mid] <= n) lo = mid; else hi = mid;
    }
    meta_s[0] = lo;
  }
  __syncthreads();
  const int b = meta_s[0];
  const int node0 = p.node_offsets[b];
  const int T = p.node_offsets[b + 1] - node0;
  const int C = p.ctx_lens[b];
  const int N = C + T;
  const int i = n - node0;
  bool bad_shape = T < 1 || T > p.max_nodes || node0 < 0 || node0 + T > p.n_total || C < 0 || i < 0 || i >= T;
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
  if (invalid) {
    if (threadIdx.x == 0) atomicMax(p.dev_status, (int)PTD_ERR_INVALID_TREE);
    for (int d = threadIdx.x; d < D; d += blockDim.x) O[qrow + d] = 0.f;
    return;
  }
  if (threadIdx.x == 0) {
    uint32_t m[4] = {0, 0, 0, 0};
    for (int a = i; a >= 0; a = par_s[a]) m[a >> 5] |= 1u << (a & 31);
    for (int w = 0; w < 4; ++w) anc_s[w] = m[w];
  }
  const float* Q = static_cast<const float*>(p.q);
  for (int d = threadIdx.x; d < D; d += blockDim.x) q_s[d] = Q[qrow + d];
  __syncthreads();
  const uint32_t a0 = anc_s[0], a1 = anc_s[1], a2 = anc_s[2], a3 = anc_s[3];

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

  float m = -INFINITY, l = 0.f;
  float acc[DPL];
#pragma unroll
  for (int c = 0; c < DPL; ++c) acc[c] = 0.f;
  for (int k0 = warp * 32; k0 < N; k0 += kWarps * 32) {
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
      const float4* qr = reinterpret_cast<const float4*>(q_s);
      float4 kv[D / 4];
#pragma unroll
      for (int c = 0; c < D / 4; ++c) kv[c] = __ldg(kr + c);
      float d0 = 0.f, d1 = 0.f;
#pragma unroll
      for (int c = 0; c < D / 4; c += 2) {
        const float4 q0 = qr[c], q1 = qr[c + 1];
        d0 = fmaf(q0.x, kv[c].x, d0);
        d0 = fmaf(q0.y, kv[c].y, d0);
        d0 = fmaf(q0.z, kv[c].z, d0);
        d0 = fmaf(q0.w, kv[c].w, d0);
        d1 = fmaf(q1.x, kv[c + 1].x, d1);
        d1 = fmaf(q1.y, kv[c + 1].y, d1);
        d1 = fmaf(q1.z, kv[c + 1].z, d1);
        d1 = fmaf(q1.w, kv[c + 1].w, d1);
      }
      s = (d0 + d1) * p.scale;
    }
    const float m_new = fmaxf(m, warp_max(s));
    if (m_new == -INFINITY) continue;   // nothing visible yet (warp-uniform)
    const float alpha = m == -INFINITY ? 0.f : expf(m - m_new);
    const float pj = vis ? expf(s - m_new) : 0.f;
    l = l * alpha + warp_sum(pj);
#pragma unroll
    for (int c = 0; c < DPL; ++c) acc[c] *= alpha;
    // all 32 V rows of the chunk at once (rows past the sequence are not read)
    const int nk = min(32, N - k0);
    float v[32][DPL];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const float* vr = Vc + slot_row(j < nk ? k0 + j : k0);
#pragma unroll
      for (int c = 0; c < DPL; ++c) v[j][c] = j < nk ? __ldg(vr + c * 32 + lane) : 0.f;
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const float pjj = __shfl_sync(0xffffffffu, pj, j);
#pragma unroll
      for (int c = 0; c < DPL; ++c) acc[c] = fmaf(pjj, v[j][c], acc[c]);
    }
    m = m_new;
  }
  // combine the four warps' partial softmax states
  if (lane == 0) {
    m_s[warp] = m;
    l_s[warp] = l;
  }
#pragma unroll
  for (int c = 0; c < DPL; ++c) o_s[warp][c * 32 + lane] = acc[c];
  __syncthreads();
  if (warp == 0) {
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) M = fmaxf(M, m_s[w]);
    float L = 0.f, wgt[kWarps];
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      wgt[w] = (m_s[w] == -INFINITY) ? 0.f : expf(m_s[w] - M);
      L += l_s[w] * wgt[w];
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
    for (int c = 0; c < DPL; ++c) {
      float o = 0.f;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) o = fmaf(wgt[w], o_s[w][c * 32 + lane], o);
      O[qrow + c * 32 + lane] = o * inv;
    }
  }
}

}  // namespace simt

cudaError_t launch_tree_attn_simt(const AttnParams& p, cudaStream_t stream) {
  if (p.hq > 65535 || p.n_total > 65535 || p.layers > 65535) return cudaErrorInvalidValue;
  const dim3 grid((unsigned)p.hq, (unsigned)p.n_total, (unsigned)p.layers);
  switch (p.head_dim) {
    case 32:
      simt::tree_attn_simt_kernel<32><<<grid, simt::kWarps * 32, 0, stream>>>(p);
      break;
    case 64:
      simt::tree_attn_simt_kernel<64><<<grid, simt::kWarps * 32, 0, stream>>>(p);
      break;
    case 128:
      simt::tree_attn_simt_kernel<128><<<grid, simt::kWarps * 32, 0, stream>>>(p);
      break;
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace ptd
