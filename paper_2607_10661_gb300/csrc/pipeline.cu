// Host-buffer steps with copies and compute overlapped: a software pipeline over two
// caller-owned device buffer sets (the end-to-end path of the tree-verify step).
//
// Streams: the caller's compute stream, plus one host-to-device and one device-to-host
// stream owned by the pipeline.  For step i on slot s = i % 2:
//   h2d:     wait compute_done[s] (step i - 2 no longer reads slot s's inputs); copy the
//            inputs into slot s, the tree's K/V rows into slot s's staging buffer; record
//            inputs_ready[s];
//   compute: wait inputs_ready[s] and results_ready[s] (step i - 2's results are out of
//            slot s's output buffers); clear the status word; copy the staged K/V rows into
//            the cache slots C_b + i (device to device: one 2-D copy per tree and K/V for a
//            contiguous cache, one scatter kernel through the block table for a paged one);
//            the step; record compute_done[s];
//   d2h:     wait compute_done[s]; copy the results to the step's host buffers; record
//            results_ready[s].
// So step i + 1's uploads run while step i computes, and step i's downloads while step
// i + 1 computes.  The cache is shared: steps compute in submission order.
#include <cuda_runtime.h>

#include <cstdint>
#include <cstring>
#include <new>

#include "../../include/ptd.h"
#include "step_checks.cuh"

struct ptd_pipeline {
  ptd_kv_cache cache;
  ptd_tree tree[2];
  ptd_step_args args[2];
  void* staging[2];
  size_t staging_bytes;
  cudaStream_t compute, h2d, d2h;
  cudaEvent_t inputs_ready[2], compute_done[2], results_ready[2];
  int64_t submitted;
};

namespace {

size_t elem_size(ptd_dtype d) { return d == PTD_BF16 ? 2 : 4; }

// Staged tree rows into a paged cache: CTA (layer, node, K/V) copies staging row
// [K/V][layer][node] (slot_bytes) to slot C_b + i of tree b, i = node - node_offsets[b],
// through the block table.  A slot outside the sequence's pages is skipped and reported.
__global__ void __launch_bounds__(128)
    tree_rows_to_pages_kernel(const uint8_t* __restrict__ staging, uint8_t* __restrict__ k_cache,
                              uint8_t* __restrict__ v_cache, int slot_bytes, int n_total, int batch,
                              const int32_t* __restrict__ node_offsets, const int32_t* __restrict__ ctx_lens,
                              const int32_t* __restrict__ block_table, int max_pages, int page_size, int num_pages,
                              int32_t* __restrict__ dev_status) {
  const int layer = blockIdx.x, n = blockIdx.y, kv = blockIdx.z;
  int lo = 0, hi = batch;   // tree b with node_offsets[b] <= n < node_offsets[b + 1]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (node_offsets[mid] <= n) lo = mid; else hi = mid;
  }
  const int b = lo, i = n - node_offsets[b], slot = ctx_lens[b] + i;
  const int pi = slot / page_size;
  const int pg = (i >= 0 && slot >= 0 && pi < max_pages) ? block_table[(size_t)b * max_pages + pi] : -1;
  if (pg < 0 || pg >= num_pages) {
    if (threadIdx.x == 0) atomicMax(dev_status, (int)PTD_ERR_INVALID_TREE);
    return;
  }
  const size_t L = gridDim.x;
  const uint4* src = reinterpret_cast<const uint4*>(staging + (((size_t)kv * L + layer) * n_total + n) * slot_bytes);
  uint4* dst = reinterpret_cast<uint4*>((kv ? v_cache : k_cache) +
                                        (((size_t)layer * num_pages + pg) * page_size + slot % page_size) * slot_bytes);
  for (int c = threadIdx.x; c < slot_bytes / 16; c += blockDim.x) dst[c] = src[c];
}

ptd_status cuda_st(cudaError_t e) { return e == cudaSuccess ? PTD_OK : PTD_ERR_CUDA; }

}  // namespace

extern "C" {

ptd_status ptd_pipeline_create(const ptd_kv_cache* cache, const ptd_tree* trees, const ptd_step_args* args,
                               void* const* staging, size_t staging_bytes, void* compute_stream,
                               ptd_pipeline** out) {
  if (!cache || !trees || !args || !staging || !staging[0] || !staging[1] || !out) return PTD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(staging[0]) | reinterpret_cast<uintptr_t>(staging[1])) % 16 != 0)
    return PTD_ERR_INVALID_ARG;
  for (int s = 0; s < 2; ++s) {
    if (trees[s].batch != trees[0].batch || trees[s].total_nodes != trees[0].total_nodes) return PTD_ERR_INVALID_ARG;
    // the step's own checks now, so that a bad argument never leaves uploads enqueued
    const ptd_status st = ptd::check_step_args(&trees[s], cache, &args[s]);
    if (st != PTD_OK) return st;
  }
  const size_t need = 2ull * cache->num_layers * trees[0].total_nodes * cache->num_kv_heads * cache->head_dim *
                      elem_size(cache->dtype);
  if (staging_bytes < need) return PTD_ERR_WORKSPACE;
  ptd_pipeline* p = new (std::nothrow) ptd_pipeline;
  if (!p) return PTD_ERR_CUDA;
  std::memset(p, 0, sizeof(*p));
  p->cache = *cache;
  for (int s = 0; s < 2; ++s) {
    p->tree[s] = trees[s];
    p->args[s] = args[s];
    p->staging[s] = staging[s];
  }
  p->staging_bytes = staging_bytes;
  p->compute = static_cast<cudaStream_t>(compute_stream);
  cudaError_t e = cudaStreamCreateWithFlags(&p->h2d, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&p->d2h, cudaStreamNonBlocking);
  for (int s = 0; s < 2 && e == cudaSuccess; ++s) {
    e = cudaEventCreateWithFlags(&p->inputs_ready[s], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p->compute_done[s], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&p->results_ready[s], cudaEventDisableTiming);
  }
  if (e != cudaSuccess) {
    ptd_pipeline_destroy(p);
    return PTD_ERR_CUDA;
  }
  *out = p;
  return PTD_OK;
}

ptd_status ptd_pipeline_submit(ptd_pipeline* p, const ptd_host_io* io, int64_t* ticket) {
  if (!p || !io || !ticket) return PTD_ERR_INVALID_ARG;
  if (!io->q_h || !io->logits_h || !io->tokens_h || !io->parents_h || !io->node_offsets_h || !io->ctx_lens_h ||
      !io->tree_k_h || !io->tree_v_h || !io->topk_idx_h || !io->topk_val_h || !io->accepted_h ||
      !io->accept_len_h || !io->bonus_h || !io->new_ctx_h || !io->status_h)
    return PTD_ERR_INVALID_ARG;
  const int s = (int)(p->submitted & 1);
  const ptd_tree& tree = p->tree[s];
  const ptd_step_args& a = p->args[s];
  const ptd_kv_cache& cache = p->cache;
  const int B = tree.batch, N = tree.total_nodes, L = cache.num_layers;
  const size_t es = elem_size(cache.dtype);
  const size_t slot_bytes = (size_t)cache.num_kv_heads * cache.head_dim * es;
  const size_t kv_bytes = (size_t)L * N * slot_bytes;
  // the host tree layout must describe this slot's tree and fit the cache (checked before
  // anything is enqueued: the staged rows are read by these offsets)
  const ptd_status layout = ptd::check_host_tree_layout(&tree, &cache, io->node_offsets_h, io->ctx_lens_h);
  if (layout != PTD_OK) return layout;
  // ---- uploads
  cudaError_t e = cudaStreamWaitEvent(p->h2d, p->compute_done[s], 0);
  auto h2d = [&](const void* dst, const void* src, size_t n) {
    if (e == cudaSuccess) e = cudaMemcpyAsync(const_cast<void*>(dst), src, n, cudaMemcpyHostToDevice, p->h2d);
  };
  h2d(a.q, io->q_h, (size_t)L * N * a.num_q_heads * cache.head_dim * es);
  h2d(a.logits, io->logits_h, (size_t)N * a.vocab * elem_size(a.logits_dtype));
  h2d(a.tokens, io->tokens_h, (size_t)N * 4);
  h2d(tree.parents, io->parents_h, (size_t)N * 4);
  h2d(tree.node_offsets, io->node_offsets_h, (size_t)(B + 1) * 4);
  h2d(tree.ctx_lens, io->ctx_lens_h, (size_t)B * 4);
  h2d(p->staging[s], io->tree_k_h, kv_bytes);
  h2d(static_cast<uint8_t*>(p->staging[s]) + kv_bytes, io->tree_v_h, kv_bytes);
  if (e == cudaSuccess) e = cudaEventRecord(p->inputs_ready[s], p->h2d);
  // ---- compute
  if (e == cudaSuccess) e = cudaStreamWaitEvent(p->compute, p->inputs_ready[s], 0);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(p->compute, p->results_ready[s], 0);
  if (e == cudaSuccess) e = cudaMemsetAsync(a.dev_status, 0, 4, p->compute);
  if (cache.page_size > 0 && e == cudaSuccess) {
    tree_rows_to_pages_kernel<<<dim3((unsigned)L, (unsigned)N, 2), 128, 0, p->compute>>>(
        static_cast<const uint8_t*>(p->staging[s]), static_cast<uint8_t*>(cache.k), static_cast<uint8_t*>(cache.v),
        (int)slot_bytes, N, B, tree.node_offsets, tree.ctx_lens, cache.block_table, cache.max_pages,
        cache.page_size, cache.num_pages, a.dev_status);
    e = cudaGetLastError();
  }
  const size_t layer_pitch = (size_t)B * cache.seq_capacity * slot_bytes;
  for (int b = 0; b < B && cache.page_size == 0 && e == cudaSuccess; ++b) {
    const int off = io->node_offsets_h[b], T = io->node_offsets_h[b + 1] - off, C = io->ctx_lens_h[b];
    const size_t dst_off = ((size_t)b * cache.seq_capacity + C) * slot_bytes;
    for (int kv = 0; kv < 2 && e == cudaSuccess; ++kv) {
      uint8_t* dst = static_cast<uint8_t*>(kv ? cache.v : cache.k) + dst_off;
      const uint8_t* src = static_cast<const uint8_t*>(p->staging[s]) + (size_t)kv * kv_bytes + (size_t)off * slot_bytes;
      e = cudaMemcpy2DAsync(dst, layer_pitch, src, (size_t)N * slot_bytes, (size_t)T * slot_bytes, (size_t)L,
                            cudaMemcpyDeviceToDevice, p->compute);
    }
  }
  if (e != cudaSuccess) return cuda_st(e);
  ptd_status st = ptd_tree_verify_step(&tree, &cache, &a, p->compute);
  if (st != PTD_OK) return st;
  e = cudaEventRecord(p->compute_done[s], p->compute);
  // ---- downloads
  if (e == cudaSuccess) e = cudaStreamWaitEvent(p->d2h, p->compute_done[s], 0);
  auto d2h = [&](void* dst, const void* src, size_t n) {
    if (e == cudaSuccess) e = cudaMemcpyAsync(dst, src, n, cudaMemcpyDeviceToHost, p->d2h);
  };
  d2h(io->topk_idx_h, a.topk_idx, (size_t)N * a.k * 4);
  d2h(io->topk_val_h, a.topk_val, (size_t)N * a.k * 4);
  d2h(io->accepted_h, a.accepted_nodes, (size_t)B * tree.max_nodes * 4);
  d2h(io->accept_len_h, a.accept_len, (size_t)B * 4);
  d2h(io->bonus_h, a.bonus_token, (size_t)B * 4);
  d2h(io->new_ctx_h, a.new_ctx_lens, (size_t)B * 4);
  d2h(io->status_h, a.dev_status, 4);
  if (e == cudaSuccess) e = cudaEventRecord(p->results_ready[s], p->d2h);
  if (e != cudaSuccess) return cuda_st(e);
  *ticket = p->submitted++;
  return PTD_OK;
}

ptd_status ptd_pipeline_wait(ptd_pipeline* p, int64_t ticket) {
  if (!p || ticket < 0 || ticket >= p->submitted) return PTD_ERR_INVALID_ARG;
  // the slot's event belongs to the latest step on it; that step's computation waited for
  // this ticket's results, so waiting for it covers this ticket too
  return cuda_st(cudaEventSynchronize(p->results_ready[ticket & 1]));
}

ptd_status ptd_pipeline_destroy(ptd_pipeline* p) {
  if (!p) return PTD_ERR_INVALID_ARG;
  if (p->h2d) cudaStreamSynchronize(p->h2d);
  if (p->d2h) cudaStreamSynchronize(p->d2h);
  for (int s = 0; s < 2; ++s) {
    if (p->inputs_ready[s]) cudaEventDestroy(p->inputs_ready[s]);
    if (p->compute_done[s]) cudaEventDestroy(p->compute_done[s]);
    if (p->results_ready[s]) cudaEventDestroy(p->results_ready[s]);
  }
  if (p->h2d) cudaStreamDestroy(p->h2d);
  if (p->d2h) cudaStreamDestroy(p->d2h);
  delete p;
  return PTD_OK;
}

}  // extern "C"
