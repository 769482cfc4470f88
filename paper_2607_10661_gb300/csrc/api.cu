// C ABI of the PTD tree-verify step: host-side argument checks, scratch sizing, TMA
// descriptor encoding and kernel launches.  No allocation, no synchronisation: every
// call enqueues on the caller's stream (declared in include/ptd.h).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstddef>
#include <cstdint>
#include <cstring>
#include <atomic>
#include <mutex>

#include "../../include/ptd.h"
#include "verify_sampling.cuh"
#include "draft_update.cuh"
#include "pool.cuh"
#include "tree_rope.cuh"
#include "lm_head.cuh"

namespace ptd {
cudaError_t launch_bounded_wait_check(int32_t* dev_status, cudaStream_t stream);
}
#include "attention.cuh"
#include "topk.cuh"
#include "verify_compact.cuh"
#include "step_checks.cuh"

namespace {

thread_local int32_t g_last_launches = 0;

constexpr int kMaxDevices = 64;

int num_sms_of_current_device() {
  static int cache[kMaxDevices] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (dev >= 0 && dev < kMaxDevices && cache[dev] > 0) return cache[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
  if (dev >= 0 && dev < kMaxDevices) cache[dev] = n;
  return n;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t dtype_size(ptd_dtype d) { return d == PTD_BF16 ? 2 : 4; }

ptd_status check_tree(const ptd_tree* t) {
  if (!t || t->batch < 1 || t->total_nodes < 1 || t->max_nodes < 1 || t->max_nodes > PTD_MAX_TREE_NODES ||
      t->max_ctx < 0 || !t->node_offsets || !t->parents || !t->ctx_lens)
    return PTD_ERR_INVALID_ARG;
  if ((int64_t)t->total_nodes > (int64_t)t->batch * t->max_nodes) return PTD_ERR_INVALID_ARG;
  return PTD_OK;
}

ptd_status check_cache(const ptd_kv_cache* c) {
  if (!c || !c->k || !c->v || c->num_layers < 1 || c->num_kv_heads < 1 || c->head_dim < 1) return PTD_ERR_INVALID_ARG;
  if (c->dtype != PTD_BF16 && c->dtype != PTD_F32) return PTD_ERR_INVALID_ARG;
  if (c->page_size < 0) return PTD_ERR_INVALID_ARG;
  if (c->page_size == 0) {
    if (c->seq_capacity < 1) return PTD_ERR_INVALID_ARG;
  } else {
    if (c->page_size != 16 && c->page_size != 32 && c->page_size != 64 && c->page_size != 128)
      return PTD_ERR_UNSUPPORTED;
    if (c->num_pages < 1 || c->max_pages < 1 || !c->block_table) return PTD_ERR_INVALID_ARG;
  }
  if (!aligned16(c->k) || !aligned16(c->v)) return PTD_ERR_INVALID_ARG;
  if (((size_t)c->num_kv_heads * c->head_dim * dtype_size(c->dtype)) % 16 != 0) return PTD_ERR_UNSUPPORTED;
  return PTD_OK;
}

int64_t cache_rows_per_layer(const ptd_kv_cache* c, int batch) {
  return c->page_size > 0 ? (int64_t)c->num_pages * c->page_size : (int64_t)batch * c->seq_capacity;
}

bool use_tensor_cores(const ptd_kv_cache* c) { return c->dtype == PTD_BF16 && c->head_dim == 128; }

// Number of 256-row M-tile pairs per (tree, KV head) and work units of the tensor-core path.
void tc_geometry(const ptd_tree* t, const ptd_kv_cache* c, int hq, int layers, int* pairs, int* units,
                 int* n_kt_max) {
  const int G = hq / c->num_kv_heads;
  const int rows = t->max_nodes * G;
  const int tiles = (rows + 127) / 128;
  *pairs = (tiles + 1) / 2;
  *units = layers * t->batch * c->num_kv_heads * (*pairs);
  *n_kt_max = (t->max_ctx + t->max_nodes + 127) / 128;
}

// Persistent schedule: one CTA per SM (fewer for tiny problems); per-(unit, 32-row block)
// piece counters and two partial slots per CTA (the pieces at either end of its range).
int persistent_ctas(int units, int n_kt, int sms) {
  const long long w = (long long)units * n_kt;
  return (int)(w < sms ? w : sms);
}

size_t counters_bytes(int units) { return (((size_t)units * 8 * sizeof(unsigned long long)) + 255) / 256 * 256; }

// Epoch of an attention launch: the kernel's piece counters hold (epoch << 32) | count, so a
// counter left by another launch reads as zero and the scratch needs no clearing.  Unique
// per launch in the process (never 0).
uint32_t next_epoch() {
  static std::atomic<uint32_t> epoch{0};
  uint32_t e = epoch.fetch_add(1u) + 1u;
  if (e == 0) e = epoch.fetch_add(1u) + 1u;
  return e;
}

size_t persistent_workspace_bytes(int units, int ctas, int head_dim) {
  return counters_bytes(units) + (size_t)2 * ctas * 256 * ((size_t)head_dim + 2) * sizeof(float);
}

// The step's tail counters (rows done per tree, cleared by the attention's CTA 0), after the
// attention's scratch.
size_t tail_counters_bytes(int batch) { return ((size_t)batch * sizeof(unsigned int) + 255) / 256 * 256; }

// The streaming top-k's tail: the counters per tree and per row (cleared together by the
// attention's CTA 0), then its part slots.
size_t stream_counters_bytes(int batch, int rows) {
  return (((size_t)batch + (size_t)rows) * sizeof(unsigned int) + 255) / 256 * 256;
}
size_t stream_tail_bytes(int batch, int rows, int sms) {
  return stream_counters_bytes(batch, rows) + (ptd::topk_stream_slot_bytes(rows, sms) + 255) / 256 * 256;
}

// Which schedule the shapes favour, from the host-known maxima (estimates in microseconds
// measured on GB300 with these kernels): a key tile costs ~1.75 us for a unit of two 128-row
// M tiles (~1.2 us for one), a CTA needs ~6.5 us to its first tile, and under the balanced
// cut the last piece of a unit merges the others' partials, ~9 us plus ~4 us per partial.
// One CTA per unit (no pieces, no merges) wins when units are few and short, e.g. a single
// MHA layer over a short context; the balanced cut wins as soon as units are long or outnumber
// the SMs.
// Where the pieces of split units are merged: fewer units than CTAs means many pieces per
// unit, merged best by tree_attn_merge_kernel over many CTAs after the attention; otherwise
// the last piece of each unit merges inside the attention, overlapping other CTAs' tiles.
bool defer_merge(int units, int ctas) { return units < ctas; }

bool grid_schedule_cheaper(int units, int n_kt, int m_tiles, int sms) {
  const double t_tile = m_tiles >= 2 ? 1.75 : 1.2;
  const double waves = (double)((units + sms - 1) / sms);
  const double t_grid = 6.5 + waves * n_kt * t_tile;
  const double W = (double)units * n_kt;
  const int ctas = (int)(W < sms ? W : sms);
  const double w = W / ctas;
  const int pieces = (int)((n_kt + w - 1e-9) / w);   // pieces of a unit, about
  double merge = 1.5;
  if (pieces > 1) merge = defer_merge(units, ctas) ? 4.0 + 1.0 * pieces : 9.0 + 4.0 * (pieces - 1);
  const double t_pers = 6.5 + w * t_tile + merge;
  return t_grid < t_pers;
}

// Tile indices of the persistent schedule are 32-bit.
bool persistent_fits(int units, int n_kt) { return (long long)units * n_kt < (1ll << 30); }

ptd_status cuda_status(cudaError_t e) { return e == cudaSuccess ? PTD_OK : PTD_ERR_CUDA; }

}  // namespace

extern "C" {

const char* ptd_status_string(ptd_status s) {
  switch (s) {
    case PTD_OK:
      return "ok";
    case PTD_ERR_INVALID_ARG:
      return "invalid argument";
    case PTD_ERR_INVALID_TREE:
      return "invalid tree (parent array is not a rooted tree in topological order)";
    case PTD_ERR_UNSUPPORTED:
      return "unsupported shape or dtype";
    case PTD_ERR_CUDA:
      return "CUDA error";
    case PTD_ERR_TIMEOUT:
      return "device wait timed out";
    case PTD_ERR_WORKSPACE:
      return "workspace missing or too small";
    case PTD_ERR_POOL_FULL:
      return "candidate pool full: merge refused";
  }
  return "unknown status";
}

int32_t ptd_last_launch_count(void) { return g_last_launches; }

size_t ptd_attention_workspace_size(const ptd_tree* tree, const ptd_kv_cache* cache, int32_t num_q_heads,
                                    int32_t num_layers) {
  if (check_tree(tree) != PTD_OK || check_cache(cache) != PTD_OK || num_q_heads < 1 || num_layers < 1 ||
      num_q_heads % cache->num_kv_heads != 0 || !use_tensor_cores(cache))
    return 0;
  int pairs, units, n_kt;
  tc_geometry(tree, cache, num_q_heads, num_layers, &pairs, &units, &n_kt);
  if (units <= 0 || n_kt <= 0) return 0;
  const int sms = num_sms_of_current_device();
  if (!persistent_fits(units, n_kt)) return 0;
  return persistent_workspace_bytes(units, persistent_ctas(units, n_kt, sms), cache->head_dim);
}

size_t ptd_step_workspace_size(const ptd_tree* tree, const ptd_kv_cache* cache, int32_t num_q_heads) {
  if (check_tree(tree) != PTD_OK || check_cache(cache) != PTD_OK) return 0;
  const size_t attn = ptd_attention_workspace_size(tree, cache, num_q_heads, cache->num_layers);
  return (attn + 255) / 256 * 256 + stream_tail_bytes(tree->batch, tree->total_nodes, num_sms_of_current_device());
}

// ptd_tree_attention, and besides: the tensor-core kernel's CTA 0 clears zero_count words at
// zero_ptr after its dependency wait (the step's tail counters).
static ptd_status tree_attention(const ptd_tree* tree, const ptd_kv_cache* cache, int32_t layer_begin,
                                 int32_t num_layers, const void* q, int32_t num_q_heads, float scale, void* out,
                                 void* workspace, size_t workspace_bytes, int32_t* dev_status, unsigned int* zero_ptr,
                                 int zero_count, void* stream) {
  g_last_launches = 0;
  ptd_status st = check_tree(tree);
  if (st != PTD_OK) return st;
  if ((st = check_cache(cache)) != PTD_OK) return st;
  if (!q || !out || !dev_status || num_q_heads < 1 || num_layers < 1 || layer_begin < 0 ||
      layer_begin + num_layers > cache->num_layers || num_q_heads % cache->num_kv_heads != 0)
    return PTD_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out)) return PTD_ERR_INVALID_ARG;
  const int D = cache->head_dim;
  ptd::AttnParams p = {};
  p.q = q;
  p.out = out;
  p.node_offsets = tree->node_offsets;
  p.parents = tree->parents;
  p.ctx_lens = tree->ctx_lens;
  p.block_table = cache->block_table;
  p.k = cache->k;
  p.v = cache->v;
  p.dev_status = dev_status;
  p.batch = tree->batch;
  p.hq = num_q_heads;
  p.hkv = cache->num_kv_heads;
  p.group = num_q_heads / cache->num_kv_heads;
  p.head_dim = D;
  p.layer_begin = layer_begin;
  p.layers = num_layers;
  p.n_total = tree->total_nodes;
  p.max_nodes = tree->max_nodes;
  p.page_size = cache->page_size;
  p.seq_capacity = cache->seq_capacity;
  p.num_pages = cache->num_pages;
  p.max_pages = cache->max_pages;
  const float sc = scale > 0.f ? scale : 1.0f / std::sqrt((float)D);
  p.scale = sc;
  p.scale_log2 = sc * 1.4426950408889634f;
  p.zero_ptr = zero_ptr;
  p.zero_count = zero_ptr != nullptr ? zero_count : 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);

  if (cache->dtype == PTD_F32) {
    if (D != 32 && D != 64 && D != 128) return PTD_ERR_UNSUPPORTED;
    p.pairs = 1;
    st = cuda_status(ptd::launch_tree_attn_simt(p, s));
    if (st == PTD_OK) g_last_launches = 1;
    return st;
  }
  if (!use_tensor_cores(cache)) return PTD_ERR_UNSUPPORTED;

  int pairs, units, n_kt;
  tc_geometry(tree, cache, num_q_heads, num_layers, &pairs, &units, &n_kt);
  if (units <= 0 || n_kt <= 0) return PTD_ERR_INVALID_ARG;
  p.pairs = pairs;
  const int sms = num_sms_of_current_device();
  const int ctas = persistent_ctas(units, n_kt, sms);
  const int m_tiles = (tree->max_nodes * (num_q_heads / cache->num_kv_heads) + 127) / 128;
  const bool persistent = persistent_fits(units, n_kt) && workspace != nullptr && aligned16(workspace) &&
                          workspace_bytes >= persistent_workspace_bytes(units, ctas, D) &&
                          !grid_schedule_cheaper(units, n_kt, m_tiles, sms);
  dim3 grid;
  if (persistent) {
    p.persistent = 1;
    p.counters = static_cast<unsigned long long*>(workspace);
    p.epoch = next_epoch();
    p.part_o = reinterpret_cast<float*>(static_cast<uint8_t*>(workspace) + counters_bytes(units));
    p.part_ml = p.part_o + (size_t)2 * ctas * 256 * D;
    p.defer_merge = defer_merge(units, ctas) ? 1 : 0;
    p.ctas = ctas;
    grid = dim3((unsigned)ctas, 1, 1);
  } else {
    p.persistent = 0;   // one CTA per unit, no scratch
    grid = dim3((unsigned)units, 1, 1);
  }

  PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
  if (!enc) return PTD_ERR_CUDA;
  const int64_t rows_per_layer = cache_rows_per_layer(cache, tree->batch);
  const cuuint64_t gdim[3] = {(cuuint64_t)D, (cuuint64_t)cache->num_kv_heads,
                              (cuuint64_t)(rows_per_layer * cache->num_layers)};
  const cuuint64_t gstride[2] = {(cuuint64_t)D * 2, (cuuint64_t)cache->num_kv_heads * D * 2};
  const cuuint32_t box[3] = {64, 1, (cuuint32_t)(cache->page_size > 0 ? cache->page_size : 128)};
  const cuuint32_t estride[3] = {1, 1, 1};
  CUtensorMap map_k, map_v;
  if (enc(&map_k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, cache->k, gdim, gstride, box, estride,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return PTD_ERR_CUDA;
  if (enc(&map_v, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, cache->v, gdim, gstride, box, estride,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return PTD_ERR_CUDA;

  // Q tiles by TMA: one M tile is 128 / G nodes x G heads, a 3-D box over [rows][Hq][D]
  CUtensorMap map_q;
  std::memset(&map_q, 0, sizeof(map_q));
  const int G = p.group;
  p.q_tma = 0;
  if (G >= 1 && G <= 128 && 128 % G == 0 && aligned16(q)) {
    const cuuint64_t qdim[3] = {(cuuint64_t)D, (cuuint64_t)num_q_heads, (cuuint64_t)num_layers * tree->total_nodes};
    const cuuint64_t qstride[2] = {(cuuint64_t)D * 2, (cuuint64_t)num_q_heads * D * 2};
    const cuuint32_t qbox[3] = {64, (cuuint32_t)G, (cuuint32_t)(128 / G)};
    if (enc(&map_q, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), qdim, qstride, qbox, estride,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS)
      p.q_tma = 1;
  }
  if ((st = cuda_status(ptd::launch_tree_attn_tc(map_k, map_v, map_q, p, grid, s))) != PTD_OK) return st;
  g_last_launches = 1;
  if (p.persistent && p.defer_merge) {
    if ((st = cuda_status(ptd::launch_tree_attn_merge(p, units, sms, s))) != PTD_OK) return st;
    g_last_launches = 2;
  }
  return PTD_OK;
}

ptd_status ptd_tree_attention(const ptd_tree* tree, const ptd_kv_cache* cache, int32_t layer_begin,
                              int32_t num_layers, const void* q, int32_t num_q_heads, float scale, void* out,
                              void* workspace, size_t workspace_bytes, int32_t* dev_status, void* stream) {
  return tree_attention(tree, cache, layer_begin, num_layers, q, num_q_heads, scale, out, workspace, workspace_bytes,
                        dev_status, nullptr, 0, stream);
}

// Host checks of ptd_topk_draft's arguments (no launch).
static ptd_status check_topk_args(const void* logits, ptd_dtype dtype, int64_t rows, int32_t vocab,
                                  int64_t row_stride, int32_t k, const int32_t* out_idx, const float* out_val) {
  if (!logits || !out_idx || !out_val || rows < 1 || vocab < 1 || row_stride < vocab || k < 1 ||
      k > PTD_MAX_TOPK || k > vocab)
    return PTD_ERR_INVALID_ARG;
  if (dtype != PTD_BF16 && dtype != PTD_F32) return PTD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(logits) % dtype_size(dtype)) != 0) return PTD_ERR_INVALID_ARG;
  return PTD_OK;
}

static ptd_status topk_draft(const void* logits, ptd_dtype dtype, int64_t rows, int32_t vocab, int64_t row_stride,
                             int32_t k, int32_t* out_idx, float* out_val, void* stream) {
  g_last_launches = 0;
  ptd_status st0 = check_topk_args(logits, dtype, rows, vocab, row_stride, k, out_idx, out_val);
  if (st0 != PTD_OK) return st0;
  const ptd_status st = cuda_status(ptd::launch_topk(logits, dtype == PTD_BF16, rows, vocab, row_stride, k, out_idx,
                                                     out_val, nullptr, nullptr, static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 1;
  return st;
}

ptd_status ptd_topk_draft(const void* logits, ptd_dtype dtype, int64_t rows, int32_t vocab, int64_t row_stride,
                          int32_t k, int32_t* out_idx, float* out_val, void* stream) {
  return topk_draft(logits, dtype, rows, vocab, row_stride, k, out_idx, out_val, stream);
}

ptd_status ptd_verify_greedy(const ptd_tree* tree, const int32_t* tokens, const int32_t* target,
                             int32_t target_stride, int32_t* accepted_nodes, int32_t* accept_len,
                             int32_t* bonus_token, int32_t* dev_status, void* stream) {
  g_last_launches = 0;
  ptd_status st = check_tree(tree);
  if (st != PTD_OK) return st;
  if (!tokens || !target || target_stride < 1 || !accepted_nodes || !accept_len || !bonus_token || !dev_status)
    return PTD_ERR_INVALID_ARG;
  st = cuda_status(ptd::launch_verify(tree->node_offsets, tree->parents, tokens, target, target_stride, tree->batch,
                                      tree->total_nodes, tree->max_nodes, accepted_nodes, accept_len, bonus_token,
                                      dev_status, static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 1;
  return st;
}

ptd_status ptd_kv_compact(const ptd_tree* tree, const ptd_kv_cache* cache, const int32_t* accepted_nodes,
                          const int32_t* accept_len, int32_t* new_ctx_lens, void* stream) {
  g_last_launches = 0;
  ptd_status st = check_tree(tree);
  if (st != PTD_OK) return st;
  if ((st = check_cache(cache)) != PTD_OK) return st;
  if (!accepted_nodes || !accept_len || !new_ctx_lens) return PTD_ERR_INVALID_ARG;
  if (new_ctx_lens == tree->ctx_lens) return PTD_ERR_INVALID_ARG;   // other CTAs still read ctx_lens
  const int row_bytes = cache->num_kv_heads * cache->head_dim * (int)dtype_size(cache->dtype);
  st = cuda_status(ptd::launch_compact(cache->k, cache->v, row_bytes, cache->num_layers, tree->batch,
                                       cache->page_size, cache->seq_capacity, cache->num_pages, cache->block_table,
                                       cache->max_pages, tree->ctx_lens, accepted_nodes, accept_len,
                                       tree->max_nodes, new_ctx_lens, static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 1;
  return st;
}

ptd_status ptd_verify_sampling(const ptd_tree* tree, const int32_t* tokens, const void* logits, ptd_dtype dtype,
                               int32_t vocab, int64_t row_stride, float temperature, const float* u_accept,
                               const float* u_bonus, int32_t* accepted_nodes, int32_t* accept_len,
                               int32_t* bonus_token, int32_t* dev_status, void* stream) {
  g_last_launches = 0;
  ptd_status st = check_tree(tree);
  if (st != PTD_OK) return st;
  if (!tokens || !logits || !u_accept || !u_bonus || !accepted_nodes || !accept_len || !bonus_token || !dev_status)
    return PTD_ERR_INVALID_ARG;
  if (dtype != PTD_BF16 && dtype != PTD_F32) return PTD_ERR_INVALID_ARG;
  if (vocab < 1 || row_stride < vocab || !(temperature > 0.f) || !std::isfinite(temperature))
    return PTD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(logits) % dtype_size(dtype)) != 0) return PTD_ERR_INVALID_ARG;
  st = cuda_status(ptd::launch_verify_sampling(tree->node_offsets, tree->parents, tokens, logits, dtype == PTD_BF16,
                                               vocab, row_stride, 1.0f / temperature, u_accept, u_bonus, tree->batch,
                                               tree->total_nodes, tree->max_nodes, accepted_nodes, accept_len,
                                               bonus_token, dev_status, static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 1;
  return st;
}

// Host checks of ptd_verify_and_compact's arguments (no launch).
static ptd_status check_verify_compact_args(const ptd_tree* tree, const ptd_kv_cache* cache, const int32_t* tokens,
                                            const int32_t* target, int32_t target_stride,
                                            const int32_t* accepted_nodes, const int32_t* accept_len,
                                            const int32_t* bonus_token, const int32_t* new_ctx_lens,
                                            const int32_t* dev_status) {
  ptd_status st = check_tree(tree);
  if (st != PTD_OK) return st;
  if ((st = check_cache(cache)) != PTD_OK) return st;
  if (!tokens || !target || target_stride < 1 || !accepted_nodes || !accept_len || !bonus_token || !dev_status ||
      !new_ctx_lens)
    return PTD_ERR_INVALID_ARG;
  if (new_ctx_lens == tree->ctx_lens) return PTD_ERR_INVALID_ARG;   // other CTAs still read ctx_lens
  return PTD_OK;
}

static ptd_status verify_and_compact(const ptd_tree* tree, const ptd_kv_cache* cache, const int32_t* tokens,
                                     const int32_t* target, int32_t target_stride, int32_t* accepted_nodes,
                                     int32_t* accept_len, int32_t* bonus_token, int32_t* new_ctx_lens,
                                     int32_t* dev_status, void* stream) {
  g_last_launches = 0;
  ptd_status st = check_verify_compact_args(tree, cache, tokens, target, target_stride, accepted_nodes, accept_len,
                                            bonus_token, new_ctx_lens, dev_status);
  if (st != PTD_OK) return st;
  const int row_bytes = cache->num_kv_heads * cache->head_dim * (int)dtype_size(cache->dtype);
  st = cuda_status(ptd::launch_verify_compact(
      tree->node_offsets, tree->parents, tokens, target, target_stride, tree->total_nodes, tree->max_nodes,
      accepted_nodes, accept_len, bonus_token, dev_status, cache->k, cache->v, row_bytes, cache->num_layers,
      tree->batch, cache->page_size, cache->seq_capacity, cache->num_pages, cache->block_table, cache->max_pages,
      tree->ctx_lens, new_ctx_lens, static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 1;
  return st;
}

ptd_status ptd_verify_and_compact(const ptd_tree* tree, const ptd_kv_cache* cache, const int32_t* tokens,
                                  const int32_t* target, int32_t target_stride, int32_t* accepted_nodes,
                                  int32_t* accept_len, int32_t* bonus_token, int32_t* new_ctx_lens,
                                  int32_t* dev_status, void* stream) {
  return verify_and_compact(tree, cache, tokens, target, target_stride, accepted_nodes, accept_len, bonus_token,
                            new_ctx_lens, dev_status, stream);
}

ptd_status ptd_draft_tree_update(int32_t batch, int32_t in_stride, const int32_t* in_count, const int32_t* in_parents,
                                 const int32_t* in_tokens, const int32_t* drafts, int32_t draft_stride, int32_t expand,
                                 int32_t width, int32_t max_depth, int32_t capacity, int32_t* out_count,
                                 int32_t* out_parents, int32_t* out_tokens, int32_t* out_depths, int32_t* old_to_new,
                                 int32_t* dev_status, void* stream) {
  g_last_launches = 0;
  if (batch < 1 || batch > 65535 || in_stride < 1 || capacity < 1 || capacity > PTD_MAX_TREE_NODES ||
      expand < 0 || expand > ptd::kMaxExpand || draft_stride < 1 || expand > draft_stride || width < 0 ||
      max_depth < 1)
    return PTD_ERR_INVALID_ARG;
  if (!in_count || !in_parents || !in_tokens || !drafts || !out_count || !out_parents || !out_tokens ||
      !out_depths || !old_to_new || !dev_status)
    return PTD_ERR_INVALID_ARG;
  // the output must not alias the input (other threads of the CTA still read it)
  if (out_parents == in_parents || out_tokens == in_tokens || out_count == in_count) return PTD_ERR_INVALID_ARG;
  const ptd_status st = cuda_status(ptd::launch_draft_update(
      batch, in_stride, in_count, in_parents, in_tokens, drafts, draft_stride, expand, width, max_depth, capacity,
      out_count, out_parents, out_tokens, out_depths, old_to_new, dev_status, static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 1;
  return st;
}

namespace {
bool pool_capacity_ok(int32_t capacity) {
  return capacity >= 16 && capacity <= (1 << 28) && (capacity & (capacity - 1)) == 0;
}
}  // namespace

size_t ptd_pool_bytes(int32_t capacity) { return pool_capacity_ok(capacity) ? ptd::pool_bytes(capacity) : 0; }

ptd_status ptd_pool_init(void* pool, int32_t capacity, void* stream) {
  g_last_launches = 0;
  if (!pool || !pool_capacity_ok(capacity) || !aligned16(pool)) return PTD_ERR_INVALID_ARG;
  return cuda_status(ptd::pool_init(pool, capacity, static_cast<cudaStream_t>(stream)));
}

ptd_status ptd_pool_merge(void* pool, int32_t capacity, int32_t max_load, int32_t step, const int32_t* count,
                          const int32_t* parents, const int32_t* tokens, int32_t* dev_status, void* stream) {
  g_last_launches = 0;
  if (!pool || !pool_capacity_ok(capacity) || !aligned16(pool) || max_load < 0 || max_load > capacity ||
      step < 0 || !count || !parents || !tokens || !dev_status)
    return PTD_ERR_INVALID_ARG;
  const ptd_status st = cuda_status(ptd::launch_pool_merge(pool, capacity, max_load, step, count, parents, tokens,
                                                           dev_status, static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 1;
  return st;
}

ptd_status ptd_pool_retrieve(const void* pool, int32_t capacity, const int32_t* root_token, int32_t width,
                             int32_t max_depth, int32_t max_nodes, int32_t* out_count, int32_t* out_parents,
                             int32_t* out_tokens, void* stream) {
  g_last_launches = 0;
  if (!pool || !pool_capacity_ok(capacity) || !aligned16(pool) || !root_token || width < 1 ||
      width > ptd::kPoolKids || max_depth < 1 || max_nodes < 1 || max_nodes > PTD_MAX_TREE_NODES || !out_count ||
      !out_parents || !out_tokens)
    return PTD_ERR_INVALID_ARG;
  const ptd_status st =
      cuda_status(ptd::launch_pool_retrieve(pool, capacity, root_token, width, max_depth, max_nodes, out_count,
                                            out_parents, out_tokens, static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 1;
  return st;
}

ptd_status ptd_tree_rope_append(const ptd_tree* tree, const ptd_kv_cache* cache, int32_t layer_begin,
                                int32_t num_layers, void* q, int32_t num_q_heads, const void* k, const void* v,
                                float rope_base, int32_t* positions_out, int32_t* dev_status, void* stream) {
  g_last_launches = 0;
  ptd_status st = check_tree(tree);
  if (st != PTD_OK) return st;
  if ((st = check_cache(cache)) != PTD_OK) return st;
  const int D = cache->head_dim, hkv = cache->num_kv_heads;
  if (layer_begin < 0 || num_layers < 1 || num_layers > 65535 || layer_begin + num_layers > cache->num_layers ||
      num_q_heads < hkv || num_q_heads % hkv != 0 || D % 2 != 0 ||
      D / 2 > ptd::kMaxRopeHalf || !q || !k || !v || !dev_status || !(rope_base > 1.f) || !std::isfinite(rope_base))
    return PTD_ERR_INVALID_ARG;
  const size_t es = dtype_size(cache->dtype);
  if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k) | reinterpret_cast<uintptr_t>(v)) % es != 0)
    return PTD_ERR_INVALID_ARG;
  ptd::RopeFreqs f = {};
  for (int j = 0; j < D / 2; ++j) {
    const double x = std::pow((double)rope_base, -2.0 * j / D);
    f.hi[j] = (float)x;
    f.lo[j] = (float)(x - (double)f.hi[j]);
  }
  st = cuda_status(ptd::launch_tree_rope(tree->node_offsets, tree->parents, tree->ctx_lens, tree->batch,
                                         tree->total_nodes, cache->dtype == PTD_BF16, D, num_q_heads, hkv, q, k, v,
                                         cache->k, cache->v, layer_begin, num_layers, cache->page_size,
                                         cache->seq_capacity,
                                         cache->num_pages, cache->block_table, cache->max_pages, f, positions_out,
                                         dev_status, static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 1;
  return st;
}

ptd_status ptd_check_bounded_wait(int32_t* dev_status, void* stream) {
  g_last_launches = 0;
  if (!dev_status) return PTD_ERR_INVALID_ARG;
  const ptd_status st = cuda_status(ptd::launch_bounded_wait_check(dev_status, static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 1;
  return st;
}

size_t ptd_lm_head_topk_workspace_size(int32_t rows, int32_t vocab) {
  if (rows < 1 || rows > PTD_MAX_TREE_NODES || vocab < 1) return 0;
  return ptd::lm_head_workspace_bytes(ptd::lm_head_ctas(num_sms_of_current_device(), vocab), rows);
}

ptd_status ptd_lm_head_topk(const void* hidden, int32_t rows, int64_t hidden_stride, const void* weight,
                            int32_t vocab, int64_t weight_stride, int32_t d_model, int32_t k, int32_t* out_idx,
                            float* out_val, void* workspace, size_t workspace_bytes, int32_t* dev_status,
                            void* stream) {
  g_last_launches = 0;
  if (!hidden || !weight || !out_idx || !out_val || !dev_status) return PTD_ERR_INVALID_ARG;
  if (rows < 1 || rows > PTD_MAX_TREE_NODES || d_model < 64 || d_model % 64 != 0 || k < 1 || k > ptd::kLmMaxK ||
      vocab < k || hidden_stride < d_model || weight_stride < d_model || hidden_stride % 8 != 0 ||
      weight_stride % 8 != 0 || !aligned16(hidden) || !aligned16(weight))
    return PTD_ERR_INVALID_ARG;
  const int ctas = ptd::lm_head_ctas(num_sms_of_current_device(), vocab);
  if (!workspace || workspace_bytes < ptd::lm_head_workspace_bytes(ctas, rows) || !aligned16(workspace))
    return PTD_ERR_WORKSPACE;
  PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
  if (!enc) return PTD_ERR_CUDA;
  CUtensorMap map_h, map_w;
  const cuuint32_t box[2] = {64, 128}, estride[2] = {1, 1};
  const cuuint64_t hdim[2] = {(cuuint64_t)d_model, (cuuint64_t)rows};
  const cuuint64_t hstride[1] = {(cuuint64_t)hidden_stride * 2};
  const cuuint64_t wdim[2] = {(cuuint64_t)d_model, (cuuint64_t)vocab};
  const cuuint64_t wstride[1] = {(cuuint64_t)weight_stride * 2};
  if (enc(&map_h, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(hidden), hdim, hstride, box, estride,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return PTD_ERR_CUDA;
  if (enc(&map_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(weight), wdim, wstride, box, estride,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return PTD_ERR_CUDA;
  const ptd_status st = cuda_status(ptd::launch_lm_head_topk(map_h, map_w, rows, d_model, vocab, k, out_idx, out_val,
                                                              workspace, ctas, dev_status,
                                                              static_cast<cudaStream_t>(stream)));
  if (st == PTD_OK) g_last_launches = 2;
  return st;
}

namespace {
std::atomic<int> g_step_topk{PTD_STEP_TOPK_AUTO};

constexpr int kTailSeparate = 0, kTailClustered = 1, kTailStreamed = 2;

// The step's tail for checked arguments.  The streaming top-k needs rows back to back on
// 16-byte vectors and the whole tail of ptd_step_workspace_size; the clustered one only the
// per-tree counters; both need the tensor-core attention (which clears the counters) and bf16
// logits.  With both possible the policy decides (auto: stream when the clustered grid, at
// three CTAs per SM, would need more than one wave).
int step_tail(const ptd_tree* tree, const ptd_kv_cache* cache, const ptd_step_args* a, size_t* attn_ws_out,
              int* sms_out) {
  const size_t attn_ws = (ptd_attention_workspace_size(tree, cache, a->num_q_heads, cache->num_layers) + 255) /
                         256 * 256;
  const int sms = num_sms_of_current_device();
  *attn_ws_out = attn_ws;
  *sms_out = sms;
  const bool tail_ok = use_tensor_cores(cache) && a->logits_dtype == PTD_BF16 && a->workspace &&
                       aligned16(a->workspace);
  const bool can_stream = tail_ok && ptd::topk_stream_ok(a->logits, a->vocab) &&
                          a->workspace_bytes >= attn_ws + stream_tail_bytes(tree->batch, tree->total_nodes, sms);
  const bool can_cluster = tail_ok && ptd::topk_can_verify(true, a->vocab) &&
                           a->workspace_bytes >= attn_ws + tail_counters_bytes(tree->batch);
  if (can_stream && can_cluster) {
    const int policy = g_step_topk.load();
    const int64_t cluster_ctas = (int64_t)tree->total_nodes * ptd::topk_cluster_size(a->vocab);
    const bool stream = policy == PTD_STEP_TOPK_STREAMED ||
                        (policy == PTD_STEP_TOPK_AUTO && cluster_ctas > 3 * (int64_t)sms);
    return stream ? kTailStreamed : kTailClustered;
  }
  return can_stream ? kTailStreamed : (can_cluster ? kTailClustered : kTailSeparate);
}
}  // namespace

int32_t ptd_step_tail(const ptd_tree* tree, const ptd_kv_cache* cache, const ptd_step_args* a) {
  if (!a || !tree || !cache || check_tree(tree) != PTD_OK || check_cache(cache) != PTD_OK || a->num_q_heads < 1)
    return -1;
  size_t attn_ws = 0;
  int sms = 0;
  return step_tail(tree, cache, a, &attn_ws, &sms);
}

int32_t ptd_step_topk_policy(int32_t policy) {
  if (policy != PTD_STEP_TOPK_AUTO && policy != PTD_STEP_TOPK_CLUSTERED && policy != PTD_STEP_TOPK_STREAMED) return -1;
  return g_step_topk.exchange(policy);
}

ptd_status ptd_tree_verify_step(const ptd_tree* tree, const ptd_kv_cache* cache, const ptd_step_args* a,
                                void* stream) {
  g_last_launches = 0;
  if (!a) return PTD_ERR_INVALID_ARG;
  // Every host check of the three parts before the first launch, so that an error enqueues
  // nothing (the attention call checks its own arguments before it launches).
  ptd_status st = check_verify_compact_args(tree, cache, a->tokens, a->topk_idx, a->k, a->accepted_nodes,
                                            a->accept_len, a->bonus_token, a->new_ctx_lens, a->dev_status);
  if (st != PTD_OK) return st;
  if ((st = check_topk_args(a->logits, a->logits_dtype, tree->total_nodes, a->vocab, a->vocab, a->k, a->topk_idx,
                            a->topk_val)) != PTD_OK)
    return st;
  // The tail: with room for its counters after the attention's scratch (the size given by
  // ptd_step_workspace_size), the tensor-core attention (which clears those counters) and bf16
  // logits on the clustered path, the top-k kernel also verifies every tree (the cluster that
  // writes a tree's last row does it) and a copy kernel compacts.  Otherwise the top-k, then
  // verification + compaction in one launch.  Each launch may be placed while the previous one
  // drains; it reads its inputs only after that one has completed (the top-k's logits come from
  // the step's forward pass).
  size_t attn_ws = 0;
  int sms = 0;
  const int tail = step_tail(tree, cache, a, &attn_ws, &sms);
  const bool streamed = tail == kTailStreamed;
  const bool fused = tail != kTailSeparate;
  unsigned int* tail_counters =
      fused ? reinterpret_cast<unsigned int*>(static_cast<uint8_t*>(a->workspace) + attn_ws) : nullptr;
  const int zero_count = streamed ? tree->batch + tree->total_nodes : tree->batch;
  int total = 0;
  st = tree_attention(tree, cache, 0, cache->num_layers, a->q, a->num_q_heads, a->scale, a->attn_out, a->workspace,
                      a->workspace_bytes, a->dev_status, tail_counters, zero_count, stream);
  if (st != PTD_OK) return st;
  total += g_last_launches;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (fused) {
    ptd::VerifyArgs va = {};
    va.node_offsets = tree->node_offsets;
    va.parents = tree->parents;
    va.tokens = a->tokens;
    va.ctx_lens = tree->ctx_lens;
    va.counters = tail_counters;
    va.batch = tree->batch;
    va.n_total = tree->total_nodes;
    va.max_nodes = tree->max_nodes;
    va.accepted = a->accepted_nodes;
    va.accept_len = a->accept_len;
    va.bonus = a->bonus_token;
    va.dev_status = a->dev_status;
    if (streamed) {
      unsigned long long* slots = reinterpret_cast<unsigned long long*>(
          static_cast<uint8_t*>(a->workspace) + attn_ws + stream_counters_bytes(tree->batch, tree->total_nodes));
      st = cuda_status(ptd::launch_topk_stream(a->logits, tree->total_nodes, a->vocab, a->k, a->topk_idx, a->topk_val,
                                               a->dev_status, va, tail_counters + tree->batch, slots, sms, s));
    } else {
      st = cuda_status(ptd::launch_topk(a->logits, true, tree->total_nodes, a->vocab, a->vocab, a->k, a->topk_idx,
                                        a->topk_val, a->dev_status, &va, s));
    }
    if (st != PTD_OK) return st;
    const int row_bytes = cache->num_kv_heads * cache->head_dim * (int)dtype_size(cache->dtype);
    if ((st = cuda_status(ptd::launch_compact(cache->k, cache->v, row_bytes, cache->num_layers, tree->batch,
                                              cache->page_size, cache->seq_capacity, cache->num_pages,
                                              cache->block_table, cache->max_pages, tree->ctx_lens, a->accepted_nodes,
                                              a->accept_len, tree->max_nodes, a->new_ctx_lens, s))) != PTD_OK)
      return st;
    g_last_launches = total + 2;
    return PTD_OK;
  }
  st = topk_draft(a->logits, a->logits_dtype, tree->total_nodes, a->vocab, a->vocab, a->k, a->topk_idx,
                  a->topk_val, stream);
  if (st != PTD_OK) return st;
  total += g_last_launches;
  st = verify_and_compact(tree, cache, a->tokens, a->topk_idx, a->k, a->accepted_nodes, a->accept_len,
                          a->bonus_token, a->new_ctx_lens, a->dev_status, stream);
  if (st != PTD_OK) return st;
  total += g_last_launches;
  g_last_launches = total;
  return PTD_OK;
}

ptd_status ptd_tree_verify_step_host(const ptd_tree* tree, const ptd_kv_cache* cache, const ptd_step_args* a,
                                     const ptd_host_io* io, void* stream) {
  if (!a || !io) return PTD_ERR_INVALID_ARG;
  ptd_status st = check_tree(tree);
  if (st != PTD_OK) return st;
  if ((st = check_cache(cache)) != PTD_OK) return st;
  if (cache->page_size != 0) return PTD_ERR_UNSUPPORTED;
  if (!io->q_h || !io->logits_h || !io->tokens_h || !io->parents_h || !io->node_offsets_h || !io->ctx_lens_h ||
      !io->tree_k_h || !io->tree_v_h || !io->topk_idx_h || !io->topk_val_h || !io->accepted_h ||
      !io->accept_len_h || !io->bonus_h || !io->new_ctx_h || !io->status_h)
    return PTD_ERR_INVALID_ARG;
  // the checks of the step itself and of the host tree layout before the first copy, so
  // that an error enqueues nothing
  if (!a->q || !a->logits) return PTD_ERR_INVALID_ARG;
  if ((st = check_verify_compact_args(tree, cache, a->tokens, a->topk_idx, a->k, a->accepted_nodes, a->accept_len,
                                      a->bonus_token, a->new_ctx_lens, a->dev_status)) != PTD_OK)
    return st;
  if ((st = check_topk_args(a->logits, a->logits_dtype, tree->total_nodes, a->vocab, a->vocab, a->k, a->topk_idx,
                            a->topk_val)) != PTD_OK)
    return st;
  if ((st = ptd::check_host_tree_layout(tree, cache, io->node_offsets_h, io->ctx_lens_h)) != PTD_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int B = tree->batch, N = tree->total_nodes, L = cache->num_layers;
  const size_t es = dtype_size(cache->dtype);
  const size_t slot_bytes = (size_t)cache->num_kv_heads * cache->head_dim * es;
  const size_t qbytes = (size_t)L * N * a->num_q_heads * cache->head_dim * es;
  const size_t lbytes = (size_t)N * a->vocab * dtype_size(a->logits_dtype);
  auto h2d = [&](void* dst, const void* src, size_t n) {
    return cudaMemcpyAsync(dst, src, n, cudaMemcpyHostToDevice, s);
  };
  cudaError_t e = cudaSuccess;
  if (e == cudaSuccess) e = h2d(const_cast<void*>(a->q), io->q_h, qbytes);
  if (e == cudaSuccess) e = h2d(const_cast<void*>(a->logits), io->logits_h, lbytes);
  if (e == cudaSuccess) e = h2d(const_cast<int32_t*>(a->tokens), io->tokens_h, (size_t)N * 4);
  if (e == cudaSuccess) e = h2d(const_cast<int32_t*>(tree->parents), io->parents_h, (size_t)N * 4);
  if (e == cudaSuccess) e = h2d(const_cast<int32_t*>(tree->node_offsets), io->node_offsets_h, (size_t)(B + 1) * 4);
  if (e == cudaSuccess) e = h2d(const_cast<int32_t*>(tree->ctx_lens), io->ctx_lens_h, (size_t)B * 4);
  if (e == cudaSuccess) e = cudaMemsetAsync(a->dev_status, 0, 4, s);
  // the tree's own K/V rows go to slots C_b .. C_b + T_b - 1 of every layer
  const size_t layer_pitch = (size_t)B * cache->seq_capacity * slot_bytes;
  for (int b = 0; b < B && e == cudaSuccess; ++b) {
    const int off = io->node_offsets_h[b], T = io->node_offsets_h[b + 1] - off, C = io->ctx_lens_h[b];
    const size_t dst_off = ((size_t)b * cache->seq_capacity + C) * slot_bytes;
    const size_t src_off = (size_t)off * slot_bytes;
    for (int kv = 0; kv < 2 && e == cudaSuccess; ++kv) {
      uint8_t* dst = static_cast<uint8_t*>(kv ? cache->v : cache->k) + dst_off;
      const uint8_t* src = static_cast<const uint8_t*>(kv ? io->tree_v_h : io->tree_k_h) + src_off;
      e = cudaMemcpy2DAsync(dst, layer_pitch, src, (size_t)N * slot_bytes, (size_t)T * slot_bytes, (size_t)L,
                            cudaMemcpyHostToDevice, s);
    }
  }
  if (e != cudaSuccess) return PTD_ERR_CUDA;
  st = ptd_tree_verify_step(tree, cache, a, stream);
  if (st != PTD_OK) return st;
  const int32_t launches = g_last_launches;
  auto d2h = [&](void* dst, const void* src, size_t n) {
    return cudaMemcpyAsync(dst, src, n, cudaMemcpyDeviceToHost, s);
  };
  if (e == cudaSuccess) e = d2h(io->topk_idx_h, a->topk_idx, (size_t)N * a->k * 4);
  if (e == cudaSuccess) e = d2h(io->topk_val_h, a->topk_val, (size_t)N * a->k * 4);
  if (e == cudaSuccess) e = d2h(io->accepted_h, a->accepted_nodes, (size_t)B * tree->max_nodes * 4);
  if (e == cudaSuccess) e = d2h(io->accept_len_h, a->accept_len, (size_t)B * 4);
  if (e == cudaSuccess) e = d2h(io->bonus_h, a->bonus_token, (size_t)B * 4);
  if (e == cudaSuccess) e = d2h(io->new_ctx_h, a->new_ctx_lens, (size_t)B * 4);
  if (e == cudaSuccess) e = d2h(io->status_h, a->dev_status, 4);
  g_last_launches = launches;
  return e == cudaSuccess ? PTD_OK : PTD_ERR_CUDA;
}

}  // extern "C"

namespace ptd {
ptd_status check_host_tree_layout(const ptd_tree* tree, const ptd_kv_cache* cache, const int32_t* node_offsets_h,
                                  const int32_t* ctx_lens_h) {
  if (!tree || !cache || !node_offsets_h || !ctx_lens_h) return PTD_ERR_INVALID_ARG;
  if (node_offsets_h[0] != 0 || node_offsets_h[tree->batch] != tree->total_nodes) return PTD_ERR_INVALID_ARG;
  for (int b = 0; b < tree->batch; ++b) {
    const int64_t T = (int64_t)node_offsets_h[b + 1] - node_offsets_h[b], C = ctx_lens_h[b];
    const int64_t cap = cache->page_size > 0 ? (int64_t)cache->max_pages * cache->page_size : cache->seq_capacity;
    if (T < 1 || T > tree->max_nodes || C < 0 || C + T > cap) return PTD_ERR_INVALID_ARG;
  }
  return PTD_OK;
}

ptd_status check_step_args(const ptd_tree* tree, const ptd_kv_cache* cache, const ptd_step_args* a) {
  if (!a || !a->q || !a->logits) return PTD_ERR_INVALID_ARG;
  ptd_status st = check_verify_compact_args(tree, cache, a->tokens, a->topk_idx, a->k, a->accepted_nodes,
                                            a->accept_len, a->bonus_token, a->new_ctx_lens, a->dev_status);
  if (st != PTD_OK) return st;
  return check_topk_args(a->logits, a->logits_dtype, tree->total_nodes, a->vocab, a->vocab, a->k, a->topk_idx,
                         a->topk_val);
}
}  // namespace ptd
