// Tree attention without a caller workspace: the scratch is a file-scope device array of
// PTD_STATIC_SCRATCH_BYTES (declared in include/ptd.h).
//
// In host code the array's name only stands for the symbol; its device address is looked
// up once per device with cudaGetSymbolAddress (with that device current) and cached for
// the life of the process (a device reset, which reloads the module, is not supported).
// The piece counters at the front of the scratch carry the launch's epoch, so a value left by
// an earlier call counts as zero; the partials written by one call are read back only by that
// same call, and each partial row is written before it is read, so nothing needs clearing.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "../../include/ptd.h"

namespace {

constexpr int kMaxNoallocDevices = 64;

static __device__ __align__(256) unsigned char g_attention_scratch[PTD_STATIC_SCRATCH_BYTES];

std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxNoallocDevices] = {};

// Device address of the scratch array on the current device (set up on first use).
ptd_status scratch_on_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return PTD_ERR_CUDA;
  if (dev < 0 || dev >= kMaxNoallocDevices) return PTD_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_attention_scratch) != cudaSuccess || p == nullptr) return PTD_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return PTD_OK;
}

}  // namespace

extern "C" ptd_status ptd_tree_attention_noalloc(const ptd_tree* tree, const ptd_kv_cache* cache,
                                                 int32_t layer_begin, int32_t num_layers, const void* q,
                                                 int32_t num_q_heads, float scale, void* out, int32_t* dev_status,
                                                 void* stream) {
  // the cheap argument checks first: an invalid call returns before the symbol lookup
  if (!tree || !cache || !q || !out || !dev_status || num_q_heads < 1 || num_layers < 1 || layer_begin < 0 ||
      layer_begin + num_layers > cache->num_layers)
    return PTD_ERR_INVALID_ARG;
  const size_t need = ptd_attention_workspace_size(tree, cache, num_q_heads, num_layers);
  if (need > PTD_STATIC_SCRATCH_BYTES) return PTD_ERR_WORKSPACE;
  void* scratch = nullptr;
  const ptd_status st = scratch_on_current_device(&scratch);
  if (st != PTD_OK) return st;
  return ptd_tree_attention(tree, cache, layer_begin, num_layers, q, num_q_heads, scale, out, scratch,
                            PTD_STATIC_SCRATCH_BYTES, dev_status, stream);
}
