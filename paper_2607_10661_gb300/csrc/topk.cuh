// Internal launcher of the per-node top-k kernel (not part of the C ABI).
#pragma once
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

namespace ptd {
// Greedy verification of each tree by the top-k cluster that completes the tree's rows (the
// step's tail): rows are the trees' nodes, back to back.
struct VerifyArgs {
  const int32_t* node_offsets;   // [batch + 1]
  const int32_t* parents;        // [n_total]
  const int32_t* tokens;         // [n_total]
  const int32_t* ctx_lens;       // [batch]
  unsigned int* counters;        // [batch] rows done per tree, zero before the launch
  int batch, n_total, max_nodes;
  int32_t* accepted;             // [batch][max_nodes]
  int32_t* accept_len;           // [batch]
  int32_t* bonus;                // [batch]
  int32_t* dev_status;
};

// The step's streaming top-k with verification (bf16 rows back to back, vocab a multiple of 8,
// logits 16-byte aligned): a persistent grid of at most 2 * sms CTAs, each over an equal share
// of the rows' bytes.  row_counters [rows] (and va.counters) must be zero before the launch;
// part_keys holds topk_stream_slot_bytes(rows, sms) bytes of scratch (no clearing needed).
bool topk_stream_ok(const void* logits, int vocab);
size_t topk_stream_slot_bytes(int64_t rows, int sms);
cudaError_t launch_topk_stream(const void* logits, int64_t rows, int vocab, int k, int32_t* out_idx, float* out_val,
                               int32_t* dev_status, const VerifyArgs& va, unsigned int* row_counters,
                               unsigned long long* part_keys, int sms, cudaStream_t stream);

// CTAs per row of the clustered bf16 top-k (one cluster per row).
int topk_cluster_size(int vocab);

// Whether launch_topk can verify for these logits (bf16 rows within the clustered fast path).
bool topk_can_verify(bool bf16, int vocab);

// Launched with programmatic stream serialization: the kernel waits for the stream's previous
// grid before its first global access and lets the next grid be placed early.  With `va`
// (bf16 fast path only) it also verifies every tree, as ptd_verify_greedy on its column 0 would;
// the node_offsets / parents / tokens it reads must have been complete before the stream's
// previous grid began.
cudaError_t launch_topk(const void* logits, bool bf16, int64_t rows, int vocab, int64_t row_stride, int k,
                        int32_t* out_idx, float* out_val, int32_t* dev_status, const VerifyArgs* va,
                        cudaStream_t stream);
}  // namespace ptd
