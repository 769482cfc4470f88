/*
 * ptd.h -- C ABI of the Progressive Tree Drafting (PTD) tree-verify step on one GPU.
 *
 * One step of PTD (Alg. 1, steps 2 and 5-6) runs the target model once over the
 * committed prefix X followed by a rooted token tree (the draft tree T and the
 * retrieved candidate tree C_X hang below the current token, Sec. 3.2), reads the
 * greedy token of every tree node, accepts the longest root path whose edges are
 * eligible, and appends it to X.  This library exposes the data-parallel part of
 * that step as four calls:
 *
 *   ptd_tree_attention   tree-masked attention, ancestor-only visibility (Sec. 3.1)
 *   ptd_topk_draft       per-node top-k of the logits: draft tokens d_v, width
 *                        control, greedy verification tokens V_n (Sec. 3.1, 3.2)
 *   ptd_verify_greedy    eligible edges I and accepted sequence X' (Sec. 3.2)
 *   ptd_kv_compact       move the accepted nodes' K/V behind the prefix (Alg. 1 step 6)
 *
 * plus ptd_verify_sampling (verification under the sampling strategy, Alg. 2),
 * ptd_draft_tree_update (the draft forest's expansion and depth control, Alg. 1 step 3),
 * ptd_pool_* (the candidate pool: merge of the draft subtrees and retrieval of the
 * candidate tree, Alg. 1 steps 4 and 1), ptd_tree_rope_append (tree positions, the
 * rotary encoding and the tree's K/V into the cache), ptd_lm_head_topk (the LM-head
 * product with a fused top-k: the logits are never written),
 * ptd_verify_and_compact (the last two as one launch) and ptd_tree_verify_step (the
 * whole step: attention, top-k, verification and compaction on one stream)
 *
 * Conventions shared by every call
 *   - Pointers are DEVICE pointers unless a comment says "host".  The caller owns
 *     all memory; the library never allocates, frees or synchronises.  Scratch
 *     space, where a call needs any, is passed in by the caller.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     Every call only enqueues work on that stream and returns.
 *   - Errors the host can see (null pointer, bad size, unsupported shape) return
 *     synchronously and enqueue nothing.  Errors only the device can see (an
 *     invalid parent array) are reported through `dev_status` (one int32 in device
 *     memory, written with atomicMax of the status code, so the caller zeroes it
 *     before the step and reads it after); the affected sequence's outputs are then
 *     defined (zeros, accept_len 0) instead of garbage.
 *   - A failed kernel launch returns PTD_ERR_CUDA.  No C++ exception crosses the ABI.
 *
 * Tree layout (ptd_tree): B trees stored back to back; tree b owns nodes
 * [node_offsets[b], node_offsets[b+1]); parents are tree-local indices with
 * parents[first] = -1 and 0 <= parents[i] < i (topological order, e.g. BFS).
 * Node 0 of a tree is the current input token; node i of tree b has its K/V at
 * cache slot ctx_lens[b] + i, right after the b-th committed prefix.
 */
#ifndef PTD_H_
#define PTD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  PTD_OK = 0,
  PTD_ERR_INVALID_ARG = 1,   /* null pointer, size out of range, inconsistent shapes      */
  PTD_ERR_INVALID_TREE = 2,  /* (device) a parent array is not a topological rooted tree  */
  PTD_ERR_UNSUPPORTED = 3,   /* valid but not implemented (dtype / head_dim combination)  */
  PTD_ERR_CUDA = 4,          /* a CUDA runtime call or kernel launch failed              */
  PTD_ERR_TIMEOUT = 5,       /* (device) a bounded on-chip wait gave up; outputs invalid  */
  PTD_ERR_WORKSPACE = 6,     /* workspace pointer null or smaller than required          */
  PTD_ERR_POOL_FULL = 7      /* (device) a candidate-pool merge was refused: no room     */
} ptd_status;

typedef enum { PTD_F32 = 0, PTD_BF16 = 1 } ptd_dtype;

/* Maximum nodes of one tree (the ancestor bitmask of a node is 4 x 32 bits). */
#define PTD_MAX_TREE_NODES 128
/* Maximum k of ptd_topk_draft. */
#define PTD_MAX_TOPK 16

/* A batch of draft/candidate trees (Sec. 3.1 "Tree Construction": every node has a
 * unique parent P(v); node v sees pi(v) = {v} U pi(P(v))). */
typedef struct {
  int32_t batch;               /* host: B >= 1                                        */
  int32_t total_nodes;         /* host: N_tot = node_offsets[B]                       */
  int32_t max_nodes;           /* host: max_b T_b, 1..PTD_MAX_TREE_NODES              */
  int32_t max_ctx;             /* host: upper bound of every ctx_lens[b] (>= 0)       */
  const int32_t* node_offsets; /* [B+1], node_offsets[0] = 0, non-decreasing          */
  const int32_t* parents;      /* [N_tot], tree-local parent index, -1 for the root   */
  const int32_t* ctx_lens;     /* [B], committed prefix length C_b                    */
} ptd_tree;

/* The per-layer K/V cache of the target model.
 * Contiguous (page_size == 0): k, v are [num_layers][B][seq_capacity][Hkv][D].
 * Paged (page_size in {16, 32, 64, 128}): k, v are [num_layers][num_pages][page_size][Hkv][D]
 *   and slot s of sequence b lives in page block_table[b * max_pages + s / page_size]
 *   (the same page index in every layer).
 * Element type `dtype`; rows of one slot (all KV heads) are contiguous. */
typedef struct {
  void* k;
  void* v;
  ptd_dtype dtype;
  int32_t num_layers;
  int32_t num_kv_heads;        /* Hkv                                                  */
  int32_t head_dim;            /* D: 128 for bf16; 32, 64 or 128 for f32               */
  int32_t page_size;           /* 0 = contiguous                                       */
  int32_t seq_capacity;        /* contiguous: slots per sequence (>= C_b + T_b)        */
  int32_t num_pages;           /* paged: pages per layer                               */
  const int32_t* block_table;  /* paged: [B][max_pages]                                */
  int32_t max_pages;           /* paged: entries per block-table row                   */
} ptd_kv_cache;

/* Bytes of scratch `ptd_tree_attention` wants for these shapes (0 if it needs none):
 * per-block counters and the fp32 partials of the units that the balanced schedule splits
 * between neighbouring SMs (one CTA per SM, two partial slots each: about 266 KB per SM).
 * Passing less (even 0 with a NULL pointer) is allowed: the call then computes each (layer,
 * tree, KV head, 256-row block) in one CTA, which needs no scratch but leaves SMs idle when
 * such units are few or their count is not a multiple of the SM count.  With the scratch, the
 * call still takes one CTA per unit when an estimate from the shapes favours it; with fewer
 * units than SMs (every unit then cut into several pieces) the pieces' partials are merged by
 * a second kernel launched right after the attention, otherwise inside it. */
size_t ptd_attention_workspace_size(const ptd_tree* tree, const ptd_kv_cache* cache,
                                    int32_t num_q_heads, int32_t num_layers);

/* Bytes of scratch the one-call step (ptd_tree_verify_step and the host-buffer and pipelined
 * steps built on it) wants as ptd_step_args.workspace: the attention's scratch
 * (ptd_attention_workspace_size, rounded up to 256 bytes) followed by the tail's: one 4-byte
 * counter per tree and one per node row (together rounded up to 256 bytes), then one slot of
 * 16 eight-byte keys per node row and two per SM of the current device (rounded up to 256
 * bytes).  With that much (and a bf16 cache and bf16 logits whose rows start on 16 bytes,
 * vocab a multiple of 8), a persistent top-k streams the rows back to back, one equal share
 * per CTA, and also verifies every tree (the CTA that completes a tree's last row does it);
 * a copy kernel compacts.  With the tree counters alone the clustered top-k (one cluster per
 * row) verifies instead; with less, the top-k is followed by ptd_verify_and_compact, every
 * CTA of which verifies its tree before copying.  The scratch needs no clearing: the
 * attention kernel clears the tail's counters and tags its own with the launch.  0 for
 * invalid arguments. */
size_t ptd_step_workspace_size(const ptd_tree* tree, const ptd_kv_cache* cache, int32_t num_q_heads);

/* Tree-masked attention (Sec. 3.1 ancestor-only visibility; Sec. 3.2 one pass over
 * [X; T; C_X]).  For every layer l in [layer_begin, layer_begin + num_layers), tree b,
 * node i and query head h (KV head h / (Hq / Hkv)):
 *     out[l'][n][h] = sum_j softmax_j(scale * <q[l'][n][h], K[l][b][j]>) V[l][b][j]
 * over the slots j in [0, C_b) U { C_b + a : a in pi(i) }, where n = node_offsets[b] + i
 * and l' = l - layer_begin.
 *   q, out: [num_layers][N_tot][num_q_heads][D], element type = cache->dtype (fp32
 *           accumulation; bf16 output rounded to nearest even).
 *   scale:  <= 0 selects 1/sqrt(D).
 *   workspace/workspace_bytes: scratch from ptd_attention_workspace_size (may be less).
 *   dev_status: device int32, atomicMax'ed with PTD_ERR_INVALID_TREE if a tree is
 *           invalid (that tree's outputs are zero) or PTD_ERR_TIMEOUT.
 * The tree's own K/V must already be in slots C_b .. C_b + T_b - 1 (position
 * encoding is applied by the caller before the call).  One launch, or two when the partials
 * of split units are merged by a kernel of their own (see ptd_attention_workspace_size). */
ptd_status ptd_tree_attention(const ptd_tree* tree, const ptd_kv_cache* cache,
                              int32_t layer_begin, int32_t num_layers,
                              const void* q, int32_t num_q_heads, float scale, void* out,
                              void* workspace, size_t workspace_bytes,
                              int32_t* dev_status, void* stream);

/* Tree-masked attention for callers that cannot allocate device memory.  Some embedders
 * hand this library only their input and output buffers: a plugin running inside another
 * runtime's engine may have no allocator of its own to ask, and a latency-critical decode
 * loop may not tolerate cudaMalloc, whose implicit device synchronisation stalls every
 * stream.  This variant computes exactly what ptd_tree_attention computes, with the same
 * schedule, but takes its scratch from a fixed array that the library
 * holds in device memory (PTD_STATIC_SCRATCH_BYTES = 48 MiB, enough for the partials of one
 * CTA per SM on a 152-SM GPU plus the counters of ~100k units; every GPU that loads the
 * library keeps it until the process exits) instead of from a caller workspace.  The paper
 * has no counterpart of this entry point.
 *   - Arguments are those of ptd_tree_attention without workspace / workspace_bytes.
 *   - If these shapes need more than PTD_STATIC_SCRATCH_BYTES of scratch
 *     (ptd_attention_workspace_size > PTD_STATIC_SCRATCH_BYTES) the call returns
 *     PTD_ERR_WORKSPACE and enqueues nothing; use ptd_tree_attention with a workspace then.
 *   - The first call on each device resolves the array's device address on that device
 *     (make that device current); issue that first call before any stream capture.  The
 *     address is kept for the life of the process: a device reset (cudaDeviceReset) after
 *     the first call is not supported.
 *   - Every call on a device shares the one array and it keeps the previous call's
 *     contents.  The kernels write every scratch entry they later read, so nothing needs
 *     clearing, but calls whose kernels overlap on the GPU (different streams without
 *     ordering between them) race on the array: serialise them.
 *   - Calls no allocator (no cudaMalloc/cudaFree, no allocating library routine). */
#define PTD_STATIC_SCRATCH_BYTES ((size_t)48 << 20)
ptd_status ptd_tree_attention_noalloc(const ptd_tree* tree, const ptd_kv_cache* cache, int32_t layer_begin,
                                      int32_t num_layers, const void* q, int32_t num_q_heads, float scale,
                                      void* out, int32_t* dev_status, void* stream);

/* Per-node top-k of the logits (Sec. 3.1 "Progressive Expansion": each node's draft
 * token d_v; "Width Control": at most k children; Sec. 3.2: greedy V_n = entry 0).
 *   logits: [rows][row_stride] of `dtype`, the first `vocab` entries of a row are used.
 *   out_idx: [rows][k] int32, out_val: [rows][k] fp32 (exact value of the logit).
 *   Order: value descending; equal values by lower index first; -0.0 equals +0.0.
 *   NaN logits are not supported (their placement is unspecified).
 *   1 <= k <= min(PTD_MAX_TOPK, vocab). */
ptd_status ptd_topk_draft(const void* logits, ptd_dtype dtype, int64_t rows, int32_t vocab,
                          int64_t row_stride, int32_t k, int32_t* out_idx, float* out_val,
                          void* stream);

/* Greedy verification (Sec. 3.2): with V_n = target[n * target_stride] (the greedy
 * token of node n, e.g. column 0 of ptd_topk_draft's out_idx with stride k), the
 * eligible edges are I = {(n, c) : c child of n, tokens[c] = V_n}; the accepted path is
 * the longest root path n_0 = 0, n_1, ..., n_m with every edge in I (ties: the
 * lexicographically smallest node sequence), and X' = (n_0, ..., n_m, V_{n_m}).
 *   tokens: [N_tot] token of each node;  target: greedy token per node (stride in int32s).
 *   accepted_nodes: [B][max_nodes] tree-local node ids of the path (entries >= accept_len
 *       are set to -1);  accept_len: [B] = m + 1 (0 if the tree is invalid);
 *   bonus_token: [B] = V_{n_m} (-1 if the tree is invalid). */
ptd_status ptd_verify_greedy(const ptd_tree* tree, const int32_t* tokens, const int32_t* target,
                             int32_t target_stride, int32_t* accepted_nodes, int32_t* accept_len,
                             int32_t* bonus_token, int32_t* dev_status, void* stream);

/* KV-cache compaction (Alg. 1 step 6: X' joins the prefix): for every layer, K and V,
 * slot C_b + j receives the pre-call content of slot C_b + accepted_nodes[b][j] for
 * j < accept_len[b]; slots below C_b are untouched; new_ctx_lens[b] = C_b + accept_len[b]
 * (C_b when accept_len[b] = 0).  Overlapping sources and destinations are handled
 * (the result equals a copy from a snapshot).  Slots >= new_ctx_lens[b] are left with
 * unspecified content.  accepted_nodes must be a root path of tree b (as written by
 * ptd_verify_greedy); it is read with stride tree->max_nodes. */
ptd_status ptd_kv_compact(const ptd_tree* tree, const ptd_kv_cache* cache,
                          const int32_t* accepted_nodes, const int32_t* accept_len,
                          int32_t* new_ctx_lens, void* stream);

/* Sampling verification (Sec. 3.2, "sampling decoding strategy"; Alg. 2, Candidate Tree
 * Recursive Sampling; App. E proves that the emitted token follows P).  For every tree,
 * from the root: P_v = softmax(logits_v / temperature); the children of the current node
 * v are tried once each, in node order; child n is accepted when u_accept[n] <
 * P_v(tokens[n]) / S, where S is the mass of P_v not yet rejected, and a rejected child's
 * token gets probability 0 (a later sibling with the same token is then rejected too).
 * An accepted child becomes the current node.  When no child is accepted (or at a leaf)
 * the bonus token is the inverse CDF, in vocabulary order, of the residual P_v / S at
 * u_bonus[b].  The random numbers are inputs, so the result is a function of them.
 *   logits: rows of `vocab` entries, `row_stride` elements apart, one per node (dtype
 *           bf16 or f32); temperature > 0.
 *   u_accept: [N_tot] fp32 in [0, 1), the draw of node n's test (the root's is unused);
 *   u_bonus: [B] fp32 in [0, 1), the draw of tree b's bonus token.
 *   accepted_nodes, accept_len, bonus_token, dev_status: as in ptd_verify_greedy.
 * Probabilities use fp32 exponentials, compensated fp32 sums over short runs of the
 * vocabulary and fp64 sums across them: a uniform within ~1e-6 of the probability it is
 * compared with may decide either way.  One thread-block cluster (up to 8 CTAs) per tree. */
ptd_status ptd_verify_sampling(const ptd_tree* tree, const int32_t* tokens, const void* logits, ptd_dtype dtype,
                               int32_t vocab, int64_t row_stride, float temperature, const float* u_accept,
                               const float* u_bonus, int32_t* accepted_nodes, int32_t* accept_len,
                               int32_t* bonus_token, int32_t* dev_status, void* stream);

/* ptd_verify_greedy followed by ptd_kv_compact, in one launch: the same outputs (accepted
 * path, accept length, bonus token, status, compacted cache, new context lengths) with the
 * same arguments and rules, computed by one kernel in which every CTA of the compaction
 * grid verifies its tree first.  This is what ptd_tree_verify_step uses.  The paper has no
 * separate counterpart: it is Alg. 1 steps 5-6 as one call. */
ptd_status ptd_verify_and_compact(const ptd_tree* tree, const ptd_kv_cache* cache, const int32_t* tokens,
                                  const int32_t* target, int32_t target_stride, int32_t* accepted_nodes,
                                  int32_t* accept_len, int32_t* bonus_token, int32_t* new_ctx_lens,
                                  int32_t* dev_status, void* stream);

/* Draft tree update: one step of the draft forest's evolution T^{t-1} -> T^t (Sec. 3.1
 * "Progressive Expansion": every node's draft token joins the tree as its child,
 * V^t = V^{t-1} U {d_v}, E^t = E^{t-1} U {(v, d_v)}; "Width Control"; "Stepping Mechanism
 * (Depth Control)"; Alg. 1 step 3: expand, then StepAndPrune past d_max).
 *
 * A draft forest is a set of seed subtrees in creation order: parents[i] = -1 (a seed) or
 * 0 <= parents[i] < i, so "earliest added" is "lowest index".  Forest b's input nodes are
 * in_parents / in_tokens [b * in_stride, b * in_stride + in_count[b]) (device); its output
 * goes to out_parents / out_tokens / out_depths [b * capacity, (b + 1) * capacity), the
 * first out_count[b] entries valid and the rest -1.
 *   Expansion: node v, in index order, tries the first `expand` (<= 16) tokens of its draft
 *   row drafts[(b * in_stride + v) * draft_stride ..] (a top-k row), in rank order; a token
 *   equal to an existing child's token is that child (nothing is added); otherwise a new
 *   child is appended while v has fewer than `width` children and the forest fewer than
 *   `capacity` (<= PTD_MAX_TREE_NODES) nodes.
 *   Depth control: depth counts nodes on a seed-to-leaf path (a lone seed has depth 1);
 *   a seed subtree deeper than `max_depth` (>= 1) keeps only the subtree of the seed's
 *   lowest-index child, which becomes a seed; the rest of it is dropped.  Once per call.
 *   Survivors keep their relative order; out_depths[i] = |pi(i)| in the new forest (the
 *   node's position offset, Sec. 3.1); old_to_new[b * in_stride + j] is the new index of
 *   input node j, or -1 (also for j >= in_count[b]).
 * A forest that is not one (a parent that is neither -1 nor earlier, in_count[b] < 0 or
 * above in_stride or capacity) sets PTD_ERR_INVALID_TREE in dev_status and gets
 * out_count[b] = 0.  Outputs must not alias inputs.  One launch, one CTA per forest. */
ptd_status ptd_draft_tree_update(int32_t batch, int32_t in_stride, const int32_t* in_count, const int32_t* in_parents,
                                 const int32_t* in_tokens, const int32_t* drafts, int32_t draft_stride, int32_t expand,
                                 int32_t width, int32_t max_depth, int32_t capacity, int32_t* out_count,
                                 int32_t* out_parents, int32_t* out_tokens, int32_t* out_depths, int32_t* old_to_new,
                                 int32_t* dev_status, void* stream);

/* Candidate pool (Sec. 3.1 "Draft Extraction via Merging": any subtree T' of the draft tree
 * is merged, by M, into the cached candidate tree with the same root value; Sec. 3.2 and
 * Alg. 1 step 1: the candidate tree C_X retrieved for the decoded sequence X).
 *
 * The pool lives in one caller buffer of ptd_pool_bytes(capacity) bytes (device), a hash
 * table of `capacity` trie nodes (a power of two, 16 .. 2^28); its first int32 is the
 * number of nodes held.  ptd_pool_init empties it.  Pool calls on one buffer must be
 * ordered (one stream); a pool is one sequence's. */
size_t ptd_pool_bytes(int32_t capacity);                        /* 0 if capacity is invalid */
ptd_status ptd_pool_init(void* pool, int32_t capacity, void* stream);

/* Merge (Alg. 1 step 4): for every node v of the draft forest (count[0] nodes, parents /
 * tokens device arrays in creation order, a seed's parent -1, at most PTD_MAX_TREE_NODES),
 * in index order, the subtree rooted at v joins the pool entry of token(v), created when
 * absent: M is the union of tries (a child whose token is new joins with its subtree, a
 * child whose token is there merges recursively).  Children keep the order in which the
 * sequential merge inserts them (step, then v, then the draft node); `step` must grow
 * from call to call.  A merge that could take the node count past max_load (<= capacity)
 * is refused as a whole with PTD_ERR_POOL_FULL in dev_status; an invalid forest sets
 * PTD_ERR_INVALID_TREE.  One launch. */
ptd_status ptd_pool_merge(void* pool, int32_t capacity, int32_t max_load, int32_t step, const int32_t* count,
                          const int32_t* parents, const int32_t* tokens, int32_t* dev_status, void* stream);

/* Retrieval (Alg. 1 step 1): the candidate tree for a sequence whose last token is
 * *root_token (device int32, e.g. the previous step's bonus token): node 0 is the root
 * token; then breadth first, each node's earliest-inserted children, at most `width`
 * (1 .. 8) per node, nodes of depth at most max_depth (>= 1, the root has depth 1), at
 * most max_nodes (1 .. PTD_MAX_TREE_NODES) in all.  A token with no entry gives the lone
 * root.  Writes out_count[0] and out_parents / out_tokens [max_nodes] (-1 past the count):
 * the tree layout of ptd_tree (parents[0] = -1, parents[i] < i).  One launch. */
ptd_status ptd_pool_retrieve(const void* pool, int32_t capacity, const int32_t* root_token, int32_t width,
                             int32_t max_depth, int32_t max_nodes, int32_t* out_count, int32_t* out_parents,
                             int32_t* out_tokens, void* stream);

/* Tree positions and the tree's K/V append (Sec. 3.1 "Tree Construction": the position of
 * node v is set by |pi(v)|).  Node i of tree b sits at p = C_b + |pi(i)| - 1 (the root at
 * C_b, where plain decoding would put the next token).  For the cache layers
 * l in [layer_begin, layer_begin + num_layers), with l' = l - layer_begin:
 *   q [num_layers][N_tot][num_q_heads][D] (device, cache->dtype) is rotated in place;
 *   k, v [num_layers][N_tot][num_kv_heads][D]: k[l'] rotated, k[l'] and v[l'] written to
 *   cache layer l, slot C_b + i;
 * rotation: for j < D/2 the pair (x_j, x_{j+D/2}) turns by p * rope_base^(-2j/D)
 * (RoFormer's rotary encoding in the rotate-half layout of Llama-family models; the angle
 * is carried as an fp32 pair from inverse frequencies computed in double, about 1e-7
 * relative).  positions_out [N_tot] (device, may be NULL)
 * receives p.  A tree that is not one, or a slot outside the cache (or a page outside the
 * pool), sets PTD_ERR_INVALID_TREE in dev_status; that node writes nothing.  q must not
 * alias k or v.  One launch, one CTA per (node, layer).  This is what puts the tree's K/V
 * where ptd_tree_attention expects them. */
ptd_status ptd_tree_rope_append(const ptd_tree* tree, const ptd_kv_cache* cache, int32_t layer_begin,
                                int32_t num_layers, void* q, int32_t num_q_heads, const void* k, const void* v,
                                float rope_base, int32_t* positions_out, int32_t* dev_status, void* stream);

/* LM head with a fused top-k: for every node row r of hidden, the logits h_r W^T (the
 * model's next-token scores P(y_T | ...) of Alg. 1 step 2) and their k largest entries,
 * as ptd_topk_draft would give them (descending, the lower token first on equal values,
 * -0.0 == +0.0; Sec. 3.1 draft tokens d_v, Sec. 3.2 verification tokens V_n), without the
 * logits ever reaching memory.
 *   hidden: [rows][hidden_stride] bf16 (device), rows 1 .. PTD_MAX_TREE_NODES;
 *   weight: [vocab][weight_stride] bf16 (device); d_model a multiple of 64; strides
 *           multiples of 8 elements, both base pointers 16-byte aligned;
 *   out_idx [rows][k] int32, out_val [rows][k] fp32 (the fp32-accumulated logits);
 *           k in 1 .. 16.
 * Logits are accumulated in fp32 by the tensor cores in an order of their own: entries
 * within ~1e-6 relative of each other may swap places against an exact evaluation.
 * workspace: ptd_lm_head_topk_workspace_size(rows, vocab) bytes, 16-byte aligned (per-CTA
 * candidate lists).  Two launches: the product with per-CTA top-k, then a per-row merge. */
size_t ptd_lm_head_topk_workspace_size(int32_t rows, int32_t vocab);
ptd_status ptd_lm_head_topk(const void* hidden, int32_t rows, int64_t hidden_stride, const void* weight,
                            int32_t vocab, int64_t weight_stride, int32_t d_model, int32_t k, int32_t* out_idx,
                            float* out_val, void* workspace, size_t workspace_bytes, int32_t* dev_status,
                            void* stream);

/* One whole tree-verify step on device buffers: attention over all cache layers,
 * top-k of the logits, greedy verification on top-k column 0, KV compaction.
 * Equivalent to ptd_tree_attention, ptd_topk_draft and ptd_verify_and_compact in that
 * order on `stream` (three launches, or four with the attention's merge kernel); when the
 * workspace holds ptd_step_workspace_size
 * bytes and the logits are bf16 (vocab a multiple of 8, or vocab <= 262143), the top-k's
 * CTAs verify the trees instead and the third launch only copies the accepted rows (node_offsets must then run
 * from 0 to total_nodes without decreasing, as ptd_tree states; a tree with an empty or
 * out-of-range node range is reported as PTD_ERR_INVALID_TREE with accept_len 0, and when
 * the offsets decrease the outputs of the other trees are unspecified).  Each launch may be
 * placed on the SMs while the one before it drains (programmatic dependent launch); it reads
 * its inputs only after that one has completed, so every kernel sees the previous one's
 * writes, as stream order would give. */
typedef struct {
  const void* q;               /* [L][N_tot][Hq][D]                                    */
  int32_t num_q_heads;
  float scale;                 /* <= 0: 1/sqrt(D)                                      */
  void* attn_out;              /* [L][N_tot][Hq][D]                                    */
  const void* logits;          /* [N_tot][vocab] of logits_dtype                       */
  ptd_dtype logits_dtype;
  int32_t vocab;
  int32_t k;
  const int32_t* tokens;       /* [N_tot]                                              */
  int32_t* topk_idx;           /* [N_tot][k]                                           */
  float* topk_val;             /* [N_tot][k]                                           */
  int32_t* accepted_nodes;     /* [B][max_nodes]                                       */
  int32_t* accept_len;         /* [B]                                                  */
  int32_t* bonus_token;        /* [B]                                                  */
  int32_t* new_ctx_lens;       /* [B]                                                  */
  int32_t* dev_status;         /* [1]                                                  */
  void* workspace;
  size_t workspace_bytes;
} ptd_step_args;

ptd_status ptd_tree_verify_step(const ptd_tree* tree, const ptd_kv_cache* cache,
                                const ptd_step_args* args, void* stream);

/* Which top-k the one-call step (and the steps built on it) uses when its workspace allows
 * both: AUTO streams the rows back to back when the clustered top-k (one cluster per row, at
 * most three CTAs per SM) would take more than one wave of the device's SMs, and clusters
 * otherwise (measured on GB300: 266 rows of 128256 logits and 128 rows of 152064 stream
 * faster, 63 rows of 128256 and 31 of 32000 run faster clustered); CLUSTERED and STREAMED force one where
 * it applies (streaming needs vocab a multiple of 8 and 16-byte aligned rows; clustering needs
 * vocab <= 262143).  Process-wide; returns the previous policy, or -1 (nothing changed) for
 * an unknown value.  Results are identical either way. */
typedef enum { PTD_STEP_TOPK_AUTO = 0, PTD_STEP_TOPK_CLUSTERED = 1, PTD_STEP_TOPK_STREAMED = 2 } ptd_step_topk;
int32_t ptd_step_topk_policy(int32_t policy);

/* The tail ptd_tree_verify_step would run for these arguments under the current policy (host
 * only; reads the sizes, the pointers' presence and alignment, and the device's SM count;
 * enqueues nothing): 2 = the streamed top-k verifies the trees, 1 = the clustered top-k does,
 * 0 = the top-k is followed by ptd_verify_and_compact; -1 for a missing or invalid tree,
 * cache or argument block. */
int32_t ptd_step_tail(const ptd_tree* tree, const ptd_kv_cache* cache, const ptd_step_args* args);

/* The same step fed from and drained to HOST memory (pinned for asynchronous copies):
 * copies the host inputs into the device buffers named by `tree`, `cache` and `args`,
 * runs ptd_tree_verify_step, and copies the small results back.  Contiguous caches only.
 * Host inputs: q_h [L][N_tot][Hq][D]; logits_h [N_tot][vocab]; tokens_h [N_tot];
 *   parents_h [N_tot]; node_offsets_h [B+1]; ctx_lens_h [B] (also used on the host to
 *   place the tree rows); tree_k_h, tree_v_h [L][N_tot][Hkv][D] (node n of tree b goes to
 *   slot ctx_lens_h[b] + (n - node_offsets_h[b])).
 * Host outputs: topk_idx_h, topk_val_h [N_tot][k]; accepted_h [B][max_nodes];
 *   accept_len_h, bonus_h, new_ctx_h [B]; status_h [1].
 * The host tree layout is checked before anything is enqueued: node_offsets_h[0] = 0,
 * node_offsets_h[B] = total_nodes, every tree has 1 .. max_nodes nodes and every
 * ctx_lens_h[b] >= 0 with ctx_lens_h[b] + T_b <= seq_capacity (else PTD_ERR_INVALID_ARG).
 * Returns after enqueueing; the host outputs are valid after the stream synchronises. */
typedef struct {
  const void* q_h;
  const void* logits_h;
  const int32_t* tokens_h;
  const int32_t* parents_h;
  const int32_t* node_offsets_h;
  const int32_t* ctx_lens_h;
  const void* tree_k_h;
  const void* tree_v_h;
  int32_t* topk_idx_h;
  float* topk_val_h;
  int32_t* accepted_h;
  int32_t* accept_len_h;
  int32_t* bonus_h;
  int32_t* new_ctx_h;
  int32_t* status_h;
} ptd_host_io;

ptd_status ptd_tree_verify_step_host(const ptd_tree* tree, const ptd_kv_cache* cache,
                                     const ptd_step_args* args, const ptd_host_io* io,
                                     void* stream);

/* Host-buffer steps with the copies overlapped (a software pipeline over two device buffer
 * sets): step i + 1's inputs go up, and step i - 1's results come down, while step i
 * computes.  Each submitted step is ptd_tree_verify_step_host's step (the same inputs,
 * outputs and rules), except that the tree's K/V rows first land in a staging buffer and
 * reach the cache slots from there at the start of the step's computation, so that an
 * upload never touches rows the previous step still reads.  Contiguous and paged caches
 * (for a paged cache the rows are scattered through the device block table by one extra
 * kernel; a slot outside a sequence's pages sets PTD_ERR_INVALID_TREE in the status).
 *   trees[2], args[2]: two complete sets of device buffers (slot s serves steps
 *           s, s + 2, ...); they share `cache`.
 *   staging[2]: device buffers of at least 2 * L * N_tot * Hkv * D elements each.
 *   compute_stream: where the steps compute, in submission order.
 * The pipeline creates two streams and six events of its own (freed by destroy); the
 * device memory stays the caller's.  submit enqueues one step and returns its ticket; the
 * step's host outputs are valid once wait(ticket) returns.  submit checks each step's host
 * tree layout as ptd_tree_verify_step_host does and, on a bad one, returns
 * PTD_ERR_INVALID_ARG with nothing enqueued and no ticket used.  A step's `io` buffers must
 * stay untouched until then; alternate two `io` sets to keep two steps in flight. */
typedef struct ptd_pipeline ptd_pipeline;
ptd_status ptd_pipeline_create(const ptd_kv_cache* cache, const ptd_tree* trees, const ptd_step_args* args,
                               void* const* staging, size_t staging_bytes, void* compute_stream,
                               ptd_pipeline** out);
ptd_status ptd_pipeline_submit(ptd_pipeline* pipeline, const ptd_host_io* io, int64_t* ticket);
ptd_status ptd_pipeline_wait(ptd_pipeline* pipeline, int64_t ticket);
ptd_status ptd_pipeline_destroy(ptd_pipeline* pipeline);

/* Diagnostic of the failure path: one thread waits on an mbarrier that nothing arrives on,
 * through the bounded wait every kernel here uses; after its limit (2 s of %globaltimer)
 * it atomicMax'es PTD_ERR_TIMEOUT into dev_status and the kernel returns, the context
 * still usable.  No fault, trap or endless loop is involved. */
ptd_status ptd_check_bounded_wait(int32_t* dev_status, void* stream);

/* Number of kernels the last successful call of each entry point enqueued on this
 * host thread (a diagnostic for launch accounting). */
int32_t ptd_last_launch_count(void);

/* Static description of a status code. */
const char* ptd_status_string(ptd_status status);

#ifdef __cplusplus
}
#endif

#endif /* PTD_H_ */
