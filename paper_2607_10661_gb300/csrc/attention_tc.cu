// Tree-masked attention on the 5th-generation tensor cores (tcgen05 + TMEM + TMA), bf16.
//
// What it computes (Sec. 3.1 visibility pi(v) = {v} U pi(P(v)); Sec. 3.2 one pass over
// [X; T; C_X]): for every layer, tree b, KV head, query head h of that KV head's group and
// tree node i, the softmax-weighted sum of V over the committed slots [0, C_b) and the
// slots C_b + a of i's ancestors a (itself included).
//
// Work decomposition.  All G = Hq/Hkv query heads of one KV head and all T_b nodes of a
// tree form the rows of one dense problem: row r = node * G + g, so M = T_b * G rows share
// every K/V tile.  A unit is one (layer, tree, KV head, pair of 128-row M tiles), e.g. 63
// nodes x 4 heads = 252 rows, and its keys are cut into 128-key tiles.  Each K/V tile is
// loaded from HBM once by TMA and used by both M tiles.
//
// Schedules.  Persistent (the default when the caller's scratch allows it): the flattened
// (unit, key tile) space is cut into one equal contiguous range per CTA, one CTA per SM, so
// every SM gets the same number of key tiles whatever the unit count.  Each warp walks its
// CTA's range as segments (whole units, or a piece of a unit at either end of the range).
// Whole units are written directly.  Of the pieces of a unit cut by range ends, all but the
// last leave an fp32 partial (O unnormalised, running max, row sum); the warp that finishes
// the last one merges those partials with its own O, still in TMEM.  The softmax warps load
// the next segment's Q before the epilogue of the current one, so the tensor core does not
// wait on it.  Grid (fallback without scratch): one CTA per unit.
//
// Warp roles (320 threads):
//   warp 0      TMA producer: K and V tiles into two stage pairs (K_j, V_j | K_j+1, V_j+1).
//   warp 1      TMEM allocator and MMA issuer (one thread issues tcgen05.mma):
//                 S_t = Q_t K_j^T    (Q and K from shared memory, fp32 S in TMEM)
//                 O_t += P_t V_j     (P from TMEM, where the softmax wrote it over S_t;
//                                     V from shared memory)
//               in the order S_0, S_1 | PV_0, S_0', PV_1, S_1' | ... so the softmax of one
//               M tile overlaps the tensor work of the other.
//   warps 2-5   softmax of M tile 0, warps 6-9 of M tile 1 (thread = row = TMEM lane
//               (warp % 4) * 32 + lane): row max, lazy rescaling of O (only when the
//               running max grows by more than 2^8), exp2, bf16 P back into TMEM, row sum;
//               at the end O / l (or a piece's partial).  Tiles that lie entirely inside the
//               committed prefix skip the mask arithmetic.
// TMEM: S_0 | S_1 | O_0 | O_1, 128 fp32 columns each = all 512 columns of the SM; P_t
// takes the first 64 columns of S_t (two bf16 per column).
// The ancestor mask of a row's node (up to 128 bits) lives in 4 registers of its thread.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <climits>
#include <cmath>
#include <cstdint>

#include "attention.cuh"
#include "ptd_device.cuh"

namespace ptd {
namespace tc {

constexpr int kThreads = 320;
constexpr int kStages = 2;                // K/V stage pairs (K tile then V tile)
constexpr uint32_t kTileBytes = 32768;   // 128 rows x 128 bf16
constexpr uint32_t kHalfBytes = 16384;   // 128 rows x 64 bf16 (one 128-byte swizzle column)
constexpr uint32_t kStageBytes = 2 * kTileBytes;
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffRing = 2 * kTileBytes;
constexpr uint32_t kOffBar = kOffRing + kStages * kStageBytes;
// barriers: full_k[2], full_v[2], empty_k[2], v_load[2], s_full[2], p_full[2], o_full[2], drain, q_ready[2],
// empty_v[2]
constexpr uint32_t kNumBars = 5 * kStages + 9;
constexpr uint32_t kOffTmemPtr = kOffBar + kNumBars * 8;
constexpr uint32_t kOffAbort = kOffTmemPtr + 4;
constexpr uint32_t kOffSched = (kOffAbort + 4 + 15) / 16 * 16;   // schedule constants + one slot per warp
constexpr uint32_t kSchedBytes = 1024;
constexpr uint32_t kOffWarp = kOffSched + kSchedBytes;   // one WarpArea per softmax warp (below)
constexpr uint32_t kTmemCols = 512;
constexpr float kRescaleLog2 = 8.0f;                // lazy rescale threshold (log2 units)

constexpr uint32_t kIdescS = idesc_bf16_f32(128, 128, 0, 0);    // Q (K-major) x K (K-major)
constexpr uint32_t kIdescPV = idesc_bf16_f32(128, 128, 0, 1);   // P (K-major) x V (MN-major)

// Bits [a0, a0+32) of "is slot C + a visible": a < 0 is committed context (visible),
// 0 <= a < 128 reads the node's ancestor mask, a >= 128 is past the tree.
__device__ __forceinline__ uint32_t vis_word(int a0, uint32_t m0, uint32_t m1, uint32_t m2, uint32_t m3) {
  if (a0 <= -32) return 0xFFFFFFFFu;
  if (a0 < 0) {
    const int sh = -a0;   // 1..31
    return (m0 << sh) | ((1u << sh) - 1u);
  }
  if (a0 >= 128) return 0u;
  const int w = a0 >> 5, sh = a0 & 31;
  const uint32_t lo = w == 0 ? m0 : w == 1 ? m1 : w == 2 ? m2 : m3;
  const uint32_t hi = w == 0 ? m1 : w == 1 ? m2 : w == 2 ? m3 : 0u;
  return __funnelshift_r(lo, hi, sh);
}

// One segment of work: key tiles [kt_begin, kt_end) of one unit.
struct Seg {
  int lq, b, hkv, mp;          // layer within the call, tree, KV head, M-tile pair
  int node0, T, C, N;          // the tree's first node, size, committed context, keys
  int n_kt, nt;                // key tiles of the unit, M tiles of the pair (1 or 2)
  int kt_begin, kt_end;
  int unit;                    // canonical unit id (layer, tree, KV head, pair)
  int ug0;                     // global index of the unit's key tile 0 (persistent)
  int slot;                    // partial slot, or -1 when the segment is the whole unit
  int valid;                   // 0: no more segments
};

// A segment taken by a softmax warp, with the validity of its tree.
struct SegRun {
  Seg s;
  int invalid;
  int pad;
};

// Shared memory of one softmax warp.
struct WarpArea {
  int parents[128];            // parent array of the last tree seen
  SegRun run[2];               // the segment being computed and the next one
  int tree_node0, tree_T;      // which tree `parents` holds
  int tree_invalid;            // that tree failed the parent check
  int mask_mp;                 // M-tile pair the ancestor masks in registers were built for
};
// Geometry of every tree of the call, read from global memory once per CTA at the start (the
// schedule walkers decode it at every segment boundary); calls with more trees read it from
// global memory each time instead.
struct TreeInfo {
  int node0, T, C, n_kt, pairs, wb;
};
constexpr int kMaxCachedTrees = 256;
constexpr uint32_t kOffTrees = kOffWarp + 8 * sizeof(WarpArea);
constexpr uint32_t kSmemUsed = kOffTrees + kMaxCachedTrees * sizeof(TreeInfo);
constexpr uint32_t kSmemBytes = kSmemUsed + 1024;   // slack to align the base to 1024 B
static_assert(kSmemBytes <= 232448, "shared memory budget");

// Persistent schedule constants: CTA c owns global key tiles [c*W/P, (c+1)*W/P).
struct WalkConst {
  int persistent, W, Wl, P, c, r0, r1;
};

// Tree b: first node, size, context, key tiles and M-tile pairs; returns the key tiles of all
// its units in one layer (0 for a malformed entry, which is skipped and reported).  From the
// CTA's shared copy `ti` when there is one.
__device__ __forceinline__ int seq_info(const AttnParams& p, const TreeInfo* ti, int b, int& node0, int& T, int& C,
                                        int& n_kt, int& pairs) {
  if (ti != nullptr) {
    const TreeInfo x = ti[b];
    node0 = x.node0;
    T = x.T;
    C = x.C;
    n_kt = x.n_kt;
    pairs = x.pairs;
    return x.wb;
  }
  node0 = p.node_offsets[b];
  T = p.node_offsets[b + 1] - node0;
  C = p.ctx_lens[b];
  const int N = C + T;
  const bool bad = T < 1 || T > p.max_nodes || node0 < 0 || node0 + T > p.n_total || C < 0 ||
                   (p.page_size > 0 ? N > p.max_pages * p.page_size : N > p.seq_capacity);
  if (bad) {
    n_kt = 0;
    pairs = 0;
    return 0;
  }
  n_kt = (N + 127) >> 7;
  pairs = ((T * p.group + 127) / 128 + 1) / 2;
  return p.hkv * pairs * n_kt;
}

__device__ __forceinline__ void fill_seg(const AttnParams& p, Seg& s, int b, int node0, int T, int C, int n_kt) {
  s.b = b;
  s.node0 = node0;
  s.T = T;
  s.C = C;
  s.N = C + T;
  s.n_kt = n_kt;
  s.nt = min(2, (T * p.group + 127) / 128 - 2 * s.mp);
  s.unit = ((s.lq * p.batch + b) * p.hkv + s.hkv) * p.pairs + s.mp;
}

__device__ __forceinline__ int range_start(const WalkConst& wc, int c) {
  return (int)((long long)c * wc.W / wc.P);
}
__device__ __forceinline__ int owner_cta(const WalkConst& wc, int g) {
  return (int)(((long long)(g + 1) * wc.P - 1) / wc.W);
}

// Returns false (schedule inconsistent with the tree arrays) if g maps to no tree.
__device__ __noinline__ bool decode_tile(const AttnParams& p, const TreeInfo* ti, int Wl, int g, Seg& s) {
  s.lq = g / Wl;
  int r = g - s.lq * Wl;
  for (int b = 0; b < p.batch; ++b) {
    int node0, T, C, n_kt, pairs;
    const int wb = seq_info(p, ti, b, node0, T, C, n_kt, pairs);
    if (r < wb) {
      const int idx = r / n_kt;
      const int tile = r - idx * n_kt;
      s.hkv = idx / pairs;
      s.mp = idx - s.hkv * pairs;
      fill_seg(p, s, b, node0, T, C, n_kt);
      s.ug0 = g - tile;
      return true;
    }
    r -= wb;
  }
  return false;
}

__device__ __noinline__ void make_walk_const(const AttnParams& p, const TreeInfo* ti, WalkConst& wc) {
  wc.persistent = p.persistent;
  if (!p.persistent) return;
  int wl = 0;
  for (int b = 0; b < p.batch; ++b) {
    int node0, T, C, n_kt, pairs;
    const int w = seq_info(p, ti, b, node0, T, C, n_kt, pairs);
    if (w == 0 && blockIdx.x == 0) atomicMax(p.dev_status, (int)PTD_ERR_INVALID_TREE);   // malformed sizes
    wl += w;
  }
  wc.Wl = wl;
  wc.W = wl * p.layers;
  wc.P = (int)gridDim.x;
  wc.c = (int)blockIdx.x;
  wc.r0 = range_start(wc, wc.c);
  wc.r1 = range_start(wc, wc.c + 1);
}

// A walker's cursor before its first step (a walk's cursors lie in [0, W]).
constexpr int kWalkStart = INT_MIN;

// Next segment of this CTA for one walker (cursor starts at kWalkStart); s.valid = 0 when done.
__device__ __noinline__ void next_segment(const AttnParams& p, const TreeInfo* ti, const WalkConst& wc, int& cursor,
                                          Seg& s) {
  s.valid = 0;
  if (!wc.persistent) {
    // grid schedule: CTA u computes unit u whole
    if (cursor != kWalkStart) return;
    cursor = 0;
    int u = blockIdx.x;
    s.mp = u % p.pairs;
    u /= p.pairs;
    s.hkv = u % p.hkv;
    u /= p.hkv;
    const int b = u % p.batch;
    s.lq = u / p.batch;
    int node0, T, C, n_kt, pairs;
    if (seq_info(p, ti, b, node0, T, C, n_kt, pairs) == 0) {
      atomicMax(p.dev_status, (int)PTD_ERR_INVALID_TREE);   // malformed sizes
      return;
    }
    if (s.mp >= pairs) return;
    fill_seg(p, s, b, node0, T, C, n_kt);
    s.ug0 = 0;
    s.kt_begin = 0;
    s.kt_end = n_kt;
    s.slot = -1;
    s.valid = 1;
    return;
  }
  if (wc.W <= 0) return;
  if (cursor == kWalkStart) cursor = wc.r0;
  if (cursor >= wc.r1) return;
  // self-check: every step must decode and move the cursor forward (the walk then ends)
  if (!decode_tile(p, ti, wc.Wl, cursor, s) || s.ug0 + s.n_kt <= cursor || s.ug0 > cursor) {
    atomicMax(p.dev_status, (int)PTD_ERR_TIMEOUT);
    cursor = wc.r1;
    return;
  }
  const int g0 = cursor;
  const int g1 = min(s.ug0 + s.n_kt, wc.r1);
  cursor = g1;
  s.kt_begin = g0 - s.ug0;
  s.kt_end = g1 - s.ug0;
  if (s.kt_begin == 0 && s.kt_end == s.n_kt) {
    s.slot = -1;
  } else {
    s.slot = wc.c * 2 + ((wc.r0 >= s.ug0 && wc.r0 < s.ug0 + s.n_kt) ? 0 : 1);
  }
  s.valid = 1;
}

// Partial slot of CTA c's piece of the unit starting at global tile ug0 (c owns a piece).
__device__ __forceinline__ int piece_slot(const WalkConst& wc, int c, int ug0, int ug1) {
  const int rs = range_start(wc, c);
  return c * 2 + ((rs >= ug0 && rs < ug1) ? 0 : 1);
}

// Rare path of the softmax, kept out of the hot loop: O_t (n_o 16-column groups) and the
// bf16 P chunks [0, c) of S_t scaled by alpha.  Warp-collective.
__device__ __noinline__ void rescale_tmem(uint32_t tO, uint32_t tS, int n_o, int c, float alpha) {
  for (int q = 0; q < n_o; ++q) {
    uint32_t o16[16];
    tmem_ld16(tO + (uint32_t)q * 16u, o16);
    tmem_ld_wait();
#pragma unroll
    for (int e = 0; e < 16; ++e) o16[e] = __float_as_uint(__uint_as_float(o16[e]) * alpha);
    tmem_st16(tO + (uint32_t)q * 16u, o16);
  }
  if (c > 0) tmem_st_wait();
  for (int q = 0; q < c; ++q) {
    uint32_t p16[16];
    tmem_ld16(tS + (uint32_t)q * 16u, p16);
    tmem_ld_wait();
#pragma unroll
    for (int e = 0; e < 16; ++e)
      p16[e] = pack_bf16x2(__uint_as_float(p16[e] << 16) * alpha, __uint_as_float(p16[e] & 0xFFFF0000u) * alpha);
    tmem_st16(tS + (uint32_t)q * 16u, p16);
  }
}

template <bool kPaged, bool kQTma>
__global__ void __launch_bounds__(kThreads, 1)
    tree_attn_tc_kernel(const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_v,
                        const __grid_constant__ CUtensorMap map_q, const AttnParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint32_t base = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (base & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  base += pad;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = p.group;

  auto bar = [&](int i) { return base + kOffBar + 8u * (uint32_t)i; };
  auto fullk_bar = [&](int s) { return bar(s); };
  auto fullv_bar = [&](int s) { return bar(kStages + s); };
  // K of a stage is free once both S GEMMs of its tile are done, V only after both PV GEMMs:
  // separate barriers let the producer refill K about one softmax earlier.
  auto emptyk_bar = [&](int s) { return bar(2 * kStages + s); };
  auto emptyv_bar = [&](int s) { return bar(4 * kStages + 9 + s); };
  // V of a tile that reaches past the sequence lands on v_load (waited on by the producer
  // only); the producer zeroes the tail rows and then arrives on full_v itself, so the MMA
  // issuer always waits on full_v, once per use of the stage.
  auto vload_bar = [&](int s) { return bar(3 * kStages + s); };
  auto sfull_bar = [&](int t) { return bar(4 * kStages + t); };
  auto pfull_bar = [&](int t) { return bar(4 * kStages + 2 + t); };
  auto ofull_bar = [&](int t) { return bar(4 * kStages + 4 + t); };
  const uint32_t drain_bar = bar(4 * kStages + 6);
  auto qready_bar = [&](int t) { return bar(4 * kStages + 7 + t); };
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffAbort);
  WalkConst* wc_s = reinterpret_cast<WalkConst*>(smem + kOffSched);
  Seg* my_seg = reinterpret_cast<Seg*>(smem + kOffSched + 64) + warp;   // this warp's schedule slot
  static_assert(64 + (kThreads / 32) * sizeof(Seg) <= kSchedBytes, "schedule area");

  // A grid launched after this one with programmatic stream serialization (the step's top-k)
  // may be scheduled now; its CTAs take the SMs this grid's CTAs leave at its end.
  if (threadIdx.x == 0) grid_launch_dependents();
  // set-up that reads no global memory: it may overlap the stream's previous grid
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(fullk_bar(s), 1);
      mbar_init(fullv_bar(s), 1);
      mbar_init(emptyk_bar(s), 1);
      mbar_init(emptyv_bar(s), 1);
      mbar_init(vload_bar(s), 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(sfull_bar(t), 1);
      mbar_init(pfull_bar(t), 4);    // one arrival per softmax warp
      mbar_init(ofull_bar(t), 1);
      mbar_init(qready_bar(t), kQTma ? 1 : 4);   // the TMA issuer, or one arrival per softmax warp
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&map_k);
    prefetch_tensormap(&map_v);
  }
  if (warp == 1) {
    tmem_alloc(base + kOffTmemPtr, kTmemCols);
    tmem_relinquish();
    tc_fence_before();
  }
  // every input (trees, Q, the cache) and output belongs to the stream's previous work
  grid_dependency_wait();
  if (blockIdx.x == 0)   // counters of the work that follows this kernel in the step (see AttnParams)
    for (int i = threadIdx.x; i < p.zero_count; i += kThreads) p.zero_ptr[i] = 0u;
  TreeInfo* const trees_s = reinterpret_cast<TreeInfo*>(smem + kOffTrees);
  const TreeInfo* const ti = p.batch <= kMaxCachedTrees ? trees_s : nullptr;
  if (ti != nullptr) {
    for (int b = threadIdx.x; b < p.batch; b += kThreads) {
      TreeInfo x;
      x.wb = seq_info(p, nullptr, b, x.node0, x.T, x.C, x.n_kt, x.pairs);
      trees_s[b] = x;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) make_walk_const(p, ti, *wc_s);
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + kOffTmemPtr);
  const WalkConst& wc = *wc_s;
  int cursor = kWalkStart;   // this warp's position in the schedule (lane 0 walks, the warp reads)
  volatile Seg* sgv = my_seg;
  auto advance = [&]() -> bool {
    __syncwarp();
    if (lane == 0) next_segment(p, ti, wc, cursor, *my_seg);
    __syncwarp();
    return sgv->valid != 0;
  };

  if (warp == 0) {
    // ================================================================ TMA producer
    bool ok = true;
    int gt = 0;                    // key tiles issued by this CTA (ring position)
    // K and V lines leave L2 first: the stream of them (read once per M-tile pair) does not push
    // out what the step's next kernels read (their code, the trees, the top-k rows)
    const uint64_t kv_policy = l2_policy_evict_first();
    int vloads[kStages] = {0, 0};  // v_load completions per stage (waited on here only)
    while (ok && advance()) {
      const int layer = p.layer_begin + sgv->lq;
      const int b = sgv->b, hkv = sgv->hkv, N = sgv->N;
      const int kt_end = sgv->kt_end;
      for (int kt = sgv->kt_begin; kt < kt_end && ok; ++kt, ++gt) {
        const int t0 = kt * 128;
        const int st = gt % kStages;
        const uint32_t ph = (uint32_t)((gt / kStages) & 1);
        const bool zero_tail = t0 + 128 > N;
        if (lane == 0) {
          const uint32_t dst = base + kOffRing + (uint32_t)st * kStageBytes;
          // paged: the tile's page numbers, loaded together before the waits (K and V use the
          // same pages), so that the copies do not each wait for their own block-table read
          int phys[kPaged ? 8 : 1];
          int nvalid = 0;
          if (kPaged) {
            const int ps = p.page_size;
            const int first_page = t0 / ps;
            nvalid = min(128 / ps, (N + ps - 1) / ps - first_page);
            const int* bt = p.block_table + (size_t)b * p.max_pages + first_page;
#pragma unroll
            for (int pg = 0; pg < (kPaged ? 8 : 1); ++pg) phys[pg] = pg < nvalid ? bt[pg] : 0;
          }
          for (int which = 0; which < 2 && ok; ++which) {
            ok = mbar_wait(which ? emptyv_bar(st) : emptyk_bar(st), ph ^ 1u, abort_flag, p.dev_status);
            if (ok) {
              const CUtensorMap* map = which ? &map_v : &map_k;
              const uint32_t fb = which ? (zero_tail ? vload_bar(st) : fullv_bar(st)) : fullk_bar(st);
              const uint32_t d = dst + (uint32_t)which * kTileBytes;
              if (!kPaged) {
                const int row0 = (layer * p.batch + b) * p.seq_capacity + t0;
                mbar_arrive_expect_tx(fb, kTileBytes);
                tma_load_3d_hint(d, map, fb, 0, hkv, row0, kv_policy);
                tma_load_3d_hint(d + kHalfBytes, map, fb, 64, hkv, row0, kv_policy);
              } else {
                const int ps = p.page_size;
                mbar_arrive_expect_tx(fb, (uint32_t)(nvalid * 2 * ps * 128));
#pragma unroll
                for (int pg = 0; pg < (kPaged ? 8 : 1); ++pg) {
                  if (pg < nvalid) {
                    const int row0 = (layer * p.num_pages + phys[pg]) * ps;
                    const uint32_t off = (uint32_t)(pg * ps * 128);
                    tma_load_3d_hint(d + off, map, fb, 0, hkv, row0, kv_policy);
                    tma_load_3d_hint(d + kHalfBytes + off, map, fb, 64, hkv, row0, kv_policy);
                  }
                }
              }
            }
          }
        }
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (ok && zero_tail) {
          // V rows past the sequence: zero them so that P = 0 never meets a non-finite value
          ok = mbar_wait_warp(vload_bar(st), (uint32_t)(vloads[st] & 1), abort_flag, p.dev_status);
          vloads[st] += 1;
          if (ok) {
            const uint32_t vbase = base + kOffRing + (uint32_t)st * kStageBytes + kTileBytes;
            const int r0 = N - t0;
            for (int c = lane; c < (128 - r0) * 16; c += 32) {
              const int r = r0 + (c >> 4), hc = c & 15;
              st_shared_v4(vbase + (uint32_t)(hc >> 3) * kHalfBytes + (uint32_t)r * 128u + (uint32_t)(hc & 7) * 16u,
                           0, 0, 0, 0);
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(fullv_bar(st));
          }
        }
      }
    }
    if (!ok && lane == 0) {
      // drain the copies already issued (bounded) before the CTA can exit
      for (int back = 1; back <= kStages && gt - back >= 0; ++back) {
        const int j2 = gt - back;
        mbar_drain(fullk_bar(j2 % kStages), (uint32_t)((j2 / kStages) & 1), 100000000ull);
        mbar_drain(fullv_bar(j2 % kStages), (uint32_t)((j2 / kStages) & 1), 100000000ull);
        mbar_drain(vload_bar(j2 % kStages), (uint32_t)((vloads[j2 % kStages] + 1) & 1), 100000000ull);
      }
    }
  } else if (warp == 1) {
    // ================================================================ MMA issuer (one thread)
    const uint32_t q_base = base + kOffQ, ring = base + kOffRing;
    auto issue_s = [&](int tt, int st) {
      const uint32_t d = tmem + (uint32_t)tt * 128u;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t koff = (uint32_t)(kk >> 2) * kHalfBytes + (uint32_t)(kk & 3) * 32u;
        const uint64_t a = smem_desc_sw128(q_base + (uint32_t)tt * kTileBytes + koff, 16, 1024);
        const uint64_t bd = smem_desc_sw128(ring + (uint32_t)st * kStageBytes + koff, 16, 1024);
        mma_bf16_ss(d, a, bd, kIdescS, kk > 0 ? 1u : 0u);
      }
    };
    auto issue_pv = [&](int tt, int st, bool acc) {
      const uint32_t d = tmem + 256u + (uint32_t)tt * 128u;
      const uint32_t a = tmem + (uint32_t)tt * 128u;   // P: 16 keys = 8 packed columns per step
      const uint32_t vb = ring + (uint32_t)st * kStageBytes + kTileBytes;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint64_t bd = smem_desc_sw128(vb + (uint32_t)kk * 2048u, kHalfBytes, 1024);
        mma_bf16_ts(d, a + (uint32_t)kk * 8u, bd, kIdescPV, (acc || kk > 0) ? 1u : 0u);
      }
    };
    bool ok = true;
    int gt = 0;
    int tiles_t[2] = {0, 0}, segs_t[2] = {0, 0};
    // The whole warp walks the schedule together; lane 0 issues, and its status is
    // broadcast after every segment so that no lane is left waiting on the others.
    while (ok && advance()) {
      if (lane == 0) {
        const int n = sgv->kt_end - sgv->kt_begin;
        const int nt = sgv->nt;
        if (n > 0) {
          // Q of this segment is in shared memory
          for (int t = 0; t < nt && ok; ++t)
            ok = mbar_wait(qready_bar(t), (uint32_t)(segs_t[t] & 1), abort_flag, p.dev_status);
          if (ok) ok = mbar_wait(fullk_bar(gt % kStages), (uint32_t)((gt / kStages) & 1), abort_flag, p.dev_status);
          if (ok) {
            tc_fence_after();
            issue_s(0, gt % kStages);
            mma_commit(sfull_bar(0));
            if (nt == 2) {
              issue_s(1, gt % kStages);
              mma_commit(sfull_bar(1));
            }
            mma_commit(emptyk_bar(gt % kStages));   // K of this tile is no longer read
          }
          for (int jj = 0; jj < n && ok; ++jj, ++gt) {
            const int st = gt % kStages;
            const uint32_t ph = (uint32_t)((gt / kStages) & 1);
            if (!(ok = mbar_wait(fullv_bar(st), ph, abort_flag, p.dev_status))) break;
            if (!(ok = mbar_wait(pfull_bar(0), (uint32_t)(tiles_t[0] & 1), abort_flag, p.dev_status))) break;
            tc_fence_after();
            issue_pv(0, st, jj > 0);
            const bool more = jj + 1 < n;
            const int st1 = (gt + 1) % kStages;
            if (more) {
              if (!(ok = mbar_wait(fullk_bar(st1), (uint32_t)(((gt + 1) / kStages) & 1), abort_flag,
                                   p.dev_status)))
                break;
              tc_fence_after();
              issue_s(0, st1);
              mma_commit(sfull_bar(0));
              if (nt == 1) mma_commit(emptyk_bar(st1));
            }
            if (nt == 2) {
              if (!(ok = mbar_wait(pfull_bar(1), (uint32_t)(tiles_t[1] & 1), abort_flag, p.dev_status))) break;
              tc_fence_after();
              issue_pv(1, st, jj > 0);
            }
            mma_commit(emptyv_bar(st));   // V of this stage is no longer read
            if (more && nt == 2) {
              issue_s(1, st1);
              mma_commit(sfull_bar(1));
              mma_commit(emptyk_bar(st1));
            }
            ++tiles_t[0];
            if (nt == 2) ++tiles_t[1];
          }
          if (ok) {
            mma_commit(ofull_bar(0));
            ++segs_t[0];
            if (nt == 2) {
              mma_commit(ofull_bar(1));
              ++segs_t[1];
            }
          }
        }
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    }
    if (lane == 0 && !ok) {
      // error path: let the tensor core finish what was issued before TMEM is freed
      mma_commit(drain_bar);
      mbar_drain(drain_bar, 0, 100000000ull);
    }
  } else {
    // ================================================================ softmax / epilogue
    const int t = (warp - 2) >> 2;
    const int row = (warp & 3) * 32 + lane;   // = TMEM lane this warp may access
    const float sl2 = p.scale_log2;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + lane_base + (uint32_t)t * 128u;
    const uint32_t tO = tmem + lane_base + 256u + (uint32_t)t * 128u;
    const unsigned long long sl2x2 = f2_pack(sl2, sl2);
    const uint32_t qrow_smem = base + kOffQ + (uint32_t)t * kTileBytes + (uint32_t)row * 128u;
    WarpArea* wa = reinterpret_cast<WarpArea*>(smem + kOffWarp) + (warp - 2);
    volatile WarpArea* wv = wa;
    if (lane == 0) {
      wa->tree_node0 = -1;
      wa->tree_T = -1;
      wa->mask_mp = -1;
    }
    __syncwarp();
    uint32_t am0 = 0, am1 = 0, am2 = 0, am3 = 0;   // ancestor mask of this row's node
    int tiles = 0, segs = 0;
    bool ok = true;
    uint32_t r[32];

    // Next segment of the range that has rows in this warp's M tile.
    auto next_mine = [&]() -> bool {
      while (advance())
        if (t < sgv->nt) return true;
      return false;
    };
    // Takes the segment just walked to as run slot k: tree check and ancestor masks (the
    // parents of the last tree seen are kept in shared memory), Q rows, q_ready.
    auto prepare = [&](int k) {
      const int T = sgv->T, node0 = sgv->node0, mp = sgv->mp;
      const int grow = (2 * mp + t) * 128 + row;
      const int node = grow / G, g = grow - node * G;
      const bool row_valid = node < T;
      const bool has_keys = sgv->kt_end > sgv->kt_begin;
      // Q rows first: their loads overlap the tree work below (per-thread path only)
      uint4 v[16];
      if constexpr (!kQTma) {
        const size_t orow = (((size_t)sgv->lq * p.n_total + node0 + node) * p.hq + (size_t)sgv->hkv * G + g) * 128;
        const uint4* srcq = reinterpret_cast<const uint4*>(p.q) + (row_valid ? orow : 0) / 8;
#pragma unroll
        for (int c = 0; c < 16; ++c) v[c] = (row_valid && has_keys) ? __ldg(srcq + c) : make_uint4(0, 0, 0, 0);
      }
      if (node0 != wv->tree_node0 || T != wv->tree_T) {
        // tree validity (parents[0] = -1, 0 <= parents[i] < i), checked by every warp on its own
        bool bad = false;
        for (int i = lane; i < T; i += 32) {
          const int pp = __ldg(p.parents + node0 + i);
          wv->parents[i] = pp;
          bad = bad || (i == 0 ? (pp != -1) : (pp < 0 || pp >= i));
        }
        const bool invalid = __any_sync(0xffffffffu, bad);
        __syncwarp();
        if (lane == 0) {
          wa->tree_node0 = node0;
          wa->tree_T = T;
          wa->tree_invalid = invalid ? 1 : 0;
          wa->mask_mp = -1;
        }
        __syncwarp();
      }
      const bool invalid = wv->tree_invalid != 0;
      if (mp != wv->mask_mp) {
        // ancestor bitmask of this row's node (walk up the parent pointers, strictly decreasing)
        am0 = am1 = am2 = am3 = 0;
        if (row_valid && !invalid) {
          for (int q = node; q >= 0; q = wv->parents[q]) {
            const uint32_t bit = 1u << (q & 31);
            const int w = q >> 5;
            am0 |= w == 0 ? bit : 0u;
            am1 |= w == 1 ? bit : 0u;
            am2 |= w == 2 ? bit : 0u;
            am3 |= w == 3 ? bit : 0u;
          }
        }
        __syncwarp();
        if (lane == 0) wa->mask_mp = mp;
      }
      // keep the segment for the epilogue (the walker's slot moves on before it runs)
      constexpr int kSegWords = (int)(sizeof(Seg) / 4);
      if (lane < kSegWords)
        reinterpret_cast<volatile int*>(&wa->run[k].s)[lane] = reinterpret_cast<const volatile int*>(sgv)[lane];
      if (lane == 0) wa->run[k].invalid = invalid ? 1 : 0;
      if (kQTma && has_keys) {
        // Q tile of this segment by TMA (every S_t GEMM of the previous segment has
        // completed): 128 / G nodes x G heads of the pair's M tile, two 64-column halves
        if ((warp & 3) == 0 && lane == 0) {
          const int qrow = sgv->lq * p.n_total + node0 + ((2 * mp + t) * 128) / G;
          const uint32_t dst = base + kOffQ + (uint32_t)t * kTileBytes;
          mbar_arrive_expect_tx(qready_bar(t), 2 * kHalfBytes);
          tma_load_3d(dst, &map_q, qready_bar(t), 0, sgv->hkv * G, qrow);
          tma_load_3d(dst + kHalfBytes, &map_q, qready_bar(t), 64, sgv->hkv * G, qrow);
        }
      } else if (has_keys) {
        // Q rows of this segment (every S_t GEMM of the previous segment has completed)
#pragma unroll
        for (int c = 0; c < 16; ++c) {
          const int half = c >> 3, j = c & 7;
          const uint4 q4 = invalid ? make_uint4(0, 0, 0, 0) : v[c];
          st_shared_v4(qrow_smem + (uint32_t)half * kHalfBytes + (uint32_t)((j ^ (row & 7)) << 4), q4.x, q4.y,
                       q4.z, q4.w);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(qready_bar(t));
      }
      __syncwarp();
    };

    // Output rows of one 32-row block from all pieces of its unit:
    // O = sum_c 2^(m_c - M) O_c / sum_c 2^(m_c - M) l_c (pieces with l_c = 0 saw no key).
    // With `own`, this warp's piece is still in TMEM (O_t, m_own, l_own) rather than a partial.
    // M is the maximum over the pieces, and both sums run over the pieces in CTA order with
    // this warp's own piece at its CTA's place, so the result does not depend on which piece
    // happened to finish last: every launch writes the same bits.
    auto merge = [&](const volatile SegRun* rec, bool own, float m_own, float l_own) {
      const int ug0 = rec->s.ug0, ug1 = ug0 + rec->s.n_kt;
      const int T = rec->s.T, mp = rec->s.mp;
      const bool invalid = rec->invalid != 0;
      const int grow = (2 * mp + t) * 128 + row;
      const int node = grow / G, g = grow - node * G;
      const bool row_valid = node < T;
      const int first = owner_cta(wc, ug0), last = owner_cta(wc, ug1 - 1);
      const float2* pml = reinterpret_cast<const float2*>(p.part_ml) + (size_t)t * 128 + row;
      // CTAs whose partial is read (an empty range owns no piece; with `own`, skip this CTA)
      auto partial_of = [&](int c) {
        return c <= last && range_start(wc, c + 1) > range_start(wc, c) && !(own && c == wc.c);
      };
      auto piece_ml = [&](int c) -> float2 {
        if (own && c == wc.c) return make_float2(m_own, l_own);
        return partial_of(c) ? __ldcg(pml + (size_t)piece_slot(wc, c, ug0, ug1) * 256) : make_float2(-INFINITY, 0.f);
      };
      float M = -INFINITY, L = 0.f;
      for (int c = first; c <= last; ++c) {
        const float2 ml = piece_ml(c);
        if (ml.y > 0.f) M = fmaxf(M, ml.x);
      }
      for (int c = first; c <= last; ++c) {
        const float2 ml = piece_ml(c);
        if (ml.y > 0.f) L += ml.y * ptx_exp2(ml.x - M);
      }
      const float inv = (L > 0.f && !invalid) ? 1.f / L : 0.f;
      const float w_own = (own && l_own > 0.f) ? ptx_exp2(m_own - M) : 0.f;
      const size_t orow = (((size_t)rec->s.lq * p.n_total + rec->s.node0 + node) * p.hq + (size_t)rec->s.hkv * G + g) * 128;
      uint4* dst = reinterpret_cast<uint4*>(p.out) + (row_valid ? orow : 0) / 8;
#pragma unroll 1
      for (int h = 0; h < 4; ++h) {   // 32 output columns at a time
        float acc[32];
#pragma unroll
        for (int d = 0; d < 32; ++d) acc[d] = 0.f;
        for (int c = first; c <= last; ++c) {
          if (own && c == wc.c) {   // warp-uniform: this warp's piece, from TMEM
            tmem_ld32(tO + (uint32_t)h * 32u, r);
            tmem_ld_wait();
#pragma unroll
            for (int d = 0; d < 32; ++d) acc[d] = w_own > 0.f ? fmaf(w_own, __uint_as_float(r[d]), acc[d]) : acc[d];
            continue;
          }
          if (!partial_of(c)) continue;
          const size_t q = (size_t)piece_slot(wc, c, ug0, ug1);
          const float2 ml = __ldcg(pml + q * 256);
          // partial layout [slot][M tile][column / 4][128 rows][4]: four columns of a row in 16 bytes
          const float4* po = reinterpret_cast<const float4*>(p.part_o + (q * 2 + t) * (128 * 128)) +
                             (size_t)(h * 8) * 128 + row;
          float o[32];
#pragma unroll
          for (int g = 0; g < 8; ++g) {
            const float4 v4 = __ldcg(po + (size_t)g * 128);
            o[4 * g] = v4.x;
            o[4 * g + 1] = v4.y;
            o[4 * g + 2] = v4.z;
            o[4 * g + 3] = v4.w;
          }
          // rows of a piece that saw no key were not written: weight 0 and never read into acc
          const float wgt = ml.y > 0.f ? ptx_exp2(ml.x - M) : 0.f;
#pragma unroll
          for (int d = 0; d < 32; ++d) acc[d] = wgt > 0.f ? fmaf(wgt, o[d], acc[d]) : acc[d];
        }
        if (row_valid) {
#pragma unroll
          for (int c8 = 0; c8 < 4; ++c8) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) w[e] = pack_bf16x2(acc[c8 * 8 + 2 * e] * inv, acc[c8 * 8 + 2 * e + 1] * inv);
            dst[h * 4 + c8] = make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
      }
    };

    bool have = next_mine();
    int k = 0;   // run slot of the current segment
    if (have) prepare(0);
    while (have) {
      const volatile SegRun* cur = &wv->run[k];
      const int kt_begin = cur->s.kt_begin;
      const int C = cur->s.C;
      const int n = cur->s.kt_end - kt_begin;
      // Reference max m_run (log2 units) against which P = 2^(s*scale*log2e - m_run) is
      // taken.  It only moves up, and only when a 32-column chunk exceeds it by more than
      // 2^8; then the row sum, O and the P chunks already written for this tile are rescaled.
      float m_run = -INFINITY, l_run = 0.f;
      for (int jj = 0; jj < n; ++jj, ++tiles) {
        if (!(ok = mbar_wait_warp(sfull_bar(t), (uint32_t)(tiles & 1), abort_flag, p.dev_status))) break;
        tc_fence_after();
        const int t0 = (kt_begin + jj) * 128;
        const bool need_mask = t0 + 128 > C;   // warp-uniform
        unsigned long long sum = f2_pack(0.f, 0.f);
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          tmem_ld32(tS + (uint32_t)c * 32u, r);
          tmem_ld_wait();
          if (need_mask) {
            const uint32_t vw = vis_word(t0 + c * 32 - C, am0, am1, am2, am3);
#pragma unroll
            for (int e = 0; e < 32; ++e) r[e] = ((vw >> e) & 1u) ? r[e] : __float_as_uint(-INFINITY);
          }
          float cm;
          {
            float a0 = -INFINITY, a1 = -INFINITY;
#pragma unroll
            for (int e = 0; e < 32; e += 4) {
              a0 = fmax3(a0, __uint_as_float(r[e]), __uint_as_float(r[e + 1]));
              a1 = fmax3(a1, __uint_as_float(r[e + 2]), __uint_as_float(r[e + 3]));
            }
            cm = fmaxf(a0, a1) * sl2;
          }
          // The TMEM accesses of a rescale are warp-collective, so the whole warp takes the
          // branch when any of its rows needs it; the other rows rescale by exactly 1.  (Rows
          // differ when a piece starts on a key tile past the committed context: each row
          // first meets a visible ancestor in whichever chunk holds one.)
          const bool raise = cm > m_run + kRescaleLog2;
          if (__any_sync(0xffffffffu, raise)) {
            // raise the reference: rescale everything taken against the old one
            float alpha = 1.f;
            if (raise) {
              alpha = m_run == -INFINITY ? 0.f : ptx_exp2(m_run - cm);
              m_run = cm;
            }
            float s0, s1;
            f2_unpack(sum, s0, s1);
            sum = f2_pack(s0 * alpha, s1 * alpha);
            l_run *= alpha;
            rescale_tmem(tO, tS, jj > 0 ? 8 : 0, c, alpha);
          }
          const float m_use = m_run == -INFINITY ? 0.f : m_run;   // -inf only while nothing is visible
          const unsigned long long negm = f2_pack(-m_use, -m_use);
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            const unsigned long long x =
                f2_fma(f2_pack(__uint_as_float(r[e]), __uint_as_float(r[e + 1])), sl2x2, negm);
            float x0, x1;
            f2_unpack(x, x0, x1);
            const float p0 = ptx_exp2(x0), p1 = ptx_exp2(x1);
            sum = f2_add(sum, f2_pack(p0, p1));
            pk[e >> 1] = pack_bf16x2(p0, p1);
          }
          tmem_st16(tS + (uint32_t)c * 16u, pk);   // P chunk c: columns [16c, 16c+16) of S_t
        }
        {
          float s0, s1;
          f2_unpack(sum, s0, s1);
          l_run += s0 + s1;
        }
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(pfull_bar(t));
      }
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      // A piece: how many of its unit's pieces have left their partials, read now so that the
      // load overlaps the drain of this segment's last PV (the count only grows; a stale one
      // sends this warp down the partial path, which counts again).
      int seen = -1;
      if (cur->s.slot >= 0 && lane == 0 && !p.defer_merge)
        seen = epoch_read(p.counters + (size_t)cur->s.unit * 8 + t * 4 + (warp & 3), p.epoch);
      // Every S_t GEMM of this segment has completed (its last s_full was seen), so the next
      // segment's Q can go in now: the tensor core starts on it while this epilogue runs.
      const bool have_next = next_mine();
      if (have_next) prepare(k ^ 1);
      // ---- epilogue of the segment
      if (n > 0) {
        if (!(ok = mbar_wait_warp(ofull_bar(t), (uint32_t)(segs & 1), abort_flag, p.dev_status))) break;
        ++segs;
        tc_fence_after();
      }
      const bool invalid = cur->invalid != 0;
      const bool have_o = n > 0 && !invalid;
      if (invalid && lane == 0) atomicMax(p.dev_status, (int)PTD_ERR_INVALID_TREE);
      const int slot = cur->s.slot;
      if (slot < 0) {
        // the whole unit: normalised bf16 output
        const int T = cur->s.T;
        const int grow = (2 * cur->s.mp + t) * 128 + row;
        const int node = grow / G, g = grow - node * G;
        const bool row_valid = node < T;
        const size_t orow =
            (((size_t)cur->s.lq * p.n_total + cur->s.node0 + node) * p.hq + (size_t)cur->s.hkv * G + g) * 128;
        const float inv = (have_o && l_run > 0.f) ? 1.f / l_run : 0.f;
        uint4* dst = reinterpret_cast<uint4*>(p.out) + (row_valid ? orow : 0) / 8;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          if (n > 0) {
            tmem_ld32(tO + (uint32_t)c * 32u, r);
            tmem_ld_wait();
          }
          if (row_valid) {
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) {
              uint32_t w[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float a0 = have_o ? __uint_as_float(r[q4 * 8 + 2 * e]) * inv : 0.f;
                const float a1 = have_o ? __uint_as_float(r[q4 * 8 + 2 * e + 1]) * inv : 0.f;
                w[e] = pack_bf16x2(a0, a1);
              }
              dst[c * 4 + q4] = make_uint4(w[0], w[1], w[2], w[3]);
            }
          }
        }
      } else {
        // A piece.  If every other piece of this 32-row block has left its partial, this warp
        // finishes the block from its own O in TMEM.  Otherwise it leaves a partial (O
        // unnormalised, running max in log2 units, row sum; four columns of a row per 16 bytes,
        // rows consecutive, so each store of the warp is 512 contiguous bytes) and counts
        // itself in; if that makes it the last, it merges the partials.  (Ranges are walked forward, so the piece at the start
        // of a range is normally done long before the piece that ends the previous range.)
        const int ug0 = cur->s.ug0;
        const int ug1 = ug0 + cur->s.n_kt;
        const int first = owner_cta(wc, ug0);
        const int last = owner_cta(wc, ug1 - 1);
        unsigned long long* counter = p.counters + (size_t)cur->s.unit * 8 + t * 4 + (warp & 3);
        int pieces = 0, done = 0;
        if (lane == 0) {
          for (int c = first; c <= last; ++c) pieces += range_start(wc, c + 1) > range_start(wc, c) ? 1 : 0;
          done = seen == pieces - 1;
        }
        done = __shfl_sync(0xffffffffu, done, 0) && !p.defer_merge;
        if (done) {
          __threadfence();
          merge(cur, true, have_o ? m_run : -INFINITY, have_o ? l_run : 0.f);
        } else {
          float4* po = reinterpret_cast<float4*>(p.part_o + ((size_t)slot * 2 + t) * (128 * 128)) + row;
#pragma unroll 1
          for (int c = 0; c < 4; ++c) {
            tmem_ld32(tO + (uint32_t)c * 32u, r);
            tmem_ld_wait();
            if (have_o) {
#pragma unroll
              for (int g = 0; g < 8; ++g)
                po[(size_t)(c * 8 + g) * 128] = make_float4(__uint_as_float(r[4 * g]), __uint_as_float(r[4 * g + 1]),
                                                            __uint_as_float(r[4 * g + 2]), __uint_as_float(r[4 * g + 3]));
            }
          }
          reinterpret_cast<float2*>(p.part_ml)[(size_t)slot * 256 + (size_t)t * 128 + row] =
              have_o ? make_float2(m_run, l_run) : make_float2(-INFINITY, 0.f);
          int is_last = 0;
          if (!p.defer_merge) {   // count in; the last piece merges (else the merge kernel does)
            __threadfence();
            __syncwarp();
            if (lane == 0) {
              const int now = epoch_increment(counter, p.epoch);
              if (now < 0) atomicMax(p.dev_status, (int)PTD_ERR_TIMEOUT);
              is_last = now == pieces;
            }
            is_last = __shfl_sync(0xffffffffu, is_last, 0);
          }
          if (is_last) {
            __threadfence();
            merge(cur, false, 0.f, 0.f);
          }
        }
      }
      tc_fence_before();
      k ^= 1;
      have = have_next;
    }
  }

  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------- merge of split units
// CTA (unit, column part) of the persistent cut, 256 threads = (M tile t, row); the unit's
// 128 output columns are cut into `hsplit` parts (1, 2 or 4) of 128 / hsplit columns.  A unit
// whose key tiles fall in one CTA's range was written whole by the attention; otherwise
// every piece left a partial and the rows are
//   O = sum_c 2^(m_c - M) O_c / sum_c 2^(m_c - M) l_c   over the pieces in CTA order
// (M the maximum over the pieces; a piece that saw no key has l_c = 0 and weight 0).
constexpr int kMergeThreads = 256;
constexpr int kMergeBatch = 2;   // pieces whose partial columns are in flight at a time
constexpr int kMergeMl = 8;      // pieces whose (m, l) stay in registers

__global__ void __launch_bounds__(kMergeThreads, 2) tree_attn_merge_kernel(const AttnParams p, int hsplit) {
  if (threadIdx.x == 0) grid_launch_dependents();   // the next grid may be placed now; it waits for this one
  grid_dependency_wait();   // the partials and the trees belong to the attention grid before this one
  int u = blockIdx.x / hsplit;
  const int hs = blockIdx.x - u * hsplit;
  const int mp = u % p.pairs;
  u /= p.pairs;
  const int hkv = u % p.hkv;
  u /= p.hkv;
  const int b = u % p.batch;
  const int lq = u / p.batch;
  int node0, T, C, n_kt, pairs_b;
  if (seq_info(p, nullptr, b, node0, T, C, n_kt, pairs_b) == 0 || mp >= pairs_b) return;
  // the flattened (unit, key tile) position of the unit, as the attention's walk decodes it
  int wl = 0, before = 0;
  for (int bb = 0; bb < p.batch; ++bb) {
    int n0, tt, cc, nk, pr;
    const int w = seq_info(p, nullptr, bb, n0, tt, cc, nk, pr);
    if (bb < b) before += w;
    wl += w;
  }
  WalkConst wc;
  wc.persistent = 1;
  wc.Wl = wl;
  wc.W = wl * p.layers;
  wc.P = p.ctas;
  wc.c = 0;
  wc.r0 = wc.r1 = 0;
  const int ug0 = lq * wl + before + (hkv * pairs_b + mp) * n_kt, ug1 = ug0 + n_kt;
  const int first = owner_cta(wc, ug0), last = owner_cta(wc, ug1 - 1);
  if (first == last) return;   // whole: written by the attention
  const int t = threadIdx.x >> 7, row = threadIdx.x & 127;
  const int nt = min(2, (T * p.group + 127) / 128 - 2 * mp);
  if (t >= nt) return;
  const int G = p.group;
  const int grow = (2 * mp + t) * 128 + row;
  const int node = grow / G, g = grow - node * G;
  if (node >= T) return;   // padding row of the M tile: no output
  const float2* pml = reinterpret_cast<const float2*>(p.part_ml) + (size_t)t * 128 + row;
  auto has_piece = [&](int c) { return c <= last && range_start(wc, c + 1) > range_start(wc, c); };
  auto piece_ml = [&](int c) -> float2 {
    return has_piece(c) ? __ldcg(pml + (size_t)piece_slot(wc, c, ug0, ug1) * 256) : make_float2(-INFINITY, 0.f);
  };
  float2 mlc[kMergeMl];
#pragma unroll
  for (int q = 0; q < kMergeMl; ++q) mlc[q] = piece_ml(first + q);
  float M = -INFINITY, L = 0.f;
#pragma unroll
  for (int q = 0; q < kMergeMl; ++q)
    if (mlc[q].y > 0.f) M = fmaxf(M, mlc[q].x);
  for (int c = first + kMergeMl; c <= last; ++c) {
    const float2 ml = piece_ml(c);
    if (ml.y > 0.f) M = fmaxf(M, ml.x);
  }
#pragma unroll
  for (int q = 0; q < kMergeMl; ++q)
    if (mlc[q].y > 0.f) L += mlc[q].y * ptx_exp2(mlc[q].x - M);
  for (int c = first + kMergeMl; c <= last; ++c) {
    const float2 ml = piece_ml(c);
    if (ml.y > 0.f) L += ml.y * ptx_exp2(ml.x - M);
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  const size_t orow = (((size_t)lq * p.n_total + node0 + node) * p.hq + (size_t)hkv * G + g) * 128;
  uint4* dst = reinterpret_cast<uint4*>(p.out) + orow / 8;
  const int h_per = 4 / hsplit;
#pragma unroll 1
  for (int h = hs * h_per; h < (hs + 1) * h_per; ++h) {   // 32 output columns at a time
    float acc[32];
#pragma unroll
    for (int d = 0; d < 32; ++d) acc[d] = 0.f;
    for (int c0 = first; c0 <= last; c0 += kMergeBatch) {
      float4 o[kMergeBatch][8];
      float wgt[kMergeBatch];
#pragma unroll
      for (int q = 0; q < kMergeBatch; ++q) {
        const int c = c0 + q;
        wgt[q] = 0.f;
        if (has_piece(c)) {
          const size_t sl = (size_t)piece_slot(wc, c, ug0, ug1);
          const float2 ml = __ldcg(pml + sl * 256);
          const float4* po = reinterpret_cast<const float4*>(p.part_o + (sl * 2 + t) * (128 * 128)) +
                             (size_t)(h * 8) * 128 + row;
#pragma unroll
          for (int gg = 0; gg < 8; ++gg) o[q][gg] = __ldcg(po + (size_t)gg * 128);
          // rows of a piece that saw no key were not written: weight 0 and never read into acc
          wgt[q] = ml.y > 0.f ? ptx_exp2(ml.x - M) : 0.f;
        }
      }
#pragma unroll
      for (int q = 0; q < kMergeBatch; ++q) {
        if (wgt[q] > 0.f) {
#pragma unroll
          for (int gg = 0; gg < 8; ++gg) {
            acc[4 * gg] = fmaf(wgt[q], o[q][gg].x, acc[4 * gg]);
            acc[4 * gg + 1] = fmaf(wgt[q], o[q][gg].y, acc[4 * gg + 1]);
            acc[4 * gg + 2] = fmaf(wgt[q], o[q][gg].z, acc[4 * gg + 2]);
            acc[4 * gg + 3] = fmaf(wgt[q], o[q][gg].w, acc[4 * gg + 3]);
          }
        }
      }
    }
#pragma unroll
    for (int c8 = 0; c8 < 4; ++c8) {
      uint32_t w[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) w[e] = pack_bf16x2(acc[c8 * 8 + 2 * e] * inv, acc[c8 * 8 + 2 * e + 1] * inv);
      dst[h * 4 + c8] = make_uint4(w[0], w[1], w[2], w[3]);
    }
  }
}

}  // namespace tc

// ------------------------------------------------------------------- host launchers
size_t tc_smem_bytes() { return tc::kSmemBytes; }

cudaError_t launch_tree_attn_merge(const AttnParams& p, int units, int sms, cudaStream_t stream) {
  // column parts per unit: about two CTAs per SM over the grid (1, 2 or 4)
  const int want = units > 0 ? 2 * sms / units : 1;
  const int hsplit = want >= 4 ? 4 : (want >= 2 ? 2 : 1);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(units * hsplit), 1, 1);
  cfg.blockDim = dim3(tc::kMergeThreads, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // placed while the attention drains
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, tc::tree_attn_merge_kernel, p, hsplit);
}

cudaError_t launch_tree_attn_tc(const CUtensorMap& map_k, const CUtensorMap& map_v, const CUtensorMap& map_q,
                                const AttnParams& p, dim3 grid, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(tc::kThreads, 1, 1);
  cfg.dynamicSmemBytes = tc::kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // set-up overlaps the previous kernel
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
#define PTD_TC_LAUNCH(PAGED, QTMA)                                                                            \
  do {                                                                                                       \
    cudaError_t e = cudaFuncSetAttribute(tc::tree_attn_tc_kernel<PAGED, QTMA>,                               \
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tc::kSmemBytes);  \
    if (e != cudaSuccess) return e;                                                                          \
    return cudaLaunchKernelEx(&cfg, tc::tree_attn_tc_kernel<PAGED, QTMA>, map_k, map_v, map_q, p);           \
  } while (0)
  if (p.page_size > 0) {
    if (p.q_tma)
      PTD_TC_LAUNCH(true, true);
    else
      PTD_TC_LAUNCH(true, false);
  } else {
    if (p.q_tma)
      PTD_TC_LAUNCH(false, true);
    else
      PTD_TC_LAUNCH(false, false);
  }
#undef PTD_TC_LAUNCH
}


}  // namespace ptd
