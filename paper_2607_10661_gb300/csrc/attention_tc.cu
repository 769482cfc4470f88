// Tree-masked attention on the 5th-generation tensor cores (tcgen05 + TMEM + TMA), bf16.
//
// What it computes (Sec. 3.1 visibility pi(v) = {v} U pi(P(v)); Sec. 3.2 one pass over
// [X; T; C_X]): for every layer, tree b, KV head, query head h of that KV head's group and
// tree node i, the softmax-weighted sum of V over the committed slots [0, C_b) and the
// slots C_b + a of i's ancestors a (itself included).
//
// Work decomposition.  All G = Hq/Hkv query heads of one KV head and all T_b nodes of a
// tree form the rows of one dense problem: row r = node * G + g, so M = T_b * G rows share
// every K/V tile.  A CTA owns two 128-row M tiles (256 rows, e.g. 63 nodes x 4 heads) of
// one (layer, tree, KV head) and a contiguous range of 128-key tiles (a KV split).  Each
// K/V tile is loaded from HBM once by TMA and used by both M tiles.
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
//               at the end O / l (or a split partial).  Tiles that lie entirely inside the
//               committed prefix skip the mask arithmetic.
// TMEM: S_0 | S_1 | O_0 | O_1, 128 fp32 columns each = all 512 columns of the SM; P_t
// takes the first 64 columns of S_t (two bf16 per column).
// The ancestor mask of a row's node (up to 128 bits) lives in 4 registers of its thread.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

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
constexpr uint32_t kOffScratch = kOffRing + kStageBytes + kTileBytes;   // setup only (V of stage 1)
constexpr uint32_t kOffBar = kOffRing + kStages * kStageBytes;
// barriers: full_k[2], full_v[2], empty[2], vzero, s_full[2], p_full[2], o_full[2], drain
constexpr uint32_t kNumBars = 3 * kStages + 8;
constexpr uint32_t kOffTmemPtr = kOffBar + kNumBars * 8;
constexpr uint32_t kOffAbort = kOffTmemPtr + 4;
constexpr uint32_t kSmemUsed = kOffAbort + 4;
constexpr uint32_t kSmemBytes = kSmemUsed + 1024;   // slack to align the base to 1024 B
static_assert(kSmemBytes <= 232448, "shared memory budget");
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

template <bool kPaged>
__global__ void __launch_bounds__(kThreads, 1)
    tree_attn_tc_kernel(const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_v,
                        const AttnParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint32_t base = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (base & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  base += pad;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // ---- work unit
  int u = blockIdx.x;
  const int unit = u;
  const int mp = u % p.pairs;
  u /= p.pairs;
  const int hkv = u % p.hkv;
  u /= p.hkv;
  const int b = u % p.batch;
  const int lq = u / p.batch;
  const int layer = p.layer_begin + lq;
  const int split = blockIdx.y;
  const int G = p.group;

  const int node0 = p.node_offsets[b];
  const int T = p.node_offsets[b + 1] - node0;
  const int C = p.ctx_lens[b];
  const int N = C + T;
  bool bad_shape = T < 1 || T > p.max_nodes || node0 < 0 || node0 + T > p.n_total || C < 0;
  if (!bad_shape) {
    if (kPaged)
      bad_shape = N > p.max_pages * p.page_size;
    else
      bad_shape = N > p.seq_capacity;
  }
  if (bad_shape) {
    if (threadIdx.x == 0) atomicMax(p.dev_status, (int)PTD_ERR_INVALID_TREE);
    return;
  }
  const int rows = T * G;
  const int tiles_b = (rows + 127) >> 7;
  const int nt = min(2, tiles_b - 2 * mp);
  if (nt <= 0) return;   // this pair of M tiles is past the tree (uniform over the CTA)

  const int n_kt = (N + 127) >> 7;
  const int tps = (n_kt + p.splits - 1) / p.splits;
  const int kt_begin = split * tps;
  const int n_local = max(0, min(n_kt, kt_begin + tps) - kt_begin);

  auto bar = [&](int i) { return base + kOffBar + 8u * (uint32_t)i; };
  auto fullk_bar = [&](int s) { return bar(s); };
  auto fullv_bar = [&](int s) { return bar(kStages + s); };
  auto empty_bar = [&](int s) { return bar(2 * kStages + s); };
  const uint32_t vzero_bar = bar(3 * kStages);
  auto sfull_bar = [&](int t) { return bar(3 * kStages + 1 + t); };
  auto pfull_bar = [&](int t) { return bar(3 * kStages + 3 + t); };
  auto ofull_bar = [&](int t) { return bar(3 * kStages + 5 + t); };
  const uint32_t drain_bar = bar(3 * kStages + 7);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffAbort);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(fullk_bar(s), 1);
      mbar_init(fullv_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(vzero_bar, 1);
    for (int t = 0; t < 2; ++t) {
      mbar_init(sfull_bar(t), 1);
      mbar_init(pfull_bar(t), 4);   // one arrival per softmax warp
      mbar_init(ofull_bar(t), 1);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(base + kOffTmemPtr, kTmemCols);
    tmem_relinquish();
    tc_fence_before();
  }

  // ---- tree: validate and build ancestor masks (scratch in the last ring slot)
  int* par_s = reinterpret_cast<int*>(smem + kOffScratch);
  uint32_t* anc_s = reinterpret_cast<uint32_t*>(smem + kOffScratch + 512);
  bool bad = false;
  if (threadIdx.x < T) {
    const int pp = p.parents[node0 + threadIdx.x];
    par_s[threadIdx.x] = pp;
    bad = threadIdx.x == 0 ? (pp != -1) : (pp < 0 || pp >= (int)threadIdx.x);
  }
  const int invalid = __syncthreads_or(bad);
  if (!invalid && threadIdx.x < T) {
    uint32_t m0 = 0, m1 = 0, m2 = 0, m3 = 0;
    for (int a = threadIdx.x; a >= 0; a = par_s[a]) {   // parents strictly decrease
      const uint32_t bit = 1u << (a & 31);
      const int w = a >> 5;
      m0 |= w == 0 ? bit : 0u;
      m1 |= w == 1 ? bit : 0u;
      m2 |= w == 2 ? bit : 0u;
      m3 |= w == 3 ? bit : 0u;
    }
    anc_s[threadIdx.x * 4 + 0] = m0;
    anc_s[threadIdx.x * 4 + 1] = m1;
    anc_s[threadIdx.x * 4 + 2] = m2;
    anc_s[threadIdx.x * 4 + 3] = m3;
  }
  __syncthreads();

  // ---- softmax-thread identity, ancestor mask and Q row
  const bool is_sm = warp >= 2;
  const int t = is_sm ? (warp - 2) >> 2 : 0;
  const int row = (warp & 3) * 32 + lane;   // = TMEM lane this warp may access
  const int grow = (2 * mp + t) * 128 + row;
  const int node = grow / G;
  const int g = grow - node * G;
  const bool active_t = is_sm && t < nt;
  const bool row_valid = active_t && node < T;
  uint32_t am0 = 0, am1 = 0, am2 = 0, am3 = 0;
  if (row_valid && !invalid) {
    am0 = anc_s[node * 4 + 0];
    am1 = anc_s[node * 4 + 1];
    am2 = anc_s[node * 4 + 2];
    am3 = anc_s[node * 4 + 3];
  }
  const size_t qo_row = row_valid ? ((((size_t)lq * p.n_total + node0 + node) * p.hq + (size_t)hkv * G + g) * 128)
                                  : 0;
  if (active_t && !invalid) {
    const uint32_t qrow = base + kOffQ + (uint32_t)t * kTileBytes + (uint32_t)row * 128u;
    const uint4* src = reinterpret_cast<const uint4*>(p.q) + qo_row / 8;
#pragma unroll
    for (int c = 0; c < 16; ++c) {
      uint4 v = make_uint4(0, 0, 0, 0);
      if (row_valid) v = __ldg(src + c);
      const int half = c >> 3, j = c & 7;
      st_shared_v4(qrow + (uint32_t)half * kHalfBytes + (uint32_t)((j ^ (row & 7)) << 4), v.x, v.y, v.z, v.w);
    }
  }
  fence_proxy_async_smem();
  __syncthreads();   // Q visible to the tensor core; the scratch slot is free again
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + kOffTmemPtr);

  const size_t part_base = ((size_t)unit * p.splits + split) * 256;   // pair-local row base

  if (invalid) {
    // A malformed parent array: define the outputs as zero and report it.
    if (threadIdx.x == 0) atomicMax(p.dev_status, (int)PTD_ERR_INVALID_TREE);
    if (row_valid) {
      if (p.splits == 1) {
        uint4* dst = reinterpret_cast<uint4*>(p.out) + qo_row / 8;
        for (int c = 0; c < 16; ++c) dst[c] = make_uint4(0, 0, 0, 0);
      } else {
        const size_t pr = part_base + (size_t)t * 128 + row;
        p.part_ml[pr * 2 + 0] = -INFINITY;
        p.part_ml[pr * 2 + 1] = 0.f;
      }
    }
  } else if (warp == 0) {
    // ================================================================ TMA producer
    if (n_local > 0) {
      if (lane == 0) {
        prefetch_tensormap(&map_k);
        prefetch_tensormap(&map_v);
      }
      bool ok = true;
      int jj = 0;
      for (; jj < n_local && ok; ++jj) {
        const int t0 = (kt_begin + jj) * 128;
        const int st = jj % kStages;
        const uint32_t ph = (uint32_t)((jj / kStages) & 1);
        if (lane == 0) {
          ok = mbar_wait(empty_bar(st), ph ^ 1u, abort_flag, p.dev_status);
          if (ok) {
            const uint32_t dst = base + kOffRing + (uint32_t)st * kStageBytes;
            for (int which = 0; which < 2; ++which) {
              const CUtensorMap* map = which ? &map_v : &map_k;
              const uint32_t fb = which ? fullv_bar(st) : fullk_bar(st);
              const uint32_t d = dst + (uint32_t)which * kTileBytes;
              if (!kPaged) {
                const int row0 = (layer * p.batch + b) * p.seq_capacity + t0;
                mbar_arrive_expect_tx(fb, kTileBytes);
                tma_load_3d(d, map, fb, 0, hkv, row0);
                tma_load_3d(d + kHalfBytes, map, fb, 64, hkv, row0);
              } else {
                const int ps = p.page_size;
                const int first_page = t0 / ps;
                const int seq_pages = (N + ps - 1) / ps;
                const int nvalid = min(128 / ps, seq_pages - first_page);
                mbar_arrive_expect_tx(fb, (uint32_t)(nvalid * 2 * ps * 128));
                for (int pg = 0; pg < nvalid; ++pg) {
                  const int phys = p.block_table[(size_t)b * p.max_pages + first_page + pg];
                  const int row0 = (layer * p.num_pages + phys) * ps;
                  const uint32_t off = (uint32_t)(pg * ps * 128);
                  tma_load_3d(d + off, map, fb, 0, hkv, row0);
                  tma_load_3d(d + kHalfBytes + off, map, fb, 64, hkv, row0);
                }
              }
            }
          }
        }
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (ok && t0 + 128 > N) {
          // V rows past the sequence: zero them so that P = 0 never meets a non-finite value
          if ((ok = mbar_wait_warp(fullv_bar(st), ph, abort_flag, p.dev_status))) {
            const uint32_t vbase = base + kOffRing + (uint32_t)st * kStageBytes + kTileBytes;
            const int r0 = N - t0;
            for (int c = lane; c < (128 - r0) * 16; c += 32) {
              const int r = r0 + (c >> 4), hc = c & 15;
              st_shared_v4(vbase + (uint32_t)(hc >> 3) * kHalfBytes + (uint32_t)r * 128u + (uint32_t)(hc & 7) * 16u,
                           0, 0, 0, 0);
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(vzero_bar);
          }
        }
      }
      if (!ok && lane == 0) {
        // drain the copies already issued (bounded) before the CTA can exit
        for (int back = 1; back <= kStages && jj - back >= 0; ++back) {
          const int j2 = jj - back;
          mbar_drain(fullk_bar(j2 % kStages), (uint32_t)((j2 / kStages) & 1), 100000000ull);
          mbar_drain(fullv_bar(j2 % kStages), (uint32_t)((j2 / kStages) & 1), 100000000ull);
        }
      }
    }
  } else if (warp == 1) {
    // ================================================================ MMA issuer (one thread)
    if (n_local > 0 && lane == 0) {
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
      bool ok = mbar_wait(fullk_bar(0), 0, abort_flag, p.dev_status);
      tc_fence_after();
      if (ok) {
        issue_s(0, 0);
        mma_commit(sfull_bar(0));
        if (nt == 2) {
          issue_s(1, 0);
          mma_commit(sfull_bar(1));
        }
      }
      for (int jj = 0; jj < n_local && ok; ++jj) {
        const int st = jj % kStages;
        const uint32_t ph = (uint32_t)((jj / kStages) & 1);
        const int t0 = (kt_begin + jj) * 128;
        // V of this tile (zeroed past the sequence by the producer warp on the last tile)
        if (!(ok = (t0 + 128 > N) ? mbar_wait(vzero_bar, 0, abort_flag, p.dev_status)
                                  : mbar_wait(fullv_bar(st), ph, abort_flag, p.dev_status)))
          break;
        if (!(ok = mbar_wait(pfull_bar(0), (uint32_t)(jj & 1), abort_flag, p.dev_status))) break;
        tc_fence_after();
        issue_pv(0, st, jj > 0);
        const bool more = jj + 1 < n_local;
        const int st1 = (jj + 1) % kStages;
        if (more) {
          if (!(ok = mbar_wait(fullk_bar(st1), (uint32_t)(((jj + 1) / kStages) & 1), abort_flag, p.dev_status)))
            break;
          tc_fence_after();
          issue_s(0, st1);
          mma_commit(sfull_bar(0));
        }
        if (nt == 2) {
          if (!(ok = mbar_wait(pfull_bar(1), (uint32_t)(jj & 1), abort_flag, p.dev_status))) break;
          tc_fence_after();
          issue_pv(1, st, jj > 0);
        }
        mma_commit(empty_bar(st));   // K and V of this stage are no longer read
        if (more && nt == 2) {
          issue_s(1, st1);
          mma_commit(sfull_bar(1));
        }
      }
      mma_commit(ofull_bar(0));
      if (nt == 2) mma_commit(ofull_bar(1));
      if (!ok) {
        // error path: let the tensor core finish what was issued before TMEM is freed
        mma_commit(drain_bar);
        mbar_drain(drain_bar, 0, 100000000ull);
      }
    }
  } else if (active_t) {
    // ================================================================ softmax / epilogue
    const float sl2 = p.scale_log2;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t tS = tmem + lane_base + (uint32_t)t * 128u;
    const uint32_t tO = tmem + lane_base + 256u + (uint32_t)t * 128u;
    const unsigned long long sl2x2 = f2_pack(sl2, sl2);
    // Reference max m_run (log2 units) against which P = 2^(s*scale*log2e - m_run) is taken.
    // It only moves up, and only when a 32-column chunk exceeds it by more than 2^8; then the
    // row sum, O and the P chunks already written for this tile are rescaled (rare).
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    uint32_t r[32];
    for (int jj = 0; jj < n_local; ++jj) {
      if (!(ok = mbar_wait_warp(sfull_bar(t), (uint32_t)(jj & 1), abort_flag, p.dev_status))) break;
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
        // differ when a split starts on a key tile past the committed context: each row
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
          if (jj > 0) {
            // O_t is idle here: PV_t of the previous tile completed before S_t of this one
#pragma unroll 1
            for (int q = 0; q < 8; ++q) {
              uint32_t o16[16];
              tmem_ld16(tO + (uint32_t)q * 16u, o16);
              tmem_ld_wait();
#pragma unroll
              for (int e = 0; e < 16; ++e) o16[e] = __float_as_uint(__uint_as_float(o16[e]) * alpha);
              tmem_st16(tO + (uint32_t)q * 16u, o16);
            }
          }
          if (c > 0) {
            tmem_st_wait();
#pragma unroll 1
            for (int q = 0; q < c; ++q) {   // bf16 P of the earlier chunks of this tile
              uint32_t p16[16];
              tmem_ld16(tS + (uint32_t)q * 16u, p16);
              tmem_ld_wait();
#pragma unroll
              for (int e = 0; e < 16; ++e)
                p16[e] = pack_bf16x2(__uint_as_float(p16[e] << 16) * alpha,
                                     __uint_as_float(p16[e] & 0xFFFF0000u) * alpha);
              tmem_st16(tS + (uint32_t)q * 16u, p16);
            }
          }
        }
        const float m_use = m_run == -INFINITY ? 0.f : m_run;   // -inf only when nothing is visible yet
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
    // ---- epilogue
    ok = __all_sync(0xffffffffu, ok);
    if (ok && n_local > 0) ok = mbar_wait_warp(ofull_bar(t), 0, abort_flag, p.dev_status);
    tc_fence_after();
    const bool have_o = ok && n_local > 0;
    if (p.splits == 1) {
      const float inv = (have_o && l_run > 0.f) ? 1.f / l_run : 0.f;
      uint4* dst = reinterpret_cast<uint4*>(p.out) + qo_row / 8;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        if (have_o) {
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
      const size_t pr = part_base + (size_t)t * 128 + row;
      float4* po = reinterpret_cast<float4*>(p.part_o + pr * 128);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        if (have_o) {
          tmem_ld32(tO + (uint32_t)c * 32u, r);
          tmem_ld_wait();
        }
        if (row_valid && have_o) {
#pragma unroll
          for (int q4 = 0; q4 < 8; ++q4)
            po[c * 8 + q4] = make_float4(__uint_as_float(r[q4 * 4 + 0]), __uint_as_float(r[q4 * 4 + 1]),
                                         __uint_as_float(r[q4 * 4 + 2]), __uint_as_float(r[q4 * 4 + 3]));
        }
      }
      if (row_valid) {
        p.part_ml[pr * 2 + 0] = have_o ? m_run : -INFINITY;
        p.part_ml[pr * 2 + 1] = have_o ? l_run : 0.f;
      }
    }
    tc_fence_before();
  }

  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Merge the per-split partials (O unnormalised, running max m in log2 units, sum l) of
// every row: O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s.  One warp per row.
__global__ void __launch_bounds__(256) attn_combine_kernel(const AttnParams p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int u = blockIdx.x;
  const int unit = u;
  const int mp = u % p.pairs;
  u /= p.pairs;
  const int hkv = u % p.hkv;
  u /= p.hkv;
  const int b = u % p.batch;
  const int lq = u / p.batch;
  const int G = p.group;
  const int node0 = p.node_offsets[b];
  const int T = p.node_offsets[b + 1] - node0;
  if (T < 1 || T > p.max_nodes || node0 < 0 || node0 + T > p.n_total) return;
  const int prow = blockIdx.y * 8 + warp;   // 0..255
  const int grow = mp * 256 + prow;
  const int node = grow / G, g = grow - node * G;
  if (node >= T) return;
  float M = -INFINITY;
  for (int s = 0; s < p.splits; ++s) {
    const size_t pr = ((size_t)unit * p.splits + s) * 256 + prow;
    if (p.part_ml[pr * 2 + 1] > 0.f) M = fmaxf(M, p.part_ml[pr * 2 + 0]);
  }
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float L = 0.f;
  for (int s = 0; s < p.splits; ++s) {
    const size_t pr = ((size_t)unit * p.splits + s) * 256 + prow;
    const float l = p.part_ml[pr * 2 + 1];
    if (!(l > 0.f)) continue;
    const float w = ptx_exp2(p.part_ml[pr * 2 + 0] - M);
    L += w * l;
    const float4 o = reinterpret_cast<const float4*>(p.part_o + pr * 128)[lane];
    acc.x = fmaf(w, o.x, acc.x);
    acc.y = fmaf(w, o.y, acc.y);
    acc.z = fmaf(w, o.z, acc.z);
    acc.w = fmaf(w, o.w, acc.w);
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  const size_t orow = (((size_t)lq * p.n_total + node0 + node) * p.hq + (size_t)hkv * G + g) * 128;
  uint2 w2;
  w2.x = pack_bf16x2(acc.x * inv, acc.y * inv);
  w2.y = pack_bf16x2(acc.z * inv, acc.w * inv);
  reinterpret_cast<uint2*>(reinterpret_cast<__nv_bfloat16*>(p.out) + orow)[lane] = w2;
}

}  // namespace tc

// ------------------------------------------------------------------- host launchers
size_t tc_smem_bytes() { return tc::kSmemBytes; }

cudaError_t launch_tree_attn_tc(const CUtensorMap& map_k, const CUtensorMap& map_v, const AttnParams& p,
                                int units, cudaStream_t stream) {
  const dim3 grid((unsigned)units, (unsigned)p.splits);
  if (p.page_size > 0) {
    cudaError_t e = cudaFuncSetAttribute(tc::tree_attn_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)tc::kSmemBytes);
    if (e != cudaSuccess) return e;
    tc::tree_attn_tc_kernel<true><<<grid, tc::kThreads, tc::kSmemBytes, stream>>>(map_k, map_v, p);
  } else {
    cudaError_t e = cudaFuncSetAttribute(tc::tree_attn_tc_kernel<false>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tc::kSmemBytes);
    if (e != cudaSuccess) return e;
    tc::tree_attn_tc_kernel<false><<<grid, tc::kThreads, tc::kSmemBytes, stream>>>(map_k, map_v, p);
  }
  return cudaGetLastError();
}

cudaError_t launch_attn_combine(const AttnParams& p, int units, cudaStream_t stream) {
  tc::attn_combine_kernel<<<dim3((unsigned)units, 32), 256, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace ptd
