// Routed anchor attention on sm_103a tensor cores (Eq. block, App. B.4, App. B.5).
//
// One CTA computes two 128-row query tiles (Q0, Q1: 256 consecutive rows) of one
// (anchor i, head h):
//   O = softmax(scale Q K^T) V over every token of the current chunk followed by the tokens
//   of the routed history blocks idx[i, h, :].
// Both query tiles consume every K/V tile, so each tile fetched from L2 feeds 256 rows.
// Warp roles (384 threads = three warpgroups, one CTA per SM, 193 KB shared memory, all 512
// TMEM columns; warpgroup 0 gives registers to the two softmax warpgroups with setmaxnreg):
//   warp 0       TMA producers: lane 0 loads Q0/Q1 and the K tiles, lane 1 the V tiles, each
//                into a two-stage ring (128 tokens x d, 128-byte swizzle, 64-element boxes);
//                current-chunk tiles come from a 2-D map, history tiles from a 3-D map
//                [block, token, channel] so a tile never reads past its block, or, with
//                (1, 8, 8) spatial blocks of history frames, from a 4-D map
//                [frame, y, x, channel] whose 8 x 8-token boxes put two routed blocks in one
//                tile (rows 0-63 and 64-127; grid-edge tokens read as zero and are masked).
//   warp 1       TMEM owner and single-thread UMMA issuer, order
//                S0_0 S1_0 | PV0_0 S0_1 PV1_0 S1_1 | PV0_1 S0_2 PV1_1 S1_2 | ...
//                (S_t = Q_t K^T, kind::f16, M=N=128, f32 in TMEM; PV_t: O_t += P_t V with P_t
//                read from TMEM over the S_t columns and V read MN-major).
//   warps 2, 3   idle (they complete warpgroup 0 for the register hand-over)
//   warps 4..7   softmax of Q0, warps 8..11 softmax of Q1: one query row per thread,
//                tcgen05.ld of the S row, masking, exp2-domain online softmax with lazy
//                rescaling (O_t and l rescaled only when the running max grows by more than
//                8 = log2 256), P packed to bf16 and stored with tcgen05.st, epilogue O / l.
// While one warpgroup runs its softmax the tensor core works on the other tile.  UMMAs of
// one thread execute in issue order, so S_t for tile j+1 (issued after PV_t of tile j)
// certifies that PV_t of tile j has completed: O_t may then be rescaled in place.
// Load balance: a unit is one CTA's pair of query tiles with all its K/V tiles.  Units fill
// whole rounds of one CTA per SM; the units of a last, partial round are split along the K/V
// axis over all SMs, each part writes its unnormalised O with its row max and sum, and the
// part that arrives last merges them (exp2-weighted by the row maxima).
// Every wait is bounded; on a timeout the CTA records an error word, drains its UMMAs and
// frees TMEM before leaving.
// Inside the block step the kernel is a programmatic dependent of the routing kernel: its CTAs
// start on the current-chunk tiles while routing finishes, and each thread that reads the
// routed block indices waits on the grid dependency just before its first history tile.
#include <cuda_bf16.h>

#include <cmath>

#include "internal.h"
#include "ptx.cuh"

namespace cast {
namespace {

__device__ unsigned int g_attn_error;

constexpr int BM = 128, BN = 128, kStages = 2;
constexpr int kThreads = 384;
// Registers: every thread starts with kLaunchRegs; warpgroup 0 (producer, MMA issuer, two
// idle warps) drops to kRegsCtl and the softmax warpgroups rise to kRegsSoftmax.
constexpr int kLaunchRegs = 168, kRegsCtl = 96, kRegsSoftmax = 200;
static_assert(128 * kRegsCtl + 256 * kRegsSoftmax <= kThreads * kLaunchRegs,
              "register split exceeds the launch allocation");
static_assert(kThreads * kLaunchRegs <= 65536, "launch allocation exceeds the register file");
constexpr int kTmemCols = 512;   // S0/P0 at 0, S1/P1 at 128, O0 at 256, O1 at 384
constexpr float kRescaleThreshold = 8.f;

template <int HD>
struct Cfg {
  static constexpr int Q_BYTES = BM * HD * 2;
  static constexpr int KV_BYTES = BN * HD * 2;
  static constexpr int OFF_Q = 0;                                   // Q0, Q1
  static constexpr int OFF_K = OFF_Q + 2 * Q_BYTES;                 // kStages K tiles
  static constexpr int OFF_V = OFF_K + kStages * KV_BYTES;          // kStages V tiles
  static constexpr int OFF_BAR = OFF_V + kStages * KV_BYTES;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;   // + barriers + alignment slack
};

struct AttnKArgs {
  int S, H, n_pairs, n_single, n_anchors, n_cur_tiles, tiles_per_block, K_eff, M, cur_rows, B_v;
  int n_hist_tiles;                 // history K/V tiles
  int spatial, hHg, hWg, nby, nbx;  // CAST_HIST_FRAMES: frame grid, 8x8 block grid
  int n_full;        // units run whole (CTAs 0 .. n_full-1)
  int n_split;       // parts of every remaining unit
  int chunk;         // K/V tiles per part
  float* part_o;     // [tail unit][part][2][128][HD] unnormalised O of the parts
  float* part_ml;    // [tail unit][part][2][128][2] row max (log2 domain) and row sum
  unsigned* counters;   // [tail unit] parts finished
  const int* idx;
  void* o;
  int o_f32;
  float* lse;
  float scale_log2;
  unsigned long long wait_ns;
  int q_frame[CAST_MAX_ANCHORS];
  int o_frame[CAST_MAX_ANCHORS];
};

struct Bars {
  uint64_t q_full;
  uint64_t k_full[kStages], k_empty[kStages], v_full[kStages], v_empty[kStages];
  uint64_t s_full[2], p_full[2];
  uint64_t fin, part_done, merge_go;
  uint32_t tmem_base;
  int abort;
  int last;
};

// 2^x in one MUFU op (flush-to-zero; 2^-inf = 0)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Whole-CTA barrier reached from the code of different roles (non-aligned form, barrier 1).
__device__ __forceinline__ void end_barrier() {
  asm volatile("barrier.sync 1, %0;" ::"n"(kThreads) : "memory");
}

// Waits (once per thread) until the grid this one depends on has completed and its writes
// (the routed block indices) are visible; a no-op for an ordinary launch.
__device__ __forceinline__ void wait_routing(bool& waited) {
  if (!waited) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    waited = true;
  }
}

__device__ __forceinline__ bool aborted(const Bars* b) {
  return *reinterpret_cast<const volatile int*>(&b->abort) != 0;
}
__device__ __forceinline__ void set_abort(Bars* b) {
  atomicExch(&b->abort, 1);
  atomicExch(&g_attn_error, 1u);
}

// Routed block k of (anchor i, head h); an index outside [0, M) records an error and reads 0.
__device__ __forceinline__ int routed_block(const AttnKArgs& a, int i, int h, int k) {
  int m = __ldg(a.idx + ((int64_t)i * a.H + h) * a.K_eff + k);
  if (m < 0 || m >= a.M) {
    atomicExch(&g_attn_error, 2u);
    m = 0;
  }
  return m;
}

// Spatial block m: (frame, first row, first column) in the history frames and the mask of its
// 64 key positions (bit 8 yl + xl set iff row yl, column xl lie inside the frame grid).
struct SpatialBlock {
  int f, y0, x0;
  uint64_t valid;
};
__device__ __forceinline__ SpatialBlock spatial_block(const AttnKArgs& a, int m) {
  SpatialBlock b;
  const int per_frame = a.nby * a.nbx;
  b.f = m / per_frame;
  const int rem = m - b.f * per_frame;
  const int by = rem / a.nbx, bx = rem - by * a.nbx;
  b.y0 = 8 * by;
  b.x0 = 8 * bx;
  const int hv = min(8, a.hHg - b.y0), wv = min(8, a.hWg - b.x0);
  const uint64_t row = (1ull << wv) - 1ull;                 // columns 0 .. wv-1 of one row
  const uint64_t rows = row * 0x0101010101010101ull;        // ... of every row
  b.valid = hv >= 8 ? rows : rows & ((1ull << (8 * hv)) - 1ull);
  return b;
}

// (tensor map, row, block) of K/V tile j: current-chunk tiles first, then the routed blocks.
// Spatial history: tile jj holds routed blocks 2jj (rows 0-63) and 2jj+1 (rows 64-127); when
// K_eff is odd the last tile repeats block 2jj in its second half, which is masked.
struct TileCoord {
  bool cur;
  int y, z;
  int m0, m1;   // spatial: the two blocks
};
__device__ __forceinline__ TileCoord tile_coord(const AttnKArgs& a, int i, int h, int j) {
  TileCoord c;
  c.cur = j < a.n_cur_tiles;
  c.m0 = c.m1 = 0;
  if (c.cur) {
    c.y = j * BN;
    c.z = 0;
  } else if (a.spatial) {
    const int jj = j - a.n_cur_tiles;
    c.y = c.z = 0;
    c.m0 = routed_block(a, i, h, 2 * jj);
    c.m1 = 2 * jj + 1 < a.K_eff ? routed_block(a, i, h, 2 * jj + 1) : c.m0;
  } else {
    const int jj = j - a.n_cur_tiles;
    const int blk = jj / a.tiles_per_block;
    c.y = (jj - blk * a.tiles_per_block) * BN;
    c.z = routed_block(a, i, h, blk);
  }
  return c;
}

template <int HD>
__global__ void __launch_bounds__(kThreads, 1)
    k_attn(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kc,
           const __grid_constant__ CUtensorMap tm_vc, const __grid_constant__ CUtensorMap tm_kh,
           const __grid_constant__ CUtensorMap tm_vh, const __grid_constant__ AttnKArgs a) {
  using C = Cfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  uint8_t* sQ = smem + C::OFF_Q;
  uint8_t* sK = smem + C::OFF_K;
  uint8_t* sV = smem + C::OFF_V;
  Bars* bars = reinterpret_cast<Bars*>(smem + C::OFF_BAR);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Unit of this CTA (whole, or one K/V part of a tail unit).  Units are ordered longest
  // first: every pair of query tiles, then the single remainder tiles (S mod 256 <= 128).
  // Head slowest within each group: CTAs resident together share the head's current-chunk
  // K/V in L2.
  const int n_tiles_all = a.n_cur_tiles + a.n_hist_tiles;
  int u, part = 0, k0 = 0, k1 = n_tiles_all;
  const bool split = (int)blockIdx.x >= a.n_full;
  if (!split) {
    u = blockIdx.x;
  } else {
    const int t = blockIdx.x - a.n_full;
    u = a.n_full + t / a.n_split;
    part = t % a.n_split;
    k0 = part * a.chunk;
    k1 = min(n_tiles_all, k0 + a.chunk);
  }
  const int tail_unit = u - a.n_full;
  int qp, rest;
  const int n_pair_units = a.n_pairs * a.n_anchors * a.H;
  if (u < n_pair_units) {
    qp = u % a.n_pairs;
    rest = u / a.n_pairs;
  } else {
    qp = a.n_pairs;
    rest = u - n_pair_units;
  }
  const int i = rest % a.n_anchors;
  const int h = rest / a.n_anchors;
  const int n_tiles = k1 - k0;   // K/V tiles of this CTA: global tiles k0 .. k1-1
  const int row0 = qp * 2 * BM;
  const bool has_q1 = row0 + BM < a.S;

  if (threadIdx.x == 0) {
    mbar_init(&bars->q_full, 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bars->k_full[s], 1);
      mbar_init(&bars->k_empty[s], 1);
      mbar_init(&bars->v_full[s], 1);
      mbar_init(&bars->v_empty[s], 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(&bars->s_full[t], 1);
      mbar_init(&bars->p_full[t], 128);
    }
    mbar_init(&bars->fin, 1);
    mbar_init(&bars->part_done, (has_q1 ? 2 : 1) * 128);
    mbar_init(&bars->merge_go, 1);
    bars->abort = 0;
    bars->last = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(&bars->tmem_base, kTmemCols);
    tmem_relinquish();
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;
  const uint64_t lim = a.wait_ns;

  if (warp < 4) {
  setmaxnreg_dec<kRegsCtl>();
  if (warp == 0) {
    // ------------------------------------------------------------ TMA producers
    if (lane == 0) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_kc);
      tma_prefetch_desc(&tm_kh);
      mbar_arrive_expect_tx(&bars->q_full, (has_q1 ? 2 : 1) * C::Q_BYTES);
      for (int t = 0; t < (has_q1 ? 2 : 1); ++t)
#pragma unroll
        for (int b = 0; b < HD / 64; ++b)
          tma_load_3d(sQ + t * C::Q_BYTES + b * BM * 128, &tm_q, &bars->q_full, h * HD + b * 64,
                      row0 + t * BM, a.q_frame[i]);
      bool waited = false;
      for (int j = 0; j < n_tiles; ++j) {
        if (k0 + j >= a.n_cur_tiles) wait_routing(waited);
        const TileCoord c = tile_coord(a, i, h, k0 + j);
        const int s = j % kStages;
        if (aborted(bars) || !mbar_wait(&bars->k_empty[s], ((uint32_t)(j / kStages) & 1u) ^ 1u, lim)) {
          set_abort(bars);
          break;
        }
        mbar_arrive_expect_tx(&bars->k_full[s], C::KV_BYTES);
        if (!c.cur && a.spatial) {
          const SpatialBlock b0 = spatial_block(a, c.m0), b1 = spatial_block(a, c.m1);
#pragma unroll
          for (int b = 0; b < HD / 64; ++b) {
            uint8_t* dst = sK + s * C::KV_BYTES + b * BN * 128;
            tma_load_4d(dst, &tm_kh, &bars->k_full[s], h * HD + b * 64, b0.x0, b0.y0, b0.f);
            tma_load_4d(dst + 64 * 128, &tm_kh, &bars->k_full[s], h * HD + b * 64, b1.x0, b1.y0, b1.f);
          }
        } else {
#pragma unroll
          for (int b = 0; b < HD / 64; ++b) {
            uint8_t* dst = sK + s * C::KV_BYTES + b * BN * 128;
            if (c.cur) tma_load_2d(dst, &tm_kc, &bars->k_full[s], h * HD + b * 64, c.y);
            else tma_load_3d(dst, &tm_kh, &bars->k_full[s], h * HD + b * 64, c.y, c.z);
          }
        }
      }
    } else if (lane == 1) {
      tma_prefetch_desc(&tm_vc);
      tma_prefetch_desc(&tm_vh);
      bool waited = false;
      for (int j = 0; j < n_tiles; ++j) {
        if (k0 + j >= a.n_cur_tiles) wait_routing(waited);
        const TileCoord c = tile_coord(a, i, h, k0 + j);
        const int s = j % kStages;
        if (aborted(bars) || !mbar_wait(&bars->v_empty[s], ((uint32_t)(j / kStages) & 1u) ^ 1u, lim)) {
          set_abort(bars);
          break;
        }
        mbar_arrive_expect_tx(&bars->v_full[s], C::KV_BYTES);
        if (!c.cur && a.spatial) {
          const SpatialBlock b0 = spatial_block(a, c.m0), b1 = spatial_block(a, c.m1);
#pragma unroll
          for (int b = 0; b < HD / 64; ++b) {
            uint8_t* dst = sV + s * C::KV_BYTES + b * BN * 128;
            tma_load_4d(dst, &tm_vh, &bars->v_full[s], h * HD + b * 64, b0.x0, b0.y0, b0.f);
            tma_load_4d(dst + 64 * 128, &tm_vh, &bars->v_full[s], h * HD + b * 64, b1.x0, b1.y0, b1.f);
          }
        } else {
#pragma unroll
          for (int b = 0; b < HD / 64; ++b) {
            uint8_t* dst = sV + s * C::KV_BYTES + b * BN * 128;
            if (c.cur) tma_load_2d(dst, &tm_vc, &bars->v_full[s], h * HD + b * 64, c.y);
            else tma_load_3d(dst, &tm_vh, &bars->v_full[s], h * HD + b * 64, c.y, c.z);
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ UMMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(BM, BN, false, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(BM, HD, false, true);
      const uint32_t q_addr = smem_u32(sQ), k_addr = smem_u32(sK), v_addr = smem_u32(sV);
      const int nq = has_q1 ? 2 : 1;
      // Descriptors of the first k-slice of each operand; a k-slice, query tile or stage
      // further on adds its byte offset / 16 to the 14-bit start-address field (the whole
      // shared-memory window is below 256 KB, so the field never carries).  This keeps the
      // single issuing thread at a few instructions per UMMA.
      static_assert(C::SMEM + 1024 <= 256 * 1024, "descriptor start-address field would carry");
      static_assert(BM == BN, "Q and K tiles share their k-slice offsets");
      const uint64_t dq = sdesc_sw128(q_addr, 16, 1024);
      const uint64_t dk = sdesc_sw128(k_addr, 16, 1024);
      const uint64_t dv = sdesc_sw128(v_addr, BN * 128, 1024);
      // S_t = Q_t K_j^T into the S_t columns (t * 128)
      auto qk = [&](int t, int j) {
        const uint64_t aq = dq + (uint64_t)((t * C::Q_BYTES) >> 4);
        const uint64_t bk = dk + (uint64_t)(((j % kStages) * C::KV_BYTES) >> 4);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint64_t off = (uint64_t)(((kk >> 2) * (BM * 128) + (kk & 3) * 32) >> 4);
          umma_bf16_ss(tmem + t * BN, aq + off, bk + off, idesc_qk, kk > 0 ? 1u : 0u);
        }
        umma_commit(&bars->s_full[t]);
      };
      // O_t += P_t V_j, P_t read from TMEM over the S_t columns
      auto pv = [&](int t, int j) {
        const uint64_t bv = dv + (uint64_t)(((j % kStages) * C::KV_BYTES) >> 4);
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk)
          umma_bf16_ts(tmem + 256 + t * 128, tmem + t * BN + kk * 8,
                       bv + (uint64_t)((kk * 16 * 128) >> 4), idesc_pv, (j > 0 || kk > 0) ? 1u : 0u);
      };
      bool ok = mbar_wait(&bars->q_full, 0, lim) && mbar_wait(&bars->k_full[0], 0, lim);
      tc_fence_after();
      if (ok && n_tiles > 0) {
        for (int t = 0; t < nq; ++t) qk(t, 0);
        umma_commit(&bars->k_empty[0]);
      }
      for (int j = 0; ok && j < n_tiles; ++j) {
        const int s = j % kStages;
        const uint32_t ph = (uint32_t)j & 1u;
        const bool more = j + 1 < n_tiles;
        // K_{j+1} is awaited with V_j, while P_0 is still being formed, so that S_0 of tile
        // j+1 follows PV_0 of tile j without a wait (its load was released two tiles ago)
        if (aborted(bars) || !mbar_wait(&bars->v_full[s], (uint32_t)(j / kStages) & 1u, lim) ||
            (more && !mbar_wait(&bars->k_full[(j + 1) % kStages], (uint32_t)((j + 1) / kStages) & 1u, lim)) ||
            !mbar_wait(&bars->p_full[0], ph, lim)) { ok = false; break; }
        tc_fence_after();
        pv(0, j);
        if (more) qk(0, j + 1);
        if (nq == 2) {
          if (aborted(bars) || !mbar_wait(&bars->p_full[1], ph, lim)) { ok = false; break; }
          tc_fence_after();
          pv(1, j);
        }
        umma_commit(&bars->v_empty[s]);
        if (more) {
          if (nq == 2) qk(1, j + 1);
          umma_commit(&bars->k_empty[(j + 1) % kStages]);
        }
      }
      if (!ok) set_abort(bars);
      // every issued UMMA has completed before the epilogue reads O and TMEM is released
      umma_commit(&bars->fin);
      mbar_wait(&bars->fin, 0, lim);
    }
  }
  // the last UMMA has completed (fin) and every softmax thread has read TMEM
  tc_fence_before();
  end_barrier();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  } else {
  setmaxnreg_inc<kRegsSoftmax>();
  if (warp < 8 || has_q1) {
    // ------------------------------------------------------------ softmax + epilogue
    const int t = warp < 8 ? 0 : 1;
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const uint32_t colS = t * BN, colO = 256 + t * 128;
    float m_ref = -INFINITY, l = 0.f;
    bool ok = true;
    bool waited = false;
    for (int j = 0; j < n_tiles; ++j) {
      const int jg = k0 + j;   // global K/V tile
      // spatial history tile: the routed block indices are fetched before the wait
      int sm0 = -1, sm1 = -1;
      if (a.spatial && jg >= a.n_cur_tiles) {
        wait_routing(waited);
        const int jj = jg - a.n_cur_tiles;
        sm0 = routed_block(a, i, h, 2 * jj);
        sm1 = 2 * jj + 1 < a.K_eff ? routed_block(a, i, h, 2 * jj + 1) : -1;
      }
      bool w = !aborted(bars) && mbar_wait(&bars->s_full[t], (uint32_t)j & 1u, lim);
      if (!__all_sync(0xffffffffu, w)) { ok = false; break; }
      tc_fence_after();
      uint32_t sr[BN];
      tmem_ld_x64(tl + colS, sr);
      tmem_ld_x64(tl + colS + 64, sr + 64);
      if (sm0 >= 0) {
        // key positions outside a truncated block, and the unused half of a last odd tile
        const uint64_t v0 = spatial_block(a, sm0).valid;
        const uint64_t v1 = sm1 >= 0 ? spatial_block(a, sm1).valid : 0ull;
        if ((v0 & v1) != ~0ull) {
          const uint32_t w4[4] = {(uint32_t)v0, (uint32_t)(v0 >> 32), (uint32_t)v1, (uint32_t)(v1 >> 32)};
#pragma unroll
          for (int c = 0; c < BN; ++c)
            if (!((w4[c >> 5] >> (c & 31)) & 1u)) sr[c] = __float_as_uint(-INFINITY);
        }
      } else {
        int valid;
        if (jg < a.n_cur_tiles) {
          valid = min(BN, a.cur_rows - jg * BN);
        } else {
          const int jj = jg - a.n_cur_tiles;
          valid = min(BN, a.B_v - (jj % a.tiles_per_block) * BN);
        }
        // columns past the chunk / block end (only in a ragged last tile) get -inf
        if (valid < BN) {
#pragma unroll
          for (int c = 0; c < BN; ++c)
            if (c >= valid) sr[c] = __float_as_uint(-INFINITY);
        }
      }
      // raw-logit max (scale > 0 commutes with max): 3-input max, 8 independent chains
      float m8[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) m8[e] = fmaxf(__uint_as_float(sr[2 * e]), __uint_as_float(sr[2 * e + 1]));
#pragma unroll
      for (int c = 16; c < BN; c += 16)
#pragma unroll
        for (int e = 0; e < 8; ++e)
          m8[e] = max3(m8[e], __uint_as_float(sr[c + 2 * e]), __uint_as_float(sr[c + 2 * e + 1]));
      const float mxr = max3(max3(m8[0], m8[1], m8[2]), max3(m8[3], m8[4], m8[5]), fmaxf(m8[6], m8[7]));
      const float mx = mxr * a.scale_log2;
      const bool need = mx > m_ref + kRescaleThreshold;
      float corr = 1.f;
      if (need) {
        corr = ex2_approx(m_ref - mx);   // 0 on the first tile (m_ref = -inf)
        m_ref = mx;
        l *= corr;
      }
      // P = 2^(s * scale_log2 - m_ref): packed f32x2 FMA and sums, one MUFU op per element,
      // packed to bf16 pairs over the first 64 S columns of this lane
      const float2 sc2 = make_float2(a.scale_log2, a.scale_log2);
      const float2 nm2 = make_float2(-m_ref, -m_ref);
      float2 s4[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                      make_float2(0.f, 0.f)};
#pragma unroll
      for (int c = 0; c < BN; c += 2) {
        const float2 x = __ffma2_rn(make_float2(__uint_as_float(sr[c]), __uint_as_float(sr[c + 1])),
                                    sc2, nm2);
        const float2 p = make_float2(ex2_approx(x.x), ex2_approx(x.y));
        s4[(c >> 1) & 3] = __fadd2_rn(s4[(c >> 1) & 3], p);
        __nv_bfloat162 b2 = __floats2bfloat162_rn(p.x, p.y);
        sr[c / 2] = *reinterpret_cast<uint32_t*>(&b2);
      }
      const float2 s2 = __fadd2_rn(__fadd2_rn(s4[0], s4[1]), __fadd2_rn(s4[2], s4[3]));
      l += s2.x + s2.y;
      tmem_st_x64(tl + colS, sr);
      if (j > 0 && __any_sync(0xffffffffu, need)) {
        // O_t holds P_0..P_{j-1} V and is final: S_t of tile j was issued after PV_t of
        // tile j-1, and PV_t of tile j waits for p_full below
#pragma unroll
        for (int half = 0; half < HD / 64; ++half) {
          uint32_t orr[64];
          tmem_ld_x64(tl + colO + half * 64, orr);
#pragma unroll
          for (int c = 0; c < 64; ++c) orr[c] = __float_as_uint(__uint_as_float(orr[c]) * corr);
          tmem_st_x64(tl + colO + half * 64, orr);
        }
      }
      tc_fence_before();
      mbar_arrive(&bars->p_full[t]);
    }
    if (ok) {
      bool w = !aborted(bars) && mbar_wait(&bars->fin, 0, lim);
      ok = __all_sync(0xffffffffu, w);
    }
    if (!ok) set_abort(bars);
    tc_fence_after();
    const int s = row0 + t * BM + row;
    const int64_t D = (int64_t)a.H * HD;
    const int64_t off = ((int64_t)a.o_frame[i] * a.S + s) * D + (int64_t)h * HD;
    // final row: O scaled by inv, written as bf16 or f32
    auto store_half = [&](int half, const float* v, float inv) {
      if (a.o_f32) {
        float* dst = static_cast<float*>(a.o) + off + half * 64;
#pragma unroll
        for (int c = 0; c < 64; c += 4)
          *reinterpret_cast<float4*>(dst + c) =
              make_float4(v[c] * inv, v[c + 1] * inv, v[c + 2] * inv, v[c + 3] * inv);
      } else {
        __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(a.o) + off + half * 64;
#pragma unroll
        for (int c = 0; c < 64; c += 8) {
          uint32_t pk4[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            __nv_bfloat162 b2 = __floats2bfloat162_rn(v[c + 2 * e] * inv, v[c + 2 * e + 1] * inv);
            pk4[e] = *reinterpret_cast<uint32_t*>(&b2);
          }
          *reinterpret_cast<uint4*>(dst + c) = make_uint4(pk4[0], pk4[1], pk4[2], pk4[3]);
        }
      }
    };
    if (!split) {
      if (ok) {
        const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
        for (int half = 0; half < HD / 64; ++half) {
          uint32_t orr[64];
          tmem_ld_x64(tl + colO + half * 64, orr);   // warp-collective: every lane loads
          if (s < a.S) store_half(half, reinterpret_cast<const float*>(orr), inv);
        }
        if (a.lse && s < a.S)
          a.lse[((int64_t)i * a.H + h) * a.S + s] = (m_ref + log2f(l)) * 0.69314718055994531f;
      }
    } else {
      // this part's unnormalised O with its row max (log2 domain) and row sum
      const int64_t slot0 = ((int64_t)tail_unit * a.n_split) * 2 * BM + t * BM + row;
      if (ok) {
        const int64_t slot = slot0 + (int64_t)part * 2 * BM;
#pragma unroll
        for (int half = 0; half < HD / 64; ++half) {
          uint32_t orr[64];
          tmem_ld_x64(tl + colO + half * 64, orr);
          float4* dst = reinterpret_cast<float4*>(a.part_o + slot * HD + half * 64);
#pragma unroll
          for (int c = 0; c < 64; c += 4)
            __stcg(dst + c / 4, make_float4(__uint_as_float(orr[c]), __uint_as_float(orr[c + 1]),
                                            __uint_as_float(orr[c + 2]), __uint_as_float(orr[c + 3])));
        }
        __stcg(reinterpret_cast<float2*>(a.part_ml) + slot, make_float2(m_ref, l));
      }
      // every softmax thread arrives (also after a failure, so nobody waits forever); one
      // thread then counts this part in, and the part that completes the count merges
      mbar_arrive(&bars->part_done);
      if (warp == 4 && lane == 0) {
        const bool w = mbar_wait(&bars->part_done, 0, lim);
        int last = 0;
        if (w && !aborted(bars)) {
          __threadfence();
          last = atomicAdd(&a.counters[tail_unit], 1u) == (unsigned)(a.n_split - 1);
          __threadfence();
        } else {
          set_abort(bars);
        }
        bars->last = last;
        mbar_arrive(&bars->merge_go);
      }
      const bool go = mbar_wait(&bars->merge_go, 0, lim);
      if (go && ok && *reinterpret_cast<volatile int*>(&bars->last) && s < a.S) {
        const float2* ml = reinterpret_cast<const float2*>(a.part_ml);
        float mm = -INFINITY, lsum = 0.f;
        for (int p = 0; p < a.n_split; ++p) mm = fmaxf(mm, __ldcg(ml + slot0 + (int64_t)p * 2 * BM).x);
        for (int p = 0; p < a.n_split; ++p) {
          const float2 v = __ldcg(ml + slot0 + (int64_t)p * 2 * BM);
          lsum += ex2_approx(v.x - mm) * v.y;
        }
        const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
#pragma unroll
        for (int half = 0; half < HD / 64; ++half) {
          float acc[64];
#pragma unroll
          for (int c = 0; c < 64; ++c) acc[c] = 0.f;
          for (int p = 0; p < a.n_split; ++p) {
            const int64_t sp = slot0 + (int64_t)p * 2 * BM;
            const float wgt = ex2_approx(__ldcg(ml + sp).x - mm);
            const float4* src = reinterpret_cast<const float4*>(a.part_o + sp * HD + half * 64);
#pragma unroll
            for (int c = 0; c < 64; c += 4) {
              const float4 v = __ldcg(src + c / 4);
              acc[c] = fmaf(wgt, v.x, acc[c]);
              acc[c + 1] = fmaf(wgt, v.y, acc[c + 1]);
              acc[c + 2] = fmaf(wgt, v.z, acc[c + 2]);
              acc[c + 3] = fmaf(wgt, v.w, acc[c + 3]);
            }
          }
          store_half(half, acc, inv);
        }
        if (a.lse)
          a.lse[((int64_t)i * a.H + h) * a.S + s] = (mm + log2f(lsum)) * 0.69314718055994531f;
      }
    }
  }
  tc_fence_before();
  end_barrier();
  }
}

// ---------------------------------------------------------------- host side
// bf16 tensor [depth][rows][inner] (rank 2 when depth == 0), box 64 x 128 (x 1), 128-B swizzle
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows,
              uint64_t row_stride_bytes, uint64_t depth, uint64_t depth_stride_bytes) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[3] = {inner, rows, depth};
  cuuint64_t strides[2] = {row_stride_bytes, depth_stride_bytes};
  cuuint32_t box[3] = {64, 128, 1};
  cuuint32_t es[3] = {1, 1, 1};
  const cuuint32_t rank = depth ? 3 : 2;
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides, box,
            es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// bf16 history frames [frames][Hg][Wg][inner], box 64 channels x 8 x 8 tokens x 1 frame
// (one (1, 8, 8) block), 128-B swizzle; tokens outside the grid read as zero
bool make_map_frames(CUtensorMap* m, const void* base, uint64_t inner, uint64_t Wg, uint64_t Hg,
                     uint64_t frames, uint64_t row_stride_bytes) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[4] = {inner, Wg, Hg, frames};
  cuuint64_t strides[3] = {row_stride_bytes, row_stride_bytes * Wg, row_stride_bytes * Wg * Hg};
  cuuint32_t box[4] = {64, 8, 8, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int HD>
cast_status launch_hd(const cast_attn_args& a, const AttnPlan& pl, int o_frame_of_anchor, void* ws,
                      cudaStream_t st, bool after_route) {
  using C = Cfg<HD>;
  const int D = a.H * HD;
  CUtensorMap mq, mkc, mvc, mkh, mvh;
  const uint64_t cur_rows = (uint64_t)a.n_frames * a.S;
  bool ok = make_map(&mq, a.q, D, a.S, a.q_row_stride * 2, a.n_frames, (uint64_t)a.S * a.q_row_stride * 2) &&
            make_map(&mkc, a.k_cur, D, cur_rows, a.cur_row_stride * 2, 0, 0) &&
            make_map(&mvc, a.v_cur, D, cur_rows, a.cur_row_stride * 2, 0, 0);
  const HistGeom hg = hist_geom(a.hist);
  if (ok && a.M > 0 && hg.spatial) {
    ok = make_map_frames(&mkh, a.k_hist, D, hg.Wg, hg.Hg, hg.frames, a.hist_row_stride * 2) &&
         make_map_frames(&mvh, a.v_hist, D, hg.Wg, hg.Hg, hg.frames, a.hist_row_stride * 2);
  } else if (ok && a.M > 0) {
    ok = make_map(&mkh, a.k_hist, D, a.B_v, a.hist_row_stride * 2, a.M,
                  (uint64_t)a.B_v * a.hist_row_stride * 2) &&
         make_map(&mvh, a.v_hist, D, a.B_v, a.hist_row_stride * 2, a.M,
                  (uint64_t)a.B_v * a.hist_row_stride * 2);
  } else if (ok) {
    mkh = mkc;
    mvh = mvc;
  }
  if (!ok) return fail(CAST_ERR_CUDA, "attention: cuTensorMapEncodeTiled failed");
  AttnKArgs k{};
  k.S = a.S;
  k.H = a.H;
  k.n_pairs = pl.n_pairs;
  k.n_single = pl.n_single;
  k.n_anchors = a.n_anchors;
  k.n_cur_tiles = pl.n_cur_tiles;
  k.tiles_per_block = pl.tiles_per_block;
  k.n_hist_tiles = pl.n_hist_tiles;
  k.spatial = hg.spatial ? 1 : 0;
  k.hHg = hg.Hg;
  k.hWg = hg.Wg;
  k.nby = hg.nby;
  k.nbx = hg.nbx;
  k.K_eff = a.M > 0 ? a.K_eff : 0;
  k.M = a.M;
  k.cur_rows = (int)cur_rows;
  k.B_v = a.B_v;
  k.idx = a.idx;
  k.o = a.o;
  k.o_f32 = a.o_dtype == CAST_F32;
  k.lse = a.lse;
  k.n_full = pl.n_full;
  k.n_split = pl.n_split;
  k.chunk = pl.chunk;
  char* w = static_cast<char*>(ws);
  k.part_o = reinterpret_cast<float*>(w);
  k.part_ml = reinterpret_cast<float*>(w + pl.part_o_bytes);
  k.counters = reinterpret_cast<unsigned*>(w + pl.part_o_bytes + pl.part_ml_bytes);
  const float scale = a.scale > 0.f ? a.scale : 1.f / sqrtf((float)HD);
  k.scale_log2 = scale * 1.4426950408889634f;
  k.wait_ns = 2000000000ull;
  for (int j = 0; j < a.n_anchors; ++j) {
    k.q_frame[j] = a.anchors[j];
    k.o_frame[j] = o_frame_of_anchor ? a.anchors[j] : j;
  }
  static std::atomic<uint64_t> attr_done{0};
  cast_status setup_status = CAST_OK;
  const bool set_up = once_per_device(attr_done, [&] {
    // the register hand-over in the kernel assumes exactly kLaunchRegs per thread at launch
    cudaFuncAttributes fa{};
    if (cudaFuncGetAttributes(&fa, k_attn<HD>) != cudaSuccess) {
      setup_status = check_launch("attention kernel attributes");
      return false;
    }
    if (fa.numRegs != kLaunchRegs) {
      setup_status = fail(CAST_ERR_UNSUPPORTED,
                          "attention kernel built with %d registers per thread, expected %d",
                          fa.numRegs, kLaunchRegs);
      return false;
    }
    if (cudaFuncSetAttribute(k_attn<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM) !=
        cudaSuccess) {
      setup_status = check_launch("attention smem attribute");
      return false;
    }
    return true;
  });
  if (!set_up) return setup_status != CAST_OK ? setup_status : check_launch("attention setup");
  // after routing the caller has reset the tail counters before the routing launches, so that
  // this launch follows the routing kernel directly (programmatic dependent launch)
  if (!after_route && pl.n_tail > 0 &&
      cudaMemsetAsync(k.counters, 0, (size_t)pl.n_tail * sizeof(unsigned), st) != cudaSuccess)
    return check_launch("attention counter reset");
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(pl.grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = after_route ? 1 : 0;
  if (cudaLaunchKernelEx(&cfg, k_attn<HD>, mq, mkc, mvc, mkh, mvh, k) != cudaSuccess)
    return check_launch("attention kernel");
  return check_launch("attention kernel");
}

}  // namespace

AttnPlan attention_plan(const cast_attn_args& a) {
  AttnPlan p{};
  p.n_pairs = a.S / (2 * BM) + (a.S % (2 * BM) > BM ? 1 : 0);
  p.n_single = (a.S % (2 * BM) > 0 && a.S % (2 * BM) <= BM) ? 1 : 0;
  p.n_cur_tiles = (int)(((int64_t)a.n_frames * a.S + BN - 1) / BN);
  p.tiles_per_block = a.M > 0 ? (a.B_v + BN - 1) / BN : 0;
  const int keff = a.M > 0 ? a.K_eff : 0;
  p.n_hist_tiles = hist_geom(a.hist).spatial ? (keff + 1) / 2 : keff * p.tiles_per_block;
  const int n_tiles = p.n_cur_tiles + p.n_hist_tiles;
  const int units = (p.n_pairs + p.n_single) * a.n_anchors * a.H;
  int dev = 0, nsm = 148;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  if (nsm < 1) nsm = 1;
  // whole rounds of one unit per SM run unsplit; the units of the last, partial round are
  // split along K/V over the SMs (never into parts of fewer than 4 tiles)
  const int rounds = units / nsm;
  const int tail = units - rounds * nsm;
  int n_split = tail > 0 ? nsm / tail : 1;
  if (n_split > n_tiles / 4) n_split = n_tiles / 4;
  if (n_split < 2) {
    p.n_full = units;
    p.n_tail = 0;
    p.n_split = 1;
    p.chunk = n_tiles;
  } else {
    p.chunk = (n_tiles + n_split - 1) / n_split;
    n_split = (n_tiles + p.chunk - 1) / p.chunk;   // no empty part
    p.n_full = rounds * nsm;
    p.n_tail = tail;
    p.n_split = n_split;
  }
  p.grid = p.n_full + p.n_tail * p.n_split;
  const size_t rows = (size_t)p.n_tail * p.n_split * 2 * BM;
  p.part_o_bytes = align_up(rows * a.d * sizeof(float));
  p.part_ml_bytes = align_up(rows * 2 * sizeof(float));
  p.counter_bytes = align_up((size_t)(p.n_tail > 0 ? p.n_tail : 1) * sizeof(unsigned));
  p.total_bytes = p.n_tail > 0 ? p.part_o_bytes + p.part_ml_bytes + p.counter_bytes : 0;
  return p;
}

cast_status launch_attention(const cast_attn_args& a, int o_frame_of_anchor, void* ws,
                             cudaStream_t st, bool after_route) {
  const AttnPlan pl = attention_plan(a);
  if (a.d == 128) return launch_hd<128>(a, pl, o_frame_of_anchor, ws, st, after_route);
  return launch_hd<64>(a, pl, o_frame_of_anchor, ws, st, after_route);
}

cast_status attention_reset_counters(const cast_attn_args& a, void* ws, cudaStream_t st) {
  const AttnPlan pl = attention_plan(a);
  if (pl.n_tail == 0) return CAST_OK;
  char* w = static_cast<char*>(ws);
  if (cudaMemsetAsync(w + pl.part_o_bytes + pl.part_ml_bytes, 0, (size_t)pl.n_tail * sizeof(unsigned),
                      st) != cudaSuccess)
    return check_launch("attention counter reset");
  return CAST_OK;
}

namespace {
// One thread waits on an mbarrier that nothing ever arrives on, with a deadline of limit_ns on
// %globaltimer; when the deadline passes it records the timeout like a kernel of the path.
__global__ void k_bounded_wait_selftest(unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_barrier_init();
  if (!mbar_wait(&bar, 0, limit_ns)) atomicExch(&g_attn_error, 1u);
}
}  // namespace

cast_status launch_bounded_wait_selftest(uint64_t limit_ns, cudaStream_t st) {
  k_bounded_wait_selftest<<<1, 32, 0, st>>>(limit_ns);
  return check_launch("bounded-wait self-test");
}

unsigned int attention_error_word(cudaStream_t st, bool clear) {
  unsigned int v = 0;
  cudaMemcpyFromSymbolAsync(&v, g_attn_error, sizeof(v), 0, cudaMemcpyDeviceToHost, st);
  cudaStreamSynchronize(st);
  if (clear && v) {
    const unsigned int z = 0;
    cudaMemcpyToSymbolAsync(g_attn_error, &z, sizeof(z), 0, cudaMemcpyHostToDevice, st);
    cudaStreamSynchronize(st);
  }
  return v;
}

}  // namespace cast
