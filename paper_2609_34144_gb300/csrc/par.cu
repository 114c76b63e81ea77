// Phase-Aware Reconstruction of skipped frames (Section 4.3, Eqs. cross, confidence, gate,
// fcpasm; App. A.2), one fused persistent kernel.
//
// Work is split into items (spectral tile p, channel chunk of 128 channels); one thread owns
// one channel of the tile.  Thread 0 streams the item's anchor tiles through a TMA 4-D map
// ([frame][row][col][channel], out-of-range rows/cols/channels arrive as zeros) into a
// shared-memory stage, issuing anchor j+1 while the CTA transforms anchor j; the current
// spectrum stays in registers and the previous one in shared memory.
//   stats item  : walks the anchors in order, forms each anchor's spectrum once, and for every
//                 adjacent anchor pair with targets reduces Z = sum_c w_c F_b conj(F_a) and
//                 W = sum_c w_c |F_b||F_a| over the chunk's channels into a partial record.
//   recon item  : waits until every chunk of its tile has published its partials, walks the
//                 anchors again (re-read mostly from L2), sums the partial records of each pair
//                 in a fixed order, derives eta, reliability, principal phases, the tile
//                 confidence c and the gate g, and for every target t of the pair writes
//                 R_t = IRFFT2((1-alpha) F_a e^{i g alpha theta} + alpha F_b e^{-i g (1-alpha) theta}).
// Items are claimed from a ticket counter in an order where every stats item of a tile is
// claimed before any recon item of that tile, so a waiting recon item only ever waits on
// items already held by running CTAs (no deadlock); the wait is also bounded in time.
#include <cuda_bf16.h>

#include <cmath>

#include "dft.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace cast {
namespace {

constexpr int kThreads = 128;      // channels per item
constexpr int kNB = 40;            // stored bins of an 8-wide tile: 8 x 5
constexpr int kNV = 3 * kNB;       // (Re Z, Im Z, W) per bin, record index = 3 * bin + component
constexpr int kMaxSeg = 128;
constexpr int kCoefBatch = 4;
constexpr int kSpecFloats = 2 * kNB * kThreads;   // one spectrum per thread, [value][thread]

__device__ unsigned int g_par_error;   // 1: a wait gave up

// Non-redundant (bin, component) values of an 8x8 tile's Z / W record, encoded bin * 4 +
// component (0: Re Z, 1: Im Z, 2: W): mirrors (ky > 4 in the kx = 0 and kx = 4 columns) are
// conjugates of their representatives, the self-conjugate bins have Im Z = 0, and DC needs
// only W (reduced separately).  96 values = three 32-value transpose groups.
__host__ __device__ __forceinline__ constexpr int fast_value(int n) {
  return
      n == 0 ? 4 :
      n == 1 ? 5 :
      n == 2 ? 6 :
      n == 3 ? 8 :
      n == 4 ? 9 :
      n == 5 ? 10 :
      n == 6 ? 12 :
      n == 7 ? 13 :
      n == 8 ? 14 :
      n == 9 ? 16 :
      n == 10 ? 18 :
      n == 11 ? 20 :
      n == 12 ? 21 :
      n == 13 ? 22 :
      n == 14 ? 24 :
      n == 15 ? 25 :
      n == 16 ? 26 :
      n == 17 ? 28 :
      n == 18 ? 29 :
      n == 19 ? 30 :
      n == 20 ? 32 :
      n == 21 ? 33 :
      n == 22 ? 34 :
      n == 23 ? 36 :
      n == 24 ? 37 :
      n == 25 ? 38 :
      n == 26 ? 40 :
      n == 27 ? 41 :
      n == 28 ? 42 :
      n == 29 ? 44 :
      n == 30 ? 45 :
      n == 31 ? 46 :
      n == 32 ? 48 :
      n == 33 ? 49 :
      n == 34 ? 50 :
      n == 35 ? 52 :
      n == 36 ? 53 :
      n == 37 ? 54 :
      n == 38 ? 56 :
      n == 39 ? 57 :
      n == 40 ? 58 :
      n == 41 ? 60 :
      n == 42 ? 61 :
      n == 43 ? 62 :
      n == 44 ? 64 :
      n == 45 ? 65 :
      n == 46 ? 66 :
      n == 47 ? 68 :
      n == 48 ? 69 :
      n == 49 ? 70 :
      n == 50 ? 72 :
      n == 51 ? 73 :
      n == 52 ? 74 :
      n == 53 ? 76 :
      n == 54 ? 77 :
      n == 55 ? 78 :
      n == 56 ? 80 :
      n == 57 ? 82 :
      n == 58 ? 84 :
      n == 59 ? 85 :
      n == 60 ? 86 :
      n == 61 ? 88 :
      n == 62 ? 89 :
      n == 63 ? 90 :
      n == 64 ? 92 :
      n == 65 ? 93 :
      n == 66 ? 94 :
      n == 67 ? 96 :
      n == 68 ? 98 :
      n == 69 ? 104 :
      n == 70 ? 105 :
      n == 71 ? 106 :
      n == 72 ? 108 :
      n == 73 ? 109 :
      n == 74 ? 110 :
      n == 75 ? 112 :
      n == 76 ? 113 :
      n == 77 ? 114 :
      n == 78 ? 124 :
      n == 79 ? 125 :
      n == 80 ? 126 :
      n == 81 ? 128 :
      n == 82 ? 129 :
      n == 83 ? 130 :
      n == 84 ? 132 :
      n == 85 ? 133 :
      n == 86 ? 134 :
      n == 87 ? 144 :
      n == 88 ? 145 :
      n == 89 ? 146 :
      n == 90 ? 148 :
      n == 91 ? 149 :
      n == 92 ? 150 :
      n == 93 ? 152 :
      n == 94 ? 153 :
      n == 95 ? 154 :
      0;
}

struct ParKArgs {
  char* r;
  const float* wch;
  int F, Hg, Wg, C;
  int th, tw, tiles_x, n_tile, n_chunk;
  int n_anchor;
  int anchor_frame[CAST_MAX_ANCHORS];
  int pair_tbeg[CAST_MAX_ANCHORS + 1];   // targets of pair j (anchors j-1, j) in [tbeg[j], tbeg[j+1])
  int target_frame[CAST_MAX_FRAMES];
  float target_alpha[CAST_MAX_FRAMES];
  int n_seg;
  int seg_first[kMaxSeg + 1];            // first ticket of each segment
  int seg_tile0[kMaxSeg];                // first tile of the segment's slab
  unsigned char seg_recon[kMaxSeg];
  int total_tickets;
  float tau_low, tau_high, q, T, eps, eta_rel, eta_abs, band;
  int gate_mode;
  unsigned long long wait_ns;
  // 8x8 tiles: record entry t (3 * bin + component) = sign * reduced value |fast_src[t]| - 1,
  // 0 = not needed (Z at DC) or identically zero (Im Z at self-conjugate bins)
  signed char fast_src[kNV];
};

template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }


__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

struct TileGeom {
  int y0, x0, h, w;
};

__device__ __forceinline__ TileGeom tile_geom(const ParKArgs& a, int tile) {
  TileGeom g;
  const int ty = tile / a.tiles_x, tx = tile - ty * a.tiles_x;
  g.y0 = ty * a.th;
  g.x0 = tx * a.tw;
  g.h = min(a.th, a.Hg - g.y0);
  g.w = min(a.tw, a.Wg - g.x0);
  return g;
}

// Warp transpose-reduction of 32 values: lane l returns the warp sum of v[l].
__device__ __forceinline__ float warp_transpose_sum(float (&v)[32], int lane) {
#pragma unroll
  for (int off = 16, n = 16; off > 0; off >>= 1, n >>= 1) {
    const bool hi = (lane & off) != 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      if (i < n) {
        const float send = hi ? v[i] : v[i + n];
        const float keep = hi ? v[i + n] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, off);
      }
    }
  }
  return v[0];
}

// Per-tile transport of one anchor pair (warp 0): theta and g per stored bin (App. A.2).
__device__ void tile_transport(const ParKArgs& a, const TileGeom& g, const float* zw, float* th,
                               float* gate, float* own_th, int* own_rel, int lane) {
  const float inv_hw = 1.f / (float)(g.h * g.w);
  const int hw2 = g.w / 2;
  float Zr[2], Zi[2], Wv[2], Za[2];
  bool valid[2];
  float wmax = 0.f;
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const int b = lane + 32 * s;
    const int ky = b / 5, kx = b % 5;
    valid[s] = b < kNB && ky < g.h && kx <= hw2;
    Zr[s] = valid[s] ? zw[3 * b] * inv_hw : 0.f;
    Zi[s] = valid[s] ? zw[3 * b + 1] * inv_hw : 0.f;
    Wv[s] = valid[s] ? zw[3 * b + 2] * inv_hw : 0.f;
    Za[s] = sqrtf(Zr[s] * Zr[s] + Zi[s] * Zi[s]);
    if (valid[s]) wmax = fmaxf(wmax, Wv[s]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) wmax = fmaxf(wmax, __shfl_xor_sync(0xffffffffu, wmax, o));
  const float eta = a.eta_rel * wmax + a.eta_abs;
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const int b = lane + 32 * s;
    if (b < kNB) {
      float t = atan2f(Zi[s], Zr[s]);
      if (t <= -3.14159265358979f) t = 3.14159265358979f;   // principal branch (-pi, pi]
      own_th[b] = t;
      own_rel[b] = valid[s] && Wv[s] > eta && Za[s] > eta;
    }
  }
  __syncwarp();
  float num = 0.f, den = 0.f;
  int any = 0;
  float thv[2];
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const int b = lane + 32 * s;
    const int ky = b / 5, kx = b % 5;
    const bool edge = kx == 0 || ((g.w % 2 == 0) && kx == hw2);
    const bool selfc = edge && (ky == 0 || ((g.h % 2 == 0) && 2 * ky == g.h));
    const bool mirror = edge && !selfc && 2 * ky > g.h;
    const int rep = mirror ? (g.h - ky) * 5 + kx : b;
    const bool rel = valid[s] && b < kNB && own_rel[rep < kNB ? rep : 0];
    float t = (b < kNB) ? own_th[rep < kNB ? rep : 0] : 0.f;
    if (mirror) t = -t;
    if (!rel || selfc) t = 0.f;
    thv[s] = t;
    if (rel && b != 0) {
      const float kap = edge ? 1.f : 2.f;
      num += kap * Za[s];
      den += kap * Wv[s];
      any = 1;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    num += __shfl_xor_sync(0xffffffffu, num, o);
    den += __shfl_xor_sync(0xffffffffu, den, o);
    any |= __shfl_xor_sync(0xffffffffu, any, o);
  }
  const float c = any ? num / (den + a.eps) : 0.f;
  const float hh = (float)(g.h / 2) / (float)g.h, ww = (float)hw2 / (float)g.w;
  const float rmax = sqrtf(hh * hh + ww * ww);
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const int b = lane + 32 * s;
    if (b >= kNB) continue;
    const int ky = b / 5, kx = b % 5;
    const int kys = ky <= (g.h - 1) / 2 ? ky : ky - g.h;
    const float fy = (float)kys / (float)g.h, fx = (float)kx / (float)g.w;
    const float nu = rmax > 0.f ? sqrtf(fy * fy + fx * fx) / rmax : 0.f;
    const float tau = a.tau_low + (a.tau_high - a.tau_low) * powf(nu, a.q);
    float gv = 1.f / (1.f + expf(-(c - tau) / a.T));
    if (a.gate_mode == CAST_GATE_ZERO) gv = 0.f;
    if (a.gate_mode == CAST_GATE_ONE) gv = 1.f;
    if (a.band >= 0.f) {
      const float ry = (float)kys * 8.f / (float)g.h, rx = (float)kx * 8.f / (float)g.w;
      if (sqrtf(ry * ry + rx * rx) > a.band) gv = 0.f;
    }
    th[b] = any ? thv[s] : 0.f;
    gate[b] = gv;
  }
}

template <typename T>
constexpr size_t stage_bytes() { return (size_t)64 * kThreads * sizeof(T); }
template <typename T>
constexpr size_t par_dyn_smem() {
  return 2 * stage_bytes<T>() + kSpecFloats * sizeof(float) + 128;   // in, out, previous spectrum
}

template <typename T>
__global__ void __launch_bounds__(kThreads, 2)
    k_par(const __grid_constant__ CUtensorMap tm, const __grid_constant__ ParKArgs a,
          float* __restrict__ partial, unsigned* __restrict__ counters) {
  extern __shared__ uint8_t dsm_raw[];
  const uint32_t raw = smem_u32(dsm_raw);
  uint8_t* dsm = dsm_raw + (((raw + 127u) & ~127u) - raw);   // TMA boxes without swizzle: 128 B
  const T* stage = reinterpret_cast<const T*>(dsm);          // [y][x][channel] of one anchor tile
  float* s_fprev = reinterpret_cast<float*>(dsm + stage_bytes<T>());   // [value][thread]
  T* ostage = reinterpret_cast<T*>(dsm + stage_bytes<T>() + kSpecFloats * sizeof(float));
  __shared__ float s_red[kThreads / 32][128];
  __shared__ float s_zw[kNV];
  __shared__ float s_th[kNB], s_g[kNB], s_own_th[kNB];
  __shared__ int s_own_rel[kNB];
  __shared__ float4 s_coef[kCoefBatch][kNB];
  __shared__ int s_ticket;
  __shared__ __align__(8) uint64_t s_full;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // bytes one TMA box delivers: 128 channels x tile_w x tile_h (must match the tensor map)
  const uint32_t kStageBytes = (uint32_t)(kThreads * a.tw * a.th * sizeof(T));
  if (tid == 0) {
    mbar_init(&s_full, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tm);
  }
  __syncthreads();
  uint32_t n_loaded = 0;   // tiles consumed so far (phase of s_full)

  for (;;) {
    if (tid == 0) s_ticket = (int)atomicAdd(&counters[0], 1u);
    __syncthreads();
    const int t = s_ticket;
    __syncthreads();
    if (t >= a.total_tickets) break;
    int q = 0;
    while (q + 1 < a.n_seg && a.seg_first[q + 1] <= t) ++q;
    const int local = t - a.seg_first[q];
    const int tile = a.seg_tile0[q] + local / a.n_chunk;
    const int chunk = local % a.n_chunk;
    const bool recon = a.seg_recon[q] != 0;
    const TileGeom g = tile_geom(a, tile);
    const int c = chunk * kThreads + tid;
    const bool active = c < a.C;
    const float wc = active ? (a.wch ? __ldg(a.wch + c) : 1.f) : 0.f;

    if (tid == 0) {
      if (recon) {
        // every chunk of this tile must have published its partial records (bounded wait)
        const uint64_t t0 = global_ns();
        while (ld_acquire(&counters[1 + tile]) < (unsigned)a.n_chunk) {
          if (global_ns() - t0 > a.wait_ns) {
            atomicExch(&g_par_error, 1u);
            break;
          }
          __nanosleep(128);
        }
      }
      mbar_arrive_expect_tx(&s_full, kStageBytes);
      tma_load_4d(const_cast<T*>(stage), &tm, &s_full, chunk * kThreads, g.x0, g.y0, a.anchor_frame[0]);
    }
    if (recon) __syncthreads();

    for (int j = 0; j < a.n_anchor; ++j) {
      float re[8][5], im[8][5];
      {
        const bool ok = mbar_wait(&s_full, n_loaded & 1u, a.wait_ns);
        ++n_loaded;
        float x[8][8];
        if (a.tw == 8 && a.th == 8) {
#pragma unroll
          for (int y = 0; y < 8; ++y)
#pragma unroll
            for (int xx = 0; xx < 8; ++xx) x[y][xx] = to_f32(stage[(y * 8 + xx) * kThreads + tid]);
        } else {
#pragma unroll
          for (int y = 0; y < 8; ++y)
#pragma unroll
            for (int xx = 0; xx < 8; ++xx)
              x[y][xx] = (y < a.th && xx < a.tw) ? to_f32(stage[(y * a.tw + xx) * kThreads + tid]) : 0.f;
        }
        // the stage is free: prefetch the next anchor while transforming this one.  A tile
        // that never arrived ends the kernel for every thread of the CTA (error word set);
        // the barrier is never re-armed in an incomplete phase.
        if (__syncthreads_or(!ok)) {
          if (tid == 0) atomicExch(&g_par_error, 1u);
          return;
        }
        if (tid == 0 && j + 1 < a.n_anchor) {
          mbar_arrive_expect_tx(&s_full, kStageBytes);
          tma_load_4d(const_cast<T*>(stage), &tm, &s_full, chunk * kThreads, g.x0, g.y0,
                      a.anchor_frame[j + 1]);
        }
        dft::fwd2d(x, g.h, g.w, re, im);
      }
      const bool has_targets = j > 0 && a.pair_tbeg[j + 1] > a.pair_tbeg[j];
      const float* fa = s_fprev;   // spectrum of anchor j-1 (this thread's column)
      if (has_targets && !recon) {
        // ---- partial Z = sum w F_b conj(F_a), W = sum w |F_b||F_a| over the chunk (Eq. cross)
        if (g.h == 8 && g.w == 8) {
          // the 96 non-redundant values in three transpose groups, W at DC by a warp sum
#pragma unroll
          for (int grp = 0; grp < 3; ++grp) {
            float v[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              const int code = fast_value(grp * 32 + e);
              const int b = code >> 2, comp = code & 3;
              const float ar = fa[(2 * b) * kThreads + tid], ai = fa[(2 * b + 1) * kThreads + tid];
              const float br = re[b / 5][b % 5], bi = im[b / 5][b % 5];
              v[e] = comp == 0 ? wc * (br * ar + bi * ai)
                   : comp == 1 ? wc * (bi * ar - br * ai)
                               : wc * sqrtf((ar * ar + ai * ai) * (br * br + bi * bi));
            }
            s_red[warp][grp * 32 + lane] = warp_transpose_sum(v, lane);
          }
          float wdc = wc * fabsf(re[0][0]) * fabsf(fa[tid]);
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) wdc += __shfl_xor_sync(0xffffffffu, wdc, o);
          if (lane == 0) s_red[warp][96] = wdc;
          __syncthreads();
          if (tid < kNV) {
            const int src = a.fast_src[tid];
            float sum = 0.f;
            if (src != 0) {
              const int k = (src > 0 ? src : -src) - 1;
#pragma unroll
              for (int w = 0; w < kThreads / 32; ++w) sum += s_red[w][k];
              if (src < 0) sum = -sum;
            }
            partial[(((int64_t)j * a.n_tile + tile) * a.n_chunk + chunk) * kNV + tid] = sum;
          }
          __syncthreads();
        } else {
#pragma unroll
          for (int grp = 0; grp < 4; ++grp) {
            float v[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              const int vi = grp * 32 + e;
              if (vi < kNV) {
                const int b = vi / 3, comp = vi % 3;
                const float ar = fa[(2 * b) * kThreads + tid], ai = fa[(2 * b + 1) * kThreads + tid];
                const float br = re[b / 5][b % 5], bi = im[b / 5][b % 5];
                v[e] = comp == 0 ? wc * (br * ar + bi * ai)
                     : comp == 1 ? wc * (bi * ar - br * ai)
                                 : wc * sqrtf((ar * ar + ai * ai) * (br * br + bi * bi));
              } else {
                v[e] = 0.f;
              }
            }
            s_red[warp][grp * 32 + lane] = warp_transpose_sum(v, lane);
          }
          __syncthreads();
          if (tid < kNV) {
            float sum = 0.f;
#pragma unroll
            for (int w = 0; w < kThreads / 32; ++w) sum += s_red[w][tid];
            partial[(((int64_t)j * a.n_tile + tile) * a.n_chunk + chunk) * kNV + tid] = sum;
          }
          __syncthreads();
        }
      } else if (has_targets && recon) {
        // ---- transport of pair (j-1, j) on this tile
        if (tid < kNV) {
          // fixed-order sum over the chunks, 4 independent loads in flight
          const float* p = partial + ((int64_t)j * a.n_tile + tile) * a.n_chunk * kNV + tid;
          float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
          int k = 0;
          for (; k + 3 < a.n_chunk; k += 4) {
            s0 += __ldcg(p + (int64_t)k * kNV);
            s1 += __ldcg(p + (int64_t)(k + 1) * kNV);
            s2 += __ldcg(p + (int64_t)(k + 2) * kNV);
            s3 += __ldcg(p + (int64_t)(k + 3) * kNV);
          }
          for (; k < a.n_chunk; ++k) s0 += __ldcg(p + (int64_t)k * kNV);
          s_zw[tid] = (s0 + s1) + (s2 + s3);
        }
        __syncthreads();
        if (warp == 0) tile_transport(a, g, s_zw, s_th, s_g, s_own_th, s_own_rel, lane);
        __syncthreads();
        const float inv_hw = 1.f / (float)(g.h * g.w);
        for (int t0 = a.pair_tbeg[j]; t0 < a.pair_tbeg[j + 1]; t0 += kCoefBatch) {
          const int nt = min(kCoefBatch, a.pair_tbeg[j + 1] - t0);
          for (int e = tid; e < nt * kNB; e += kThreads) {
            const int k = e / kNB, b = e % kNB;
            const float al = a.target_alpha[t0 + k];
            float sa, ca, sb, cb;
            sincosf(s_g[b] * al * s_th[b], &sa, &ca);
            sincosf(-s_g[b] * (1.f - al) * s_th[b], &sb, &cb);
            const float fa_ = (1.f - al) * inv_hw, fb_ = al * inv_hw;
            s_coef[k][b] = make_float4(fa_ * ca, fa_ * sa, fb_ * cb, fb_ * sb);
          }
          __syncthreads();
          for (int k = 0; k < nt; ++k) {
            // Eq. (fcpasm): (1-alpha) F_a U^{g alpha} + alpha F_b U^{-g (1-alpha)}, ortho scale folded
            float hr[8][5], hi[8][5];
#pragma unroll
            for (int b = 0; b < kNB; ++b) {
              const int ky = b / 5, kx = b % 5;
              const float4 cf = s_coef[k][b];
              const float ar = fa[(2 * b) * kThreads + tid], ai = fa[(2 * b + 1) * kThreads + tid];
              const float br = re[ky][kx], bi = im[ky][kx];
              hr[ky][kx] = cf.x * ar - cf.y * ai + cf.z * br - cf.w * bi;
              hi[ky][kx] = cf.x * ai + cf.y * ar + cf.z * bi + cf.w * br;
            }
            // the previous tile store must have finished reading the out stage
            if (tid == 0) bulk_wait_read_all();
            __syncthreads();
            const int tw = a.tw;
            dft::inv2d_emit(hr, hi, g.h, g.w, [&](int yy, const float* row) {
              if (tw == 8) {
#pragma unroll
                for (int xx = 0; xx < 8; ++xx) ostage[(yy * 8 + xx) * kThreads + tid] = T(row[xx]);
              } else {
#pragma unroll
                for (int xx = 0; xx < 8; ++xx)
                  if (xx < tw) ostage[(yy * tw + xx) * kThreads + tid] = T(row[xx]);
              }
            });
            fence_proxy_async_smem();
            __syncthreads();
            if (tid == 0) {
              tma_store_4d(&tm, ostage, chunk * kThreads, g.x0, g.y0, a.target_frame[t0 + k]);
              bulk_commit();
            }
          }
          __syncthreads();
        }
      }
      // this anchor's spectrum becomes the previous one (thread-private column)
      if (j + 1 < a.n_anchor) {
#pragma unroll
        for (int b = 0; b < kNB; ++b) {
          s_fprev[(2 * b) * kThreads + tid] = re[b / 5][b % 5];
          s_fprev[(2 * b + 1) * kThreads + tid] = im[b / 5][b % 5];
        }
      }
    }
    if (!recon) {
      __syncthreads();
      if (tid == 0) {
        __threadfence();
        atomicAdd(&counters[1 + tile], 1u);
      }
    }
  }
  if (tid == 0) bulk_wait_all();   // tile stores complete before the CTA's shared memory goes
}

// 4-D map [F][Hg][Wg][C], box (128 channels, tw, th, 1), zero fill out of range
bool make_r_map(CUtensorMap* m, const cast_par_args& a) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (!fn) return false;
  const cuuint64_t elt = a.dtype == CAST_BF16 ? 2 : 4;
  cuuint64_t dims[4] = {(cuuint64_t)a.C, (cuuint64_t)a.Wg, (cuuint64_t)a.Hg, (cuuint64_t)a.F};
  cuuint64_t strides[3] = {a.C * elt, (cuuint64_t)a.Wg * a.C * elt, (cuuint64_t)a.Hg * a.Wg * a.C * elt};
  cuuint32_t box[4] = {(cuuint32_t)kThreads, (cuuint32_t)a.params.tile_w, (cuuint32_t)a.params.tile_h, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, a.dtype == CAST_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
            4, a.r, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <typename T>
cast_status launch_typed(const CUtensorMap& tm, const ParKArgs& k, int tickets, float* partial,
                         unsigned* counters, cudaStream_t st) {
  static bool attr_set = false;
  constexpr size_t smem = par_dyn_smem<T>();
  if (!attr_set) {
    if (cudaFuncSetAttribute(k_par<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
        cudaSuccess)
      return check_launch("PAR smem attribute");
    attr_set = true;
  }
  int dev = 0, nsm = 0, occ = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k_par<T>, kThreads, smem);
  if (occ < 1) occ = 1;
  int grid = nsm * occ;
  if (grid > tickets) grid = tickets;
  k_par<T><<<grid, kThreads, smem, st>>>(tm, k, partial, counters);
  return check_launch("PAR kernel");
}

}  // namespace

ParPlan par_plan(const cast_par_args& a) {
  ParPlan p{};
  int na = 0;
  for (int f = 0; f < a.F; ++f) na += a.anchor_mask[f] ? 1 : 0;
  p.n_anchor = na;
  p.n_pair = na > 0 ? na - 1 : 0;
  p.n_target = a.F - na;
  const int th = a.params.tile_h, tw = a.params.tile_w;
  p.tiles_y = (a.Hg + th - 1) / th;
  p.tiles_x = (a.Wg + tw - 1) / tw;
  p.n_tile = p.tiles_y * p.tiles_x;
  p.chunk = kThreads;
  p.n_chunk = (a.C + kThreads - 1) / kThreads;
  // slab: tiles whose anchor bytes stay well inside L2 between the stats and recon passes
  const double elt = a.dtype == CAST_BF16 ? 2.0 : 4.0;
  const double tile_bytes = (double)na * th * tw * a.C * elt;
  int slab = (int)(24.0e6 / (tile_bytes > 1 ? tile_bytes : 1));
  if (slab < 1) slab = 1;
  if (slab > p.n_tile) slab = p.n_tile;
  while ((p.n_tile + slab - 1) / slab > kMaxSeg / 2) ++slab;
  p.slab_tiles = slab;
  p.n_slab = (p.n_tile + slab - 1) / slab;
  p.partial_bytes = align_up((size_t)(na > 0 ? na : 1) * p.n_tile * p.n_chunk * kNV * sizeof(float));
  p.counter_bytes = align_up((size_t)(1 + p.n_tile) * sizeof(unsigned));
  p.total_bytes = p.partial_bytes + p.counter_bytes;
  return p;
}

cast_status launch_par(const cast_par_args& a, void* ws, cudaStream_t st) {
  const ParPlan p = par_plan(a);
  if (p.n_target == 0) return CAST_OK;   // every frame is an anchor: reconstruction bypassed
  ParKArgs k{};
  k.r = static_cast<char*>(a.r);
  k.wch = a.channel_weight;
  k.F = a.F;
  k.Hg = a.Hg;
  k.Wg = a.Wg;
  k.C = a.C;
  k.th = a.params.tile_h;
  k.tw = a.params.tile_w;
  k.tiles_x = p.tiles_x;
  k.n_tile = p.n_tile;
  k.n_chunk = p.n_chunk;
  int anchors[CAST_MAX_FRAMES];
  int na = 0;
  for (int f = 0; f < a.F; ++f)
    if (a.anchor_mask[f]) anchors[na++] = f;
  k.n_anchor = na;
  for (int j = 0; j < na; ++j) k.anchor_frame[j] = anchors[j];
  // targets grouped by pair j (anchors j-1, j), j = 1..na-1 (Eq. block)
  int nt = 0;
  for (int j = 0; j <= na; ++j) k.pair_tbeg[j] = 0;
  for (int j = 1; j < na; ++j) {
    k.pair_tbeg[j] = nt;
    const int a0 = anchors[j - 1], a1 = anchors[j];
    auto add = [&](int t) {
      k.target_frame[nt] = t;
      k.target_alpha[nt] = (float)((double)(t - a0) / (double)(a1 - a0));
      ++nt;
    };
    if (j == 1)
      for (int t = 0; t < a0; ++t) add(t);
    for (int t = a0 + 1; t < a1; ++t) add(t);
    if (j == na - 1)
      for (int t = a1 + 1; t < a.F; ++t) add(t);
  }
  k.pair_tbeg[na] = nt;
  // ticket schedule: S(0), S(1), R(0), S(2), R(1), ..., R(n-1)
  int nseg = 0, ticket = 0;
  auto seg = [&](int slab, bool recon) {
    const int t0 = slab * p.slab_tiles;
    const int nt_ = (t0 + p.slab_tiles <= p.n_tile ? p.slab_tiles : p.n_tile - t0);
    k.seg_first[nseg] = ticket;
    k.seg_tile0[nseg] = t0;
    k.seg_recon[nseg] = recon ? 1 : 0;
    ticket += nt_ * p.n_chunk;
    ++nseg;
  };
  seg(0, false);
  for (int s = 1; s < p.n_slab; ++s) {
    seg(s, false);
    seg(s - 1, true);
  }
  seg(p.n_slab - 1, true);
  k.n_seg = nseg;
  k.seg_first[nseg] = ticket;
  k.total_tickets = ticket;
  const cast_par_params& pp = a.params;
  k.tau_low = pp.tau_low;
  k.tau_high = pp.tau_high;
  k.q = pp.q;
  k.T = pp.T;
  k.eps = pp.eps;
  k.eta_rel = pp.eta_rel;
  k.eta_abs = pp.eta_abs;
  k.band = pp.band_radius;
  k.gate_mode = pp.gate_mode;
  k.wait_ns = 2000000000ull;
  {
    // record entry t = 3 * bin + comp of an 8x8 tile from the 96 reduced values (+ W at DC = 96)
    int pos[40 * 4];
    for (int q = 0; q < 160; ++q) pos[q] = -1;
    for (int n = 0; n < 96; ++n) pos[fast_value(n)] = n;
    for (int t = 0; t < kNV; ++t) {
      const int b = t / 3, comp = t % 3, ky = b / 5, kx = b % 5;
      const bool edge = kx == 0 || kx == 4;
      const bool selfc = edge && (ky == 0 || ky == 4);
      const bool mirror = edge && !selfc && ky > 4;
      const int r = mirror ? (8 - ky) * 5 + kx : b;
      int src = 0;
      if (r == 0) src = comp == 2 ? 96 + 1 : 0;                 // DC: only W
      else if (comp == 1 && selfc) src = 0;                     // Im Z of a real bin
      else src = (pos[r * 4 + comp] + 1) * ((mirror && comp == 1) ? -1 : 1);
      k.fast_src[t] = (signed char)src;
    }
  }

  CUtensorMap tm;
  if (!make_r_map(&tm, a)) return fail(CAST_ERR_CUDA, "PAR: cuTensorMapEncodeTiled failed");
  char* w = static_cast<char*>(ws);
  float* partial = reinterpret_cast<float*>(w);
  unsigned* counters = reinterpret_cast<unsigned*>(w + p.partial_bytes);
  if (cudaMemsetAsync(counters, 0, (size_t)(1 + p.n_tile) * sizeof(unsigned), st) != cudaSuccess)
    return check_launch("PAR counter reset");
  if (a.dtype == CAST_BF16) return launch_typed<__nv_bfloat16>(tm, k, ticket, partial, counters, st);
  return launch_typed<float>(tm, k, ticket, partial, counters, st);
}

unsigned int par_error_word(cudaStream_t st, bool clear) {
  unsigned int v = 0;
  cudaMemcpyFromSymbolAsync(&v, g_par_error, sizeof(v), 0, cudaMemcpyDeviceToHost, st);
  cudaStreamSynchronize(st);
  if (clear && v) {
    const unsigned int z = 0;
    cudaMemcpyToSymbolAsync(g_par_error, &z, sizeof(z), 0, cudaMemcpyHostToDevice, st);
    cudaStreamSynchronize(st);
  }
  return v;
}

}  // namespace cast
