// Phase-Aware Reconstruction of skipped frames (Section 4.3, Eqs. cross, confidence, gate,
// fcpasm; App. A.2) in three passes per tile kind (full 8x8 tiles / truncated edge tiles):
//
//   K_stats (tile, channel chunk): one thread per channel streams the anchors of the tile in
//       time order through a TMA 4-D map ([frame][row][col][channel], out-of-range rows/cols/
//       channels arrive as zeros), forms each tile spectrum in registers (the previous anchor's
//       spectrum stays in shared memory) and, for every anchor pair with targets, reduces
//       Z = sum_c w_c F_b conj(F_a) and W = sum_c w_c |F_b||F_a| over the chunk's channels
//       (warp transpose reductions) into one record in the workspace.
//   K_transport (tile, pair[, target]): sums the records of the tile's channel chunks in chunk
//       order (deterministic) and derives eta, reliability, principal phases, the confidence c
//       and the gate g per bin; writes theta and g (and, for bf16, one target's blend matrix).
//   K_blend (tile, channel chunk): streams the anchors again (an L2 hit at these sizes), forms
//       their spectra and writes every target straight from registers:
//       R_t = IRFFT2((1-alpha) F_a e^{i g alpha theta} + alpha F_b e^{-i g (1-alpha) theta}).
//       This is the f32 blend.  For bf16 residuals the blend runs on the tensor cores instead
//       (K_blend_tc below): on one tile, Eq. (fcpasm) is exactly two circular convolutions,
//         R_t = h_a (*) R_a + h_b (*) R_b,  h = IDFT2 of the Hermitian-extended phasors
//         phi_a = (1-alpha) e^{i g alpha theta}, phi_b = alpha e^{-i g (1-alpha) theta},
//       so K_transport also writes each target's 64 x 128 matrix [H_a | H_b] (two bf16 pieces,
//       laid out as a swizzled UMMA operand) and one UMMA chain per pair of targets computes
//       [H_t1 ; H_t2] [X_a ; X_b] for 128 channels (M = 128 output rows, K = 128 tokens).
// The CTAs of a pass never wait on each other, so the passes fill the GPU whatever the number
// of anchor pairs; the passes are chained as programmatic dependents (the transport releases
// the blend at its end), the full-tile chain on the caller's stream and the edge-tile chain on
// a second stream.  Global traffic beyond the algorithmic bytes: a second read of the anchors,
// the records (120 floats per tile, pair and chunk) and, for bf16, the blend matrices (32 KB
// per tile and target, read from L2 by every channel chunk).
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>
#include <mutex>

#include "dft.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace cast {
namespace {

constexpr int kCC = 128;           // channels per CTA (one thread each)
constexpr int kNB = 40;            // stored bins of an 8-wide tile: 8 x 5
constexpr int kNV = 3 * kNB;       // (Re Z, Im Z, W) per bin, record index = 3 * bin + component
constexpr int kRec = kNV;          // record slots per chunk (96 + 1 used for 8x8 tiles)
constexpr int kCoefBatch = 4;

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
  float* rec;     // workspace [tile][pair j][chunk][kRec]: each chunk's Z / W record
  float* trans;   // workspace [tile][pair j][2][kNB]: theta and g per bin
  char* img;      // workspace [tile][target][kImgBytes]: blend matrices (bf16 runs), or null
  int n_target;
  int F, Hg, Wg, C, n_chunk;             // n_chunk: channel chunks of kCC channels
  int tile_base;                         // global index of tile 0 of this launch's kind
  int th, tw, tiles_x, tiles_y, n_tile, n_tseg;
  int n_anchor;
  int anchor_frame[CAST_MAX_ANCHORS];
  int pair_tbeg[CAST_MAX_ANCHORS + 1];   // targets of pair j (anchors j-1, j) in [tbeg[j], tbeg[j+1])
  int target_frame[CAST_MAX_FRAMES];
  float target_alpha[CAST_MAX_FRAMES];
  int seg_pair0[CAST_MAX_ANCHORS];       // time segment s covers pairs seg_pair0[s] .. seg_pair1[s]
  int seg_pair1[CAST_MAX_ANCHORS];
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


struct TileGeom {
  int y0, x0, h, w;
};

// Tile i of one kind.  With 8x8 tiles: full tiles (row-major over the full-tile grid) or edge
// tiles (the truncated last column of every tile row, then the truncated last row).  Other
// tile sides: every tile, row-major, in the edge kind.
__device__ __forceinline__ TileGeom tile_geom(const ParKArgs& a, int i, bool full) {
  TileGeom g;
  if (a.th != 8 || a.tw != 8) {
    const int ty = i / a.tiles_x, tx = i - (i / a.tiles_x) * a.tiles_x;
    g.y0 = ty * a.th;
    g.x0 = tx * a.tw;
    g.h = min(a.th, a.Hg - g.y0);
    g.w = min(a.tw, a.Wg - g.x0);
    return g;
  }
  const int fy = a.Hg / 8, fx = a.Wg / 8;   // full tiles per column / row
  int ty, tx;
  if (full) {
    ty = i / fx;
    tx = i - ty * fx;
  } else if (a.Wg % 8 != 0 && i < a.tiles_y) {
    ty = i;
    tx = fx;
  } else {
    ty = fy;
    tx = i - (a.Wg % 8 != 0 ? a.tiles_y : 0);
  }
  g.y0 = ty * 8;
  g.x0 = tx * 8;
  g.h = min(8, a.Hg - g.y0);
  g.w = min(8, a.Wg - g.x0);
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

__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float sqrt_approx(float x) {
  float y;
  asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// sin and cos of x = 2 pi k + r with |r| <= pi (Cody-Waite split of 2 pi into two parts),
// then the hardware approximations on the reduced argument.
__device__ __forceinline__ void sincos_reduced(float x, float* s, float* c) {
  const float k = rintf(x * 0.159154943091895336f);
  float r = fmaf(-k, 6.28318548202514648f, x);
  r = fmaf(-k, -1.74845553e-07f, r);
  __sincosf(r, s, c);
}

// Geometry of the stored bins of one tile shape (App. A.2), computed once per CTA: per bin
// b = ky * 5 + kx the representative (mirrors point at their conjugate), the pooling weight
// kappa (0: not stored, DC, or outside the tile), the flags, the gate threshold tau(nu) and
// whether the band cut forces g = 0.
struct BinInfo {
  float tau[kNB], kap[kNB];
  int rep[kNB];
  unsigned char valid[kNB], selfc[kNB], mirror[kNB], cut[kNB];
};

__device__ void bin_info(const ParKArgs& a, const TileGeom& g, BinInfo& bi, int tid) {
  if (tid >= kNB) return;
  const int b = tid, ky = b / 5, kx = b % 5, hw2 = g.w / 2;
  const bool valid = ky < g.h && kx <= hw2;
  const bool edge = kx == 0 || ((g.w % 2 == 0) && kx == hw2);
  const bool selfc = edge && (ky == 0 || ((g.h % 2 == 0) && 2 * ky == g.h));
  const bool mirror = edge && !selfc && 2 * ky > g.h;
  bi.valid[b] = valid;
  bi.selfc[b] = selfc;
  bi.mirror[b] = mirror;
  bi.rep[b] = mirror ? (g.h - ky) * 5 + kx : b;
  bi.kap[b] = (valid && b != 0) ? (edge ? 1.f : 2.f) : 0.f;
  const int kys = ky <= (g.h - 1) / 2 ? ky : ky - g.h;
  const float hh = (float)(g.h / 2) / (float)g.h, ww = (float)hw2 / (float)g.w;
  const float rmax = sqrtf(hh * hh + ww * ww);
  const float fy = (float)kys / (float)g.h, fx = (float)kx / (float)g.w;
  const float nu = rmax > 0.f ? sqrtf(fy * fy + fx * fx) / rmax : 0.f;
  bi.tau[b] = a.tau_low + (a.tau_high - a.tau_low) * powf(nu, a.q);
  bool cut = false;
  if (a.band >= 0.f) {
    const float ry = (float)kys * 8.f / (float)g.h, rx = (float)kx * 8.f / (float)g.w;
    cut = sqrtf(ry * ry + rx * rx) > a.band;
  }
  bi.cut[b] = cut;
}

// Per-tile transport of one anchor pair (warp 0, two bins per lane): theta and g per stored
// bin from the pooled Z, W record (App. A.2).
__device__ void tile_transport(const ParKArgs& a, const TileGeom& g, const BinInfo& bi,
                               const float* zw, float* th, float* gate, float* own_th,
                               int* own_rel, int lane) {
  const float inv_hw = 1.f / (float)(g.h * g.w);
  float Zr[2], Zi[2], Wv[2], Za[2], t[2];
  float wmax = 0.f;
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const int b = lane + 32 * s;
    const bool v = b < kNB && bi.valid[b];
    Zr[s] = v ? zw[3 * b] * inv_hw : 0.f;
    Zi[s] = v ? zw[3 * b + 1] * inv_hw : 0.f;
    Wv[s] = v ? zw[3 * b + 2] * inv_hw : 0.f;
    Za[s] = sqrt_approx(Zr[s] * Zr[s] + Zi[s] * Zi[s]);
    t[s] = atan2f(Zi[s], Zr[s]);
    if (t[s] <= -3.14159265358979f) t[s] = 3.14159265358979f;   // principal branch (-pi, pi]
    if (v) wmax = fmaxf(wmax, Wv[s]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) wmax = fmaxf(wmax, __shfl_xor_sync(0xffffffffu, wmax, o));
  const float eta = a.eta_rel * wmax + a.eta_abs;
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const int b = lane + 32 * s;
    if (b < kNB) {
      own_th[b] = t[s];
      own_rel[b] = bi.valid[b] && Wv[s] > eta && Za[s] > eta;
    }
  }
  __syncwarp();
  float num = 0.f, den = 0.f;
  int any = 0;
  float thv[2];
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const int b = lane + 32 * s;
    thv[s] = 0.f;
    if (b < kNB) {
      const int rep = bi.rep[b] < kNB ? bi.rep[b] : 0;
      const bool rel = bi.valid[b] && own_rel[rep];
      float tv = own_th[rep];
      if (bi.mirror[b]) tv = -tv;
      thv[s] = (!rel || bi.selfc[b]) ? 0.f : tv;
      if (rel && bi.kap[b] > 0.f) {
        num += bi.kap[b] * Za[s];
        den += bi.kap[b] * Wv[s];
        any = 1;
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    num += __shfl_xor_sync(0xffffffffu, num, o);
    den += __shfl_xor_sync(0xffffffffu, den, o);
    any |= __shfl_xor_sync(0xffffffffu, any, o);
  }
  const float c = any ? __fdividef(num, den + a.eps) : 0.f;
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const int b = lane + 32 * s;
    if (b >= kNB) continue;
    const float tau = bi.tau[b];
    float gv = rcp_approx(1.f + __expf((tau - c) * rcp_approx(a.T)));
    if (a.gate_mode == CAST_GATE_ZERO) gv = 0.f;
    if (a.gate_mode == CAST_GATE_ONE) gv = 1.f;
    if (bi.cut[b]) gv = 0.f;   // outside the band
    th[b] = any ? thv[s] : 0.f;
    gate[b] = gv;
  }
}

// ------------------------------------------------------------------ blend matrices
constexpr int kImgTerm = 64 * 128 * 2;   // one bf16 piece of one target's [64][128] matrix, 16 KB
constexpr int kImgBytes = 2 * kImgTerm;  // both pieces (hi, lo): 32 KB per (tile, target)

// The blend matrices of the targets t_begin <= t < t_end of one (tile, pair), written as UMMA operand images
// (K-major, 128-byte swizzle, K-blocks of 64 tokens 8 KB apart, two bf16 pieces kImgTerm apart):
// row m = output token 8 yo + xo, column 64 side + 8 yi + xi = input token of anchor a (side 0)
// or b (side 1); entry h_side((yo - yi) mod h, (xo - xi) mod w) with
// h_side(d) = (1 / (h w)) sum over stored bins of kappa' Re(phi_side e^{2 pi i (ky dy / h + kx dx / w)}),
// kappa' = 1 on the kx = 0 and Nyquist columns (every ky stored), 2 elsewhere;
// phi_a = (1 - alpha) e^{i g alpha theta}, phi_b = alpha e^{-i g (1 - alpha) theta}.  128 threads.
// FULL8: an 8x8 tile, where every twiddle is an 8th root of unity and every index a mask (the
// same values, summed in the same order, as the general form).
template <bool FULL8>
__device__ void build_blend_images(const ParKArgs& a, const TileGeom& g, const BinInfo& bi,
                                   const float* th, const float* gate, int tg, int t_begin, int t_end,
                                   int tid) {
  __shared__ float2 s_cs[64];
  __shared__ unsigned char s_ym[8][8], s_xm[5][8];
  __shared__ float4 s_phi[kNB];
  __shared__ float s_h[2][64];
  const int h = FULL8 ? 8 : g.h, w = FULL8 ? 8 : g.w, n = h * w;
  if (FULL8) {
    // e^{2 pi i q / 8} at s_cs[q]
    if (tid < 8) {
      float sv, cv;
      sincospif((float)tid / 4.f, &sv, &cv);
      s_cs[tid] = make_float2(cv, sv);
    }
  } else if (tid < 64) {
    if (tid < n) {
      float sv, cv;
      sincospif(2.f * (float)tid / (float)n, &sv, &cv);
      s_cs[tid] = make_float2(cv, sv);
    }
    s_ym[tid >> 3][tid & 7] = (unsigned char)(((tid >> 3) * (tid & 7)) % h);
  } else if (tid < 64 + 40) {
    const int e = tid - 64;
    s_xm[e >> 3][e & 7] = (unsigned char)(((e >> 3) * (e & 7)) % w);
  }
  const float inv_n = 1.f / (float)n;
  const int side = tid >> 6, d = tid & 63, dy0 = d >> 3, dx0 = d & 7;
  for (int t = t_begin; t < t_end; ++t) {
    const float al = a.target_alpha[t];
    if (tid < kNB) {
      const int b = tid, kx = b % 5;
      float4 ph = make_float4(0.f, 0.f, 0.f, 0.f);
      if (bi.valid[b]) {
        const bool edge = kx == 0 || ((w % 2 == 0) && kx == w / 2);
        const float kap = (edge ? 1.f : 2.f) * inv_n;
        float sa, ca, sb, cb;
        const float gt = gate[b] * th[b];
        sincosf(gt * al, &sa, &ca);
        sincosf(-gt * (1.f - al), &sb, &cb);
        ph = make_float4(kap * (1.f - al) * ca, kap * (1.f - al) * sa, kap * al * cb, kap * al * sb);
      }
      s_phi[b] = ph;
    }
    __syncthreads();
    if (FULL8) {
      float acc = 0.f;
#pragma unroll
      for (int ky = 0; ky < 8; ++ky) {
        const int ry = ky * dy0;
#pragma unroll
        for (int kx = 0; kx < 5; ++kx) {
          const float2 e = s_cs[(ry + kx * dx0) & 7];
          const float4 ph = s_phi[ky * 5 + kx];
          const float pr = side ? ph.z : ph.x, pi = side ? ph.w : ph.y;
          acc = fmaf(pr, e.x, fmaf(-pi, e.y, acc));
        }
      }
      s_h[side][d] = acc;
    } else {
      float acc = 0.f;
      if (dy0 < h && dx0 < w) {
        for (int b = 0; b < kNB; ++b) {
          const int ky = b / 5, kx = b % 5;
          if (ky >= h || kx > w / 2) continue;
          int p = (int)s_ym[ky][dy0] * w + (int)s_xm[kx][dx0] * h;
          if (p >= n) p -= n;
          const float2 e = s_cs[p];
          const float4 ph = s_phi[b];
          const float pr = side ? ph.z : ph.x, pi = side ? ph.w : ph.y;
          acc = fmaf(pr, e.x, fmaf(-pi, e.y, acc));
        }
      }
      s_h[side][d] = acc;
    }
    __syncthreads();
    // 16-byte chunk q = 128 it + tid of a piece: side q >> 9, output token (row) m = (q >> 3) & 63,
    // stored chunk q & 7 = input row yi ^ (m & 7); a warp writes 512 contiguous bytes per piece
    uint8_t* img = reinterpret_cast<uint8_t*>(a.img) + ((int64_t)tg * a.n_target + t) * kImgBytes;
#pragma unroll
    for (int it = 0; it < 8; ++it) {
      const int q = it * 128 + tid, sd = q >> 9, m = (q >> 3) & 63, yi = (q & 7) ^ (m & 7);
      const int yo = m >> 3, xo = m & 7;
      const bool row_ok = FULL8 || (yo < h && xo < w && yi < h);
      const int dy = FULL8 ? (yo - yi) & 7 : yo - yi + (yo < yi ? h : 0);
      float v[8];
#pragma unroll
      for (int xi = 0; xi < 8; ++xi) {
        const int dx = FULL8 ? (xo - xi) & 7 : xo - xi + (xo < xi ? w : 0);
        v[xi] = (FULL8 || (row_ok && xi < w)) ? s_h[sd][dy * 8 + dx] : 0.f;
      }
      uint32_t hi[4], lo[4];
#pragma unroll
      for (int u = 0; u < 8; u += 2) {
        const __nv_bfloat162 b1 = __floats2bfloat162_rn(v[u], v[u + 1]);
        const __nv_bfloat162 b2 = __floats2bfloat162_rn(v[u] - __low2float(b1), v[u + 1] - __high2float(b1));
        hi[u / 2] = *reinterpret_cast<const uint32_t*>(&b1);
        lo[u / 2] = *reinterpret_cast<const uint32_t*>(&b2);
      }
      const int off = q << 4;   // side * 8192 + m * 128 + ((yi ^ (m & 7)) << 4)
      *reinterpret_cast<uint4*>(img + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
      *reinterpret_cast<uint4*>(img + kImgTerm + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
    }
    __syncthreads();   // s_phi and s_h are rewritten for the next target
  }
}

__device__ __forceinline__ void grid_dependency_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Dynamic shared memory of a streaming CTA with cc channels: a ring of n_stages<T> TMA stages
// (one anchor tile each, 128-byte aligned; two for bf16, one for f32 so that three CTAs still
// fit an SM) and the previous anchor's spectrum [value][thread].
template <typename T>
__host__ __device__ constexpr int n_stages() { return sizeof(T) == 2 ? 2 : 1; }
template <typename T>
__host__ __device__ constexpr size_t stage_bytes(int cc) { return (size_t)64 * cc * sizeof(T); }
__host__ __device__ constexpr size_t spec_bytes(int cc) { return (size_t)2 * kNB * cc * sizeof(float); }
template <typename T>
__host__ __device__ constexpr size_t par_dyn_smem(int cc) {
  return n_stages<T>() * stage_bytes<T>(cc) + spec_bytes(cc) + 128;
}

// K_stats (STATS) and K_blend (!STATS): grid (n_chunk, n_tiles_of_kind * n_tseg), CC threads,
// one channel each.  A time segment covers the anchor pairs seg_pair0 .. seg_pair1 (it starts
// one anchor earlier).  FULL: every tile of the launch is 8x8 (the specialised fast path).
template <typename T, int CC, bool FULL, bool STATS>
__global__ void __launch_bounds__(CC, 3)
    k_par(const __grid_constant__ CUtensorMap tm, const __grid_constant__ ParKArgs a) {
  extern __shared__ uint8_t dsm_raw[];
  const uint32_t raw = smem_u32(dsm_raw);
  uint8_t* dsm = dsm_raw + (((raw + 127u) & ~127u) - raw);   // TMA boxes without swizzle: 128 B
  constexpr int cc = CC;
  constexpr int nwarp = CC / 32;
  constexpr int kStages = n_stages<T>();
  T* stages = reinterpret_cast<T*>(dsm);       // kStages x [y][x][channel] of one anchor tile
  float* s_fprev = reinterpret_cast<float*>(dsm + kStages * stage_bytes<T>(cc));   // [value][thread]
  __shared__ float s_red[STATS ? nwarp : 1][128];
  __shared__ float4 s_coef[STATS ? 1 : kCoefBatch][kNB];
  __shared__ __align__(8) uint64_t s_full[kStages];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int chunk = blockIdx.x;
  const int tile = blockIdx.y / a.n_tseg, seg = blockIdx.y - tile * a.n_tseg;
  const int tg = a.tile_base + tile;                  // tile index in the workspace
  const int j0 = a.seg_pair0[seg] - 1, j1 = a.seg_pair1[seg];   // anchors of this segment
  const TileGeom g = tile_geom(a, tile, FULL);
  const int c = chunk * cc + tid;
  const bool active = c < a.C;
  const float wc = active ? (a.wch ? __ldg(a.wch + c) : 1.f) : 0.f;
  // bytes one TMA box delivers: cc channels x tile_w x tile_h (must match the tensor map)
  const uint32_t box_bytes = (uint32_t)(cc * a.tw * a.th * sizeof(T));
  if (tid == 0) {
    for (int st = 0; st < kStages; ++st) mbar_init(&s_full[st], 1);
    fence_barrier_init();
    tma_prefetch_desc(&tm);
    // the first kStages anchors of the segment are in flight at once
    for (int st = 0; st < kStages && j0 + st <= j1; ++st) {
      mbar_arrive_expect_tx(&s_full[st], box_bytes);
      tma_load_4d(stages + st * (stage_bytes<T>(cc) / sizeof(T)), &tm, &s_full[st], chunk * cc, g.x0,
                  g.y0, a.anchor_frame[j0 + st]);
    }
  }
  launch_dependents();
  __syncthreads();
  // K_blend reads theta and g, written by the preceding K_transport
  if (!STATS) grid_dependency_wait();
  bool ok = true;          // CTA-uniform; after a failed wait no more TMA is issued
  const int64_t frame_elems = (int64_t)a.Hg * a.Wg * a.C;
  T* out = reinterpret_cast<T*>(a.r);

  for (int j = j0; j <= j1; ++j) {
    float re[8][5], im[8][5];
    {
      const int it = j - j0, st = it % kStages;
      const T* stage = stages + st * (stage_bytes<T>(cc) / sizeof(T));
      const bool got = ok && mbar_wait(&s_full[st], (uint32_t)(it / kStages) & 1u, a.wait_ns);
      float x[8][8];
      if (FULL) {
#pragma unroll
        for (int y = 0; y < 8; ++y)
#pragma unroll
          for (int xx = 0; xx < 8; ++xx) x[y][xx] = to_f32(stage[(y * 8 + xx) * cc + tid]);
      } else {
#pragma unroll
        for (int y = 0; y < 8; ++y)
#pragma unroll
          for (int xx = 0; xx < 8; ++xx)
            x[y][xx] = (y < g.h && xx < g.w) ? to_f32(stage[(y * a.tw + xx) * cc + tid]) : 0.f;
      }
      // the stage is free: the anchor kStages ahead goes into it while this one is transformed
      if (__syncthreads_or(ok && !got)) {
        if (tid == 0) atomicExch(&g_par_error, 1u);
        ok = false;
      }
      if (ok && tid == 0 && j + kStages <= j1) {
        mbar_arrive_expect_tx(&s_full[st], box_bytes);
        tma_load_4d(const_cast<T*>(stage), &tm, &s_full[st], chunk * cc, g.x0, g.y0,
                    a.anchor_frame[j + kStages]);
      }
      if (FULL) dft::fwd2d(x, 8, 8, re, im);
      else dft::fwd2d(x, g.h, g.w, re, im);
    }
    const bool has_targets = j > j0 && a.pair_tbeg[j + 1] > a.pair_tbeg[j];
    const float* fa = s_fprev;   // spectrum of anchor j-1 (this thread's column)
    if (STATS && has_targets) {
      // this chunk's Z = sum w F_b conj(F_a), W = sum w |F_b||F_a| (Eq. cross)
      if (FULL) {
        // the 96 non-redundant values in three transpose groups, W at DC by a warp sum
#pragma unroll
        for (int grp = 0; grp < 3; ++grp) {
          float v[32];
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const int code = fast_value(grp * 32 + e);
            const int b = code >> 2, comp = code & 3;
            const float ar = fa[(2 * b) * cc + tid], ai = fa[(2 * b + 1) * cc + tid];
            const float br = re[b / 5][b % 5], bi = im[b / 5][b % 5];
            v[e] = comp == 0 ? wc * (br * ar + bi * ai)
                 : comp == 1 ? wc * (bi * ar - br * ai)
                             : wc * sqrt_approx((ar * ar + ai * ai) * (br * br + bi * bi));
          }
          s_red[warp][grp * 32 + lane] = warp_transpose_sum(v, lane);
        }
        float wdc = wc * fabsf(re[0][0]) * fabsf(fa[tid]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) wdc += __shfl_xor_sync(0xffffffffu, wdc, o);
        if (lane == 0) s_red[warp][96] = wdc;
      } else {
#pragma unroll
        for (int grp = 0; grp < 4; ++grp) {
          float v[32];
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const int vi = grp * 32 + e;
            if (vi < kNV) {
              const int b = vi / 3, comp = vi % 3;
              const float ar = fa[(2 * b) * cc + tid], ai = fa[(2 * b + 1) * cc + tid];
              const float br = re[b / 5][b % 5], bi = im[b / 5][b % 5];
              v[e] = comp == 0 ? wc * (br * ar + bi * ai)
                   : comp == 1 ? wc * (bi * ar - br * ai)
                               : wc * sqrt_approx((ar * ar + ai * ai) * (br * br + bi * bi));
            } else {
              v[e] = 0.f;
            }
          }
          s_red[warp][grp * 32 + lane] = warp_transpose_sum(v, lane);
        }
      }
      __syncthreads();
      constexpr int nrec = FULL ? 97 : kNV;
      if (tid < nrec) {
        float sum = 0.f;
#pragma unroll
        for (int w = 0; w < nwarp; ++w) sum += s_red[w][tid];
        a.rec[(((int64_t)tg * a.n_anchor + j) * a.n_chunk + chunk) * kRec + tid] = sum;
      }
      // s_red is rewritten only after the next anchor's stage barrier
    }
    if (!STATS && has_targets) {
      // every target of the pair (Eq. fcpasm), ortho scale folded into the coefficients
      const float* th = a.trans + ((int64_t)tg * a.n_anchor + j) * 2 * kNB;
      const float* gg = th + kNB;
      const float inv_hw = 1.f / (float)(g.h * g.w);
      for (int t0 = a.pair_tbeg[j]; t0 < a.pair_tbeg[j + 1]; t0 += kCoefBatch) {
        const int nt = min(kCoefBatch, a.pair_tbeg[j + 1] - t0);
        for (int e = tid; e < nt * kNB; e += cc) {
          const int k = e / kNB, b = e % kNB;
          const float al = a.target_alpha[t0 + k];
          const float tb = __ldcg(th + b), gb = __ldcg(gg + b);
          float sa, ca, sb, cb;
          sincos_reduced(gb * al * tb, &sa, &ca);
          sincos_reduced(-gb * (1.f - al) * tb, &sb, &cb);
          const float fa_ = (1.f - al) * inv_hw, fb_ = al * inv_hw;
          s_coef[k][b] = make_float4(fa_ * ca, fa_ * sa, fb_ * cb, fb_ * sb);
        }
        __syncthreads();
        for (int k = 0; k < nt; ++k) {
          float hr[8][5], hi[8][5];
#pragma unroll
          for (int b = 0; b < kNB; ++b) {
            const int ky = b / 5, kx = b % 5;
            const float4 cf = s_coef[k][b];
            const float ar = fa[(2 * b) * cc + tid], ai = fa[(2 * b + 1) * cc + tid];
            const float br = re[ky][kx], bi = im[ky][kx];
            hr[ky][kx] = cf.x * ar - cf.y * ai + cf.z * br - cf.w * bi;
            hi[ky][kx] = cf.x * ai + cf.y * ar + cf.z * bi + cf.w * br;
          }
          T* dst = out + (int64_t)a.target_frame[t0 + k] * frame_elems +
                   ((int64_t)g.y0 * a.Wg + g.x0) * a.C + c;
          const int64_t row_step = (int64_t)a.Wg * a.C;
          const int w = FULL ? 8 : g.w, C = a.C;
          // keeps the compiler from hoisting the stores over the blend (register pressure)
          asm volatile("" ::: "memory");
          auto emit = [&](int yy, const float* row) {
            if (!active) return;
            T* d = dst + yy * row_step;
#pragma unroll
            for (int xx = 0; xx < 8; ++xx)
              if (xx < w) d[(int64_t)xx * C] = T(row[xx]);
          };
          if (FULL) dft::inv2d_emit(hr, hi, 8, 8, emit);
          else dft::inv2d_emit(hr, hi, g.h, g.w, emit);
        }
        __syncthreads();   // s_coef is rewritten by the next batch
      }
    }
    // this anchor's spectrum becomes the previous one (thread-private column)
    if (j < j1) {
#pragma unroll
      for (int b = 0; b < kNB; ++b) {
        s_fprev[(2 * b) * cc + tid] = re[b / 5][b % 5];
        s_fprev[(2 * b + 1) * cc + tid] = im[b / 5][b % 5];
      }
    }
  }
}

// K_transport: grid (n_tiles_of_kind, n_anchor - 1, z), 128 threads; block y = pair j - 1.  With
// blend matrices (bf16) block z builds the matrix of the pair's target z (z < the largest target
// count of a pair; every block of a (tile, pair) solves the same transport), else z = 0 only.
template <bool FULL>
__global__ void __launch_bounds__(128) k_par_transport(const __grid_constant__ ParKArgs a) {
  __shared__ float s_zw[kNV];
  __shared__ float s_th[kNB], s_g[kNB], s_own_th[kNB];
  __shared__ int s_own_rel[kNB];
  __shared__ BinInfo s_bins;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int tile = blockIdx.x, j = blockIdx.y + 1, tg = a.tile_base + tile;
  const int t = a.pair_tbeg[j] + (int)blockIdx.z;   // this block's target
  if (!(a.pair_tbeg[j + 1] > t)) {   // no (further) target: no record
    launch_dependents();
    return;
  }
  const TileGeom g = tile_geom(a, tile, FULL);
  bin_info(a, g, s_bins, tid);
  grid_dependency_wait();   // the records come from the preceding K_stats
  if (tid < kNV) {
    int k = tid, sign = 1;
    if (FULL) {
      const int src = a.fast_src[tid];
      k = (src > 0 ? src : -src) - 1;
      sign = src < 0 ? -1 : 1;
    }
    float sum = 0.f;
    if (k >= 0) {
      // chunk order; twelve loads in flight per round
      const float* r = a.rec + ((int64_t)tg * a.n_anchor + j) * a.n_chunk * kRec + k;
      for (int ch0 = 0; ch0 < a.n_chunk; ch0 += 12) {
        float v[12];
#pragma unroll
        for (int u = 0; u < 12; ++u) v[u] = ch0 + u < a.n_chunk ? __ldcg(r + (int64_t)(ch0 + u) * kRec) : 0.f;
#pragma unroll
        for (int u = 0; u < 12; ++u) sum += v[u];
      }
    }
    s_zw[tid] = sign < 0 ? -sum : sum;
  }
  __syncthreads();
  if (warp == 0) tile_transport(a, g, s_bins, s_zw, s_th, s_g, s_own_th, s_own_rel, lane);
  __syncthreads();
  if (tid < kNB && blockIdx.z == 0) {
    float* tr = a.trans + ((int64_t)tg * a.n_anchor + j) * 2 * kNB;
    tr[tid] = s_th[tid];
    tr[kNB + tid] = s_g[tid];
  }
  if (a.img) build_blend_images<FULL>(a, g, s_bins, s_th, s_g, tg, t, t + 1, tid);
  // the blend is released only now: a tensor-core blend CTA takes a whole SM's shared memory,
  // and released early it would leave room for too few of this grid's blocks
  launch_dependents();
}

// ------------------------------------------------------------------ K_blend_tc (bf16)
// Persistent, one CTA per SM over the (tile, 128-channel chunk) items of one tile kind, 224
// threads: warp 0 streams the anchors of each item ([8 x 8 tokens][channels] through a
// 128-byte-swizzled TMA box, the MN-major UMMA operand) through four stages (an item's first
// anchors load while the previous item's last pairs run); warp 6 streams
// the blend matrices K_transport wrote, two targets of one pair stacked per group (rows 0-63
// target 1, 64-127 target 2 of the M = 128 operand), two groups in flight;
// warp 1 issues one UMMA chain per group (2 pieces x 8 K-steps, M = 128, N = 128) into one of
// two TMEM buffers; warps 2-5 (one TMEM lane quadrant each: a target slot and 32 output tokens)
// convert the result to bf16 into a swizzled staging tile that one thread stores with TMA.
constexpr int kTbNC = 128;                      // channels per item
constexpr int kTbStages = 4;                    // 225 KB of shared memory in all
constexpr int kTbPlane = 64 * kTbNC * 2;        // one anchor tile, 16 KB
constexpr int kTbPiece = 128 * 128 * 2;         // one bf16 piece of a group's [128][128] operand, 32 KB
constexpr int kTbGroup = 2 * kTbPiece;          // both pieces, 64 KB
constexpr int kTbOut = 2 * kTbPlane;            // two targets' output tiles, 32 KB
constexpr int kTbThreads = 224;
constexpr int kTbSmem = kTbStages * kTbPlane + 2 * kTbGroup + kTbOut + 1024;

template <bool FULL>
__global__ void __launch_bounds__(kTbThreads, 1)
    k_par_blend_tc(const __grid_constant__ CUtensorMap tm, const __grid_constant__ CUtensorMap tm_out,
                   const __grid_constant__ ParKArgs a, int n_tiles) {
  extern __shared__ uint8_t dsm_raw[];
  const uint32_t raw_addr = smem_u32(dsm_raw);
  uint8_t* dsm = dsm_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);   // 128-byte swizzle atoms
  uint8_t* s_stage = dsm;
  uint8_t* s_img = dsm + kTbStages * kTbPlane;
  uint8_t* s_out = s_img + 2 * kTbGroup;
  __shared__ __align__(8) uint64_t b_full[kTbStages], b_empty[kTbStages], b_ifull[2], b_iempty[2],
      b_tfull[2], b_tempty[2];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n_anc = a.n_anchor;
  const int nck = (a.C + kTbNC - 1) / kTbNC;   // 128-channel chunks per tile
  const int n_items = nck * n_tiles;           // item = tile * nck + chunk, CTAs stride the items
  const uint64_t lim = a.wait_ns;
  auto wait = [&](uint64_t* bar, uint32_t parity) -> bool {
    if (s_abort) return false;
    if (mbar_wait(bar, parity, lim)) return true;
    s_abort = 1;
    atomicExch(&g_par_error, 1u);
    return false;
  };
  if (tid == 0) {
    for (int s = 0; s < kTbStages; ++s) {
      mbar_init(&b_full[s], 1);
      mbar_init(&b_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&b_ifull[b], 1);
      mbar_init(&b_iempty[b], 1);
      mbar_init(&b_tfull[b], 1);
      mbar_init(&b_tempty[b], 4);
    }
    fence_barrier_init();
    s_abort = 0;
  }
  if (warp == 1) {
    tmem_alloc(&s_tmem, 2 * kTbNC);
    tmem_relinquish();
  }
  launch_dependents();
  // the blend images come from the preceding K_transport (and the anchors from kernels before)
  grid_dependency_wait();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  constexpr uint32_t kAnchorBytes = (uint32_t)kTbPlane;

  if (warp == 0) {
    // ---------------------------------------------------------------- anchor producer
    // anchor load L (counted over the CTA's items) goes into stage L % kTbStages once anchor
    // L - kTbStages has been released by the UMMA issuer
    if (lane == 0) {
      tma_prefetch_desc(&tm);
      int L = 0;
      for (int item = blockIdx.x; item < n_items && !s_abort; item += gridDim.x) {
        const int tile = item / nck, c0 = (item - tile * nck) * kTbNC;
        const TileGeom g = tile_geom(a, tile, FULL);
        for (int i = 0; i < n_anc; ++i, ++L) {
          const int s = L % kTbStages;
          if (L >= kTbStages && !wait(&b_empty[s], (uint32_t)((L / kTbStages) - 1) & 1u)) break;
          mbar_arrive_expect_tx(&b_full[s], kAnchorBytes);
          tma_load_4d(s_stage + s * kTbPlane, &tm, &b_full[s], c0, g.x0, g.y0, a.anchor_frame[i]);
          tma_load_4d(s_stage + s * kTbPlane + 8192, &tm, &b_full[s], c0 + 64, g.x0, g.y0, a.anchor_frame[i]);
        }
      }
      if (s_abort)   // the copies still in flight land before the shared memory is released
        for (int l = L > kTbStages ? L - kTbStages : 0; l < L; ++l)
          mbar_wait(&b_full[l % kTbStages], (uint32_t)(l / kTbStages) & 1u, lim);
    }
  } else if (warp == 6) {
    // ---------------------------------------------------------------- image producer
    if (lane == 0) {
      int n = 0;
      for (int item = blockIdx.x; item < n_items && !s_abort; item += gridDim.x) {
        const int tg = a.tile_base + item / nck;
        for (int j = 1; j < n_anc && !s_abort; ++j)
          for (int t0 = a.pair_tbeg[j]; t0 < a.pair_tbeg[j + 1]; t0 += 2, ++n) {
            const int ib = n & 1, nt = min(2, a.pair_tbeg[j + 1] - t0);
            if (n >= 2 && !wait(&b_iempty[ib], (uint32_t)((n >> 1) - 1) & 1u)) break;
            mbar_arrive_expect_tx(&b_ifull[ib], (uint32_t)(nt * kImgBytes));
            uint8_t* dst = s_img + ib * kTbGroup;
            for (int ts = 0; ts < nt; ++ts) {
              const char* src = a.img + ((int64_t)tg * a.n_target + t0 + ts) * kImgBytes;
              // piece p, K-block kb of the target -> rows 64 ts .. 64 ts + 63 of the stacked operand
              for (int p = 0; p < 2; ++p)
                for (int kb = 0; kb < 2; ++kb)
                  bulk_load(dst + p * kTbPiece + kb * 16384 + ts * 8192, src + p * kImgTerm + kb * 8192, 8192u,
                            &b_ifull[ib]);
            }
          }
      }
      if (s_abort)   // let the images in flight land (at most the last two groups)
        for (int l = n > 2 ? n - 2 : 0; l < n; ++l) mbar_wait(&b_ifull[l & 1], (uint32_t)(l >> 1) & 1u, lim);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- UMMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, kTbNC, false, true);
      int n = 0, L = 0;
      bool ok = true;
      for (int item = blockIdx.x; ok && item < n_items; item += gridDim.x, L += n_anc) {
        if (!wait(&b_full[L % kTbStages], (uint32_t)(L / kTbStages) & 1u)) break;
        for (int j = 1; ok && j < n_anc; ++j) {
          const int La = L + j - 1, Lb = L + j;
          if (!wait(&b_full[Lb % kTbStages], (uint32_t)(Lb / kTbStages) & 1u)) { ok = false; break; }
          const uint32_t xa = smem_u32(s_stage + (La % kTbStages) * kTbPlane);
          const uint32_t xb = smem_u32(s_stage + (Lb % kTbStages) * kTbPlane);
          for (int t0 = a.pair_tbeg[j]; t0 < a.pair_tbeg[j + 1]; t0 += 2, ++n) {
            const int ib = n & 1;
            if (!wait(&b_ifull[ib], (uint32_t)(n >> 1) & 1u) ||
                (n >= 2 && !wait(&b_tempty[ib], (uint32_t)((n >> 1) - 1) & 1u))) { ok = false; break; }
            tc_fence_after();
            const uint32_t im = smem_u32(s_img + ib * kTbGroup), d = tmem + (uint32_t)(ib * kTbNC);
#pragma unroll
            for (int p = 0; p < 2; ++p)
#pragma unroll
              for (int kk = 0; kk < 8; ++kk)
                umma_bf16_ss(d, sdesc_sw128(im + p * kTbPiece + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024),
                             sdesc_sw128((kk < 4 ? xa : xb) + (kk & 3) * 2048, 8192, 1024), idesc,
                             (p | kk) ? 1u : 0u);
            umma_commit(&b_iempty[ib]);
            umma_commit(&b_tfull[ib]);
          }
          if (ok) umma_commit(&b_empty[La % kTbStages]);   // the pair's UMMAs were anchor La's last readers
        }
        if (ok) umma_commit(&b_empty[(L + n_anc - 1) % kTbStages]);   // the item's last anchor
      }
      if (s_abort && n > 0) mbar_wait(&b_tfull[(n - 1) & 1], (uint32_t)((n - 1) >> 1) & 1u, lim);
    }
  } else if (warp >= 2 && warp <= 5) {
    // ---------------------------------------------------------------- epilogue warps 2-5
    // (warp 6 has no role: it goes straight to the final barrier)
    const int ctid = tid - 64;                 // 0..127
    const int q = warp & 3;                    // TMEM lanes 32 q .. 32 q + 31
    const int ts = q >> 1;                     // target slot of this warp
    const int o = 32 * (q & 1) + lane;         // output token 8 y + x
    const int yo = o >> 3, xo = o & 7;
    const bool valid = yo < a.th && xo < a.tw;
    const int sr = yo * a.tw + xo;             // row inside the store box
    uint8_t* out = s_out + ts * kTbPlane;
    bool fail = false;
    int n = 0;
    for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
      const int tile = item / nck, c0 = (item - tile * nck) * kTbNC;
      const TileGeom g = tile_geom(a, tile, FULL);
      for (int j = 1; j < n_anc; ++j)
        for (int t0 = a.pair_tbeg[j]; t0 < a.pair_tbeg[j + 1]; t0 += 2, ++n) {
          const int ib = n & 1, nt = min(2, a.pair_tbeg[j + 1] - t0);
          if (!fail && !wait(&b_tfull[ib], (uint32_t)(n >> 1) & 1u)) fail = true;
          // the previous group's TMA stores have read the staging tiles
          if (ctid == 0) bulk_wait_read_all();
          if (bar_sync_or(1, 128, fail)) {
            fail = true;
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&b_tempty[ib]);
            continue;
          }
          tc_fence_after();
          const uint32_t ta = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(ib * kTbNC);
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            // 64 channels (one 128-byte box) at a time
            uint32_t r[64];
            tmem_ld_x64(ta + 64 * half, r);
            if (half == 1) {   // the whole buffer is in registers: it goes back to the issuer
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&b_tempty[ib]);
            }
            if (ts < nt && valid) {
#pragma unroll
              for (int c8 = 0; c8 < 8; ++c8) {
                uint32_t pk[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                  const __nv_bfloat162 b2 = __floats2bfloat162_rn(__uint_as_float(r[8 * c8 + 2 * u]),
                                                                  __uint_as_float(r[8 * c8 + 2 * u + 1]));
                  pk[u] = *reinterpret_cast<const uint32_t*>(&b2);
                }
                *reinterpret_cast<uint4*>(out + half * 8192 + sr * 128 + ((c8 ^ (sr & 7)) << 4)) =
                    make_uint4(pk[0], pk[1], pk[2], pk[3]);
              }
            }
          }
          fence_proxy_async_smem();
          bar_sync_or(1, 128, false);
          if (ctid == 0) {
            for (int u = 0; u < nt; ++u)
              for (int b = 0; b < 2; ++b)
                if (c0 + 64 * b < a.C)
                  tma_store_4d(&tm_out, s_out + u * kTbPlane + b * 8192, c0 + 64 * b, g.x0, g.y0,
                               a.target_frame[t0 + u]);
            bulk_commit();
          }
        }
    }
    if (ctid == 0) bulk_wait_all();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 2 * kTbNC);
}

// 4-D map [F][Hg][Wg][C] with a 128-byte-swizzled box (64 bf16 channels, bw, bh, 1)
bool make_r_map_sw(CUtensorMap* m, const cast_par_args& a, int bw, int bh) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[4] = {(cuuint64_t)a.C, (cuuint64_t)a.Wg, (cuuint64_t)a.Hg, (cuuint64_t)a.F};
  cuuint64_t strides[3] = {a.C * 2ull, (cuuint64_t)a.Wg * a.C * 2, (cuuint64_t)a.Hg * a.Wg * a.C * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)bw, (cuuint32_t)bh, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, a.r, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 4-D map [F][Hg][Wg][C], box (cc channels, tw, th, 1), zero fill out of range
bool make_r_map(CUtensorMap* m, const cast_par_args& a, int cc) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (!fn) return false;
  const cuuint64_t elt = a.dtype == CAST_BF16 ? 2 : 4;
  cuuint64_t dims[4] = {(cuuint64_t)a.C, (cuuint64_t)a.Wg, (cuuint64_t)a.Hg, (cuuint64_t)a.F};
  cuuint64_t strides[3] = {a.C * elt, (cuuint64_t)a.Wg * a.C * elt, (cuuint64_t)a.Hg * a.Wg * a.C * elt};
  cuuint32_t box[4] = {(cuuint32_t)cc, (cuuint32_t)a.params.tile_w, (cuuint32_t)a.params.tile_h, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, a.dtype == CAST_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
            4, a.r, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// One tile kind on one stream: K_stats, then K_transport and K_blend as programmatic dependents.
template <typename T, bool FULL>
cast_status launch_kind(const CUtensorMap& tm, const CUtensorMap* tm_sw, const CUtensorMap* tm_out,
                        const ParKArgs& k, int n_tiles, cudaStream_t st) {
  const size_t smem = par_dyn_smem<T>(kCC);
  static std::atomic<uint64_t> attr_done{0};
  if (!once_per_device(attr_done, [smem] {
        return cudaFuncSetAttribute(k_par<T, kCC, FULL, true>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) == cudaSuccess &&
               cudaFuncSetAttribute(k_par<T, kCC, FULL, false>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) == cudaSuccess &&
               cudaFuncSetAttribute(k_par_blend_tc<FULL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    kTbSmem) == cudaSuccess;
      }))
    return check_launch("PAR kernel attributes");
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(k.n_chunk, n_tiles * k.n_tseg, 1);
  cfg.blockDim = dim3(kCC, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  if (cudaLaunchKernelEx(&cfg, k_par<T, kCC, FULL, true>, tm, k) != cudaSuccess)
    return check_launch("PAR statistics kernel");
  int zmax = 1;   // one transport block per (tile, pair, target) when it writes blend matrices
  if (k.img)
    for (int j = 1; j < k.n_anchor; ++j) zmax = std::max(zmax, k.pair_tbeg[j + 1] - k.pair_tbeg[j]);
  cudaLaunchConfig_t tc{};
  tc.gridDim = dim3(n_tiles, k.n_anchor - 1, zmax);
  tc.blockDim = dim3(128, 1, 1);
  tc.stream = st;
  tc.attrs = pdl;
  tc.numAttrs = 1;
  if (cudaLaunchKernelEx(&tc, k_par_transport<FULL>, k) != cudaSuccess)
    return check_launch("PAR transport kernel");
  cfg.attrs = pdl;
  cfg.numAttrs = 1;
  if (k.img) {
    // bf16: the blend as tensor-core GEMMs over the matrices K_transport wrote
    // persistent: one CTA per SM over the (tile, 128-channel chunk) items of this kind
    int dev = 0, nsm = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    const int items = ((k.C + kTbNC - 1) / kTbNC) * n_tiles;
    cudaLaunchConfig_t bc{};
    bc.gridDim = dim3(items < nsm ? items : nsm, 1, 1);
    bc.blockDim = dim3(kTbThreads, 1, 1);
    bc.dynamicSmemBytes = kTbSmem;
    bc.stream = st;
    bc.attrs = pdl;
    bc.numAttrs = 1;
    if (cudaLaunchKernelEx(&bc, k_par_blend_tc<FULL>, *tm_sw, *tm_out, k, n_tiles) != cudaSuccess)
      return check_launch("PAR tensor-core blend kernel");
  } else if (cudaLaunchKernelEx(&cfg, k_par<T, kCC, FULL, false>, tm, k) != cudaSuccess) {
    return check_launch("PAR blend kernel");
  }
  return check_launch("PAR kernels");
}

// A second stream per device (and the events that fork it from and join it back into the
// caller's stream) for the edge-tile launch, created on first use.
struct ForkStream {
  cudaStream_t side = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
};
cast_status fork_stream(ForkStream*& out) {
  static std::mutex mu;
  static ForkStream per_dev[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return check_launch("PAR device");
  std::lock_guard<std::mutex> lock(mu);
  ForkStream& f = per_dev[dev];
  if (!f.side) {
    if (cudaStreamCreateWithFlags(&f.side, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&f.fork, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&f.join, cudaEventDisableTiming) != cudaSuccess)
      return check_launch("PAR side stream");
  }
  out = &f;
  return CAST_OK;
}

// Time segments of consecutive anchor pairs (pairs 1 .. n_anchor-1), as even as possible.
ParKArgs with_segments(const ParKArgs& k0, int nseg) {
  ParKArgs k = k0;
  const int npair = k.n_anchor - 1;
  k.n_tseg = nseg;
  int pair = 1;
  for (int sg = 0; sg < nseg; ++sg) {
    const int left = npair - (pair - 1), segs_left = nseg - sg;
    const int take = (left + segs_left - 1) / segs_left;
    k.seg_pair0[sg] = pair;
    k.seg_pair1[sg] = pair + take - 1;
    pair += take;
  }
  return k;
}

template <typename T>
cast_status launch_typed(const CUtensorMap& tm, const CUtensorMap* tm_sw, const CUtensorMap* tm_out,
                         const ParKArgs& k0, const ParPlan& p, cudaStream_t st) {
  ParKArgs kf = with_segments(k0, p.n_tseg_full), ke = with_segments(k0, p.n_tseg_edge);
  kf.tile_base = 0;
  ke.tile_base = p.n_full;
  if (p.n_edge == 0) return launch_kind<T, true>(tm, tm_sw, tm_out, kf, p.n_full, st);
  if (p.n_full == 0) return launch_kind<T, false>(tm, tm_sw, tm_out, ke, p.n_edge, st);
  // full tiles on the caller's stream, edge tiles concurrently on the side stream
  ForkStream* f = nullptr;
  cast_status s = fork_stream(f);
  if (s != CAST_OK) return s;
  if (cudaEventRecord(f->fork, st) != cudaSuccess || cudaStreamWaitEvent(f->side, f->fork, 0) != cudaSuccess)
    return check_launch("PAR fork");
  s = launch_kind<T, false>(tm, tm_sw, tm_out, ke, p.n_edge, f->side);
  if (s != CAST_OK) return s;
  s = launch_kind<T, true>(tm, tm_sw, tm_out, kf, p.n_full, st);
  if (cudaEventRecord(f->join, f->side) != cudaSuccess || cudaStreamWaitEvent(st, f->join, 0) != cudaSuccess)
    return check_launch("PAR join");
  return s;
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
  // 8x8 tiles take the specialised kernel; with smaller tile sides every tile is an edge tile
  if (th == 8 && tw == 8) {
    p.n_full = (a.Hg / 8) * (a.Wg / 8);
    p.n_edge = p.n_tile - p.n_full;
  } else {
    p.n_full = 0;
    p.n_edge = p.n_tile;
  }
  // channel chunks of kCC channels, one CTA each
  p.chunk = kCC;
  p.n_chunk = (a.C + kCC - 1) / kCC;
  // time segments: split the anchor pairs so that the CTAs of a kind cover the SMs about
  // two deep for full tiles and four deep for the (fewer, longer-running) edge tiles, which
  // run concurrently on the side stream; each segment re-reads its first anchor.  Measured at
  // the Matrix-Game size (3 pairs: full tiles 2 segments, 0.049 ms against 0.053 ms with 3)
  // and the PAR sweep (edge tiles 3 segments, 2 % faster than 2).
  int dev = 0, nsm = 148;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  if (nsm <= 0) nsm = 148;
  auto segs = [&](int n_tiles, int depth) {
    const int want_ctas = depth * nsm;
    const int per_seg = n_tiles * p.n_chunk;
    int nseg = per_seg > 0 ? (want_ctas + per_seg - 1) / per_seg : 1;
    if (nseg > p.n_pair) nseg = p.n_pair;
    return nseg < 1 ? 1 : nseg;
  };
  p.n_tseg_full = segs(p.n_full, 2);
  p.n_tseg_edge = segs(p.n_edge, 4);
  // workspace: the chunk records [tile][pair][chunk][kRec] and theta, g [tile][pair][2][kNB]
  p.rec_bytes = align_up((size_t)p.n_tile * (na > 0 ? na : 1) * p.n_chunk * kRec * sizeof(float));
  p.trans_bytes = align_up((size_t)p.n_tile * (na > 0 ? na : 1) * 2 * kNB * sizeof(float));
  // bf16: the blend matrices of every (tile, target)
  p.img_bytes = a.dtype == CAST_BF16 ? align_up((size_t)p.n_tile * (p.n_target > 0 ? p.n_target : 1) * kImgBytes) : 0;
  p.total_bytes = p.n_target > 0 ? p.rec_bytes + p.trans_bytes + p.img_bytes : 0;
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
  k.tiles_y = p.tiles_y;
  k.n_tile = p.n_tile;
  k.n_chunk = p.n_chunk;
  k.rec = static_cast<float*>(ws);
  k.trans = reinterpret_cast<float*>(static_cast<char*>(ws) + p.rec_bytes);
  k.img = p.img_bytes ? static_cast<char*>(ws) + p.rec_bytes + p.trans_bytes : nullptr;
  k.n_target = p.n_target;
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
  if (!make_r_map(&tm, a, p.chunk)) return fail(CAST_ERR_CUDA, "PAR: cuTensorMapEncodeTiled failed");
  if (a.dtype == CAST_BF16) {
    CUtensorMap tm_sw, tm_out;
    if (!make_r_map_sw(&tm_sw, a, 8, 8) || !make_r_map_sw(&tm_out, a, k.tw, k.th))
      return fail(CAST_ERR_CUDA, "PAR: cuTensorMapEncodeTiled failed");
    return launch_typed<__nv_bfloat16>(tm, &tm_sw, &tm_out, k, p, st);
  }
  return launch_typed<float>(tm, nullptr, nullptr, k, p, st);
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
