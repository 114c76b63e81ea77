// Routing of historical KV blocks (Section 4.4, Eqs. pooled, omission, topk).
//
//   K_pool     : column sums of every pooled segment (anchor query frames, history key
//                blocks, history value blocks), split over rows; HBM-bound streaming of
//                (K_f S + 2 M B_v) H d elements with 16-byte loads.
//   K_finalize : sums the row splits in a fixed order and divides by the row count
//                (deterministic means q_bar, k_bar, v_bar in f32).
//   K_score    : one CTA per (anchor, head): s, pi, o_bar, delta, u (Eq. omission, with an
//                optional Gram matrix G = P^T P of the output projection) and a warp-level
//                TopK with ties to the lower block index, written in ascending order.
//   K_refine   : optional, one CTA per head: the reconstruction-coupled fixed-budget best
//                responses of Alg. (routing) (App. B.3) starting from the TopK masks.
#include <cuda_bf16.h>

#include <cfloat>
#include <cmath>

#include "internal.h"

namespace cast {
namespace {

constexpr int kPoolThreads = 256;

struct PoolArgs {
  const char* q;          // anchor frame base = q + anchors[i] * S * q_row_stride * elt
  const char* k;
  const char* v;
  int64_t q_row_stride, hist_row_stride;   // elements
  int n_anchors, M, S, B_v, D, nsplit, elt;
  int anchors[CAST_MAX_ANCHORS];
};

template <typename T>
__device__ __forceinline__ void load_vec(const char* p, float (&x)[16 / sizeof(T)]);

template <>
__device__ __forceinline__ void load_vec<float>(const char* p, float (&x)[4]) {
  float4 v = __ldcs(reinterpret_cast<const float4*>(p));
  x[0] = v.x; x[1] = v.y; x[2] = v.z; x[3] = v.w;
}
template <>
__device__ __forceinline__ void load_vec<__nv_bfloat16>(const char* p, float (&x)[8]) {
  uint4 v = __ldcs(reinterpret_cast<const uint4*>(p));
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    x[2 * k] = __uint_as_float(w[k] << 16);
    x[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
  }
}

// grid (nsplit, n_seg); partial[(seg * nsplit + split) * D + col]
template <typename T>
__global__ void __launch_bounds__(kPoolThreads) k_pool(PoolArgs a, float* __restrict__ partial) {
  constexpr int VEC = 16 / sizeof(T);
  const int seg = blockIdx.y, split = blockIdx.x;
  const char* base;
  int64_t rs;
  int nrows;
  if (seg < a.n_anchors) {
    base = a.q + (int64_t)a.anchors[seg] * a.S * a.q_row_stride * a.elt;
    rs = a.q_row_stride;
    nrows = a.S;
  } else if (seg < a.n_anchors + a.M) {
    base = a.k + (int64_t)(seg - a.n_anchors) * a.B_v * a.hist_row_stride * a.elt;
    rs = a.hist_row_stride;
    nrows = a.B_v;
  } else {
    base = a.v + (int64_t)(seg - a.n_anchors - a.M) * a.B_v * a.hist_row_stride * a.elt;
    rs = a.hist_row_stride;
    nrows = a.B_v;
  }
  const int per = (nrows + a.nsplit - 1) / a.nsplit;
  const int r0 = split * per, r1 = min(nrows, r0 + per);
  const int ncg = a.D / VEC;                          // 16-byte column groups
  const int lanes_r = ncg >= kPoolThreads ? 1 : kPoolThreads / ncg;   // row lanes
  const int tcg = threadIdx.x % (ncg >= kPoolThreads ? kPoolThreads : ncg);
  const int trl = threadIdx.x / (ncg >= kPoolThreads ? kPoolThreads : ncg);
  __shared__ float red[kPoolThreads * 8];
  float* out = partial + ((int64_t)seg * a.nsplit + split) * a.D;
  for (int cg = tcg; cg < ncg; cg += (ncg >= kPoolThreads ? kPoolThreads : ncg)) {
    float acc[VEC];
#pragma unroll
    for (int k = 0; k < VEC; ++k) acc[k] = 0.f;
    if (trl < lanes_r) {
      const char* p = base + ((int64_t)(r0 + trl) * rs + (int64_t)cg * VEC) * a.elt;
      const int64_t step = (int64_t)lanes_r * rs * a.elt;
      int r = r0 + trl;
      for (; r + 3 * lanes_r < r1; r += 4 * lanes_r) {
        float x0[VEC], x1[VEC], x2[VEC], x3[VEC];
        load_vec<T>(p, x0);
        load_vec<T>(p + step, x1);
        load_vec<T>(p + 2 * step, x2);
        load_vec<T>(p + 3 * step, x3);
        p += 4 * step;
#pragma unroll
        for (int k = 0; k < VEC; ++k) acc[k] += (x0[k] + x1[k]) + (x2[k] + x3[k]);
      }
      for (; r < r1; r += lanes_r) {
        float x0[VEC];
        load_vec<T>(p, x0);
        p += step;
#pragma unroll
        for (int k = 0; k < VEC; ++k) acc[k] += x0[k];
      }
    }
    if (lanes_r == 1) {
#pragma unroll
      for (int k = 0; k < VEC; ++k) out[cg * VEC + k] = acc[k];
    } else {
      // reduce the row lanes of this column group through shared memory (fixed order)
      __syncthreads();
      if (trl < lanes_r) {
#pragma unroll
        for (int k = 0; k < VEC; ++k) red[(trl * ncg + cg) * VEC + k] = acc[k];
      }
      __syncthreads();
      if (trl == 0) {
        for (int l = 1; l < lanes_r; ++l)
#pragma unroll
          for (int k = 0; k < VEC; ++k) acc[k] += red[(l * ncg + cg) * VEC + k];
#pragma unroll
        for (int k = 0; k < VEC; ++k) out[cg * VEC + k] = acc[k];
      }
    }
  }
}

// pooled[seg * D + col] = (sum over splits in order) / rows(seg)
__global__ void k_finalize(const float* __restrict__ partial, float* __restrict__ qbar,
                           float* __restrict__ kbar, float* __restrict__ vbar, int n_anchors,
                           int M, int S, int B_v, int D, int nsplit) {
  const int seg = blockIdx.y;
  const int col = blockIdx.x * blockDim.x + threadIdx.x;
  if (col >= D) return;
  float s = 0.f;
  for (int k = 0; k < nsplit; ++k) s += partial[((int64_t)seg * nsplit + k) * D + col];
  if (seg < n_anchors) {
    qbar[(int64_t)seg * D + col] = s / (float)S;
  } else if (seg < n_anchors + M) {
    kbar[(int64_t)(seg - n_anchors) * D + col] = s / (float)B_v;
  } else {
    vbar[(int64_t)(seg - n_anchors - M) * D + col] = s / (float)B_v;
  }
}

constexpr int kScoreThreads = 256;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// grid (H, n_anchors).  Dynamic smem: s[M], pi[M], key[M], sel[M] (int), obar[d], qb[d],
// e[8 warps][d] scratch.
__global__ void __launch_bounds__(kScoreThreads)
    k_score_topk(const float* __restrict__ qbar, const float* __restrict__ kbar,
                 const float* __restrict__ vbar, const float* __restrict__ gram, int H, int d,
                 int M, int K_eff, float eps, int mode, int32_t* __restrict__ idx,
                 float* __restrict__ u_out) {
  extern __shared__ float sm[];
  const int h = blockIdx.x, i = blockIdx.y;
  const int D = H * d;
  float* s = sm;
  float* pi = s + M;
  float* key = pi + M;
  int* sel = reinterpret_cast<int*>(key + M);
  float* ob = reinterpret_cast<float*>(sel + M);
  float* qb = ob + d;
  float* ew = qb + d;   // [kScoreThreads/32][d]
  __shared__ float red[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = kScoreThreads / 32;
  const float scale = rsqrtf((float)d);

  for (int c = tid; c < d; c += kScoreThreads) qb[c] = qbar[(int64_t)i * D + h * d + c];
  for (int m = tid; m < M; m += kScoreThreads) sel[m] = 0;
  __syncthreads();
  // s_m = q_bar . k_bar_m / sqrt(d)   (Eq. pooled)
  for (int m = warp; m < M; m += nwarp) {
    const float* kb = kbar + (int64_t)m * D + h * d;
    float acc = 0.f;
    for (int c = lane; c < d; c += 32) acc = fmaf(qb[c], kb[c], acc);
    acc = warp_sum(acc);
    if (lane == 0) s[m] = acc * scale;
  }
  __syncthreads();
  // softmax over blocks
  float mx = -FLT_MAX;
  for (int m = tid; m < M; m += kScoreThreads) mx = fmaxf(mx, s[m]);
  mx = warp_max(mx);
  if (lane == 0) red[warp] = mx;
  __syncthreads();
  if (warp == 0) {
    float v = lane < nwarp ? red[lane] : -FLT_MAX;
    v = warp_max(v);
    if (lane == 0) red[16] = v;
  }
  __syncthreads();
  mx = red[16];
  float tot = 0.f;
  for (int m = tid; m < M; m += kScoreThreads) {
    const float e = expf(s[m] - mx);
    pi[m] = e;
    tot += e;
  }
  tot = warp_sum(tot);
  __syncthreads();
  if (lane == 0) red[warp] = tot;
  __syncthreads();
  if (warp == 0) {
    float v = lane < nwarp ? red[lane] : 0.f;
    v = warp_sum(v);
    if (lane == 0) red[17] = v;
  }
  __syncthreads();
  const float inv = 1.f / red[17];
  for (int m = tid; m < M; m += kScoreThreads) pi[m] *= inv;
  __syncthreads();
  // o_bar = sum_m pi_m v_bar_m
  for (int c = tid; c < d; c += kScoreThreads) {
    float acc = 0.f;
    for (int m = 0; m < M; ++m) acc = fmaf(pi[m], vbar[(int64_t)m * D + h * d + c], acc);
    ob[c] = acc;
  }
  __syncthreads();
  // delta_m = pi_m / (1 - pi_m + eps) (o_bar - v_bar_m);  u_m = delta^T G delta (Eq. omission)
  float* e = ew + warp * d;
  for (int m = warp; m < M; m += nwarp) {
    const float* vb = vbar + (int64_t)m * D + h * d;
    const float coef = pi[m] / (1.f - pi[m] + eps);
    float acc = 0.f;
    if (gram == nullptr) {
      for (int c = lane; c < d; c += 32) {
        const float x = ob[c] - vb[c];
        acc = fmaf(x, x, acc);
      }
    } else {
      for (int c = lane; c < d; c += 32) e[c] = ob[c] - vb[c];
      __syncwarp();
      const float* G = gram + (int64_t)h * d * d;
      for (int r = lane; r < d; r += 32) {
        float y = 0.f;
        for (int c = 0; c < d; ++c) y = fmaf(G[(int64_t)r * d + c], e[c], y);
        acc = fmaf(e[r], y, acc);
      }
      __syncwarp();
    }
    acc = warp_sum(acc);
    if (lane == 0) {
      const float u = coef * coef * acc;
      key[m] = (mode == CAST_ROUTE_SIMILARITY) ? s[m] : u;
      if (u_out) u_out[((int64_t)i * H + h) * M + m] = (mode == CAST_ROUTE_SIMILARITY) ? s[m] : u;
    }
  }
  __syncthreads();
  // TopK by repeated warp argmax (ties -> lower index), then ascending compaction
  if (warp == 0) {
    for (int k = 0; k < K_eff; ++k) {
      float best = -INFINITY;
      int bi = 0x7fffffff;   // none yet
      for (int m = lane; m < M; m += 32) {   // ascending m: strict > keeps the lower index
        if (sel[m]) continue;
        const float v = key[m];
        if (bi == 0x7fffffff || v > best) { best = v; bi = m; }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, best, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (oi != 0x7fffffff && (bi == 0x7fffffff || ov > best || (ov == best && oi < bi))) {
          best = ov;
          bi = oi;
        }
      }
      if (lane == 0 && bi != 0x7fffffff) sel[bi] = 1;
      __syncwarp();
    }
    int base = 0;
    int32_t* out = idx + ((int64_t)i * H + h) * K_eff;
    for (int m0 = 0; m0 < M; m0 += 32) {
      const int m = m0 + lane;
      const bool on = m < M && sel[m];
      const unsigned bal = __ballot_sync(0xffffffffu, on);
      if (on) out[base + __popc(bal & ((1u << lane) - 1u))] = m;
      base += __popc(bal);
    }
  }
}

// ---------------------------------------------------------------------- refinement
struct RefineArgs {
  int n_anchors, M, K_eff, H, passes;
  float lam_anc, lam_rec, tol;
  float A[CAST_MAX_ANCHORS], B[CAST_MAX_ANCHORS], C[CAST_MAX_ANCHORS];   // interval (j-1, j)
  float AL, BL, CL, AR, BR, CR;                                          // boundary sets
};

constexpr int kRefineThreads = 256;

// Warp 0: mask[m] = 1 for the K largest key[m] (ties to the lower index), 0 elsewhere.
__device__ void warp_topk_mask(const float* key, float* mask, int M, int K, int lane) {
  for (int m = lane; m < M; m += 32) mask[m] = 0.f;
  __syncwarp();
  for (int k = 0; k < K; ++k) {
    float best = -INFINITY;
    int bi = 0x7fffffff;
    for (int m = lane; m < M; m += 32) {
      if (mask[m] != 0.f) continue;
      const float v = key[m];
      if (bi == 0x7fffffff || v > best) { best = v; bi = m; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, best, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (oi != 0x7fffffff && (bi == 0x7fffffff || ov > best || (ov == best && oi < bi))) {
        best = ov;
        bi = oi;
      }
    }
    if (lane == 0 && bi != 0x7fffffff) mask[bi] = 1.f;
    __syncwarp();
  }
}

// Eq. (risk) term of one block for the anchor pair (p, q) with coefficients (A, B, C)
__device__ __forceinline__ float pair_risk(float A, float B, float C, float xp, float xq, float up,
                                           float uq) {
  return A * (1.f - xp) * up + B * (1.f - xq) * uq + 2.f * C * (1.f - xp) * (1.f - xq) * sqrtf(up * uq);
}

__device__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = 0.f;
  if (threadIdx.x < 32) {
    t = threadIdx.x < kRefineThreads / 32 ? red[threadIdx.x] : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (threadIdx.x == 0) red[31] = t;
  }
  __syncthreads();
  return red[31];
}

// Eq. (objective) of the current masks (block-wide)
__device__ float objective(const RefineArgs& r, const float* u, const float* x, float* red) {
  const int na = r.n_anchors, M = r.M;
  float v = 0.f;
  for (int m = threadIdx.x; m < M; m += kRefineThreads) {
    for (int i = 0; i < na; ++i) v += r.lam_anc * (1.f - x[i * M + m]) * u[i * M + m];
    float rec = 0.f;
    for (int j = 1; j < na; ++j)
      rec += pair_risk(r.A[j], r.B[j], r.C[j], x[(j - 1) * M + m], x[j * M + m], u[(j - 1) * M + m],
                       u[j * M + m]);
    if (na >= 2) {
      rec += pair_risk(r.AL, r.BL, r.CL, x[m], x[M + m], u[m], u[M + m]);
      rec += pair_risk(r.AR, r.BR, r.CR, x[(na - 2) * M + m], x[(na - 1) * M + m], u[(na - 2) * M + m],
                       u[(na - 1) * M + m]);
    }
    v += r.lam_rec * rec;
  }
  return block_sum(v, red);
}

// grid (H).  Dynamic smem: u [na][M], x [na][M], G [M], xn [M] (floats).
__global__ void __launch_bounds__(kRefineThreads)
    k_refine(const float* __restrict__ u_all, const __grid_constant__ RefineArgs r,
             int32_t* __restrict__ idx) {
  extern __shared__ float sm[];
  __shared__ float red[32];
  __shared__ int s_accept;
  const int h = blockIdx.x, na = r.n_anchors, M = r.M, K = r.K_eff;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float* u = sm;
  float* x = u + na * M;
  float* G = x + na * M;
  float* xn = G + M;
  for (int e = tid; e < na * M; e += kRefineThreads) {
    const int i = e / M, m = e - i * M;
    u[e] = u_all[((int64_t)i * r.H + h) * M + m];
  }
  __syncthreads();
  // initial masks: TopK of u per anchor (one warp per anchor)
  for (int i = warp; i < na; i += kRefineThreads / 32) warp_topk_mask(u + i * M, x + i * M, M, K, lane);
  __syncthreads();
  float J = objective(r, u, x, red);
  for (int pass = 1; pass <= r.passes; ++pass) {
    bool changed = false;
    for (int step = 0; step < na; ++step) {
      const int i = (pass & 1) ? step : na - 1 - step;
      // retain gains, Eqs. (gain) and (boundarygain)
      for (int m = tid; m < M; m += kRefineThreads) {
        const float ui = u[i * M + m];
        float g = r.lam_anc * ui, rec = 0.f;
        if (i >= 1) {
          const float ul = u[(i - 1) * M + m];
          rec += r.B[i] * ui + 2.f * r.C[i] * (1.f - x[(i - 1) * M + m]) * sqrtf(ul * ui);
        }
        if (i + 1 < na) {
          const float ur = u[(i + 1) * M + m];
          rec += r.A[i + 1] * ui + 2.f * r.C[i + 1] * (1.f - x[(i + 1) * M + m]) * sqrtf(ui * ur);
        }
        if (na >= 2) {
          if (i == 0) rec += r.AL * ui + 2.f * r.CL * (1.f - x[M + m]) * sqrtf(ui * u[M + m]);
          if (i == 1) rec += r.BL * ui + 2.f * r.CL * (1.f - x[m]) * sqrtf(ui * u[m]);
          if (i == na - 2) rec += r.AR * ui + 2.f * r.CR * (1.f - x[(na - 1) * M + m]) * sqrtf(ui * u[(na - 1) * M + m]);
          if (i == na - 1) rec += r.BR * ui + 2.f * r.CR * (1.f - x[(na - 2) * M + m]) * sqrtf(ui * u[(na - 2) * M + m]);
        }
        G[m] = g + r.lam_rec * rec;
      }
      __syncthreads();
      if (warp == 0) warp_topk_mask(G, xn, M, K, lane);
      __syncthreads();
      float d = 0.f;
      for (int m = tid; m < M; m += kRefineThreads) d += G[m] * (xn[m] - x[i * M + m]);
      const float gain = block_sum(d, red);
      if (tid == 0) s_accept = gain > r.tol * fmaxf(J, 1e-8f);
      __syncthreads();
      if (s_accept) {
        for (int m = tid; m < M; m += kRefineThreads) x[i * M + m] = xn[m];
        __syncthreads();
        J = objective(r, u, x, red);
        changed = true;
      }
    }
    if (!changed) break;
  }
  __syncthreads();
  // ascending block indices of every anchor's mask
  for (int i = warp; i < na; i += kRefineThreads / 32) {
    int base = 0;
    int32_t* out = idx + ((int64_t)i * r.H + h) * K;
    for (int m0 = 0; m0 < M; m0 += 32) {
      const int m = m0 + lane;
      const bool on = m < M && x[i * M + m] != 0.f;
      const unsigned bal = __ballot_sync(0xffffffffu, on);
      if (on) out[base + __popc(bal & ((1u << lane) - 1u))] = m;
      base += __popc(bal);
    }
  }
}

}  // namespace

size_t refine_smem_bytes(const cast_route_args& a) {
  return (size_t)(2 * a.n_anchors + 2) * (size_t)a.M * sizeof(float);
}

RoutePlan route_plan(const cast_route_args& a) {
  RoutePlan p{};
  const int D = a.H * a.d;
  p.n_seg = a.n_anchors + 2 * a.M;
  // enough CTAs to cover the SMs several times, each streaming >= ~128 rows
  const int64_t rows = (int64_t)a.n_anchors * a.S + 2LL * a.M * a.B_v;
  int target = 4 * 152;
  int nsplit = (int)((target + p.n_seg - 1) / p.n_seg);
  const int maxrows = a.M > 0 ? (a.S > a.B_v ? a.S : a.B_v) : a.S;
  while (nsplit > 1 && (maxrows + nsplit - 1) / nsplit < 64) --nsplit;
  if (nsplit < 1) nsplit = 1;
  (void)rows;
  p.nsplit = nsplit;
  p.partial_bytes = align_up((size_t)p.n_seg * nsplit * D * sizeof(float));
  p.pooled_bytes = align_up((size_t)p.n_seg * D * sizeof(float));
  p.u_bytes = (a.refine_passes > 0 && !a.u) ? align_up((size_t)a.n_anchors * a.H * a.M * sizeof(float)) : 0;
  p.total_bytes = p.partial_bytes + p.pooled_bytes + p.u_bytes;
  return p;
}

cast_status launch_route(const cast_route_args& a, void* ws, cudaStream_t st) {
  const RoutePlan p = route_plan(a);
  const int D = a.H * a.d;
  const int K_eff = a.K < a.M ? a.K : a.M;
  if (a.M == 0) return CAST_OK;   // nothing to route (App. B.3 bypass)
  char* w = static_cast<char*>(ws);
  float* partial = reinterpret_cast<float*>(w);
  float* pooled = reinterpret_cast<float*>(w + p.partial_bytes);
  float* qbar = a.qbar ? a.qbar : pooled;
  float* kbar = a.kbar ? a.kbar : pooled + (size_t)a.n_anchors * D;
  float* vbar = a.vbar ? a.vbar : pooled + (size_t)(a.n_anchors + a.M) * D;

  PoolArgs pa;
  pa.q = static_cast<const char*>(a.q);
  pa.k = static_cast<const char*>(a.k_hist);
  pa.v = static_cast<const char*>(a.v_hist);
  pa.q_row_stride = a.q_row_stride;
  pa.hist_row_stride = a.hist_row_stride;
  pa.n_anchors = a.n_anchors;
  pa.M = a.M;
  pa.S = a.S;
  pa.B_v = a.B_v;
  pa.D = D;
  pa.nsplit = p.nsplit;
  pa.elt = a.dtype == CAST_BF16 ? 2 : 4;
  for (int k = 0; k < a.n_anchors; ++k) pa.anchors[k] = a.anchors[k];
  dim3 grid(p.nsplit, p.n_seg);
  if (a.dtype == CAST_BF16)
    k_pool<__nv_bfloat16><<<grid, kPoolThreads, 0, st>>>(pa, partial);
  else
    k_pool<float><<<grid, kPoolThreads, 0, st>>>(pa, partial);
  cast_status s = check_launch("routing pool kernel");
  if (s != CAST_OK) return s;
  dim3 gf((D + 255) / 256, p.n_seg);
  k_finalize<<<gf, 256, 0, st>>>(partial, qbar, kbar, vbar, a.n_anchors, a.M, a.S, a.B_v, D,
                                 p.nsplit);
  s = check_launch("routing finalize kernel");
  if (s != CAST_OK) return s;
  const size_t smem = (size_t)(4 * a.M + 2 * a.d + (kScoreThreads / 32) * a.d) * sizeof(float);
  if (smem > 48 * 1024) {
    if (cudaFuncSetAttribute(k_score_topk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess)
      return fail(CAST_ERR_CUDA, "routing: cannot reserve %zu B of shared memory", smem);
  }
  const bool refine = a.refine_passes > 0 && K_eff > 0 && K_eff < a.M;
  float* u_buf = a.u ? a.u : (p.u_bytes ? reinterpret_cast<float*>(w + p.partial_bytes + p.pooled_bytes) : nullptr);
  k_score_topk<<<dim3(a.H, a.n_anchors), kScoreThreads, smem, st>>>(
      qbar, kbar, vbar, a.gram, a.H, a.d, a.M, K_eff, a.eps, a.mode, a.idx, u_buf);
  s = check_launch("routing score/TopK kernel");
  if (s != CAST_OK || !refine) return s;
  // Alg. (routing): interval and boundary coefficients of the anchor layout (Eqs. abc,
  // boundarycoeff), then the directional best-response passes on the GPU
  RefineArgs r{};
  r.n_anchors = a.n_anchors;
  r.M = a.M;
  r.K_eff = K_eff;
  r.H = a.H;
  r.passes = a.refine_passes;
  r.lam_anc = a.lambda_anc;
  r.lam_rec = a.lambda_rec;
  r.tol = a.refine_tol;
  for (int j = 1; j < a.n_anchors; ++j) {
    const int x0 = a.anchors[j - 1], x1 = a.anchors[j];
    double A = 0, B = 0, C = 0;
    for (int t = x0 + 1; t < x1; ++t) {
      const double al = (double)(t - x0) / (double)(x1 - x0);
      A += (1 - al) * (1 - al);
      B += al * al;
      C += al * (1 - al);
    }
    r.A[j] = (float)A;
    r.B[j] = (float)B;
    r.C[j] = (float)C;
  }
  if (a.n_anchors >= 2) {
    auto bset = [&](int x0, int x1, int t0, int t1, float& A, float& B, float& C) {
      double sa = 0, sb = 0, sc = 0;
      for (int t = t0; t < t1; ++t) {
        const double al = (double)(t - x0) / (double)(x1 - x0);
        sa += (1 - al) * (1 - al);
        sb += al * al;
        sc += std::fabs(al * (1 - al));
      }
      A = (float)sa;
      B = (float)sb;
      C = (float)sc;
    };
    bset(a.anchors[0], a.anchors[1], 0, a.anchors[0], r.AL, r.BL, r.CL);
    bset(a.anchors[a.n_anchors - 2], a.anchors[a.n_anchors - 1], a.anchors[a.n_anchors - 1] + 1,
         a.n_frames, r.AR, r.BR, r.CR);
  }
  const size_t rsm = refine_smem_bytes(a);
  if (rsm > 48 * 1024 &&
      cudaFuncSetAttribute(k_refine, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)rsm) != cudaSuccess)
    return fail(CAST_ERR_CUDA, "routing: cannot reserve %zu B of shared memory for refinement", rsm);
  k_refine<<<a.H, kRefineThreads, rsm, st>>>(u_buf, r, a.idx);
  return check_launch("routing refinement kernel");
}

}  // namespace cast
