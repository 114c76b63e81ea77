// Routing of historical KV blocks (Section 4.4, Eqs. pooled, omission, topk; App. B.3).
//
//   K_pool  : mean of every pooled segment (anchor query frames, history key blocks, history
//             value blocks): HBM-bound streaming of (K_f S + 2 M B_v) H d elements with 16-byte
//             loads, or, for long contiguous segments, through a ring of bulk copies into
//             shared memory.  A segment's rows are split over the CTAs of one thread-block
//             cluster; the CTAs reduce their column sums through distributed shared memory in
//             rank order (deterministic) and write q_bar, k_bar, v_bar in f32.  No partial sums
//             leave the chip.  Two launches with their own row split: the history blocks (with
//             (1, 8, 8) spatial blocks of history frames, 8 runs of up to 8 tokens each), then
//             the anchor frames (few long segments).
//   K_head_small : for M <= 32 blocks and up to 8 anchors, one CTA per head with one warp per
//             anchor for the statistics and the refinement in warp 0's registers.
//   K_head  : one CTA per head, every anchor at once, with the head's k_bar and v_bar staged in
//             shared memory: s, pi, o_bar, delta, u (Eq. omission, with an optional Gram matrix
//             G = P^T P of the output projection), the TopK mask of each anchor (ties to the
//             lower block index) and, when asked, the reconstruction-coupled best-response passes
//             of Alg. (routing); block indices are written in ascending order.
//   K_head_wide : the same for many blocks (means too large to stage): a thread-block cluster
//             per head shares the statistics, its rank-0 CTA selects (exact radix select) and
//             refines with all its threads.
// Each launch is a programmatic dependent of the one before: its CTAs become resident while
// the previous grid drains and wait on the grid dependency before reading its results.
#include <cuda_bf16.h>

#include <cfloat>
#include <cmath>

#include "internal.h"
#include "ptx.cuh"

namespace cast {
namespace {

constexpr int kPoolMaxThreads = 512;
constexpr int kPoolUnroll = 8;     // 16-byte loads in flight per thread
constexpr int kMaxClusterSplit = 8;
// bulk-copy pooling of contiguous segments: a ring of kPoolStages copies of about
// kPoolStageBytes (whole rows) per CTA, two CTAs per SM
constexpr int kPoolStages = 3;
constexpr int kPoolStageBytes = 32 * 1024;
// bulk-copy pooling only where a CTA streams at least this much: measured on GB300, 0.245 vs
// 0.253 ms for HY-World routing (2.7 MB per CTA) and 0.84 vs 0.89 ms for the stress history
// (7 MB), but 0.052 vs 0.047 ms for Matrix-Game (0.6 MB), where the ring's per-CTA latency
// chain is longer than that of eight register loads in flight per thread
constexpr int64_t kPoolBulkMinBytes = 1 << 20;
constexpr uint64_t kPoolWaitNs = 2000000000ull;

// Thread layout of the pooling CTA: cgs 16-byte column groups side by side, lanes_r row lanes.
struct PoolShape {
  int cgs, lanes_r;
};
inline PoolShape pool_shape(int D, int elt) {
  const int ncg = D / (16 / elt);
  PoolShape p;
  p.cgs = ncg >= kPoolMaxThreads ? kPoolMaxThreads : ncg;
  p.lanes_r = kPoolMaxThreads / p.cgs;
  return p;
}

struct PoolArgs {
  const char* q;          // anchor frame base = q + anchors[i] * S * q_row_stride * elt
  const char* k;
  const char* v;
  float* qbar;            // [n_anchors, D]
  float* kbar;            // [M, D]
  float* vbar;            // [M, D]
  int64_t q_row_stride, hist_row_stride;   // elements
  int n_anchors, M, S, B_v, D, nsplit, elt;
  int seg_base;           // segment of blockIdx.y == 0 (anchor frames first, then K, then V blocks)
  int bulk_rows;          // bulk-copy pooling: rows per ring stage
  int Hg, Wg, nby, nbx;   // CAST_HIST_FRAMES: history frame grid and its 8x8 block grid
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

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ float ld_dsmem(const float* local, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
               : "=r"(remote)
               : "r"((uint32_t)__cvta_generic_to_shared(local)), "r"(rank));
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(remote) : "memory");
  return v;
}
__device__ __forceinline__ void st_dsmem(float* local, uint32_t rank, float v) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;"
               : "=r"(remote)
               : "r"((uint32_t)__cvta_generic_to_shared(local)), "r"(rank));
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote), "f"(v) : "memory");
}
__device__ __forceinline__ void grid_dependency_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ unsigned int g_pool_error;   // 1: a bulk-copy wait of the pooling gave up

// Offset of the bulk-copy ring in the pooling kernel's dynamic shared memory (after colsum and
// the per-lane rows), 128-byte aligned.
__host__ __device__ inline size_t pool_ring_offset(int lanes_r, int D) {
  return ((size_t)lanes_r * D * sizeof(float) + 127) & ~(size_t)127;
}

template <typename T>
__device__ __forceinline__ void load_vec_smem(const uint8_t* p, float (&x)[16 / sizeof(T)]) {
  const uint4 v = *reinterpret_cast<const uint4*>(p);
  if (sizeof(T) == 4) {
    x[0] = __uint_as_float(v.x);
    x[1] = __uint_as_float(v.y);
    x[2] = __uint_as_float(v.z);
    x[3] = __uint_as_float(v.w);
  } else {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      x[2 * k] = __uint_as_float(w[k] << 16);
      x[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
    }
  }
}

// grid (nsplit, n_seg), cluster (nsplit, 1, 1), cgs * lanes_r threads.  Dynamic smem:
// colsum[D] and (lanes_r - 1) rows of per-lane sums (then, BULK, the copy ring).  SPATIAL: the
// history segments are (1, 8, 8) blocks of frames [frames][Hg][Wg] (hv runs of wv consecutive
// tokens, Wg tokens apart); the anchor-frame segments stay contiguous.  BULK (contiguous rows,
// one 16-byte column group per thread): the CTA's rows arrive through a ring of bulk copies of
// bulk_rows rows each, so that two CTAs keep about 190 KB of loads in flight per SM.
template <typename T, bool SPATIAL, bool BULK>
__global__ void __launch_bounds__(kPoolMaxThreads) k_pool(const __grid_constant__ PoolArgs a) {
  constexpr int VEC = 16 / sizeof(T);
  extern __shared__ float colsum[];
  launch_dependents();
  const int seg = blockIdx.y + a.seg_base, split = blockIdx.x;
  const char* base;
  int64_t rs;
  int nrows;
  int run = 1 << 30;      // SPATIAL: tokens per run (wv) and rows between runs (Wg)
  int64_t run_stride = 0;
  float* out;
  if (seg < a.n_anchors) {
    base = a.q + (int64_t)a.anchors[seg] * a.S * a.q_row_stride * a.elt;
    rs = a.q_row_stride;
    nrows = a.S;
    out = a.qbar + (int64_t)seg * a.D;
  } else {
    const bool is_k = seg < a.n_anchors + a.M;
    const int m = is_k ? seg - a.n_anchors : seg - a.n_anchors - a.M;
    rs = a.hist_row_stride;
    out = (is_k ? a.kbar : a.vbar) + (int64_t)m * a.D;
    const char* src = is_k ? a.k : a.v;
    if (SPATIAL) {
      const int per_frame = a.nby * a.nbx;
      const int f = m / per_frame, rem = m - f * per_frame;
      const int by = rem / a.nbx, bx = rem - by * a.nbx;
      const int hv = min(8, a.Hg - 8 * by), wv = min(8, a.Wg - 8 * bx);
      base = src + (((int64_t)f * a.Hg + 8 * by) * a.Wg + 8 * bx) * rs * a.elt;
      nrows = hv * wv;
      run = wv;
      run_stride = a.Wg;
    } else {
      base = src + (int64_t)m * a.B_v * rs * a.elt;
      nrows = a.B_v;
    }
  }
  const int per = (nrows + a.nsplit - 1) / a.nsplit;
  const int r0 = split * per, r1 = min(nrows, r0 + per);
  const int ncg = a.D / VEC;                                    // 16-byte column groups
  const int nthreads = blockDim.x;
  const int cgs = ncg >= kPoolMaxThreads ? kPoolMaxThreads : ncg;   // column groups per pass
  const int lanes_r = nthreads / cgs;                               // row lanes (>= 1)
  const int tcg = threadIdx.x % cgs, trl = threadIdx.x / cgs;
  float* lane_sum = colsum + a.D;                               // [lanes_r - 1][D] when lanes_r > 1
  if constexpr (BULK) {
    __shared__ __align__(8) uint64_t full[kPoolStages];
    __shared__ int s_fail;
    uint8_t* ring = reinterpret_cast<uint8_t*>(colsum) + pool_ring_offset(lanes_r, a.D);
    const int row_bytes = a.D * a.elt, rps = a.bulk_rows, stage_bytes = rps * row_bytes;
    const int nst = r1 > r0 ? (r1 - r0 + rps - 1) / rps : 0;
    if (threadIdx.x == 0) {
      for (int st = 0; st < kPoolStages; ++st) mbar_init(&full[st], 1);
      fence_barrier_init();
      s_fail = 0;
    }
    __syncthreads();
    auto issue = [&](int it) {   // thread 0: rows r0 + it * rps .. into stage it % kPoolStages
      const int st = it % kPoolStages, rr = r0 + it * rps, n = min(rps, r1 - rr);
      mbar_arrive_expect_tx(&full[st], (uint32_t)(n * row_bytes));
      bulk_load(ring + st * stage_bytes, base + (int64_t)rr * row_bytes, (uint32_t)(n * row_bytes), &full[st]);
    };
    int issued = 0;
    if (threadIdx.x == 0)
      for (; issued < kPoolStages && issued < nst; ++issued) issue(issued);
    float acc[VEC];
#pragma unroll
    for (int k = 0; k < VEC; ++k) acc[k] = 0.f;
    int it = 0;
    for (; it < nst; ++it) {
      const int st = it % kPoolStages;
      if (mbar_wait(&full[st], (uint32_t)(it / kPoolStages) & 1u, kPoolWaitNs)) {
        const int n = min(rps, r1 - (r0 + it * rps));
        const uint8_t* sp = ring + st * stage_bytes + tcg * 16;
        for (int q = trl; q < n; q += lanes_r) {
          float x[VEC];
          load_vec_smem<T>(sp + q * row_bytes, x);
#pragma unroll
          for (int k = 0; k < VEC; ++k) acc[k] += x[k];
        }
      } else {
        s_fail = 1;
      }
      __syncthreads();   // stage st has been read by every thread
      if (s_fail) break;
      if (threadIdx.x == 0 && issued < nst) {
        fence_proxy_async_smem();
        issue(issued++);
      }
    }
    if (s_fail && threadIdx.x == 0) {   // the copies in flight land before the memory is released
      atomicExch(&g_pool_error, 1u);
      for (int l = it; l < issued; ++l) mbar_wait(&full[l % kPoolStages], (uint32_t)(l / kPoolStages) & 1u, kPoolWaitNs);
    }
    if (trl == 0) {
#pragma unroll
      for (int k = 0; k < VEC; ++k) colsum[tcg * VEC + k] = acc[k];
    } else if (trl < lanes_r) {
#pragma unroll
      for (int k = 0; k < VEC; ++k) lane_sum[(int64_t)(trl - 1) * a.D + tcg * VEC + k] = acc[k];
    }
  }
  for (int cg = tcg; !BULK && cg < ncg; cg += cgs) {
    float acc[VEC];
#pragma unroll
    for (int k = 0; k < VEC; ++k) acc[k] = 0.f;
    if (SPATIAL && trl < lanes_r) {
      // row r of the segment: run r / wv, token r % wv of that run
      const char* pc = base + (int64_t)cg * VEC * a.elt;
      auto rowp = [&](int r) {
        const int y = r / run;
        return pc + ((int64_t)y * run_stride + (r - y * run)) * rs * a.elt;
      };
      int r = r0 + trl;
      for (; r + (kPoolUnroll - 1) * lanes_r < r1; r += kPoolUnroll * lanes_r) {
        float x[kPoolUnroll][VEC];
#pragma unroll
        for (int u = 0; u < kPoolUnroll; ++u) load_vec<T>(rowp(r + u * lanes_r), x[u]);
#pragma unroll
        for (int k = 0; k < VEC; ++k) {
          float s0 = 0.f, s1 = 0.f;
#pragma unroll
          for (int u = 0; u < kPoolUnroll; u += 2) {
            s0 += x[u][k];
            s1 += x[u + 1][k];
          }
          acc[k] += s0 + s1;
        }
      }
      for (; r < r1; r += lanes_r) {
        float x0[VEC];
        load_vec<T>(rowp(r), x0);
#pragma unroll
        for (int k = 0; k < VEC; ++k) acc[k] += x0[k];
      }
    } else if (trl < lanes_r) {
      const char* p = base + ((int64_t)(r0 + trl) * rs + (int64_t)cg * VEC) * a.elt;
      const int64_t step = (int64_t)lanes_r * rs * a.elt;
      int r = r0 + trl;
      for (; r + (kPoolUnroll - 1) * lanes_r < r1; r += kPoolUnroll * lanes_r) {
        float x[kPoolUnroll][VEC];
#pragma unroll
        for (int u = 0; u < kPoolUnroll; ++u) load_vec<T>(p + u * step, x[u]);
        p += kPoolUnroll * step;
#pragma unroll
        for (int k = 0; k < VEC; ++k) {
          float s0 = 0.f, s1 = 0.f;
#pragma unroll
          for (int u = 0; u < kPoolUnroll; u += 2) {
            s0 += x[u][k];
            s1 += x[u + 1][k];
          }
          acc[k] += s0 + s1;
        }
      }
      for (; r < r1; r += lanes_r) {
        float x0[VEC];
        load_vec<T>(p, x0);
        p += step;
#pragma unroll
        for (int k = 0; k < VEC; ++k) acc[k] += x0[k];
      }
    }
    if (trl == 0) {
#pragma unroll
      for (int k = 0; k < VEC; ++k) colsum[cg * VEC + k] = acc[k];
    } else if (trl < lanes_r) {
#pragma unroll
      for (int k = 0; k < VEC; ++k) lane_sum[(int64_t)(trl - 1) * a.D + cg * VEC + k] = acc[k];
    }
  }
  if (lanes_r > 1) {   // row lanes of each column, fixed order
    __syncthreads();
    for (int c = threadIdx.x; c < a.D; c += nthreads) {
      float s = colsum[c];
      for (int l = 1; l < lanes_r; ++l) s += lane_sum[(int64_t)(l - 1) * a.D + c];
      colsum[c] = s;
    }
  }
  // the cluster's column sums, reduced over its CTAs in rank order; this CTA owns one slice
  cluster_sync_all();
  const int cpr = (a.D + a.nsplit - 1) / a.nsplit;
  const int c0 = split * cpr, c1 = min(a.D, c0 + cpr);
  const float inv = 1.f / (float)nrows;
  for (int c = c0 + threadIdx.x; c < c1; c += nthreads) {
    float s = 0.f;
    for (int r = 0; r < a.nsplit; ++r) s += ld_dsmem(colsum + c, (uint32_t)r);
    out[c] = s * inv;
  }
  cluster_sync_all();   // no CTA leaves while a peer still reads its shared memory
  // the second pooling launch is a programmatic dependent of the first: it completes only after
  // the first has, so its own dependents see every mean
  grid_dependency_wait();
}

// ---------------------------------------------------------------------- per-head kernel
constexpr int kHeadThreads = 256, kHeadWarps = kHeadThreads / 32;

__device__ unsigned int g_route_error;

struct HeadArgs {
  const float* qbar;
  const float* kbar;
  const float* vbar;
  const float* gram;
  const int32_t* cand;   // optional [n_anchors, H, Mc] candidate sets
  int32_t* idx;
  float* u_out;
  int H, d, M, n_anchors, K_eff, mode, passes, Mc;
  float eps, lam_anc, lam_rec, tol;
  float A[CAST_MAX_ANCHORS], B[CAST_MAX_ANCHORS], C[CAST_MAX_ANCHORS];   // interval (j-1, j)
  float AL, BL, CL, AR, BR, CR;                                          // boundary sets
};

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
// TopK membership of key[m] among key[0..M): rank = #(larger, or equal with a lower index).
// Eight independent loads per round; the scan stops after a round that ranks K above m.
__device__ __forceinline__ bool in_topk(const float* key, int M, int K, int m) {
  const float v = key[m];
  int rank = 0, j = 0;
  for (; j + 8 <= M && rank < K; j += 8) {
    float w[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) w[t] = key[j + t];
#pragma unroll
    for (int t = 0; t < 8; ++t) rank += (w[t] > v) || (w[t] == v && j + t < m);
  }
  for (; j < M && rank < K; ++j) {
    const float w = key[j];
    rank += (w > v) || (w == v && j < m);
  }
  return rank < K;
}

// Warp-wide sum of one value per lane (every lane gets the total).
__device__ __forceinline__ float warp_total(float v) { return warp_sum(v); }

// grid (H).  Dynamic smem (floats): qb[na*d], ob[na*d], pi[na*M], key[na*M], x[na*M], G[M],
// with candidate sets Gc[M], then e[kHeadWarps*d] (Gram scratch); with candidate sets the
// membership bytes cm[na*M]; then kb[M*d], vb[M*d] (this head's means, staged).
__global__ void __launch_bounds__(kHeadThreads) k_head(const __grid_constant__ HeadArgs a) {
  extern __shared__ float sm[];
  const int h = blockIdx.x, na = a.n_anchors, M = a.M, d = a.d, K = a.K_eff;
  const int D = a.H * d;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool restricted = a.cand != nullptr;
  float* qb = sm;
  float* ob = qb + na * d;
  float* pi = ob + na * d;
  float* key = pi + na * M;
  float* x = key + na * M;
  float* G = x + na * M;
  float* Gc = G + M;                         // best-response keys restricted to C_i
  float* ew = Gc + (restricted ? M : 0);
  uint8_t* cm = reinterpret_cast<uint8_t*>(ew + kHeadWarps * d);
  // float4 stores below: the staged means start on a 16-byte boundary
  const size_t cm_bytes = restricted ? (((size_t)na * M + 15) & ~(size_t)15) : 0;
  float* kb_s = reinterpret_cast<float*>(
      reinterpret_cast<uint8_t*>(sm) +
      (((reinterpret_cast<uint8_t*>(ew + kHeadWarps * d) - reinterpret_cast<uint8_t*>(sm)) + 15) & ~(ptrdiff_t)15) +
      cm_bytes);
  float* vb_s = kb_s + (size_t)M * d;
  launch_dependents();
  grid_dependency_wait();   // the pooled means come from the preceding kernel
  // this head's slices of q_bar, k_bar and v_bar into shared memory, all loads in flight at once
  const float* kb = a.kbar + h * d;
  const float* vb = a.vbar + h * d;
  const int64_t kv_stride = d;
  {
    // rows of d/4 float4: q_bar rows of every anchor, then k_bar and v_bar rows;
    // each thread issues up to 8 loads before its first store
    const int q4 = d / 4;
    const int n_q = na * q4, n_all = n_q + 2 * M * q4;
    for (int e0 = tid; e0 < n_all; e0 += 8 * kHeadThreads) {
      float4 v[8];
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        const int e = e0 + t * kHeadThreads;
        if (e < n_q) {
          const int i = e / q4, c = (e - i * q4) * 4;
          v[t] = __ldcg(reinterpret_cast<const float4*>(a.qbar + (int64_t)i * D + h * d + c));
        } else if (e < n_all) {
          const int f = e - n_q, m = (f >> 1) / q4, c = ((f >> 1) - m * q4) * 4;
          v[t] = __ldcg(reinterpret_cast<const float4*>(((f & 1) ? vb : kb) + (int64_t)m * D + c));
        }
      }
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        const int e = e0 + t * kHeadThreads;
        if (e < n_q) {
          const int i = e / q4, c = (e - i * q4) * 4;
          *reinterpret_cast<float4*>(qb + i * d + c) = v[t];
        } else if (e < n_all) {
          const int f = e - n_q, m = (f >> 1) / q4, c = ((f >> 1) - m * q4) * 4;
          *reinterpret_cast<float4*>(((f & 1) ? vb_s : kb_s) + (int64_t)m * d + c) = v[t];
        }
      }
    }
    kb = kb_s;
    vb = vb_s;
  }
  __syncthreads();
  const float scale = rsqrtf((float)d);
  // s_{i,m} = q_bar_i . k_bar_m / sqrt(d)   (Eq. pooled); eight threads per (i, m), thread k
  // of a pair takes the float4 chunks k, k+8, ... (conflict-free shared-memory reads)
  // (rounds are block-uniform so every lane reaches the shuffles)
  const int sub = tid & 7, n4 = d / 4;
  const int n_pair = na * M, rounds = (n_pair + kHeadThreads / 8 - 1) / (kHeadThreads / 8);
  for (int rd = 0; rd < rounds; ++rd) {
    const int p = rd * (kHeadThreads / 8) + (tid >> 3);
    const bool live = p < n_pair;
    const int i = live ? p / M : 0, m = live ? p - i * M : 0;
    const float4* qv = reinterpret_cast<const float4*>(qb + i * d);
    const float4* kv = reinterpret_cast<const float4*>(kb + (int64_t)m * kv_stride);
    float acc = 0.f;
    for (int c = sub; live && c < n4; c += 8) {
      const float4 x4 = qv[c], y4 = kv[c];
      acc = fmaf(x4.x, y4.x, fmaf(x4.y, y4.y, fmaf(x4.z, y4.z, fmaf(x4.w, y4.w, acc))));
    }
    acc += __shfl_xor_sync(0xffffffffu, acc, 1);
    acc += __shfl_xor_sync(0xffffffffu, acc, 2);
    acc += __shfl_xor_sync(0xffffffffu, acc, 4);
    if (live && sub == 0) key[p] = acc * scale;
  }
  __syncthreads();
  // pi_i = softmax over blocks, one warp per anchor
  for (int i = warp; i < na; i += kHeadWarps) {
    const float* s = key + i * M;
    float mx = -FLT_MAX;
    for (int m = lane; m < M; m += 32) mx = fmaxf(mx, s[m]);
    mx = warp_max(mx);
    float tot = 0.f;
    for (int m = lane; m < M; m += 32) {
      const float e = expf(s[m] - mx);
      pi[i * M + m] = e;
      tot += e;
    }
    tot = warp_sum(tot);
    const float inv = 1.f / tot;
    for (int m = lane; m < M; m += 32) pi[i * M + m] *= inv;
  }
  __syncthreads();
  // o_bar_i = sum_m pi_{i,m} v_bar_m (four independent partial sums)
  for (int e = tid; e < na * d; e += kHeadThreads) {
    const int i = e / d, c = e - i * d;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    int m = 0;
    for (; m + 4 <= M; m += 4)
#pragma unroll
      for (int t = 0; t < 4; ++t) acc[t] = fmaf(pi[i * M + m + t], vb[(int64_t)(m + t) * kv_stride + c], acc[t]);
    for (; m < M; ++m) acc[0] = fmaf(pi[i * M + m], vb[(int64_t)m * kv_stride + c], acc[0]);
    ob[e] = (acc[0] + acc[1]) + (acc[2] + acc[3]);
  }
  __syncthreads();
  // delta_{i,m} = pi/(1 - pi + eps) (o_bar_i - v_bar_m);  u = delta^T G delta  (Eq. omission)
  if (a.mode == CAST_ROUTE_OMISSION && a.gram == nullptr) {
    // eight threads per (i, m) as for the scores
    for (int rd = 0; rd < rounds; ++rd) {
      const int p = rd * (kHeadThreads / 8) + (tid >> 3);
      const bool live = p < n_pair;
      const int i = live ? p / M : 0, m = live ? p - i * M : 0;
      const float4* ov = reinterpret_cast<const float4*>(ob + i * d);
      const float4* vv = reinterpret_cast<const float4*>(vb + (int64_t)m * kv_stride);
      float acc = 0.f;
      for (int c = sub; live && c < n4; c += 8) {
        const float4 x4 = ov[c], y4 = vv[c];
        const float t0 = x4.x - y4.x, t1 = x4.y - y4.y, t2 = x4.z - y4.z, t3 = x4.w - y4.w;
        acc = fmaf(t0, t0, fmaf(t1, t1, fmaf(t2, t2, fmaf(t3, t3, acc))));
      }
      acc += __shfl_xor_sync(0xffffffffu, acc, 1);
      acc += __shfl_xor_sync(0xffffffffu, acc, 2);
      acc += __shfl_xor_sync(0xffffffffu, acc, 4);
      if (live && sub == 0) {
        const float coef = pi[p] / (1.f - pi[p] + a.eps);
        key[p] = coef * coef * acc;
      }
    }
    __syncthreads();
  } else if (a.mode == CAST_ROUTE_OMISSION) {
    float* e = ew + warp * d;
    for (int p = warp; p < na * M; p += kHeadWarps) {
      const int i = p / M, m = p - i * M;
      const float* vm = vb + (int64_t)m * kv_stride;
      const float coef = pi[p] / (1.f - pi[p] + a.eps);
      float acc = 0.f;
      {
        for (int c = lane; c < d; c += 32) e[c] = ob[i * d + c] - vm[c];
        __syncwarp();
        const float* Gm = a.gram + (int64_t)h * d * d;
        for (int r = lane; r < d; r += 32) {
          float y = 0.f;
          for (int c = 0; c < d; ++c) y = fmaf(Gm[(int64_t)r * d + c], e[c], y);
          acc = fmaf(e[r], y, acc);
        }
        __syncwarp();
      }
      acc = warp_sum(acc);
      if (lane == 0) key[p] = coef * coef * acc;
    }
    __syncthreads();
  }
  if (a.u_out)
    for (int p = tid; p < na * M; p += kHeadThreads) {
      const int i = p / M, m = p - i * M;
      a.u_out[((int64_t)i * a.H + h) * M + m] = key[p];
    }
  if (K == 0) return;
  // candidate sets C_i (App. B.3): membership bytes; the initial TopK runs on keys that are
  // -inf outside C_i (pi is free here and holds them)
  const float* key0 = key;
  if (restricted) {
    for (int p = tid; p < na * M; p += kHeadThreads) cm[p] = 0;
    __syncthreads();
    for (int e = tid; e < na * a.Mc; e += kHeadThreads) {
      const int i = e / a.Mc, c = e - i * a.Mc;
      const int m = __ldg(a.cand + ((int64_t)i * a.H + h) * a.Mc + c);
      if (m < 0 || m >= M) atomicExch(&g_route_error, 1u);
      else cm[i * M + m] = 1;
    }
    __syncthreads();
    // a repeated index leaves its set with fewer than Mc members
    for (int i = warp; i < na; i += kHeadWarps) {
      int n = 0;
      for (int m = lane; m < M; m += 32) n += cm[i * M + m];
      n = __reduce_add_sync(0xffffffffu, n);
      if (lane == 0 && n != a.Mc) atomicExch(&g_route_error, 1u);
    }
    for (int p = tid; p < na * M; p += kHeadThreads) pi[p] = cm[p] ? key[p] : -INFINITY;
    __syncthreads();
    key0 = pi;
  }
  // initial masks: TopK of each anchor's key (Eq. topk)
  for (int p = tid; p < na * M; p += kHeadThreads) {
    const int i = p / M, m = p - i * M;
    x[p] = in_topk(key0 + i * M, M, K, m) ? 1.f : 0.f;
  }
  __syncthreads();
  if (a.passes > 0 && K < M) {
    // Alg. (routing) with u = key.  Shared state for the passes: sq[j][m] = sqrt(u_{j-1,m}
    // u_{j,m}) of every adjacent anchor pair (pi is no longer needed) and the interval
    // coefficients (o_bar is no longer needed); the boundary sets use the pairs (0, 1) and
    // (na-2, na-1), i.e. sq[1] and sq[na-1].
    const float* u = key;
    float* sq = pi;
    float* cA = ob;
    float* cB = ob + na;
    float* cC = ob + 2 * na;
    for (int p = tid; p < na * M; p += kHeadThreads)
      if (p >= M) sq[p] = sqrtf(u[p - M] * u[p]);
    for (int j = tid; j < na; j += kHeadThreads) {
      cA[j] = a.A[j];
      cB[j] = a.B[j];
      cC[j] = a.C[j];
    }
    __syncthreads();
    if (warp == 0) {
      // one warp: fixed-budget best responses on J (Eq. objective); lane l owns blocks l, l+32, ...
      const float AL = a.AL, BL = a.BL, CL = a.CL, AR = a.AR, BR = a.BR, CR = a.CR;
      const float lam_anc = a.lam_anc, lam_rec = a.lam_rec;
      float Jl = 0.f;
      for (int m = lane; m < M; m += 32) {
        for (int i = 0; i < na; ++i) Jl += lam_anc * (1.f - x[i * M + m]) * u[i * M + m];
        float rec = 0.f;
        for (int j = 1; j < na; ++j) {
          const float xp = 1.f - x[(j - 1) * M + m], xq = 1.f - x[j * M + m];
          rec += cA[j] * xp * u[(j - 1) * M + m] + cB[j] * xq * u[j * M + m] + 2.f * cC[j] * xp * xq * sq[j * M + m];
        }
        if (na >= 2) {
          const float x0 = 1.f - x[m], x1 = 1.f - x[M + m];
          rec += AL * x0 * u[m] + BL * x1 * u[M + m] + 2.f * CL * x0 * x1 * sq[M + m];
          const int r0 = (na - 2) * M + m, r1 = (na - 1) * M + m;
          const float y0 = 1.f - x[r0], y1 = 1.f - x[r1];
          rec += AR * y0 * u[r0] + BR * y1 * u[r1] + 2.f * CR * y0 * y1 * sq[r1];
        }
        Jl += lam_rec * rec;
      }
      float J = warp_total(Jl);
      for (int pass = 1; pass <= a.passes; ++pass) {
        bool changed = false;
        for (int step = 0; step < na; ++step) {
          const int i = (pass & 1) ? step : na - 1 - step;
          // retain gains, Eqs. (gain) and (boundarygain)
          for (int m = lane; m < M; m += 32) {
            const float ui = u[i * M + m];
            float rec = 0.f;
            if (i >= 1) rec += cB[i] * ui + 2.f * cC[i] * (1.f - x[(i - 1) * M + m]) * sq[i * M + m];
            if (i + 1 < na) rec += cA[i + 1] * ui + 2.f * cC[i + 1] * (1.f - x[(i + 1) * M + m]) * sq[(i + 1) * M + m];
            if (na >= 2) {
              if (i == 0) rec += AL * ui + 2.f * CL * (1.f - x[M + m]) * sq[M + m];
              if (i == 1) rec += BL * ui + 2.f * CL * (1.f - x[m]) * sq[M + m];
              if (i == na - 2) rec += AR * ui + 2.f * CR * (1.f - x[(na - 1) * M + m]) * sq[(na - 1) * M + m];
              if (i == na - 1) rec += BR * ui + 2.f * CR * (1.f - x[(na - 2) * M + m]) * sq[(na - 1) * M + m];
            }
            const float g = lam_anc * ui + lam_rec * rec;
            G[m] = g;
            if (restricted) Gc[m] = cm[i * M + m] ? g : -INFINITY;
          }
          __syncwarp();
          // best response TopK(G) (within C_i) and its gain sum_m G_m (x_new - x_i); J is
          // affine in x_i, so the accepted step lowers J by exactly that gain
          const float* Gk = restricted ? Gc : G;
          float gl = 0.f;
          uint32_t sel = 0u;   // this lane's memberships (bit r: block lane + 32 r; M <= 1024 here)
          for (int m = lane, r = 0; m < M; m += 32, ++r) {
            const bool in = in_topk(Gk, M, K, m);
            sel |= (uint32_t)in << r;
            gl += G[m] * ((in ? 1.f : 0.f) - x[i * M + m]);
          }
          const float gain = warp_total(gl);
          if (gain > a.tol * fmaxf(J, 1e-8f)) {   // uniform across the warp
            for (int m = lane, r = 0; m < M; m += 32, ++r) x[i * M + m] = ((sel >> r) & 1u) ? 1.f : 0.f;
            J -= gain;
            changed = true;
          }
          __syncwarp();
        }
        if (!changed) break;
      }
    }
  }
  __syncthreads();
  // ascending block indices of every anchor's mask
  for (int i = warp; i < na; i += kHeadWarps) {
    int base = 0;
    int32_t* out = a.idx + ((int64_t)i * a.H + h) * K;
    for (int m0 = 0; m0 < M; m0 += 32) {
      const int m = m0 + lane;
      const bool on = m < M && x[i * M + m] != 0.f;
      const unsigned bal = __ballot_sync(0xffffffffu, on);
      if (on) out[base + __popc(bal & ((1u << lane) - 1u))] = m;
      base += __popc(bal);
    }
  }
}

// ---------------------------------------------------------------------- small per-head kernel
// The same statistics, TopK and refinement for the common small case (no Gram matrix, no
// candidate sets, M <= 32 blocks, at most 8 anchors), with one warp per anchor and lane m =
// block m, so that the phases need no block-wide barriers: lane m forms s_m, the warp's
// shuffles give the softmax, lanes split o_bar by dimensions, lane m forms u_m and its rank.
// The refinement passes (Alg. routing) run in warp 0 with every anchor's u, sqrt(u u) of the
// adjacent pairs and the masks (ballots) in registers, TopK(G) ranked by shuffles.
constexpr int kSmallMaxM = 32, kSmallMaxAnchors = 8;

// shared memory (floats): qb[na][d], ob[na][d], kb[M][d + 4], vb[M][d + 4] (rows padded so
// that lane m's 16-byte reads of row m fall in distinct bank groups), key[na][32]
size_t small_head_bytes(const cast_route_args& a) {
  const int dp = a.d + 4;
  return ((size_t)2 * a.n_anchors * a.d + (size_t)2 * a.M * dp + (size_t)a.n_anchors * kSmallMaxM) * sizeof(float);
}

template <int HD>
__global__ void __launch_bounds__(kHeadThreads) k_head_small(const __grid_constant__ HeadArgs a) {
  extern __shared__ float sm[];
  constexpr int d = HD, dp = d + 4, d4 = d / 4;
  const int h = blockIdx.x, na = a.n_anchors, M = a.M, K = a.K_eff;
  const int D = a.H * d;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float* qb = sm;
  float* ob = qb + na * d;
  float* kb = ob + na * d;
  float* vb = kb + M * dp;
  float* key = vb + M * dp;
  __shared__ uint32_t s_mask[kSmallMaxAnchors];
  launch_dependents();
  grid_dependency_wait();   // the pooled means come from the preceding kernel
  {
    // q_bar rows of every anchor, then k_bar and v_bar rows; up to 8 loads in flight per thread
    const int n_q = na * d4, n_all = n_q + 2 * M * d4;
    for (int e0 = tid; e0 < n_all; e0 += 8 * kHeadThreads) {
      float4 v[8];
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        const int e = e0 + t * kHeadThreads;
        if (e < n_q) {
          const int i = e / d4, c = (e - i * d4) * 4;
          v[t] = __ldcg(reinterpret_cast<const float4*>(a.qbar + (int64_t)i * D + h * d + c));
        } else if (e < n_all) {
          const int f = e - n_q, m = (f >> 1) / d4, c = ((f >> 1) - m * d4) * 4;
          v[t] = __ldcg(reinterpret_cast<const float4*>(((f & 1) ? a.vbar : a.kbar) + (int64_t)m * D + h * d + c));
        }
      }
#pragma unroll
      for (int t = 0; t < 8; ++t) {
        const int e = e0 + t * kHeadThreads;
        if (e < n_q) {
          const int i = e / d4, c = (e - i * d4) * 4;
          *reinterpret_cast<float4*>(qb + i * d + c) = v[t];
        } else if (e < n_all) {
          const int f = e - n_q, m = (f >> 1) / d4, c = ((f >> 1) - m * d4) * 4;
          *reinterpret_cast<float4*>(((f & 1) ? vb : kb) + m * dp + c) = v[t];
        }
      }
    }
  }
  __syncthreads();
  const bool live = lane < M;
  if (warp < na) {
    const int i = warp;
    // s_m = q_bar_i . k_bar_m / sqrt(d)   (Eq. pooled)
    const float4* q4 = reinterpret_cast<const float4*>(qb + i * d);
    const float4* k4 = reinterpret_cast<const float4*>(kb + (live ? lane : 0) * dp);
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int c = 0; c < d4; ++c) {
      const float4 x = q4[c], y = k4[c];
      acc[c & 3] = fmaf(x.x, y.x, fmaf(x.y, y.y, fmaf(x.z, y.z, fmaf(x.w, y.w, acc[c & 3]))));
    }
    const float s = live ? ((acc[0] + acc[1]) + (acc[2] + acc[3])) * rsqrtf((float)d) : -FLT_MAX;
    float u;
    if (a.mode == CAST_ROUTE_OMISSION) {
      // pi = softmax over blocks; o_bar = sum pi_m v_bar_m; u_m = (pi_m / (1 - pi_m + eps))^2 |o_bar - v_bar_m|^2
      const float mx = warp_max(s);
      const float e = live ? expf(s - mx) : 0.f;
      const float pi = e / warp_sum(e);
      // pi through shared memory (this anchor's key row, rewritten with u below): the
      // dimension loop below runs on d / 4 lanes only
      if (live) key[i * kSmallMaxM + lane] = pi;
      __syncwarp();
      if (lane < d4) {
        const int c = lane;
        float4 o[2] = {make_float4(0.f, 0.f, 0.f, 0.f), make_float4(0.f, 0.f, 0.f, 0.f)};
#pragma unroll
        for (int m = 0; m < kSmallMaxM; ++m) {
          if (m < M) {
            const float pm = key[i * kSmallMaxM + m];
            const float4 v = *reinterpret_cast<const float4*>(vb + m * dp + 4 * c);
            float4& t = o[m & 1];
            t.x = fmaf(pm, v.x, t.x);
            t.y = fmaf(pm, v.y, t.y);
            t.z = fmaf(pm, v.z, t.z);
            t.w = fmaf(pm, v.w, t.w);
          }
        }
        *reinterpret_cast<float4*>(ob + i * d + 4 * c) =
            make_float4(o[0].x + o[1].x, o[0].y + o[1].y, o[0].z + o[1].z, o[0].w + o[1].w);
      }
      __syncwarp();
      const float4* o4 = reinterpret_cast<const float4*>(ob + i * d);
      const float4* v4 = reinterpret_cast<const float4*>(vb + (live ? lane : 0) * dp);
      float dist[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int c = 0; c < d4; ++c) {
        const float4 x = o4[c], y = v4[c];
        const float t0 = x.x - y.x, t1 = x.y - y.y, t2 = x.z - y.z, t3 = x.w - y.w;
        dist[c & 3] = fmaf(t0, t0, fmaf(t1, t1, fmaf(t2, t2, fmaf(t3, t3, dist[c & 3]))));
      }
      const float coef = pi / (1.f - pi + a.eps);
      u = live ? coef * coef * ((dist[0] + dist[1]) + (dist[2] + dist[3])) : 0.f;
    } else {
      u = live ? s : 0.f;   // SIMILARITY: TopK on the pooled score
    }
    if (live) {
      key[i * kSmallMaxM + lane] = u;
      if (a.u_out) a.u_out[((int64_t)i * a.H + h) * M + lane] = u;
    }
    // initial mask: TopK of u (Eq. topk), ties to the lower block index
    const float uk = live ? u : -INFINITY;
    int rank = 0;
#pragma unroll 4
    for (int l = 0; l < M; ++l) {
      const float w = __shfl_sync(0xffffffffu, uk, l);
      rank += (w > uk) || (w == uk && l < lane);
    }
    const uint32_t mask = __ballot_sync(0xffffffffu, live && rank < K);
    if (lane == 0) s_mask[i] = mask;
  }
  if (K == 0) return;
  __syncthreads();
  if (warp == 0) {
    uint32_t mk[kSmallMaxAnchors];
    float uu[kSmallMaxAnchors], sq[kSmallMaxAnchors];
#pragma unroll
    for (int k = 0; k < kSmallMaxAnchors; ++k) {
      mk[k] = k < na ? s_mask[k] : 0u;
      uu[k] = (k < na && live) ? key[k * kSmallMaxM + lane] : 0.f;
    }
#pragma unroll
    for (int k = 0; k < kSmallMaxAnchors; ++k) sq[k] = (k >= 1 && k < na) ? sqrtf(uu[k - 1] * uu[k]) : 0.f;
    if (a.passes > 0 && K < M) {
      auto xb = [&](int k) -> float {   // 1 - x_{k, lane} (omission indicator), k < na
        uint32_t v = 0u;
#pragma unroll
        for (int t = 0; t < kSmallMaxAnchors; ++t)
          if (t == k) v = mk[t];
        return ((v >> lane) & 1u) ? 0.f : 1.f;
      };
      auto pick = [&](const float* arr, int k) -> float {
        float v = 0.f;
#pragma unroll
        for (int t = 0; t < kSmallMaxAnchors; ++t)
          if (t == k) v = arr[t];
        return v;
      };
      const float AL = a.AL, BL = a.BL, CL = a.CL, AR = a.AR, BR = a.BR, CR = a.CR;
      const float lam_anc = a.lam_anc, lam_rec = a.lam_rec;
      // J of the current masks (Eq. objective)
      float Jl = 0.f;
      if (live) {
#pragma unroll
        for (int k = 0; k < kSmallMaxAnchors; ++k)
          if (k < na) Jl += lam_anc * xb(k) * uu[k];
        float rec = 0.f;
#pragma unroll
        for (int j = 1; j < kSmallMaxAnchors; ++j)
          if (j < na) {
            const float xp = xb(j - 1), xq = xb(j);
            rec += a.A[j] * xp * uu[j - 1] + a.B[j] * xq * uu[j] + 2.f * a.C[j] * xp * xq * sq[j];
          }
        if (na >= 2) {
          const float x0 = xb(0), x1 = xb(1);
          rec += AL * x0 * uu[0] + BL * x1 * uu[1] + 2.f * CL * x0 * x1 * sq[1];
          const float y0 = xb(na - 2), y1 = xb(na - 1);
          rec += AR * y0 * pick(uu, na - 2) + BR * y1 * pick(uu, na - 1) + 2.f * CR * y0 * y1 * pick(sq, na - 1);
        }
        Jl += lam_rec * rec;
      }
      float J = warp_sum(Jl);
      for (int pass = 1; pass <= a.passes; ++pass) {
        bool changed = false;
        for (int step = 0; step < na; ++step) {
          const int i = (pass & 1) ? step : na - 1 - step;
          // retain gains, Eqs. (gain) and (boundarygain)
          const float ui = pick(uu, i);
          float rec = 0.f;
          if (i >= 1) rec += a.B[i] * ui + 2.f * a.C[i] * xb(i - 1) * pick(sq, i);
          if (i + 1 < na) rec += a.A[i + 1] * ui + 2.f * a.C[i + 1] * xb(i + 1) * pick(sq, i + 1);
          if (na >= 2) {
            if (i == 0) rec += AL * ui + 2.f * CL * xb(1) * sq[1];
            if (i == 1) rec += BL * ui + 2.f * CL * xb(0) * sq[1];
            if (i == na - 2) rec += AR * ui + 2.f * CR * xb(na - 1) * pick(sq, na - 1);
            if (i == na - 1) rec += BR * ui + 2.f * CR * xb(na - 2) * pick(sq, na - 1);
          }
          const float G = live ? lam_anc * ui + lam_rec * rec : -INFINITY;
          // best response TopK(G) and its gain sum_m G_m (x_new - x_i) (J is affine in x_i)
          int rank = 0;
#pragma unroll 4
          for (int l = 0; l < M; ++l) {
            const float w = __shfl_sync(0xffffffffu, G, l);
            rank += (w > G) || (w == G && l < lane);
          }
          const bool in = live && rank < K;
          const float xi = 1.f - xb(i);
          const float gain = warp_sum(live ? G * ((in ? 1.f : 0.f) - xi) : 0.f);
          if (gain > a.tol * fmaxf(J, 1e-8f)) {   // uniform across the warp
            const uint32_t nm = __ballot_sync(0xffffffffu, in);
#pragma unroll
            for (int t = 0; t < kSmallMaxAnchors; ++t)
              if (t == i) mk[t] = nm;
            J -= gain;
            changed = true;
          }
        }
        if (!changed) break;
      }
    }
    // ascending block indices of every anchor's mask
    for (int i = 0; i < na; ++i) {
      uint32_t v = 0u;
#pragma unroll
      for (int t = 0; t < kSmallMaxAnchors; ++t)
        if (t == i) v = mk[t];
      if ((v >> lane) & 1u) a.idx[((int64_t)i * a.H + h) * K + __popc(v & ((1u << lane) - 1u))] = lane;
    }
  }
}

// ---------------------------------------------------------------------- wide per-head kernel
// For many history blocks (k_bar, v_bar of a head too large for one CTA's shared memory) the
// statistics of one head are spread over a cluster of cl CTAs, each owning a contiguous range
// of mr blocks: scores, the softmax max and sum, o_bar partial sums and the omission scores
// are exchanged through distributed shared memory (reduced in rank order).  The rank-0 CTA
// then gathers every anchor's scores and runs the TopK selections and the refinement passes
// with all its threads; each TopK is an exact radix select on a 46-bit key (the score's order
// bits, then the inverted block index, so that ties go to the lower index).
constexpr int kWideThreads = 256, kWideWarps = kWideThreads / 32;
constexpr int kWideMaxCl = 8, kWideGroup = 8;   // CTAs per head; anchors per o_bar pass
constexpr int kWideRows = 8;                    // history blocks a warp loads at once
constexpr int kRadixBins = 1024;                // 10-bit digits of the TopK radix select

__host__ __device__ inline uint32_t take_smem(size_t& o, size_t bytes) {
  const size_t r = o;
  o += (bytes + 15) & ~(size_t)15;
  return (uint32_t)r;
}

// Byte offsets of the wide kernel's shared memory.  The o_bar partials of the warps share
// their space with the rank-0 arrays, which are only written after the partials are reduced.
struct WideLayout {
  uint32_t qb, ob, obp, red, sl, pl, ew, coef, owp, u, x, sq, G, red2, hist, pre, cm;
  size_t total;
};
__host__ __device__ inline WideLayout wide_layout(int na, int M, int d, int mr, bool refine,
                                                  bool restricted) {
  WideLayout L{};
  size_t o = 0;
  const size_t naf = (size_t)na * sizeof(float);
  L.qb = take_smem(o, naf * d);
  L.ob = take_smem(o, naf * d);
  L.obp = take_smem(o, naf * d);
  L.red = take_smem(o, 2 * naf);
  L.sl = take_smem(o, naf * mr);
  L.pl = take_smem(o, naf * mr);
  L.ew = take_smem(o, (size_t)kWideWarps * d * sizeof(float));
  L.coef = take_smem(o, 3 * naf);
  const size_t region = o;
  L.owp = (uint32_t)region;
  const size_t owp_end = region + (size_t)kWideWarps * kWideGroup * d * sizeof(float);
  L.u = take_smem(o, naf * M);
  L.x = take_smem(o, naf * M);
  L.sq = refine ? take_smem(o, naf * M) : 0;
  L.G = take_smem(o, (size_t)M * sizeof(float));
  L.red2 = take_smem(o, 64 * sizeof(float));
  L.hist = take_smem(o, (size_t)2 * kRadixBins * sizeof(unsigned));
  L.pre = take_smem(o, 4 * sizeof(unsigned long long));
  L.cm = restricted ? take_smem(o, (size_t)na * M) : 0;
  L.total = o > owp_end ? o : owp_end;
  return L;
}

inline int wide_cluster(int M) {
  const int cl = (M + 63) / 64;
  return cl > kWideMaxCl ? kWideMaxCl : (cl < 1 ? 1 : cl);
}

// Order key of score v at block m (M <= 16384): larger key = selected first; -0 ranks as +0,
// -inf (outside a candidate set) below every finite score.
__device__ __forceinline__ unsigned long long order_key(float v, int m) {
  uint32_t b = __float_as_uint(v == 0.f ? 0.f : v);
  b = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  return ((unsigned long long)b << 14) | (unsigned long long)(16383 - m);
}
__device__ __forceinline__ float masked(const float* key, const uint8_t* cm, int p) {
  return (cm && !cm[p]) ? -INFINITY : key[p];
}

// Radix select of the TopK threshold of one row key[0..M) (entries with cm[m] == 0 count as
// -inf; 0 < K < M): returns the order key t such that exactly K keys of the row have
// order_key >= t.  Rounds of 10-bit digits from the top of the 46-bit key; a round whose
// chosen digit holds exactly the remaining count ends the select (its lower bits are then
// left zero).  hist holds two 1024-bin buffers, zero on entry and zero again on return; each
// round's buffer is cleared during the round after it.  Every thread of the CTA calls this.
__device__ unsigned long long topk_threshold(const float* key, const uint8_t* cm, int M, int K,
                                             unsigned* hist2, unsigned long long* sel) {
  const int tid = threadIdx.x, lane = tid & 31;
  unsigned long long pre = 0ull;
  int krem = K;
  int round = 0;
  for (int shift = 36;; shift = shift >= 10 ? shift - 10 : 0, ++round) {
    const int width = shift == 0 ? 6 : 10;   // bits 45..36, 35..26, 25..16, 15..6, 5..0
    // (the last round's 6-bit digit uses bins 0..63 of the same 1024)
    unsigned* hist = hist2 + (round & 1) * kRadixBins;
    if (round > 0)   // the previous round's buffer is free again (read before the last barrier)
      for (int e = tid; e < kRadixBins; e += kWideThreads) hist2[((round - 1) & 1) * kRadixBins + e] = 0u;
    const unsigned long long hi = ~0ull << (shift + width);
    for (int m = tid; m < M; m += kWideThreads) {
      const unsigned long long c = order_key(cm && !cm[m] ? -INFINITY : key[m], m);
      if ((c & hi) == pre) atomicAdd(&hist[(int)((c >> shift) & (unsigned long long)(kRadixBins - 1))], 1u);
    }
    __syncthreads();
    if (tid < 32) {
      // the digit where the count from the top reaches krem: lane l first sums the 32 bins
      // 1023-32l .. 992-32l (rotated so the lanes hit different banks), a warp scan picks the
      // chunk, then the warp scans that chunk's bins
      unsigned part = 0;
#pragma unroll 8
      for (int t = 0; t < 32; ++t) part += hist[kRadixBins - 1 - 32 * lane - ((t + lane) & 31)];
      unsigned inc = part;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned w = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += w;
      }
      const int l = __ffs(__ballot_sync(0xffffffffu, inc >= (unsigned)krem)) - 1;
      const unsigned carry = __shfl_sync(0xffffffffu, inc - part, l);
      const int b = kRadixBins - 1 - 32 * l - lane;
      const unsigned v = hist[b];
      unsigned inc2 = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned w = __shfl_up_sync(0xffffffffu, inc2, o);
        if (lane >= o) inc2 += w;
      }
      const int j = __ffs(__ballot_sync(0xffffffffu, carry + inc2 >= (unsigned)krem)) - 1;
      if (lane == j) {
        const unsigned before = carry + inc2 - v;
        sel[0] = pre | ((unsigned long long)b << shift);
        sel[1] = (unsigned long long)(krem - (int)before);
        sel[2] = (v == (unsigned)krem - before || shift == 0) ? 1ull : 0ull;
      }
    }
    __syncthreads();
    pre = sel[0];
    krem = (int)sel[1];
    const bool done = sel[2] != 0ull;
    if (done) {
      // clear this round's buffer before leaving (the other one is already zero)
      for (int e = tid; e < kRadixBins; e += kWideThreads) hist[e] = 0u;
      __syncthreads();
      return pre;
    }
  }
}

// Deterministic CTA-wide sum (warp sums added in warp order); every thread gets the total.
// red2 holds two slot sets used alternately (`slot` flips between calls), so a call never
// overwrites partials a slower thread is still adding from the previous call.
__device__ __forceinline__ float block_sum(float v, float* red2, int& slot) {
  v = warp_sum(v);
  float* r = red2 + slot * kWideWarps;
  slot ^= 1;
  if ((threadIdx.x & 31) == 0) r[threadIdx.x >> 5] = v;
  __syncthreads();
  float t = 0.f;
#pragma unroll
  for (int w = 0; w < kWideWarps; ++w) t += r[w];
  return t;
}

// Sums each of v[0..7] over the 32 lanes with 9 shuffles (halving the set at each of the first
// three steps); on return lane l holds the total of v[(l >> 2) & 7].
__device__ __forceinline__ float warp_sum8(float (&v)[8]) {
  const int lane = threadIdx.x & 31;
  float w[4], y[2];
  const bool b4 = lane & 16, b3 = lane & 8, b2 = lane & 4;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float keep = b4 ? v[j + 4] : v[j], give = b4 ? v[j] : v[j + 4];
    w[j] = keep + __shfl_xor_sync(0xffffffffu, give, 16);
  }
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const float keep = b3 ? w[j + 2] : w[j], give = b3 ? w[j] : w[j + 2];
    y[j] = keep + __shfl_xor_sync(0xffffffffu, give, 8);
  }
  float z = (b2 ? y[1] : y[0]) + __shfl_xor_sync(0xffffffffu, b2 ? y[0] : y[1], 4);
  z += __shfl_xor_sync(0xffffffffu, z, 2);
  z += __shfl_xor_sync(0xffffffffu, z, 1);
  return z;
}

template <int NP>
__device__ __forceinline__ void load_row(const float* p, float (&v)[NP]) {
  if constexpr (NP == 4) {
    const float4 t = __ldcg(reinterpret_cast<const float4*>(p));
    v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
  } else {
    const float2 t = __ldcg(reinterpret_cast<const float2*>(p));
    v[0] = t.x; v[1] = t.y;
  }
}

// grid (cl, H), cluster (cl, 1, 1), kWideThreads threads; lane l of a warp holds channels
// l*NP .. l*NP+NP-1 of a head vector (HD = 32 NP).
template <int HD>
__global__ void __launch_bounds__(kWideThreads) k_head_wide(const __grid_constant__ HeadArgs a) {
  constexpr int NP = HD / 32;
  extern __shared__ __align__(16) uint8_t wsm[];
  const int rank = blockIdx.x, cl = gridDim.x, h = blockIdx.y;
  const int na = a.n_anchors, M = a.M, K = a.K_eff, D = a.H * HD;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool restricted = a.cand != nullptr;
  const bool refine = a.passes > 0 && K > 0 && K < M;
  const int mr = (M + cl - 1) / cl;
  const int m0 = min(M, rank * mr), m1 = min(M, m0 + mr), nm = m1 - m0;
  const WideLayout L = wide_layout(na, M, HD, mr, refine, restricted);
  float* qb = reinterpret_cast<float*>(wsm + L.qb);
  float* ob = reinterpret_cast<float*>(wsm + L.ob);
  float* obp = reinterpret_cast<float*>(wsm + L.obp);
  float* red = reinterpret_cast<float*>(wsm + L.red);
  float* sl = reinterpret_cast<float*>(wsm + L.sl);    // [na][mr] scores s of this CTA's blocks
  float* pl = reinterpret_cast<float*>(wsm + L.pl);    // [na][mr] pi, then the omission score u
  float* ew = reinterpret_cast<float*>(wsm + L.ew);
  const float* kbar = a.kbar + h * HD;
  const float* vbar = a.vbar + h * HD;
  launch_dependents();
  grid_dependency_wait();   // the pooled means come from the preceding kernels
  for (int e = tid; e < na * (HD / 4); e += kWideThreads) {
    const int i = e / (HD / 4), c = (e - i * (HD / 4)) * 4;
    *reinterpret_cast<float4*>(qb + i * HD + c) =
        __ldcg(reinterpret_cast<const float4*>(a.qbar + (int64_t)i * D + h * HD + c));
  }
  __syncthreads();
  // s_{i,m} = q_bar_i . k_bar_m / sqrt(d)  (Eq. pooled): a warp takes kWideRows blocks at once
  const float scale = rsqrtf((float)HD);
  for (int mb = m0 + warp * kWideRows; mb < m1; mb += kWideWarps * kWideRows) {
    float kv[kWideRows][NP];
#pragma unroll
    for (int t = 0; t < kWideRows; ++t) {
      if (mb + t < m1) load_row<NP>(kbar + (int64_t)(mb + t) * D + lane * NP, kv[t]);
      else
#pragma unroll
        for (int k = 0; k < NP; ++k) kv[t][k] = 0.f;
    }
    for (int i = 0; i < na; ++i) {
      float qv[NP], p[kWideRows];
#pragma unroll
      for (int k = 0; k < NP; ++k) qv[k] = qb[i * HD + lane * NP + k];
#pragma unroll
      for (int t = 0; t < kWideRows; ++t) {
        p[t] = 0.f;
#pragma unroll
        for (int k = 0; k < NP; ++k) p[t] = fmaf(qv[k], kv[t][k], p[t]);
      }
      const float tot = warp_sum8(p);   // row (lane >> 2) & 7 of the batch
      const int t = (lane >> 2) & 7;
      if ((lane & 3) == 0 && mb + t < m1) sl[i * mr + (mb + t - m0)] = tot * scale;
    }
  }
  __syncthreads();
  // pi_i = softmax over all M blocks: cluster-wide max, then sum (both in rank order)
  for (int i = warp; i < na; i += kWideWarps) {
    float mx = -INFINITY;
    for (int m = lane; m < nm; m += 32) mx = fmaxf(mx, sl[i * mr + m]);
    mx = warp_max(mx);
    if (lane == 0) red[i] = mx;
  }
  cluster_sync_all();
  for (int i = warp; i < na; i += kWideWarps) {
    float gm = -INFINITY;
    for (int r = 0; r < cl; ++r) gm = fmaxf(gm, ld_dsmem(red + i, (uint32_t)r));
    float tot = 0.f;
    for (int m = lane; m < nm; m += 32) {
      const float e = expf(sl[i * mr + m] - gm);
      pl[i * mr + m] = e;
      tot += e;
    }
    tot = warp_sum(tot);
    if (lane == 0) red[na + i] = tot;
  }
  cluster_sync_all();
  for (int i = warp; i < na; i += kWideWarps) {
    float tot = 0.f;
    for (int r = 0; r < cl; ++r) tot += ld_dsmem(red + na + i, (uint32_t)r);
    const float inv = 1.f / tot;
    for (int m = lane; m < nm; m += 32) pl[i * mr + m] *= inv;
  }
  __syncthreads();
  // o_bar_i = sum_m pi_{i,m} v_bar_m: per-warp partials (kWideGroup anchors per pass), summed
  // over warps in order, then over the cluster's CTAs in rank order
  float* owp = reinterpret_cast<float*>(wsm + L.owp);
  for (int g0 = 0; g0 < na; g0 += kWideGroup) {
    const int ng = min(kWideGroup, na - g0);
    float acc[kWideGroup][NP];
#pragma unroll
    for (int g = 0; g < kWideGroup; ++g)
#pragma unroll
      for (int k = 0; k < NP; ++k) acc[g][k] = 0.f;
    for (int mb = m0 + warp * kWideRows; mb < m1; mb += kWideWarps * kWideRows) {
      float vv[kWideRows][NP];
#pragma unroll
      for (int t = 0; t < kWideRows; ++t) {
        if (mb + t < m1) load_row<NP>(vbar + (int64_t)(mb + t) * D + lane * NP, vv[t]);
        else
#pragma unroll
          for (int k = 0; k < NP; ++k) vv[t][k] = 0.f;
      }
#pragma unroll
      for (int g = 0; g < kWideGroup; ++g) {
        if (g < ng) {
#pragma unroll
          for (int t = 0; t < kWideRows; ++t) {
            const float w = mb + t < m1 ? pl[(g0 + g) * mr + (mb + t - m0)] : 0.f;
#pragma unroll
            for (int k = 0; k < NP; ++k) acc[g][k] = fmaf(w, vv[t][k], acc[g][k]);
          }
        }
      }
    }
#pragma unroll
    for (int g = 0; g < kWideGroup; ++g)
#pragma unroll
      for (int k = 0; k < NP; ++k) owp[(warp * kWideGroup + g) * HD + lane * NP + k] = acc[g][k];
    __syncthreads();
    for (int e = tid; e < ng * HD; e += kWideThreads) {
      const int g = e / HD, c = e - g * HD;
      float t = 0.f;
      for (int w = 0; w < kWideWarps; ++w) t += owp[(w * kWideGroup + g) * HD + c];
      obp[(g0 + g) * HD + c] = t;
    }
    __syncthreads();
  }
  cluster_sync_all();
  for (int e = tid; e < na * HD; e += kWideThreads) {
    float t = 0.f;
    for (int r = 0; r < cl; ++r) t += ld_dsmem(obp + e, (uint32_t)r);
    ob[e] = t;
  }
  __syncthreads();
  // delta_{i,m} = pi/(1 - pi + eps) (o_bar_i - v_bar_m);  u = delta^T G delta  (Eq. omission)
  if (a.mode == CAST_ROUTE_OMISSION && a.gram == nullptr) {
    for (int mb = m0 + warp * kWideRows; mb < m1; mb += kWideWarps * kWideRows) {
      float vv[kWideRows][NP];
#pragma unroll
      for (int t = 0; t < kWideRows; ++t) {
        if (mb + t < m1) load_row<NP>(vbar + (int64_t)(mb + t) * D + lane * NP, vv[t]);
        else
#pragma unroll
          for (int k = 0; k < NP; ++k) vv[t][k] = 0.f;
      }
      for (int i = 0; i < na; ++i) {
        float ov[NP], acc[kWideRows];
#pragma unroll
        for (int k = 0; k < NP; ++k) ov[k] = ob[i * HD + lane * NP + k];
#pragma unroll
        for (int t = 0; t < kWideRows; ++t) {
          acc[t] = 0.f;
#pragma unroll
          for (int k = 0; k < NP; ++k) {
            const float df = ov[k] - vv[t][k];
            acc[t] = fmaf(df, df, acc[t]);
          }
        }
        const float tot = warp_sum8(acc);   // row (lane >> 2) & 7 of the batch
        const int t = (lane >> 2) & 7;
        if ((lane & 3) == 0 && mb + t < m1) {
          const int q = i * mr + (mb + t - m0);
          const float coef = pl[q] / (1.f - pl[q] + a.eps);
          pl[q] = coef * coef * tot;
        }
      }
    }
  } else if (a.mode == CAST_ROUTE_OMISSION) {
    float* e = ew + warp * HD;
    const float* Gm = a.gram + (int64_t)h * HD * HD;
    for (int m = m0 + warp; m < m1; m += kWideWarps) {
      for (int i = 0; i < na; ++i) {
        for (int c = lane; c < HD; c += 32) e[c] = ob[i * HD + c] - vbar[(int64_t)m * D + c];
        __syncwarp();
        float acc = 0.f;
        for (int r = lane; r < HD; r += 32) {
          float y = 0.f;
          for (int c = 0; c < HD; ++c) y = fmaf(Gm[(int64_t)r * HD + c], e[c], y);
          acc = fmaf(e[r], y, acc);
        }
        __syncwarp();
        acc = warp_sum(acc);
        if (lane == 0) {
          const int q = i * mr + (m - m0);
          const float coef = pl[q] / (1.f - pl[q] + a.eps);
          pl[q] = coef * coef * acc;
        }
      }
    }
  }
  __syncthreads();
  // every CTA pushes its keys into rank 0's u[na][M] (that space held o_bar partials, which
  // every CTA finished with before the last cluster barrier); the barrier below publishes them
  const float* keyl = a.mode == CAST_ROUTE_OMISSION ? pl : sl;   // the TopK key of Eq. (topk)
  float* u = reinterpret_cast<float*>(wsm + L.u);
  for (int e = tid; e < na * nm; e += kWideThreads) {
    const int i = e / nm, ml = e - i * nm;
    const float v = keyl[i * mr + ml];
    if (a.u_out) a.u_out[((int64_t)i * a.H + h) * M + m0 + ml] = v;
    if (K > 0) st_dsmem(u + i * M + m0 + ml, 0u, v);
  }
  cluster_sync_all();
  if (rank != 0 || K == 0) return;

  float* x = reinterpret_cast<float*>(wsm + L.x);
  float* G = reinterpret_cast<float*>(wsm + L.G);
  float* red2 = reinterpret_cast<float*>(wsm + L.red2);
  unsigned* hist = reinterpret_cast<unsigned*>(wsm + L.hist);
  unsigned long long* sel = reinterpret_cast<unsigned long long*>(wsm + L.pre);
  uint8_t* cm = restricted ? wsm + L.cm : nullptr;
  // candidate sets C_i (App. B.3): membership bytes; keys outside C_i count as -inf
  if (restricted) {
    for (int p = tid; p < na * M; p += kWideThreads) cm[p] = 0;
    __syncthreads();
    for (int e = tid; e < na * a.Mc; e += kWideThreads) {
      const int i = e / a.Mc, c = e - i * a.Mc;
      const int m = __ldg(a.cand + ((int64_t)i * a.H + h) * a.Mc + c);
      if (m < 0 || m >= M) atomicExch(&g_route_error, 1u);
      else cm[i * M + m] = 1;
    }
    __syncthreads();
    for (int i = warp; i < na; i += kWideWarps) {
      int n = 0;
      for (int m = lane; m < M; m += 32) n += cm[i * M + m];
      n = __reduce_add_sync(0xffffffffu, n);
      if (lane == 0 && n != a.Mc) atomicExch(&g_route_error, 1u);
    }
  }
  for (int e = tid; e < 2 * kRadixBins; e += kWideThreads) hist[e] = 0u;
  int slot = 0;
  __syncthreads();
  // initial masks: TopK of each anchor's key (Eq. topk), within C_i
  if (K >= M) {
    for (int p = tid; p < na * M; p += kWideThreads) x[p] = 1.f;
  } else {
    for (int i = 0; i < na; ++i) {
      const uint8_t* cmi = cm ? cm + i * M : nullptr;
      const unsigned long long t = topk_threshold(u + i * M, cmi, M, K, hist, sel);
      for (int m = tid; m < M; m += kWideThreads)
        x[i * M + m] = order_key(masked(u + i * M, cmi, m), m) >= t ? 1.f : 0.f;
    }
  }
  __syncthreads();
  if (refine) {
    // Alg. (routing) with the whole CTA: sq[j][m] = sqrt(u_{j-1,m} u_{j,m}); interval
    // coefficients A, B, C of Eq. (abc); boundary sets from the pairs (0, 1) and (na-2, na-1)
    float* sq = reinterpret_cast<float*>(wsm + L.sq);
    float* cA = reinterpret_cast<float*>(wsm + L.coef);
    float* cB = cA + na;
    float* cC = cA + 2 * na;
    for (int p = tid; p < na * M; p += kWideThreads)
      if (p >= M) sq[p] = sqrtf(u[p - M] * u[p]);
    for (int j = tid; j < na; j += kWideThreads) {
      cA[j] = a.A[j];
      cB[j] = a.B[j];
      cC[j] = a.C[j];
    }
    __syncthreads();
    const float AL = a.AL, BL = a.BL, CL = a.CL, AR = a.AR, BR = a.BR, CR = a.CR;
    const float lam_anc = a.lam_anc, lam_rec = a.lam_rec;
    float Jl = 0.f;
    for (int m = tid; m < M; m += kWideThreads) {
      for (int i = 0; i < na; ++i) Jl += lam_anc * (1.f - x[i * M + m]) * u[i * M + m];
      float rec = 0.f;
      for (int j = 1; j < na; ++j) {
        const float xp = 1.f - x[(j - 1) * M + m], xq = 1.f - x[j * M + m];
        rec += cA[j] * xp * u[(j - 1) * M + m] + cB[j] * xq * u[j * M + m] + 2.f * cC[j] * xp * xq * sq[j * M + m];
      }
      if (na >= 2) {
        const float x0 = 1.f - x[m], x1 = 1.f - x[M + m];
        rec += AL * x0 * u[m] + BL * x1 * u[M + m] + 2.f * CL * x0 * x1 * sq[M + m];
        const int r0 = (na - 2) * M + m, r1 = (na - 1) * M + m;
        const float y0 = 1.f - x[r0], y1 = 1.f - x[r1];
        rec += AR * y0 * u[r0] + BR * y1 * u[r1] + 2.f * CR * y0 * y1 * sq[r1];
      }
      Jl += lam_rec * rec;
    }
    float J = block_sum(Jl, red2, slot);
    for (int pass = 1; pass <= a.passes; ++pass) {
      bool changed = false;
      for (int step = 0; step < na; ++step) {
        const int i = (pass & 1) ? step : na - 1 - step;
        // retain gains, Eqs. (gain) and (boundarygain)
        for (int m = tid; m < M; m += kWideThreads) {
          const float ui = u[i * M + m];
          float rec = 0.f;
          if (i >= 1) rec += cB[i] * ui + 2.f * cC[i] * (1.f - x[(i - 1) * M + m]) * sq[i * M + m];
          if (i + 1 < na) rec += cA[i + 1] * ui + 2.f * cC[i + 1] * (1.f - x[(i + 1) * M + m]) * sq[(i + 1) * M + m];
          if (na >= 2) {
            if (i == 0) rec += AL * ui + 2.f * CL * (1.f - x[M + m]) * sq[M + m];
            if (i == 1) rec += BL * ui + 2.f * CL * (1.f - x[m]) * sq[M + m];
            if (i == na - 2) rec += AR * ui + 2.f * CR * (1.f - x[(na - 1) * M + m]) * sq[(na - 1) * M + m];
            if (i == na - 1) rec += BR * ui + 2.f * CR * (1.f - x[(na - 2) * M + m]) * sq[(na - 1) * M + m];
          }
          G[m] = lam_anc * ui + lam_rec * rec;
        }
        __syncthreads();
        // best response TopK(G) within C_i and its gain sum_m G_m (x_new - x_i); J is affine in
        // x_i, so the accepted step lowers J by exactly that gain
        const uint8_t* cmi = cm ? cm + i * M : nullptr;
        const unsigned long long thr = topk_threshold(G, cmi, M, K, hist, sel);
        float gl = 0.f;
        for (int m = tid; m < M; m += kWideThreads) {
          const float nx = order_key(masked(G, cmi, m), m) >= thr ? 1.f : 0.f;
          gl += G[m] * (nx - x[i * M + m]);
        }
        const float gain = block_sum(gl, red2, slot);
        if (gain > a.tol * fmaxf(J, 1e-8f)) {   // uniform across the CTA
          for (int m = tid; m < M; m += kWideThreads)
            x[i * M + m] = order_key(masked(G, cmi, m), m) >= thr ? 1.f : 0.f;
          J -= gain;
          changed = true;
        }
        __syncthreads();
      }
      if (!changed) break;
    }
  }
  __syncthreads();
  // ascending block indices of every anchor's mask
  for (int i = warp; i < na; i += kWideWarps) {
    int base = 0;
    int32_t* out = a.idx + ((int64_t)i * a.H + h) * K;
    for (int mb = 0; mb < M; mb += 32) {
      const int m = mb + lane;
      const bool on = m < M && x[i * M + m] != 0.f;
      const unsigned bal = __ballot_sync(0xffffffffu, on);
      if (on) out[base + __popc(bal & ((1u << lane) - 1u))] = m;
      base += __popc(bal);
    }
  }
}

// shared state of the single-CTA head kernel without the staged means
size_t head_state_bytes(const cast_route_args& a) {
  const bool restricted = a.candidates != nullptr;
  const size_t floats = (size_t)2 * a.n_anchors * a.d + (size_t)3 * a.n_anchors * a.M + (size_t)a.M +
                        (restricted ? (size_t)a.M : 0) + (size_t)kHeadWarps * a.d;
  return floats * sizeof(float) + (restricted ? align_up((size_t)a.n_anchors * a.M, 16) : 0);
}

constexpr size_t kHeadSmemLimit = 200 * 1024;
// the single-CTA head kernel holds k_bar and v_bar of its head in shared memory
size_t head_staged_bytes(const cast_route_args& a) {
  return align_up(head_state_bytes(a), 16) + (size_t)2 * a.M * a.d * sizeof(float);
}
bool head_stages_kv(const cast_route_args& a) { return a.M <= 1024 && head_staged_bytes(a) <= kHeadSmemLimit; }

size_t wide_bytes(const cast_route_args& a) {
  const int K_eff = a.K < a.M ? a.K : a.M;
  const int cl = wide_cluster(a.M);
  const int mr = (a.M + cl - 1) / cl;
  return wide_layout(a.n_anchors, a.M, a.d, mr, a.refine_passes > 0 && K_eff > 0 && K_eff < a.M,
                     a.candidates != nullptr).total;
}

}  // namespace

size_t route_head_smem_bytes(const cast_route_args& a) {
  return head_stages_kv(a) ? head_staged_bytes(a) : wide_bytes(a);
}

size_t route_pool_smem_bytes(const cast_route_args& a) {
  const int D = a.H * a.d;
  return (size_t)pool_shape(D, a.dtype == CAST_BF16 ? 2 : 4).lanes_r * D * sizeof(float);
}

RoutePlan route_plan(const cast_route_args& a) {
  RoutePlan p{};
  const int D = a.H * a.d;
  p.n_seg = a.n_anchors + 2 * a.M;
  // per launch (anchor frames, history blocks): a cluster of up to 8 CTAs per segment, enough
  // CTAs to cover the SMs a few times, each streaming >= 64 rows
  int dev = 0, nsm = 148;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  const int target = 4 * (nsm > 0 ? nsm : 148);
  auto splits = [&](int n_seg, int rows) {
    int ns = n_seg > 0 ? (target + n_seg - 1) / n_seg : 1;
    if (ns > kMaxClusterSplit) ns = kMaxClusterSplit;
    while (ns > 1 && (rows + ns - 1) / ns < 64) --ns;
    return ns < 1 ? 1 : ns;
  };
  p.nsplit_q = splits(a.n_anchors, a.S);
  p.nsplit_kv = splits(2 * a.M, a.B_v);
  p.wide = a.M > 0 && !head_stages_kv(a);
  p.cl = p.wide ? wide_cluster(a.M) : 1;
  p.pooled_bytes = align_up((size_t)p.n_seg * D * sizeof(float));
  p.total_bytes = p.pooled_bytes;
  return p;
}

cast_status launch_route(const cast_route_args& a, void* ws, cudaStream_t st) {
  const RoutePlan p = route_plan(a);
  const int D = a.H * a.d;
  const int K_eff = a.K < a.M ? a.K : a.M;
  if (a.M == 0) return CAST_OK;   // nothing to route (App. B.3 bypass)
  float* pooled = static_cast<float*>(ws);
  float* qbar = a.qbar ? a.qbar : pooled;
  float* kbar = a.kbar ? a.kbar : pooled + (size_t)a.n_anchors * D;
  float* vbar = a.vbar ? a.vbar : pooled + (size_t)(a.n_anchors + a.M) * D;

  PoolArgs pa;
  pa.q = static_cast<const char*>(a.q);
  pa.k = static_cast<const char*>(a.k_hist);
  pa.v = static_cast<const char*>(a.v_hist);
  pa.qbar = qbar;
  pa.kbar = kbar;
  pa.vbar = vbar;
  pa.q_row_stride = a.q_row_stride;
  pa.hist_row_stride = a.hist_row_stride;
  pa.n_anchors = a.n_anchors;
  pa.M = a.M;
  pa.S = a.S;
  pa.B_v = a.B_v;
  pa.D = D;
  pa.elt = a.dtype == CAST_BF16 ? 2 : 4;
  const HistGeom hg = hist_geom(a.hist);
  pa.Hg = hg.Hg;
  pa.Wg = hg.Wg;
  pa.nby = hg.nby;
  pa.nbx = hg.nbx;
  for (int k = 0; k < a.n_anchors; ++k) pa.anchors[k] = a.anchors[k];

  const size_t psm = route_pool_smem_bytes(a);
  const PoolShape ps = pool_shape(D, pa.elt);
  const int row_bytes = D * pa.elt;
  // two launches of the pooling kernel, each with its own row split: the history blocks (the
  // larger part), then, as a programmatic dependent that fills the remaining SMs, the anchor
  // frames (few long segments; it completes only after the first, see k_pool).  A part whose
  // rows are contiguous (row stride D), whose column groups fit one per thread and whose CTAs
  // stream at least kPoolBulkMinBytes each is pooled through the bulk-copy ring.
  for (int part = 0; part < 2; ++part) {
    const bool hist = part == 0;
    const int nsplit = hist ? p.nsplit_kv : p.nsplit_q;
    const bool contiguous = hist ? (!hg.spatial && a.hist_row_stride == D) : a.q_row_stride == D;
    const int rows = hist ? a.B_v : a.S;
    const int64_t cta_bytes = (int64_t)((rows + nsplit - 1) / nsplit) * row_bytes;
    const bool bulk = contiguous && ps.cgs * (16 / pa.elt) == D && row_bytes <= kPoolStageBytes &&
                      cta_bytes >= kPoolBulkMinBytes;
    pa.nsplit = nsplit;
    pa.seg_base = hist ? a.n_anchors : 0;
    pa.bulk_rows = bulk ? kPoolStageBytes / row_bytes : 0;
    const size_t smem = bulk ? pool_ring_offset(ps.lanes_r, D) + (size_t)kPoolStages * pa.bulk_rows * row_bytes : psm;
    void (*fn)(PoolArgs);
    if (a.dtype == CAST_BF16)
      fn = bulk ? k_pool<__nv_bfloat16, false, true>
                : (hist && hg.spatial ? k_pool<__nv_bfloat16, true, false> : k_pool<__nv_bfloat16, false, false>);
    else
      fn = bulk ? k_pool<float, false, true> : (hist && hg.spatial ? k_pool<float, true, false> : k_pool<float, false, false>);
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
      return fail(CAST_ERR_CUDA, "routing: cannot reserve %zu B of shared memory for pooling", smem);
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(nsplit, hist ? 2 * a.M : a.n_anchors, 1);
    cfg.blockDim = dim3(ps.cgs * ps.lanes_r, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = nsplit;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = part == 0 ? 1 : 2;
    if (cudaLaunchKernelEx(&cfg, fn, pa) != cudaSuccess) return check_launch("routing pool kernel");
    const cast_status s = check_launch("routing pool kernel");
    if (s != CAST_OK) return s;
  }

  HeadArgs ha{};
  ha.qbar = qbar;
  ha.kbar = kbar;
  ha.vbar = vbar;
  ha.gram = a.gram;
  ha.cand = a.candidates;
  ha.Mc = a.candidates ? a.M_c : a.M;
  ha.idx = a.idx;
  ha.u_out = a.u;
  ha.H = a.H;
  ha.d = a.d;
  ha.M = a.M;
  ha.n_anchors = a.n_anchors;
  ha.K_eff = K_eff;
  ha.mode = a.mode;
  ha.passes = a.refine_passes;
  ha.eps = a.eps;
  ha.lam_anc = a.lambda_anc;
  ha.lam_rec = a.lambda_rec;
  ha.tol = a.refine_tol;
  if (a.refine_passes > 0) {
    // interval and boundary coefficients of the anchor layout (Eqs. abc, boundarycoeff) with
    // the alpha of Eq. (block)
    for (int j = 1; j < a.n_anchors; ++j) {
      const int x0 = a.anchors[j - 1], x1 = a.anchors[j];
      double A = 0, B = 0, C = 0;
      for (int t = x0 + 1; t < x1; ++t) {
        const double al = (double)(t - x0) / (double)(x1 - x0);
        A += (1 - al) * (1 - al);
        B += al * al;
        C += al * (1 - al);
      }
      ha.A[j] = (float)A;
      ha.B[j] = (float)B;
      ha.C[j] = (float)C;
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
      bset(a.anchors[0], a.anchors[1], 0, a.anchors[0], ha.AL, ha.BL, ha.CL);
      bset(a.anchors[a.n_anchors - 2], a.anchors[a.n_anchors - 1], a.anchors[a.n_anchors - 1] + 1,
           a.n_frames, ha.AR, ha.BR, ha.CR);
    }
  }
  // the small per-head kernel for the common case; the staged or wide kernel otherwise
  const bool small = !p.wide && a.gram == nullptr && a.candidates == nullptr && a.M <= kSmallMaxM &&
                     a.n_anchors <= kSmallMaxAnchors;
  const size_t hsm = small ? small_head_bytes(a) : route_head_smem_bytes(a);
  auto head_fn = small ? (a.d == 128 ? k_head_small<128> : k_head_small<64>)
                       : !p.wide ? k_head : (a.d == 128 ? k_head_wide<128> : k_head_wide<64>);
  if (hsm > 48 * 1024 &&
      cudaFuncSetAttribute(head_fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)hsm) != cudaSuccess)
    return fail(CAST_ERR_CUDA, "routing: cannot reserve %zu B of shared memory", hsm);
  cudaLaunchConfig_t hc{};
  hc.gridDim = p.wide ? dim3(p.cl, a.H, 1) : dim3(a.H, 1, 1);
  hc.blockDim = dim3(p.wide ? kWideThreads : kHeadThreads, 1, 1);
  hc.dynamicSmemBytes = hsm;
  hc.stream = st;
  cudaLaunchAttribute hat[2];
  hat[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  hat[0].val.programmaticStreamSerializationAllowed = 1;
  hat[1].id = cudaLaunchAttributeClusterDimension;
  hat[1].val.clusterDim.x = p.cl;
  hat[1].val.clusterDim.y = 1;
  hat[1].val.clusterDim.z = 1;
  hc.attrs = hat;
  hc.numAttrs = p.wide ? 2 : 1;
  if (cudaLaunchKernelEx(&hc, head_fn, ha) != cudaSuccess) return check_launch("routing head kernel");
  return check_launch("routing head kernel");
}

unsigned int route_error_word(cudaStream_t st, bool clear) {
  unsigned int v = 0, vp = 0;
  cudaMemcpyFromSymbolAsync(&v, g_route_error, sizeof(v), 0, cudaMemcpyDeviceToHost, st);
  cudaMemcpyFromSymbolAsync(&vp, g_pool_error, sizeof(vp), 0, cudaMemcpyDeviceToHost, st);
  cudaStreamSynchronize(st);
  if (clear && (v || vp)) {
    const unsigned int z = 0;
    cudaMemcpyToSymbolAsync(g_route_error, &z, sizeof(z), 0, cudaMemcpyHostToDevice, st);
    cudaMemcpyToSymbolAsync(g_pool_error, &z, sizeof(z), 0, cudaMemcpyHostToDevice, st);
    cudaStreamSynchronize(st);
  }
  return vp ? 2u : v;   // 2: a pooling wait gave up; 1: a candidate index outside [0, M) or repeated
}

}  // namespace cast
