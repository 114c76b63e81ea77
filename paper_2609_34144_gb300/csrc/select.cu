// Control-aware frame selection (Section 3, Eqs. sensitivity, debt, score; App. B.1 Eq.
// normalization).
//
//   K_sumsq  : sum of squares of every frame's control update, the frame split over several
//              CTAs (HBM-bound: one read of n_branch * N_cur * S * D elements, 16-byte loads);
//              each CTA writes one partial sum.
//   K_select : one CTA, one thread per frame: r = sqrt(sum / (S D)) summed over the splits in
//              order (deterministic), min-max normalisation per branch, d, refresh ages, debt,
//              scores, and the TopK_f by rank (ties to the lower frame index), written in
//              ascending frame order.  Launched as a programmatic dependent of K_sumsq.
#include <cuda_bf16.h>

#include <cfloat>
#include <cmath>

#include "internal.h"

namespace cast {
namespace {

constexpr int kSumThreads = 256;
constexpr int kUnroll = 8;

struct SumArgs {
  const char* delta[CAST_MAX_BRANCHES];
  int64_t frame_elems;
  int n_frames, nsplit, elt;
  float* partial;   // [branch][frame][split]
};

__device__ __forceinline__ float sumsq16(const char* p, int elt) {
  if (elt == 4) {
    const float4 v = __ldcs(reinterpret_cast<const float4*>(p));
    return fmaf(v.x, v.x, fmaf(v.y, v.y, fmaf(v.z, v.z, v.w * v.w)));
  }
  const uint4 v = __ldcs(reinterpret_cast<const uint4*>(p));
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  float acc = 0.f;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float lo = __uint_as_float(w[k] << 16), hi = __uint_as_float(w[k] & 0xFFFF0000u);
    acc = fmaf(lo, lo, fmaf(hi, hi, acc));
  }
  return acc;
}

// grid (nsplit, n_frames, n_branch): CTA (s, i, k) sums the squares of its slice of frame i
// of branch k in 16-byte groups, eight loads in flight per thread.
__global__ void __launch_bounds__(kSumThreads) k_sumsq(const __grid_constant__ SumArgs a) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int split = blockIdx.x, i = blockIdx.y, k = blockIdx.z;
  const int64_t groups = a.frame_elems * a.elt / 16;            // 16-byte groups per frame
  const int64_t per = (groups + a.nsplit - 1) / a.nsplit;
  const int64_t g0 = split * per, g1 = min(groups, g0 + per);
  const char* base = a.delta[k] + (int64_t)i * a.frame_elems * a.elt;
  float acc[2] = {0.f, 0.f};
  int64_t g = g0 + threadIdx.x;
  for (; g + (int64_t)(kUnroll - 1) * kSumThreads < g1; g += (int64_t)kUnroll * kSumThreads) {
    float v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) v[u] = sumsq16(base + (g + (int64_t)u * kSumThreads) * 16, a.elt);
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) acc[u & 1] += v[u];
  }
  for (; g < g1; g += kSumThreads) acc[0] += sumsq16(base + g * 16, a.elt);
  float s = acc[0] + acc[1];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  __shared__ float red[kSumThreads / 32];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < kSumThreads / 32; ++w) t += red[w];
    a.partial[((int64_t)k * a.n_frames + i) * a.nsplit + split] = t;
  }
}

struct SelectArgs {
  const float* partial;
  const int32_t* ages;
  const uint8_t* anchor_mask;
  int32_t* ages_out;
  int32_t* anchors_out;
  uint8_t* mask_out;
  float* rms_out;
  float* score_out;
  int64_t frame_elems;
  int n_frames, n_branch, nsplit, K_f;
  float lambda_cov, eps;
};

constexpr int kSelectThreads = CAST_MAX_FRAMES;

__device__ __forceinline__ float block_min_max(float v, bool want_max, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float w = __shfl_xor_sync(0xffffffffu, v, o);
    v = want_max ? fmaxf(v, w) : fminf(v, w);
  }
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = red[0];
  for (int w = 1; w < kSelectThreads / 32; ++w) t = want_max ? fmaxf(t, red[w]) : fminf(t, red[w]);
  return t;
}

__global__ void __launch_bounds__(kSelectThreads) k_select(const __grid_constant__ SelectArgs a) {
  __shared__ float red[kSelectThreads / 32];
  __shared__ float s_score[CAST_MAX_FRAMES];
  __shared__ int s_sel[CAST_MAX_FRAMES];
  asm volatile("griddepcontrol.wait;" ::: "memory");   // the partial sums of K_sumsq
  const int i = threadIdx.x, N = a.n_frames;
  const bool live = i < N;
  // Eq. (sensitivity) with Eq. (normalization) per branch
  float d = 0.f;
  for (int k = 0; k < a.n_branch; ++k) {
    float r = 0.f;
    if (live) {
      const float* p = a.partial + ((int64_t)k * N + i) * a.nsplit;
      float s = 0.f;
      for (int q = 0; q < a.nsplit; ++q) s += p[q];
      r = sqrtf(s / (float)a.frame_elems);
      if (a.rms_out) a.rms_out[(int64_t)k * N + i] = r;
    }
    const float rmin = block_min_max(live ? r : FLT_MAX, false, red);
    const float rmax = block_min_max(live ? r : -FLT_MAX, true, red);
    d += (r - rmin) / (rmax - rmin + a.eps);
  }
  if (a.n_branch > 0) d /= (float)a.n_branch;
  // Eqs. (debt), (score)
  int h = 0;
  float S = -FLT_MAX;
  if (live) {
    h = a.anchor_mask[i] ? 0 : a.ages[i] + 1;
    const int h_cov = (N + a.K_f - 1) / a.K_f;
    const float D = (float)h / (float)h_cov;
    S = (a.n_branch > 0 ? d : 0.f) + a.lambda_cov * D;
    s_score[i] = S;
  }
  __syncthreads();
  // TopK_f by rank: frames with a larger score, or an equal one at a lower index, come first
  const int K = a.K_f < N ? a.K_f : N;
  bool sel = false;
  if (live) {
    int rank = 0;
    for (int j = 0; j < N; ++j) {
      const float w = s_score[j];
      rank += (w > S) || (w == S && j < i);
    }
    sel = rank < K;
    s_sel[i] = sel ? 1 : 0;
  }
  __syncthreads();
  if (live) {
    int pos = 0;   // selected frames below i: position in the ascending list
    for (int j = 0; j < i; ++j) pos += s_sel[j];
    if (sel) a.anchors_out[pos] = i;
    a.ages_out[i] = h;
    if (a.mask_out) a.mask_out[i] = sel ? 1 : 0;
    if (a.score_out) a.score_out[i] = S;
  }
}

int sum_splits(const cast_select_args& a) {
  const int64_t groups = a.frame_elems * (a.dtype == CAST_BF16 ? 2 : 4) / 16;
  int dev = 0, nsm = 148;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  const int units = a.n_branch * a.n_frames;
  int nsplit = (4 * (nsm > 0 ? nsm : 148) + units - 1) / (units > 0 ? units : 1);
  // at least 64 KB per CTA
  const int64_t max_split = groups / 4096 > 0 ? groups / 4096 : 1;
  if (nsplit > max_split) nsplit = (int)max_split;
  return nsplit < 1 ? 1 : nsplit;
}

cast_status validate_select(const cast_select_args* a) {
  const char* who = "cast_select_frames";
  if (!a) return fail(CAST_ERR_INVALID_ARG, "%s: args is NULL", who);
  if (a->n_frames < 1 || a->n_frames > CAST_MAX_FRAMES)
    return fail(CAST_ERR_INVALID_ARG, "%s: n_frames %d outside 1..%d", who, a->n_frames, CAST_MAX_FRAMES);
  if (a->K_f < 1) return fail(CAST_ERR_INVALID_ARG, "%s: K_f %d < 1", who, a->K_f);
  if (a->n_branch < 0 || a->n_branch > CAST_MAX_BRANCHES)
    return fail(CAST_ERR_INVALID_ARG, "%s: n_branch %d outside 0..%d", who, a->n_branch, CAST_MAX_BRANCHES);
  if (a->dtype != CAST_F32 && a->dtype != CAST_BF16)
    return fail(CAST_ERR_INVALID_ARG, "%s: dtype %d", who, a->dtype);
  const int elt = a->dtype == CAST_BF16 ? 2 : 4;
  if (a->n_branch > 0) {
    if (a->frame_elems < 1 || (a->frame_elems * elt) % 16 != 0)
      return fail(CAST_ERR_INVALID_ARG, "%s: frame_elems %lld (x %d bytes) not a positive multiple of 16 bytes",
                  who, (long long)a->frame_elems, elt);
    for (int k = 0; k < a->n_branch; ++k)
      if (!a->delta[k] || reinterpret_cast<uintptr_t>(a->delta[k]) % 16)
        return fail(CAST_ERR_INVALID_ARG, "%s: delta[%d] NULL or not 16-byte aligned", who, k);
  }
  if (!a->ages || !a->anchor_mask || !a->ages_out || !a->anchors_out)
    return fail(CAST_ERR_INVALID_ARG, "%s: ages, anchor_mask, ages_out and anchors_out are required", who);
  if (!(a->lambda_cov >= 0.f) || !(a->eps >= 0.f))
    return fail(CAST_ERR_INVALID_ARG, "%s: lambda_cov and eps must be >= 0", who);
  return CAST_OK;
}

size_t select_workspace(const cast_select_args& a) {
  if (a.n_branch == 0) return 0;
  return align_up((size_t)a.n_branch * a.n_frames * sum_splits(a) * sizeof(float));
}

}  // namespace
}  // namespace cast

using namespace cast;

extern "C" {

size_t cast_select_workspace_size(const cast_select_args* a) {
  if (!a || a->n_frames < 1 || a->n_frames > CAST_MAX_FRAMES || a->n_branch < 0 ||
      a->n_branch > CAST_MAX_BRANCHES)
    return 0;
  return select_workspace(*a);
}

cast_status cast_select_frames(const cast_select_args* a, void* ws, size_t ws_bytes, void* stream) {
  clear_error_detail();
  cast_status s = validate_select(a);
  if (s) return s;
  const size_t need = select_workspace(*a);
  if (ws_bytes < need || (need && !ws))
    return fail(CAST_ERR_INVALID_ARG, "cast_select_frames: workspace %zu B < %zu B", ws_bytes, need);
  if (reinterpret_cast<uintptr_t>(ws) % kWsAlign)
    return fail(CAST_ERR_INVALID_ARG, "cast_select_frames: workspace not 256-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int nsplit = a->n_branch > 0 ? sum_splits(*a) : 1;
  float* partial = static_cast<float*>(ws);
  if (a->n_branch > 0) {
    SumArgs sa{};
    for (int k = 0; k < a->n_branch; ++k) sa.delta[k] = static_cast<const char*>(a->delta[k]);
    sa.frame_elems = a->frame_elems;
    sa.n_frames = a->n_frames;
    sa.nsplit = nsplit;
    sa.elt = a->dtype == CAST_BF16 ? 2 : 4;
    sa.partial = partial;
    k_sumsq<<<dim3(nsplit, a->n_frames, a->n_branch), kSumThreads, 0, st>>>(sa);
    if ((s = check_launch("frame-selection sum-of-squares kernel"))) return s;
  }
  SelectArgs ka{};
  ka.partial = partial;
  ka.ages = a->ages;
  ka.anchor_mask = a->anchor_mask;
  ka.ages_out = a->ages_out;
  ka.anchors_out = a->anchors_out;
  ka.mask_out = a->mask_out;
  ka.rms_out = a->rms_out;
  ka.score_out = a->score_out;
  ka.frame_elems = a->frame_elems;
  ka.n_frames = a->n_frames;
  ka.n_branch = a->n_branch;
  ka.nsplit = nsplit;
  ka.K_f = a->K_f;
  ka.lambda_cov = a->lambda_cov;
  ka.eps = a->eps;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(1, 1, 1);
  cfg.blockDim = dim3(kSelectThreads, 1, 1);
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, k_select, ka) != cudaSuccess) return check_launch("frame-selection kernel");
  return check_launch("frame-selection kernel");
}

}  // extern "C"
