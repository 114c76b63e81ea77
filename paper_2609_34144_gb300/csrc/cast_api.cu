// C ABI of libcast: argument validation, workspace sizing and dispatch to the kernels.
// Every entry point validates before launching anything; on an error it returns a status,
// records a message for cast_last_error_detail() and writes nothing.
#include <cuda_bf16.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "internal.h"

namespace cast {

static thread_local char g_detail[512] = "";

void clear_error_detail() { g_detail[0] = 0; }

cast_status fail(cast_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_detail, sizeof(g_detail), fmt, ap);
  va_end(ap);
  return s;
}

EncodeTiledFn tensor_map_encoder() {
  // looked up once per process (thread-safe static initialisation)
  static const EncodeTiledFn fn = []() -> EncodeTiledFn {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<EncodeTiledFn>(ptr);
    return nullptr;
  }();
  return fn;
}

cast_status check_launch(const char* what) {
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(CAST_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
  return CAST_OK;
}

namespace {

__global__ void k_residual_add_f32(float* __restrict__ x, const float* __restrict__ r, size_t n) {
  size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  const size_t n4 = n / 4;
  for (size_t k = i; k < n4; k += stride) {
    float4 a = reinterpret_cast<float4*>(x)[k];
    const float4 b = __ldcs(reinterpret_cast<const float4*>(r) + k);
    a.x += b.x; a.y += b.y; a.z += b.z; a.w += b.w;
    reinterpret_cast<float4*>(x)[k] = a;
  }
  for (size_t k = n4 * 4 + i; k < n; k += stride) x[k] += r[k];
}

__global__ void k_residual_add_bf16(__nv_bfloat16* __restrict__ x,
                                    const __nv_bfloat16* __restrict__ r, size_t n) {
  size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  for (size_t k = i; k < n / 2; k += stride) {
    __nv_bfloat162 a = reinterpret_cast<__nv_bfloat162*>(x)[k];
    const __nv_bfloat162 b = reinterpret_cast<const __nv_bfloat162*>(r)[k];
    const float2 fa = __bfloat1622float2(a), fb = __bfloat1622float2(b);
    reinterpret_cast<__nv_bfloat162*>(x)[k] = __floats2bfloat162_rn(fa.x + fb.x, fa.y + fb.y);
  }
  if (i == 0 && (n & 1))
    x[n - 1] = __float2bfloat16_rn(__bfloat162float(x[n - 1]) + __bfloat162float(r[n - 1]));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

cast_status validate_anchors(const int32_t* anchors, int n_anchors, int n_frames, const char* who) {
  if (!anchors) return fail(CAST_ERR_INVALID_ARG, "%s: anchors is NULL", who);
  if (n_anchors < 1 || n_anchors > CAST_MAX_ANCHORS)
    return fail(CAST_ERR_INVALID_ARG, "%s: n_anchors=%d outside 1..%d", who, n_anchors,
                CAST_MAX_ANCHORS);
  for (int k = 0; k < n_anchors; ++k) {
    if (anchors[k] < 0 || anchors[k] >= n_frames)
      return fail(CAST_ERR_INVALID_ARG, "%s: anchor %d = %d outside [0, %d)", who, k, anchors[k],
                  n_frames);
    if (k > 0 && anchors[k] <= anchors[k - 1])
      return fail(CAST_ERR_INVALID_ARG, "%s: anchors must be strictly ascending", who);
  }
  return CAST_OK;
}

cast_status validate_tokens(const void* p, int64_t row_stride, int H, int d, const char* name,
                            const char* who) {
  if (!p) return fail(CAST_ERR_INVALID_ARG, "%s: %s is NULL", who, name);
  if (!aligned16(p)) return fail(CAST_ERR_INVALID_ARG, "%s: %s is not 16-byte aligned", who, name);
  if (row_stride < (int64_t)H * d || row_stride % 8 != 0)
    return fail(CAST_ERR_INVALID_ARG, "%s: %s row stride %lld must be >= H*d and a multiple of 8",
                who, name, (long long)row_stride);
  return CAST_OK;
}

// History layout (App. B.5 Tab. config): CAST_HIST_FRAMES needs a positive grid, M equal to
// its (1, 8, 8) block count and the nominal block size B_v = 64.
cast_status validate_hist(const cast_hist_layout& h, int M, int B_v, const char* who) {
  if (h.kind == CAST_HIST_BLOCKS) return CAST_OK;
  if (h.kind != CAST_HIST_FRAMES) return fail(CAST_ERR_INVALID_ARG, "%s: hist.kind %d", who, h.kind);
  if (h.frames < 1 || h.Hg < 1 || h.Wg < 1)
    return fail(CAST_ERR_INVALID_ARG, "%s: history grid %d x %d x %d must be positive", who, h.frames,
                h.Hg, h.Wg);
  if ((int64_t)h.frames * h.Hg * h.Wg >= (1LL << 31))
    return fail(CAST_ERR_UNSUPPORTED, "%s: history of %lld tokens", who,
                (long long)h.frames * h.Hg * h.Wg);
  const HistGeom g = hist_geom(h);
  if (g.blocks() != M)
    return fail(CAST_ERR_INVALID_ARG, "%s: M=%d but the history frames hold %lld (1,8,8) blocks", who, M,
                (long long)g.blocks());
  if (B_v != kSpatialBlock * kSpatialBlock)
    return fail(CAST_ERR_INVALID_ARG, "%s: B_v=%d with (1,8,8) blocks (must be 64)", who, B_v);
  return CAST_OK;
}

cast_status validate_route(const cast_route_args* a) {
  const char* who = "cast_route_topk";
  if (!a) return fail(CAST_ERR_INVALID_ARG, "%s: args is NULL", who);
  if (a->dtype != CAST_BF16 && a->dtype != CAST_F32)
    return fail(CAST_ERR_INVALID_ARG, "%s: dtype %d", who, a->dtype);
  if (a->d != 64 && a->d != 128) return fail(CAST_ERR_UNSUPPORTED, "%s: head dim %d (64 or 128)", who, a->d);
  if (a->n_frames < 1 || a->S < 1 || a->H < 1)
    return fail(CAST_ERR_INVALID_ARG, "%s: n_frames, S, H must be positive", who);
  if (a->M < 0 || a->K < 0) return fail(CAST_ERR_INVALID_ARG, "%s: M and K must be >= 0", who);
  if (a->M > 0 && a->B_v < 1) return fail(CAST_ERR_INVALID_ARG, "%s: B_v must be >= 1", who);
  if (a->M > 16384) return fail(CAST_ERR_UNSUPPORTED, "%s: M=%d above 16384", who, a->M);
  cast_status s = validate_anchors(a->anchors, a->n_anchors, a->n_frames, who);
  if (s) return s;
  if ((s = validate_hist(a->hist, a->M, a->B_v, who))) return s;
  s = validate_tokens(a->q, a->q_row_stride, a->H, a->d, "q", who);
  if (s) return s;
  if (a->M > 0) {
    if ((s = validate_tokens(a->k_hist, a->hist_row_stride, a->H, a->d, "k_hist", who))) return s;
    if ((s = validate_tokens(a->v_hist, a->hist_row_stride, a->H, a->d, "v_hist", who))) return s;
    if (!a->idx && a->K > 0) return fail(CAST_ERR_INVALID_ARG, "%s: idx is NULL", who);
  }
  if (a->mode != CAST_ROUTE_OMISSION && a->mode != CAST_ROUTE_SIMILARITY)
    return fail(CAST_ERR_INVALID_ARG, "%s: mode %d", who, a->mode);
  for (const float* p : {a->qbar, a->kbar, a->vbar})
    if (reinterpret_cast<uintptr_t>(p) % 16)
      return fail(CAST_ERR_INVALID_ARG, "%s: qbar/kbar/vbar must be 16-byte aligned", who);
  if (!(a->eps >= 0.f)) return fail(CAST_ERR_INVALID_ARG, "%s: eps must be >= 0", who);
  if (a->refine_passes < 0) return fail(CAST_ERR_INVALID_ARG, "%s: refine_passes < 0", who);
  if (a->refine_passes > 0) {
    if (a->mode != CAST_ROUTE_OMISSION)
      return fail(CAST_ERR_INVALID_ARG, "%s: refinement needs CAST_ROUTE_OMISSION", who);
    if (!(a->lambda_anc >= 0.f) || !(a->lambda_rec >= 0.f) || !(a->refine_tol >= 0.f))
      return fail(CAST_ERR_INVALID_ARG, "%s: refinement weights and tolerance must be >= 0", who);
  }
  if (a->candidates) {
    const int keff = a->K < a->M ? a->K : a->M;
    if (a->M_c < 1 || a->M_c < keff || a->M_c > a->M)
      return fail(CAST_ERR_INVALID_ARG, "%s: candidate sets of M_c=%d blocks need %d <= M_c <= M=%d", who,
                  a->M_c, keff, a->M);
    if (reinterpret_cast<uintptr_t>(a->candidates) % 4)
      return fail(CAST_ERR_INVALID_ARG, "%s: candidates misaligned", who);
  }
  if (route_pool_smem_bytes(*a) > 200 * 1024)
    return fail(CAST_ERR_UNSUPPORTED, "%s: H*d = %d channels exceed the pooling kernel's shared memory",
                who, a->H * a->d);
  if (a->M > 0 && route_head_smem_bytes(*a) > 200 * 1024)
    return fail(CAST_ERR_UNSUPPORTED, "%s: %d anchors x %d blocks exceed the per-head shared memory",
                who, a->n_anchors, a->M);
  return CAST_OK;
}

cast_status validate_attn(const cast_attn_args* a) {
  const char* who = "cast_anchor_attention";
  if (!a) return fail(CAST_ERR_INVALID_ARG, "%s: args is NULL", who);
  if (a->d != 64 && a->d != 128) return fail(CAST_ERR_UNSUPPORTED, "%s: head dim %d (64 or 128)", who, a->d);
  if (a->n_frames < 1 || a->S < 1 || a->H < 1)
    return fail(CAST_ERR_INVALID_ARG, "%s: n_frames, S, H must be positive", who);
  if ((int64_t)a->n_frames * a->S >= (1LL << 31))
    return fail(CAST_ERR_UNSUPPORTED, "%s: chunk of %lld tokens", who, (long long)a->n_frames * a->S);
  if (a->M < 0 || a->K_eff < 0) return fail(CAST_ERR_INVALID_ARG, "%s: M and K_eff must be >= 0", who);
  if (a->K_eff > 0 && a->M == 0) return fail(CAST_ERR_INVALID_ARG, "%s: K_eff > 0 with M == 0", who);
  if (a->K_eff > a->M) return fail(CAST_ERR_INVALID_ARG, "%s: K_eff %d > M %d", who, a->K_eff, a->M);
  if (a->M > 0 && a->B_v < 1) return fail(CAST_ERR_INVALID_ARG, "%s: B_v must be >= 1", who);
  cast_status s = validate_anchors(a->anchors, a->n_anchors, a->n_frames, who);
  if (s) return s;
  if ((s = validate_hist(a->hist, a->M, a->B_v, who))) return s;
  if ((s = validate_tokens(a->q, a->q_row_stride, a->H, a->d, "q", who))) return s;
  if ((s = validate_tokens(a->k_cur, a->cur_row_stride, a->H, a->d, "k_cur", who))) return s;
  if ((s = validate_tokens(a->v_cur, a->cur_row_stride, a->H, a->d, "v_cur", who))) return s;
  if (a->M > 0) {
    if ((s = validate_tokens(a->k_hist, a->hist_row_stride, a->H, a->d, "k_hist", who))) return s;
    if ((s = validate_tokens(a->v_hist, a->hist_row_stride, a->H, a->d, "v_hist", who))) return s;
  }
  if (a->K_eff > 0 && !a->idx) return fail(CAST_ERR_INVALID_ARG, "%s: idx is NULL", who);
  if (!a->o || !aligned16(a->o)) return fail(CAST_ERR_INVALID_ARG, "%s: o is NULL or misaligned", who);
  if (a->o_dtype != CAST_BF16 && a->o_dtype != CAST_F32)
    return fail(CAST_ERR_INVALID_ARG, "%s: o_dtype %d", who, a->o_dtype);
  if (!(std::isfinite(a->scale))) return fail(CAST_ERR_INVALID_ARG, "%s: scale is not finite", who);
  return CAST_OK;
}

cast_status validate_par(const cast_par_args* a) {
  const char* who = "cast_par_reconstruct";
  if (!a) return fail(CAST_ERR_INVALID_ARG, "%s: args is NULL", who);
  if (a->dtype != CAST_BF16 && a->dtype != CAST_F32)
    return fail(CAST_ERR_INVALID_ARG, "%s: dtype %d", who, a->dtype);
  if (a->F < 1 || a->F > CAST_MAX_FRAMES || a->Hg < 1 || a->Wg < 1 || a->C < 1)
    return fail(CAST_ERR_INVALID_ARG, "%s: bad shape F=%d Hg=%d Wg=%d C=%d", who, a->F, a->Hg,
                a->Wg, a->C);
  if (a->C % 8 != 0) return fail(CAST_ERR_UNSUPPORTED, "%s: C=%d not a multiple of 8", who, a->C);
  if (a->C > 4096) return fail(CAST_ERR_UNSUPPORTED, "%s: C=%d above 4096", who, a->C);
  const cast_par_params& p = a->params;
  if (p.tile_h < 1 || p.tile_h > 8 || p.tile_w < 1 || p.tile_w > 8)
    return fail(CAST_ERR_UNSUPPORTED, "%s: tile %dx%d outside 1..8", who, p.tile_h, p.tile_w);
  if (!(p.T > 0.f) || !(p.q > 0.f) || !(p.tau_high >= p.tau_low))
    return fail(CAST_ERR_INVALID_ARG, "%s: gate needs T > 0, q > 0, tau_high >= tau_low", who);
  if (!(p.eps >= 0.f) || !(p.eta_rel >= 0.f) || !(p.eta_abs >= 0.f))
    return fail(CAST_ERR_INVALID_ARG, "%s: eps / eta must be >= 0", who);
  if (p.gate_mode < CAST_GATE_PAPER || p.gate_mode > CAST_GATE_ONE)
    return fail(CAST_ERR_INVALID_ARG, "%s: gate_mode %d", who, p.gate_mode);
  if (!a->anchor_mask) return fail(CAST_ERR_INVALID_ARG, "%s: anchor_mask is NULL", who);
  int na = 0;
  for (int f = 0; f < a->F; ++f) na += a->anchor_mask[f] ? 1 : 0;
  if (na > CAST_MAX_ANCHORS) return fail(CAST_ERR_UNSUPPORTED, "%s: %d anchors", who, na);
  if (na < a->F && na < 2)
    return fail(CAST_ERR_INVALID_ARG, "%s: %d anchor(s) but skipped frames exist (needs >= 2)", who, na);
  if (!a->r || !aligned16(a->r)) return fail(CAST_ERR_INVALID_ARG, "%s: r is NULL or misaligned", who);
  return CAST_OK;
}

cast_par_args par_of_block(const cast_block_args* a, uint8_t* mask) {
  cast_par_args p{};
  p.r = a->r_out;
  p.dtype = a->r_dtype;
  p.F = a->n_frames;
  p.Hg = a->Hg;
  p.Wg = a->Wg;
  p.C = a->H * a->d;
  for (int f = 0; f < a->n_frames; ++f) mask[f] = 0;
  for (int k = 0; k < a->n_anchors; ++k)
    if (a->anchors[k] >= 0 && a->anchors[k] < a->n_frames) mask[a->anchors[k]] = 1;
  p.anchor_mask = mask;
  p.channel_weight = a->channel_weight;
  p.params = a->par;
  return p;
}

cast_route_args route_of_block(const cast_block_args* a, int32_t* idx) {
  cast_route_args r{};
  r.q = a->q;
  r.q_row_stride = a->q_row_stride;
  r.n_frames = a->n_frames;
  r.S = a->Hg * a->Wg;
  r.H = a->H;
  r.d = a->d;
  r.dtype = CAST_BF16;
  r.anchors = a->anchors;
  r.n_anchors = a->n_anchors;
  r.k_hist = a->k_hist;
  r.v_hist = a->v_hist;
  r.hist_row_stride = a->hist_row_stride;
  r.M = a->M;
  r.B_v = a->B_v;
  r.gram = a->gram;
  r.K = a->K;
  r.eps = a->route_eps;
  r.mode = a->route_mode;
  r.refine_passes = a->route_refine_passes;
  r.lambda_anc = a->route_lambda_anc;
  r.lambda_rec = a->route_lambda_rec;
  r.refine_tol = a->route_refine_tol;
  r.hist = a->hist;
  r.candidates = a->route_candidates;
  r.M_c = a->route_M_c;
  r.idx = idx;
  return r;
}

cast_attn_args attn_of_block(const cast_block_args* a, const int32_t* idx) {
  cast_attn_args t{};
  t.q = a->q;
  t.k_cur = a->k_cur;
  t.v_cur = a->v_cur;
  t.q_row_stride = a->q_row_stride;
  t.cur_row_stride = a->cur_row_stride;
  t.n_frames = a->n_frames;
  t.S = a->Hg * a->Wg;
  t.H = a->H;
  t.d = a->d;
  t.anchors = a->anchors;
  t.n_anchors = a->n_anchors;
  t.k_hist = a->k_hist;
  t.v_hist = a->v_hist;
  t.hist_row_stride = a->hist_row_stride;
  t.M = a->M;
  t.B_v = a->B_v;
  t.idx = idx;
  t.K_eff = a->K < a->M ? a->K : a->M;
  t.scale = a->scale;
  t.o = a->r_out;
  t.o_dtype = a->r_dtype;
  t.lse = nullptr;
  t.hist = a->hist;
  return t;
}

// block-step workspace: [route ws][idx (when idx_out is NULL)][attention ws][par ws]
struct BlockPlan {
  size_t route_bytes, idx_bytes, attn_bytes, par_bytes, proj_bytes, total;
};
BlockPlan block_plan(const cast_block_args* a) {
  BlockPlan b{};
  int32_t dummy_idx = 0;
  cast_route_args r = route_of_block(a, &dummy_idx);
  b.route_bytes = (a->M > 0 && a->K > 0) ? route_plan(r).total_bytes : 0;
  const int keff = a->K < a->M ? a->K : a->M;
  b.idx_bytes = a->idx_out ? 0 : align_up((size_t)a->n_anchors * a->H * (keff > 0 ? keff : 1) * 4);
  cast_attn_args t = attn_of_block(a, nullptr);
  b.attn_bytes = align_up(attention_plan(t).total_bytes);
  uint8_t mask[CAST_MAX_FRAMES];
  cast_par_args p = par_of_block(a, mask);
  b.par_bytes = par_plan(p).total_bytes;
  // with W_O: the attention output [n_anchors, S, H*d] bf16
  b.proj_bytes = a->w_o ? align_up((size_t)a->n_anchors * a->Hg * a->Wg * a->H * a->d * 2) : 0;
  b.total = b.route_bytes + b.idx_bytes + b.attn_bytes + b.par_bytes + b.proj_bytes;
  return b;
}

}  // namespace
}  // namespace cast

using namespace cast;

extern "C" {

const char* cast_version(void) { return "0.1.0"; }

const char* cast_status_string(cast_status s) {
  switch (s) {
    case CAST_OK: return "CAST_OK";
    case CAST_ERR_INVALID_ARG: return "CAST_ERR_INVALID_ARG";
    case CAST_ERR_UNSUPPORTED: return "CAST_ERR_UNSUPPORTED";
    case CAST_ERR_CUDA: return "CAST_ERR_CUDA";
    case CAST_ERR_DEVICE_TIMEOUT: return "CAST_ERR_DEVICE_TIMEOUT";
    default: return "CAST_ERR_UNKNOWN";
  }
}

const char* cast_last_error_detail(void) { return g_detail; }

void cast_par_params_default(cast_par_params* p) {
  if (!p) return;
  p->tile_h = 8;
  p->tile_w = 8;
  p->tau_low = 0.25f;
  p->tau_high = 0.75f;
  p->q = 2.0f;
  p->T = 0.10f;
  p->eps = 1e-8f;
  p->eta_rel = 1e-6f;
  p->eta_abs = 1e-8f;
  p->band_radius = -1.0f;
  p->gate_mode = CAST_GATE_PAPER;
}

size_t cast_route_workspace_size(const cast_route_args* a) {
  if (!a || a->M <= 0 || a->n_anchors < 1 || a->H < 1 || a->d < 1) return 0;
  return route_plan(*a).total_bytes;
}

cast_status cast_route_topk(const cast_route_args* a, void* ws, size_t ws_bytes, void* stream) {
  g_detail[0] = 0;
  cast_status s = validate_route(a);
  if (s) return s;
  const int keff = a->K < a->M ? a->K : a->M;
  if (a->k_eff) *a->k_eff = keff;
  if (a->M == 0) return CAST_OK;
  const size_t need = route_plan(*a).total_bytes;
  if (ws_bytes < need || (need && !ws))
    return fail(CAST_ERR_INVALID_ARG, "cast_route_topk: workspace %zu B < %zu B", ws_bytes, need);
  if (reinterpret_cast<uintptr_t>(ws) % kWsAlign)
    return fail(CAST_ERR_INVALID_ARG, "cast_route_topk: workspace not 256-byte aligned");
  return launch_route(*a, ws, static_cast<cudaStream_t>(stream));
}

size_t cast_attention_workspace_size(const cast_attn_args* a) {
  if (!a || a->n_anchors < 1 || a->H < 1 || a->S < 1 || a->n_frames < 1 || (a->d != 64 && a->d != 128))
    return 0;
  return attention_plan(*a).total_bytes;
}

cast_status cast_anchor_attention(const cast_attn_args* a, void* ws, size_t ws_bytes, void* stream) {
  g_detail[0] = 0;
  cast_status s = validate_attn(a);
  if (s) return s;
  const size_t need = attention_plan(*a).total_bytes;
  if (need > 0 && (ws_bytes < need || !ws))
    return fail(CAST_ERR_INVALID_ARG, "cast_anchor_attention: workspace %zu B < %zu B", ws_bytes, need);
  if (need > 0 && reinterpret_cast<uintptr_t>(ws) % kWsAlign)
    return fail(CAST_ERR_INVALID_ARG, "cast_anchor_attention: workspace not 256-byte aligned");
  return launch_attention(*a, 0, ws, static_cast<cudaStream_t>(stream));
}

size_t cast_par_workspace_size(const cast_par_args* a) {
  if (!a || !a->anchor_mask || a->F < 1 || a->F > CAST_MAX_FRAMES || a->Hg < 1 || a->Wg < 1 ||
      a->C < 1 || a->params.tile_h < 1 || a->params.tile_w < 1)
    return 0;
  return par_plan(*a).total_bytes;
}

cast_status cast_par_reconstruct(const cast_par_args* a, void* ws, size_t ws_bytes, void* stream) {
  g_detail[0] = 0;
  cast_status s = validate_par(a);
  if (s) return s;
  const ParPlan p = par_plan(*a);
  if (p.n_target == 0) return CAST_OK;
  if (ws_bytes < p.total_bytes || (p.total_bytes && !ws))
    return fail(CAST_ERR_INVALID_ARG, "cast_par_reconstruct: workspace %zu B < %zu B", ws_bytes,
                p.total_bytes);
  if (reinterpret_cast<uintptr_t>(ws) % kWsAlign)
    return fail(CAST_ERR_INVALID_ARG, "cast_par_reconstruct: workspace not 256-byte aligned");
  return launch_par(*a, ws, static_cast<cudaStream_t>(stream));
}

size_t cast_block_workspace_size(const cast_block_args* a) {
  if (!a || !a->anchors || a->n_anchors < 1 || a->n_anchors > CAST_MAX_ANCHORS || a->n_frames < 1 ||
      a->n_frames > CAST_MAX_FRAMES || a->H < 1 || a->d < 1 || a->Hg < 1 || a->Wg < 1)
    return 0;
  return block_plan(a).total;
}

cast_status cast_block_step(const cast_block_args* a, void* ws, size_t ws_bytes, void* stream) {
  g_detail[0] = 0;
  const char* who = "cast_block_step";
  if (!a) return fail(CAST_ERR_INVALID_ARG, "%s: args is NULL", who);
  if (a->n_frames < 1 || a->n_frames > CAST_MAX_FRAMES)
    return fail(CAST_ERR_INVALID_ARG, "%s: n_frames %d outside 1..%d", who, a->n_frames, CAST_MAX_FRAMES);
  if (a->r_dtype != CAST_BF16 && a->r_dtype != CAST_F32)
    return fail(CAST_ERR_INVALID_ARG, "%s: r_dtype %d", who, a->r_dtype);
  cast_status s = validate_anchors(a->anchors, a->n_anchors, a->n_frames, who);
  if (s) return s;
  const BlockPlan bp = block_plan(a);
  int32_t* idx = a->idx_out;
  char* w = static_cast<char*>(ws);
  if (!idx) idx = reinterpret_cast<int32_t*>(w + bp.route_bytes);
  cast_route_args r = route_of_block(a, idx);
  if ((s = validate_route(&r))) return s;
  cast_attn_args t = attn_of_block(a, idx);
  if ((s = validate_attn(&t))) return s;
  uint8_t mask[CAST_MAX_FRAMES];
  cast_par_args p = par_of_block(a, mask);
  if ((s = validate_par(&p))) return s;
  if (a->x && !aligned16(a->x)) return fail(CAST_ERR_INVALID_ARG, "%s: x misaligned", who);
  if (a->w_o && (!aligned16(a->w_o) || (a->b_o && !aligned16(a->b_o))))
    return fail(CAST_ERR_INVALID_ARG, "%s: w_o / b_o misaligned", who);
  if (!a->w_o && a->b_o) return fail(CAST_ERR_INVALID_ARG, "%s: b_o given without w_o", who);
  if (ws_bytes < bp.total || (bp.total && !ws))
    return fail(CAST_ERR_INVALID_ARG, "%s: workspace %zu B < %zu B", who, ws_bytes, bp.total);
  if (reinterpret_cast<uintptr_t>(ws) % kWsAlign)
    return fail(CAST_ERR_INVALID_ARG, "%s: workspace not 256-byte aligned", who);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const bool routed = a->M > 0 && a->K > 0;
  char* aws = w + bp.route_bytes + bp.idx_bytes;
  if (routed) {
    // the attention follows the routing kernel directly: its tail counters are reset first
    if ((s = attention_reset_counters(t, aws, st))) return s;
    if ((s = launch_route(r, w, st))) return s;
  }
  if (!a->w_o) {
    if ((s = launch_attention(t, 1, aws, st, routed))) return s;
  } else {
    // attention output of the anchors into the workspace, then r_out[a] = O_a W_O^T + b_O
    char* proj = w + bp.route_bytes + bp.idx_bytes + bp.attn_bytes + bp.par_bytes;
    const int S = a->Hg * a->Wg, D = a->H * a->d;
    const size_t o_bytes = align_up((size_t)a->n_anchors * S * D * 2);
    t.o = proj;
    t.o_dtype = CAST_BF16;
    if ((s = launch_attention(t, 0, aws, st, routed))) return s;
    (void)o_bytes;
    AnchorGemm g{};
    g.a = proj;
    g.lda = D;
    g.a_frame_stride = (int64_t)S * D;
    g.a_frames = a->n_anchors;
    g.w = a->w_o;
    g.ldw = D;
    g.bias = a->b_o;
    g.bias_dtype = a->r_dtype;
    g.c = a->r_out;
    g.ldc = D;
    g.c_dtype = a->r_dtype;
    g.S = S;
    g.N = D;
    g.K = D;
    g.n_anchors = a->n_anchors;
    for (int i = 0; i < a->n_anchors; ++i) {
      g.a_frame[i] = i;
      g.c_frame[i] = a->anchors[i];
    }
    g.gelu = false;
    if ((s = gemm_anchor_rows(g, st))) return s;
  }
  if (par_plan(p).n_target > 0) {
    if ((s = launch_par(p, w + bp.route_bytes + bp.idx_bytes + bp.attn_bytes, st))) return s;
  }
  if (a->x) {
    const size_t n = (size_t)a->n_frames * a->Hg * a->Wg * a->H * a->d;
    if ((s = launch_residual_add(a->x, a->r_out, a->r_dtype, n, st))) return s;
  }
  return CAST_OK;
}

namespace cast {
namespace {
// PAR of the FFN site: the skipped frames of r_out from its anchor rows
cast_par_args par_of_ffn(const cast_ffn_args* a, uint8_t* mask) {
  cast_par_args p{};
  p.r = a->r_out;
  p.dtype = a->r_dtype;
  p.F = a->n_frames;
  p.Hg = a->Hg;
  p.Wg = a->Wg;
  p.C = a->D;
  for (int f = 0; f < a->n_frames && f < CAST_MAX_FRAMES; ++f) mask[f] = 0;
  for (int k = 0; k < a->n_anchors; ++k)
    if (a->anchors && a->anchors[k] >= 0 && a->anchors[k] < a->n_frames) mask[a->anchors[k]] = 1;
  p.anchor_mask = mask;
  p.channel_weight = a->channel_weight;
  p.params = a->par;
  return p;
}
}  // namespace
}  // namespace cast

size_t cast_ffn_workspace_size(const cast_ffn_args* a) {
  if (!a || a->Hg < 1 || a->Wg < 1 || a->D_ff < 1 || a->n_frames < 1 || a->n_frames > CAST_MAX_FRAMES ||
      a->n_anchors < 1 || a->n_anchors > CAST_MAX_ANCHORS || !a->anchors)
    return 0;
  uint8_t mask[CAST_MAX_FRAMES];
  const cast_par_args p = par_of_ffn(a, mask);
  const size_t par = (p.params.tile_h >= 1 && p.params.tile_w >= 1 && p.C >= 1) ? par_plan(p).total_bytes : 0;
  return align_up((size_t)a->n_anchors * a->Hg * a->Wg * a->D_ff * 2) + align_up(par);
}

cast_status cast_ffn_step(const cast_ffn_args* a, void* ws, size_t ws_bytes, void* stream) {
  g_detail[0] = 0;
  const char* who = "cast_ffn_step";
  if (!a) return fail(CAST_ERR_INVALID_ARG, "%s: args is NULL", who);
  if (a->n_frames < 1 || a->n_frames > CAST_MAX_FRAMES || a->Hg < 1 || a->Wg < 1 || a->D < 8 ||
      a->D_ff < 8 || a->D % 8 || a->D_ff % 8)
    return fail(CAST_ERR_INVALID_ARG, "%s: bad shape (frames %d, grid %dx%d, D %d, D_ff %d)", who,
                a->n_frames, a->Hg, a->Wg, a->D, a->D_ff);
  if (a->r_dtype != CAST_BF16 && a->r_dtype != CAST_F32)
    return fail(CAST_ERR_INVALID_ARG, "%s: r_dtype %d", who, a->r_dtype);
  cast_status s = validate_anchors(a->anchors, a->n_anchors, a->n_frames, who);
  if (s) return s;
  if (!a->x || !aligned16(a->x) || a->x_row_stride < a->D || a->x_row_stride % 8)
    return fail(CAST_ERR_INVALID_ARG, "%s: x NULL, misaligned or with a bad row stride", who);
  if (!a->w1 || !a->w2 || !aligned16(a->w1) || !aligned16(a->w2) || (a->b1 && !aligned16(a->b1)) ||
      (a->b2 && !aligned16(a->b2)))
    return fail(CAST_ERR_INVALID_ARG, "%s: weights or biases NULL or misaligned", who);
  uint8_t mask[CAST_MAX_FRAMES];
  cast_par_args p = par_of_ffn(a, mask);
  if ((s = validate_par(&p))) return s;
  const size_t need = cast_ffn_workspace_size(a);
  if (ws_bytes < need || !ws)
    return fail(CAST_ERR_INVALID_ARG, "%s: workspace %zu B < %zu B", who, ws_bytes, need);
  if (reinterpret_cast<uintptr_t>(ws) % kWsAlign)
    return fail(CAST_ERR_INVALID_ARG, "%s: workspace not 256-byte aligned", who);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int S = a->Hg * a->Wg;
  // hidden activations of every anchor [n_anchors, S, D_ff] bf16, then the PAR workspace
  char* hid = static_cast<char*>(ws);
  char* pws = hid + align_up((size_t)a->n_anchors * S * a->D_ff * 2);
  AnchorGemm g1{};
  g1.a = a->x;
  g1.lda = a->x_row_stride;
  g1.a_frame_stride = (int64_t)S * a->x_row_stride;
  g1.a_frames = a->n_frames;
  g1.w = a->w1;
  g1.ldw = a->D;
  g1.bias = a->b1;
  g1.bias_dtype = CAST_BF16;
  g1.c = hid;
  g1.ldc = a->D_ff;
  g1.c_dtype = CAST_BF16;
  g1.S = S;
  g1.N = a->D_ff;
  g1.K = a->D;
  g1.n_anchors = a->n_anchors;
  g1.gelu = true;
  AnchorGemm g2{};
  g2.a = hid;
  g2.lda = a->D_ff;
  g2.a_frame_stride = (int64_t)S * a->D_ff;
  g2.a_frames = a->n_anchors;
  g2.w = a->w2;
  g2.ldw = a->D_ff;
  g2.bias = a->b2;
  g2.bias_dtype = a->r_dtype;
  g2.c = a->r_out;
  g2.ldc = a->D;
  g2.c_dtype = a->r_dtype;
  g2.S = S;
  g2.N = a->D;
  g2.K = a->D_ff;
  g2.n_anchors = a->n_anchors;
  g2.gelu = false;
  for (int i = 0; i < a->n_anchors; ++i) {
    g1.a_frame[i] = a->anchors[i];
    g1.c_frame[i] = i;
    g2.a_frame[i] = i;
    g2.c_frame[i] = a->anchors[i];
  }
  if ((s = gemm_anchor_rows(g1, st))) return s;
  if ((s = gemm_anchor_rows(g2, st))) return s;
  if (par_plan(p).n_target > 0) return launch_par(p, pws, st);
  return CAST_OK;
}

cast_status cast_selftest_bounded_wait(uint64_t limit_ns, void* stream) {
  g_detail[0] = 0;
  if (limit_ns < 1000 || limit_ns > 2000000000ull)
    return fail(CAST_ERR_INVALID_ARG, "cast_selftest_bounded_wait: limit %llu ns outside 1 us .. 2 s",
                (unsigned long long)limit_ns);
  return launch_bounded_wait_selftest(limit_ns, static_cast<cudaStream_t>(stream));
}

cast_status cast_check_device(void* stream) {
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const cudaError_t e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return fail(CAST_ERR_CUDA, "cast_check_device: %s", cudaGetErrorString(e));
  const unsigned int wa = attention_error_word(st, true);
  const unsigned int wp = par_error_word(st, true);
  const unsigned int wr = route_error_word(st, true);
  const unsigned int wd = dense_error_word(st, true);
  if (wa == 1u || wp || wd || wr == 2u) return fail(CAST_ERR_DEVICE_TIMEOUT, "a kernel gave up on a bounded wait");
  if (wa == 2u) return fail(CAST_ERR_INVALID_ARG, "attention: a routed block index was outside [0, M)");
  if (wr) return fail(CAST_ERR_INVALID_ARG, "routing: a candidate index was outside [0, M) or repeated");
  return check_launch("cast_check_device");
}

}  // extern "C"

namespace cast {
cast_status launch_residual_add(void* x, const void* r, int dtype, size_t n, cudaStream_t st) {
  const int threads = 256;
  int blocks = (int)((n / 4 + threads - 1) / threads);
  if (blocks > 152 * 8) blocks = 152 * 8;
  if (blocks < 1) blocks = 1;
  if (dtype == CAST_F32)
    k_residual_add_f32<<<blocks, threads, 0, st>>>(static_cast<float*>(x), static_cast<const float*>(r), n);
  else
    k_residual_add_bf16<<<blocks, threads, 0, st>>>(static_cast<__nv_bfloat16*>(x),
                                                    static_cast<const __nv_bfloat16*>(r), n);
  return check_launch("residual add");
}
}  // namespace cast
