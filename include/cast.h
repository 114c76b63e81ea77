/*
 * cast.h - C ABI of the CAST per-block anchor/skip step on one GB300 (sm_103a).
 *
 * CAST (reconstruction-coupled acceleration of interactive world models) computes,
 * at each eligible residual site of a transformer block, the update of the
 * anchor frames directly and reconstructs the residual of every skipped frame
 * from the two anchors that bracket it (Section 4.1, Eq. block).  This library
 * runs the data-parallel hot path of that step:
 *
 *   cast_route_topk        pooled historical scoring and one-block omission
 *                          scores, TopK of K history blocks per (anchor, head)
 *                          (Section 4.4, Eqs. pooled, omission, topk)
 *   cast_anchor_attention  anchor queries attend to the whole current chunk plus
 *                          their routed history blocks (Eq. block, App. B.4)
 *   cast_par_reconstruct   Phase-Aware Reconstruction of the skipped frames
 *                          (Section 4.3, Eqs. cross, confidence, gate, fcpasm;
 *                          App. A.2)
 *   cast_block_step        the three in order at one attention residual site
 *
 * Conventions shared by every entry point
 *   - Tensor pointers are DEVICE pointers owned by the caller; `anchors` and
 *     `anchor_mask` are HOST arrays read during the call only.  The library
 *     allocates no device memory: scratch comes from the caller's workspace,
 *     sized by the matching cast_*_workspace_size() and at least 256-byte aligned.
 *   - Work is enqueued asynchronously on `stream` (a cudaStream_t; NULL = the
 *     legacy default stream).  No call synchronises the host with the device.
 *   - Every call validates its arguments before launching anything.  On an
 *     error nothing is written and a cast_status other than CAST_OK is
 *     returned; cast_last_error_detail() gives a message for the calling thread.
 *     CAST_ERR_CUDA reports a launch or runtime error seen after enqueuing.
 *   - Kernels never wait without bound.  A wait that exceeds its limit makes the
 *     kernel record an error word and return; cast_check_device() reads (and
 *     clears) that word and returns CAST_ERR_DEVICE_TIMEOUT.
 *   - Layouts are row-major.  Token tensors are [frames, S, H, d] with d
 *     contiguous and S = Hg * Wg tokens of a frame's latent grid in row-major
 *     (y, x) order; the token row stride (elements between consecutive tokens)
 *     must be >= H*d and a multiple of 8.  Residuals are channels-last
 *     [F, Hg, Wg, C] (the attention output viewed per frame).
 *   - bf16 is IEEE bfloat16 (round-to-nearest-even on output); f32 is IEEE float.
 */
#ifndef CAST_H_
#define CAST_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int cast_status;
#define CAST_OK 0
#define CAST_ERR_INVALID_ARG 1     /* a shape, pointer, alignment or value is wrong */
#define CAST_ERR_UNSUPPORTED 2     /* valid but outside what the kernels implement */
#define CAST_ERR_CUDA 3            /* the CUDA runtime reported an error */
#define CAST_ERR_DEVICE_TIMEOUT 4  /* a kernel gave up on a bounded wait */

#define CAST_F32 0
#define CAST_BF16 1

#define CAST_ROUTE_OMISSION 0     /* TopK on u = ||P delta||^2 (Eq. omission), the paper's */
#define CAST_ROUTE_SIMILARITY 1   /* TopK on the pooled similarity s (Eq. pooled) */

#define CAST_GATE_PAPER 0         /* g from Eq. (gate) */
#define CAST_GATE_ZERO 1          /* g = 0: direct value interpolation / extrapolation */
#define CAST_GATE_ONE 2           /* g = 1: full endpoint phase transport */

#define CAST_MAX_FRAMES 256       /* frames of one chunk (anchors + skipped) */
#define CAST_MAX_ANCHORS 64

/* ------------------------------------------------------------------------ */
/* Layout of the historical KV blocks (Section 4.4; App. B.5 Tab. config:    */
/* blocks (t, h, w) = (1, 8, 8) in token coordinates, partial blocks masked). */
/* ------------------------------------------------------------------------ */
#define CAST_HIST_BLOCKS 0        /* k_hist/v_hist [M, B_v, H, d]: block m = rows m*B_v .. m*B_v+B_v-1 */
#define CAST_HIST_FRAMES 1        /* k_hist/v_hist [frames, Hg, Wg, H, d]: (1, 8, 8) blocks */

typedef struct {
  int32_t kind;                   /* CAST_HIST_BLOCKS (zero-initialised default) or CAST_HIST_FRAMES */
  /* CAST_HIST_FRAMES only: the history frames and their token grid.  Block
     m = (f * ceil(Hg/8) + by) * ceil(Wg/8) + bx holds the tokens of frame f in rows
     8by .. min(8by+8, Hg)-1 and columns 8bx .. min(8bx+8, Wg)-1 (a block never spans frames;
     blocks at the right and bottom edges are truncated).  M must equal
     frames * ceil(Hg/8) * ceil(Wg/8) and B_v must be 64 (the nominal block size); a truncated
     block pools over its own tokens and its missing key positions are masked in attention. */
  int32_t frames, Hg, Wg;
} cast_hist_layout;

/* ------------------------------------------------------------------------ */
/* Routing: Section 4.4, Eqs. (pooled), (omission), (topk); App. B.1.        */
/* ------------------------------------------------------------------------ */
typedef struct {
  /* queries of the current chunk, [n_frames, S, H, d]; only anchor frames are read */
  const void* q;
  int64_t q_row_stride;
  int32_t n_frames, S, H, d;      /* d in {64, 128} */
  int32_t dtype;                  /* dtype of q, k_hist, v_hist: CAST_BF16 or CAST_F32 */
  const int32_t* anchors;         /* HOST, n_anchors strictly ascending frame indices */
  int32_t n_anchors;
  /* history blocks, [M, B_v, H, d] (block m is rows m*B_v .. m*B_v+B_v-1), or history frames
     in (1, 8, 8) blocks as given by hist */
  const void* k_hist;
  const void* v_hist;
  int64_t hist_row_stride;
  int32_t M, B_v;
  /* Gram matrices G_h = P_h^T P_h of the output-projection head slices P = W_O^(h),
     device f32 [H, d, d]; NULL means P = I (u = ||delta||^2) */
  const float* gram;
  int32_t K;                      /* budget K_KV; K_eff = min(K, M) blocks are kept */
  float eps;                      /* stabiliser of Eq. (omission); 1e-8 by default */
  int32_t mode;                   /* CAST_ROUTE_OMISSION | CAST_ROUTE_SIMILARITY */
  /* outputs (device unless noted) */
  int32_t* idx;                   /* [n_anchors, H, K_eff] ascending block indices */
  float* u;                       /* optional [n_anchors, H, M] routing scores used for TopK */
  float* qbar;                    /* optional [n_anchors, H, d] pooled queries (16-B aligned) */
  float* kbar;                    /* optional [M, H, d] pooled keys (16-B aligned) */
  float* vbar;                    /* optional [M, H, d] pooled values (16-B aligned) */
  int32_t* k_eff;                 /* optional HOST: receives K_eff */
  /* Reconstruction-coupled refinement (Alg. routing, App. B.3): refine_passes > 0 runs that many
     directional best-response passes (forward, backward, ...) after the TopK initialisation,
     minimising Eq. (objective) with weights lambda_anc, lambda_rec under the fixed budget K_eff,
     accepting a change only when J drops by more than refine_tol * max(J, 1e-8).  The paper:
     2 passes, (1, 1), 1e-6.  0 passes = independent TopK.  Needs CAST_ROUTE_OMISSION. */
  int32_t refine_passes;
  float lambda_anc, lambda_rec, refine_tol;
  cast_hist_layout hist;          /* layout of k_hist/v_hist; zero = CAST_HIST_BLOCKS */
  /* Optional fixed candidate sets C_i (App. B.3): device int32 [n_anchors, H, M_c], distinct
     block indices per (anchor, head), K_eff <= M_c <= M.  The TopK initialisation and the
     refinement's best responses choose within C_i only; blocks outside C_i stay unselected and
     still count as omissions in J and in the neighbours' gains.  NULL = every block
     (M_c = M, the paper's setting, Tab. config_cast). */
  const int32_t* candidates;
  int32_t M_c;
} cast_route_args;

/* Pooled mean statistics q_bar, k_bar, v_bar (mean over a frame's S tokens and over a
 * block's B_v tokens, f32 accumulation), scores s = q_bar.k_bar / sqrt(d), pi = softmax
 * over blocks, o_bar = sum pi v_bar, delta = pi/(1-pi+eps) (o_bar - v_bar),
 * u = delta^T G delta; then per (anchor, head) the K_eff largest scores (ties to the
 * lower block index), written in ascending block order.  K >= M keeps every block and
 * M == 0 writes nothing (routing bypass, App. B.3).
 * With CAST_HIST_FRAMES a block's means run over its own tokens (64, or fewer at the grid
 * edge).
 * Errors: INVALID_ARG for NULL required pointers, n_anchors < 1 or > CAST_MAX_ANCHORS,
 * anchors not ascending / out of range, K < 0, M < 0, B_v < 1 with M > 0, bad strides,
 * an unknown hist.kind, or CAST_HIST_FRAMES with a non-positive grid, M different from its
 * block count or B_v != 64,
 * a workspace smaller than cast_route_workspace_size(), refinement with a negative weight or
 * tolerance or outside CAST_ROUTE_OMISSION, candidates with M_c outside K_eff..M; a candidate
 * index outside [0, M) or repeated within a set makes the kernel record an error that
 * cast_check_device() reports as INVALID_ARG (that set then holds fewer members and its
 * selection is completed by the lowest-index other blocks); UNSUPPORTED for d not 64/128, M > 16384,
 * H*d > 51200 channels (pooling shared memory) or a per-head routing state above 200 KB of
 * shared memory (about 8 K_f M bytes, 12 K_f M with refinement, plus K_f M with candidate
 * sets, and 4 K_f d + 36 KB for the statistics). */
cast_status cast_route_topk(const cast_route_args* args, void* workspace,
                            size_t workspace_bytes, void* stream);
size_t cast_route_workspace_size(const cast_route_args* args);

/* cast_route_topk for callers that cannot allocate device memory.  The paper has no
 * counterpart: this is a deployment convenience.  Plugins inside a host framework that owns
 * all device allocations, real-time loops that must not take an allocator's locks or its
 * implicit synchronisation, and fixed-budget embedded runtimes can call this instead of
 * providing a workspace.  The scratch is a 16 MiB array that the library reserves in device
 * memory on every GPU where it is loaded, until the process exits.
 *   - Problems needing more than 16 MiB of scratch (cast_route_workspace_size() > 16 MiB)
 *     are rejected with CAST_ERR_UNSUPPORTED and a message; nothing is launched.
 *   - The first call on a device looks up the array's device address with that device
 *     current (no allocation); make that first call before any stream capture.  The address
 *     is kept for the life of the process: do not call this entry point on a device after a
 *     cudaDeviceReset() (or any other teardown of its primary context) in the same process.
 *   - All calls share the one array and the kernels fully overwrite what they read, so no
 *     clearing is needed between calls; calls whose work overlaps on the GPU (concurrent
 *     streams, or several host threads) race on it and must be serialised by the caller.
 *   - Inputs, outputs and errors are those of cast_route_topk. */
cast_status cast_route_topk_noalloc(const cast_route_args* args, void* stream);

/* ------------------------------------------------------------------------ */
/* Routed anchor attention: Eq. (block), App. B.4, App. B.5.                 */
/* ------------------------------------------------------------------------ */
typedef struct {
  const void* q;                  /* bf16 [n_frames, S, H, d], anchor rows are read */
  const void* k_cur;              /* bf16 [n_frames, S, H, d] keys of the whole current chunk */
  const void* v_cur;              /* bf16 [n_frames, S, H, d] */
  int64_t q_row_stride, cur_row_stride;
  int32_t n_frames, S, H, d;      /* d in {64, 128} */
  const int32_t* anchors;         /* HOST, strictly ascending */
  int32_t n_anchors;
  const void* k_hist;             /* bf16 [M, B_v, H, d], or frames as given by hist */
  const void* v_hist;
  int64_t hist_row_stride;
  int32_t M, B_v;
  const int32_t* idx;             /* device [n_anchors, H, K_eff] routed blocks (any order) */
  int32_t K_eff;                  /* 0 = current chunk only */
  float scale;                    /* softmax scale; <= 0 means 1/sqrt(d) */
  void* o;                        /* device [n_anchors, S, H*d], dtype o_dtype */
  int32_t o_dtype;                /* CAST_BF16 or CAST_F32 */
  float* lse;                     /* optional device f32 [n_anchors, H, S]: natural-log
                                     log-sum-exp of the scaled logits of each query row */
  cast_hist_layout hist;          /* layout of k_hist/v_hist; zero = CAST_HIST_BLOCKS */
} cast_attn_args;

/* O[i, s, h, :] = sum_j softmax_j(scale * q_i,s,h . k_j) v_j, where j runs over every
 * token of the current chunk (no causal mask inside the chunk) and every token of the
 * history blocks idx[i, h, :].  bf16 operands, f32 softmax and accumulation (Tab. config).
 * The workspace (cast_attention_workspace_size() bytes; 0 and NULL allowed when that is 0)
 * holds the partial results of query tiles whose keys are split over several SMs to fill the
 * last round of work.
 * With CAST_HIST_FRAMES the routed blocks are taken two at a time (two 8x8 token boxes per
 * 128-key tile); key positions outside a truncated block, and the empty second half of the
 * last tile when K_eff is odd, are masked (-inf logits).
 * Errors: INVALID_ARG for NULL pointers, bad shapes or strides, anchors not ascending,
 * K_eff > 0 with M == 0, a short workspace, a history layout as in cast_route_topk;
 * UNSUPPORTED for d not 64/128, S*n_frames >= 2^31, or CAST_HIST_FRAMES with
 * frames * Hg * Wg >= 2^31 tokens.  Block indices outside [0, M) make the kernel record an error and
 * read block 0 instead. */
cast_status cast_anchor_attention(const cast_attn_args* args, void* workspace,
                                  size_t workspace_bytes, void* stream);
size_t cast_attention_workspace_size(const cast_attn_args* args);

/* ------------------------------------------------------------------------ */
/* Phase-Aware Reconstruction: Section 4.3, Eqs. (cross), (confidence),      */
/* (gate), (fcpasm); App. A.2.                                               */
/* ------------------------------------------------------------------------ */
typedef struct {
  int32_t tile_h, tile_w;         /* disjoint spatial tiles, 1..8 tokens; 8x8 in the paper */
  float tau_low, tau_high, q, T;  /* gate of Eq. (gate); (0.25, 0.75, 2, 0.10) in the paper */
  float eps;                      /* 1e-8, Eq. (confidence) */
  float eta_rel, eta_abs;         /* reliability threshold eta = eta_rel max W + eta_abs */
  float band_radius;              /* < 0: every bin gated as in the paper; >= 0: bins whose
                                     radius in 8x8-tile bin units exceeds it get g = 0 */
  int32_t gate_mode;              /* CAST_GATE_PAPER | CAST_GATE_ZERO | CAST_GATE_ONE */
} cast_par_params;

/* Fills the paper's defaults (Tab. config_cast, App. A.2). */
void cast_par_params_default(cast_par_params* p);

typedef struct {
  void* r;                        /* device [F, Hg, Wg, C] in/out: anchor frames read,
                                     skipped frames overwritten */
  int32_t dtype;                  /* CAST_F32 or CAST_BF16 */
  int32_t F, Hg, Wg, C;           /* C a multiple of 8 */
  const uint8_t* anchor_mask;     /* HOST [F]: nonzero = anchor */
  const float* channel_weight;    /* optional device [C], >= 0; NULL = 1 */
  cast_par_params params;
} cast_par_args;

/* For every skipped frame t with bracketing anchors (a, b) (frames outside the anchor
 * span use the two nearest anchors and alpha < 0 or > 1), alpha = (t-a)/(b-a); per tile
 * and channel F = RFFT2_ortho(R), Z = sum_c w_c F_b conj(F_a), W = sum_c w_c |F_b||F_a|,
 * reliable bins W > eta and |Z| > eta, theta = Arg Z in (-pi, pi] on representatives
 * (mirrors negated, self-conjugate bins 0), c = sum kappa|Z| / (sum kappa W + eps) over the
 * reliable non-DC bins, g = sigmoid((c - tau(nu)) / T), and
 * R_t = IRFFT2_ortho((1-alpha) F_a e^{i g alpha theta} + alpha F_b e^{-i g (1-alpha) theta}).
 * All frames anchors: nothing to do (workspace size 0).  The workspace
 * (cast_par_workspace_size() bytes) holds each channel chunk's partial Z, W per (tile, pair)
 * and theta, g per bin: 120 ceil(C/128) + 80 floats per tile and anchor, and for bf16
 * residuals each target's blend matrix (32 KB per tile and skipped frame) for the tensor-core
 * blend (each part rounded up to 256 bytes).
 * Errors: INVALID_ARG when a frame is skipped and fewer than two anchors exist, bad shapes
 * or pointers, a short workspace; UNSUPPORTED for tile sides outside 1..8, C not a multiple
 * of 8, C > 4096. */
cast_status cast_par_reconstruct(const cast_par_args* args, void* workspace,
                                 size_t workspace_bytes, void* stream);
size_t cast_par_workspace_size(const cast_par_args* args);

/* ------------------------------------------------------------------------ */
/* One block step at an attention residual site: Eq. (block), App. B.4.      */
/* ------------------------------------------------------------------------ */
typedef struct {
  const void* q;                  /* bf16 [n_frames, S, H, d] */
  const void* k_cur;
  const void* v_cur;
  int64_t q_row_stride, cur_row_stride;
  int32_t n_frames, Hg, Wg, H, d; /* S = Hg * Wg */
  const int32_t* anchors;         /* HOST, strictly ascending; n_anchors >= 2 unless
                                     every frame is an anchor */
  int32_t n_anchors;
  const void* k_hist;             /* bf16 [M, B_v, H, d], or frames as given by hist */
  const void* v_hist;
  int64_t hist_row_stride;
  int32_t M, B_v;
  const float* gram;              /* optional, as in cast_route_args */
  int32_t K;
  float route_eps;
  int32_t route_mode;
  int32_t route_refine_passes;    /* as cast_route_args.refine_passes (0 = independent TopK) */
  float route_lambda_anc, route_lambda_rec, route_refine_tol;
  float scale;                    /* <= 0: 1/sqrt(d) */
  void* r_out;                    /* device [n_frames, S, H*d]: anchor rows = attention
                                     output, skipped rows = PAR reconstruction */
  int32_t r_dtype;                /* CAST_BF16 or CAST_F32 */
  void* x;                        /* optional device [n_frames, S, H*d] of r_dtype: x += r_out */
  int32_t* idx_out;               /* optional device [n_anchors, H, min(K, M)] */
  const float* channel_weight;    /* optional device [H*d] PAR channel weights */
  cast_par_params par;
  /* Optional output projection (App. B.1: PAR acts on the site's residual): with w_o the
     anchor rows of r_out are O_a W_O^T + b_O and PAR reconstructs the skipped rows of that
     projected residual; NULL = the attention output itself (pre-W_O). */
  const void* w_o;                /* optional device bf16 [H*d, H*d], layer layout [out, in] */
  const void* b_o;                /* optional device [H*d] of r_dtype */
  cast_hist_layout hist;          /* layout of k_hist/v_hist; zero = CAST_HIST_BLOCKS */
  const int32_t* route_candidates;   /* optional, as cast_route_args.candidates */
  int32_t route_M_c;
} cast_block_args;

/* route_topk -> anchor_attention -> (output projection) -> par_reconstruct on one stream,
 * then the optional residual update x += r_out.  The projection of every anchor's rows is
 * one tcgen05 GEMM launch (bias epilogue) on the caller's stream.  Errors: those of the steps;
 * INVALID_ARG for a misaligned w_o / b_o. */
cast_status cast_block_step(const cast_block_args* args, void* workspace,
                            size_t workspace_bytes, void* stream);
size_t cast_block_workspace_size(const cast_block_args* args);

/* ------------------------------------------------------------------------ */
/* The FFN residual site (App. B.1, B.4): the anchors' FFN is computed, the  */
/* skipped frames' FFN residuals are reconstructed by PAR with the same      */
/* anchors.                                                                   */
/* ------------------------------------------------------------------------ */
typedef struct {
  const void* x;                  /* device bf16 [n_frames, S, D] FFN input (anchor frames read) */
  int64_t x_row_stride;           /* elements between token rows, >= D, multiple of 8 */
  int32_t n_frames, Hg, Wg, D, D_ff;   /* S = Hg * Wg; D and D_ff multiples of 8 */
  const int32_t* anchors;         /* HOST, strictly ascending, as in cast_block_args */
  int32_t n_anchors;
  const void* w1;                 /* device bf16 [D_ff, D] */
  const void* b1;                 /* optional device bf16 [D_ff] */
  const void* w2;                 /* device bf16 [D, D_ff] */
  const void* b2;                 /* optional device [D] of r_dtype */
  void* r_out;                    /* device [n_frames, S, D]: anchor rows = FFN(x), skipped rows = PAR */
  int32_t r_dtype;                /* CAST_BF16 or CAST_F32 */
  const float* channel_weight;    /* optional device [D] PAR channel weights */
  cast_par_params par;
} cast_ffn_args;

/* For every anchor frame a: r_out[a] = GELU(x[a] W1^T + b1) W2^T + b2 (GELU in its tanh
 * form, the hidden activations rounded to bf16 between the two GEMMs), then
 * par_reconstruct(r_out) over the skipped frames.  Each GEMM is one tcgen05 launch over the
 * rows of every anchor (bias, and GELU, in its epilogue); the workspace holds the hidden
 * activations [n_anchors, S, D_ff] bf16 and PAR's records.  Errors: INVALID_ARG for bad
 * shapes, strides or pointers, anchors as in cast_block_step, a short workspace; those of
 * par_reconstruct. */
cast_status cast_ffn_step(const cast_ffn_args* args, void* workspace, size_t workspace_bytes,
                          void* stream);
size_t cast_ffn_workspace_size(const cast_ffn_args* args);

/* ------------------------------------------------------------------------ */
/* Control-aware frame selection: Section 3 ("Interaction sensitivity",      */
/* "Coverage debt"), Eqs. (sensitivity), (debt), (score); App. B.1 Eq.      */
/* (normalization).  Picks the anchors of block l+1 from the control-branch  */
/* updates of block l and the frames' refresh ages.                          */
/* ------------------------------------------------------------------------ */
#define CAST_MAX_BRANCHES 2       /* control branches (camera, action) */

typedef struct {
  /* device [N_cur, frame_elems] feature updates of the available control branches (the
     frame's S spatial x D channel coordinates, contiguous, 16-byte aligned); entries past
     n_branch are ignored */
  const void* delta[CAST_MAX_BRANCHES];
  int32_t n_branch;               /* 0..2; 0 = no fresh response: the score is the debt term alone */
  int32_t dtype;                  /* CAST_F32 | CAST_BF16 (of delta) */
  int32_t n_frames;               /* N_cur, 1..CAST_MAX_FRAMES */
  int64_t frame_elems;            /* S * D; frame_elems * element size a multiple of 16 bytes */
  const int32_t* ages;            /* device [N_cur] refresh ages h^l */
  const uint8_t* anchor_mask;     /* device [N_cur] anchors of block l (nonzero = anchor) */
  int32_t K_f;                    /* anchors to select, >= 1 (K_f >= N_cur selects every frame) */
  float lambda_cov;               /* debt weight, 0.5 in the paper */
  float eps;                      /* epsilon of Eq. (normalization), 1e-8 */
  int32_t* ages_out;              /* device [N_cur] h^{l+1} (may alias ages) */
  int32_t* anchors_out;           /* device [min(K_f, N_cur)] frame indices of block l+1, ascending */
  uint8_t* mask_out;              /* optional device [N_cur] anchor mask of block l+1 */
  float* rms_out;                 /* optional device [n_branch, N_cur] RMS of each update (App. B.1) */
  float* score_out;               /* optional device [N_cur] scores S^{l+1} (Eq. score) */
} cast_select_args;

/* r_{i,k} = RMS(delta_k[i]); Norm = (r - min r) / (max r - min r + eps) over the chunk per
 * branch; d_i = mean over the given branches; h^{l+1} = 0 for anchors of block l, h^l + 1
 * otherwise; D = h^{l+1} / ceil(N_cur / K_f); S = d + lambda_cov D (debt alone without a
 * branch); anchors of block l+1 = the K_f largest S, ties to the lower frame index, written in
 * ascending order.  Errors: INVALID_ARG for NULL required pointers, n_frames outside
 * 1..CAST_MAX_FRAMES, K_f < 1, n_branch outside 0..2, misaligned delta, frame_elems < 1,
 * negative lambda_cov or eps, a short workspace. */
cast_status cast_select_frames(const cast_select_args* args, void* workspace,
                               size_t workspace_bytes, void* stream);
size_t cast_select_workspace_size(const cast_select_args* args);

/* ------------------------------------------------------------------------ */
/* Status                                                                    */
/* ------------------------------------------------------------------------ */
const char* cast_status_string(cast_status s);
/* Message of the last error on the calling thread ("" if none). */
const char* cast_last_error_detail(void);
/* Synchronises `stream`, then reports CAST_ERR_DEVICE_TIMEOUT if a kernel on the current
 * device recorded a bounded-wait timeout, CAST_ERR_INVALID_ARG if one met a device-side index
 * outside its range (a routed block in attention, a routing candidate) (both records are
 * cleared), CAST_ERR_CUDA on a pending CUDA error, CAST_OK otherwise. */
cast_status cast_check_device(void* stream);
/* Failure-path self-test (no counterpart in the paper): enqueues one thread that waits on a
 * device barrier nothing ever completes, with a deadline of limit_ns (1 us .. 2 s) on the
 * GPU's global timer, exactly as the kernels of the path bound their waits.  When the
 * deadline passes it records a timeout, so the next cast_check_device() on the stream returns
 * CAST_ERR_DEVICE_TIMEOUT (and clears the record); the context stays usable.
 * Errors: INVALID_ARG for a limit outside the range. */
cast_status cast_selftest_bounded_wait(uint64_t limit_ns, void* stream);
/* Library version, "major.minor.patch". */
const char* cast_version(void);

#ifdef __cplusplus
}
#endif
#endif /* CAST_H_ */
