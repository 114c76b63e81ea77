"""ctypes binding of libcast (include/cast.h): argument marshalling only.

Every function takes torch CUDA tensors, passes their device pointers, sizes and the
current torch stream to the C entry point of the same name, and raises CastError on a
non-OK status.  Workspaces are torch allocations owned by the caller (plumbing).  There
is no fallback: without the built library, importing this module raises.
"""
from __future__ import annotations

import ctypes as C
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libcast.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"libcast is not built ({LIB_PATH} missing); run __graft_entry__.build()")
_lib = C.CDLL(LIB_PATH)

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_DEVICE_TIMEOUT = 0, 1, 2, 3, 4
F32, BF16 = 0, 1
ROUTE_OMISSION, ROUTE_SIMILARITY = 0, 1
HIST_BLOCKS, HIST_FRAMES = 0, 1
GATE_PAPER, GATE_ZERO, GATE_ONE = 0, 1, 2
MAX_FRAMES, MAX_ANCHORS = 256, 64

_vp = C.c_void_p
_i32, _i64, _f32 = C.c_int32, C.c_int64, C.c_float


class HistLayout(C.Structure):
    _fields_ = [("kind", _i32), ("frames", _i32), ("Hg", _i32), ("Wg", _i32)]


class RouteArgs(C.Structure):
    _fields_ = [("q", _vp), ("q_row_stride", _i64), ("n_frames", _i32), ("S", _i32), ("H", _i32),
                ("d", _i32), ("dtype", _i32), ("anchors", C.POINTER(_i32)), ("n_anchors", _i32),
                ("k_hist", _vp), ("v_hist", _vp), ("hist_row_stride", _i64), ("M", _i32),
                ("B_v", _i32), ("gram", _vp), ("K", _i32), ("eps", _f32), ("mode", _i32),
                ("idx", _vp), ("u", _vp), ("qbar", _vp), ("kbar", _vp), ("vbar", _vp),
                ("k_eff", C.POINTER(_i32)), ("refine_passes", _i32), ("lambda_anc", _f32),
                ("lambda_rec", _f32), ("refine_tol", _f32), ("hist", HistLayout),
                ("candidates", _vp), ("M_c", _i32)]


class AttnArgs(C.Structure):
    _fields_ = [("q", _vp), ("k_cur", _vp), ("v_cur", _vp), ("q_row_stride", _i64),
                ("cur_row_stride", _i64), ("n_frames", _i32), ("S", _i32), ("H", _i32), ("d", _i32),
                ("anchors", C.POINTER(_i32)), ("n_anchors", _i32), ("k_hist", _vp),
                ("v_hist", _vp), ("hist_row_stride", _i64), ("M", _i32), ("B_v", _i32),
                ("idx", _vp), ("K_eff", _i32), ("scale", _f32), ("o", _vp), ("o_dtype", _i32),
                ("lse", _vp), ("hist", HistLayout)]


class ParParams(C.Structure):
    _fields_ = [("tile_h", _i32), ("tile_w", _i32), ("tau_low", _f32), ("tau_high", _f32),
                ("q", _f32), ("T", _f32), ("eps", _f32), ("eta_rel", _f32), ("eta_abs", _f32),
                ("band_radius", _f32), ("gate_mode", _i32)]


class ParArgs(C.Structure):
    _fields_ = [("r", _vp), ("dtype", _i32), ("F", _i32), ("Hg", _i32), ("Wg", _i32), ("C", _i32),
                ("anchor_mask", C.POINTER(C.c_uint8)), ("channel_weight", _vp),
                ("params", ParParams)]


class BlockArgs(C.Structure):
    _fields_ = [("q", _vp), ("k_cur", _vp), ("v_cur", _vp), ("q_row_stride", _i64),
                ("cur_row_stride", _i64), ("n_frames", _i32), ("Hg", _i32), ("Wg", _i32),
                ("H", _i32), ("d", _i32), ("anchors", C.POINTER(_i32)), ("n_anchors", _i32),
                ("k_hist", _vp), ("v_hist", _vp), ("hist_row_stride", _i64), ("M", _i32),
                ("B_v", _i32), ("gram", _vp), ("K", _i32), ("route_eps", _f32),
                ("route_mode", _i32), ("route_refine_passes", _i32), ("route_lambda_anc", _f32),
                ("route_lambda_rec", _f32), ("route_refine_tol", _f32), ("scale", _f32),
                ("r_out", _vp), ("r_dtype", _i32),
                ("x", _vp), ("idx_out", _vp), ("channel_weight", _vp), ("par", ParParams),
                ("w_o", _vp), ("b_o", _vp), ("hist", HistLayout), ("route_candidates", _vp),
                ("route_M_c", _i32)]


class FfnArgs(C.Structure):
    _fields_ = [("x", _vp), ("x_row_stride", _i64), ("n_frames", _i32), ("Hg", _i32), ("Wg", _i32),
                ("D", _i32), ("D_ff", _i32), ("anchors", C.POINTER(_i32)), ("n_anchors", _i32),
                ("w1", _vp), ("b1", _vp), ("w2", _vp), ("b2", _vp), ("r_out", _vp), ("r_dtype", _i32),
                ("channel_weight", _vp), ("par", ParParams)]


class SelectArgs(C.Structure):
    _fields_ = [("delta", _vp * 2), ("n_branch", _i32), ("dtype", _i32), ("n_frames", _i32),
                ("frame_elems", _i64), ("ages", _vp), ("anchor_mask", _vp), ("K_f", _i32),
                ("lambda_cov", _f32), ("eps", _f32), ("ages_out", _vp), ("anchors_out", _vp),
                ("mask_out", _vp), ("rms_out", _vp), ("score_out", _vp)]


_lib.cast_ffn_step.argtypes = [C.POINTER(FfnArgs), _vp, C.c_size_t, _vp]
_lib.cast_ffn_workspace_size.argtypes = [C.POINTER(FfnArgs)]
_lib.cast_ffn_workspace_size.restype = C.c_size_t
_lib.cast_select_frames.argtypes = [C.POINTER(SelectArgs), _vp, C.c_size_t, _vp]
_lib.cast_select_workspace_size.argtypes = [C.POINTER(SelectArgs)]
_lib.cast_select_workspace_size.restype = C.c_size_t
_lib.cast_route_topk.argtypes = [C.POINTER(RouteArgs), _vp, C.c_size_t, _vp]
_lib.cast_route_workspace_size.argtypes = [C.POINTER(RouteArgs)]
_lib.cast_route_workspace_size.restype = C.c_size_t
_lib.cast_route_topk_noalloc.argtypes = [C.POINTER(RouteArgs), _vp]
_lib.cast_anchor_attention.argtypes = [C.POINTER(AttnArgs), _vp, C.c_size_t, _vp]
_lib.cast_attention_workspace_size.argtypes = [C.POINTER(AttnArgs)]
_lib.cast_attention_workspace_size.restype = C.c_size_t
_lib.cast_par_reconstruct.argtypes = [C.POINTER(ParArgs), _vp, C.c_size_t, _vp]
_lib.cast_par_workspace_size.argtypes = [C.POINTER(ParArgs)]
_lib.cast_par_workspace_size.restype = C.c_size_t
_lib.cast_block_step.argtypes = [C.POINTER(BlockArgs), _vp, C.c_size_t, _vp]
_lib.cast_block_workspace_size.argtypes = [C.POINTER(BlockArgs)]
_lib.cast_block_workspace_size.restype = C.c_size_t
_lib.cast_par_params_default.argtypes = [C.POINTER(ParParams)]
_lib.cast_status_string.argtypes = [C.c_int]
_lib.cast_status_string.restype = C.c_char_p
_lib.cast_last_error_detail.restype = C.c_char_p
_lib.cast_check_device.argtypes = [_vp]
_lib.cast_selftest_bounded_wait.argtypes = [C.c_uint64, _vp]
_lib.cast_selftest_bounded_wait.restype = C.c_int
_lib.cast_version.restype = C.c_char_p
for _f in ("cast_route_topk", "cast_route_topk_noalloc", "cast_anchor_attention", "cast_par_reconstruct", "cast_block_step",
           "cast_check_device"):
    getattr(_lib, _f).restype = C.c_int

EXPORTED = ["cast_select_frames", "cast_select_workspace_size", "cast_ffn_step",
            "cast_ffn_workspace_size",
            "cast_route_topk", "cast_route_workspace_size", "cast_route_topk_noalloc",
            "cast_anchor_attention", "cast_attention_workspace_size",
            "cast_par_reconstruct", "cast_par_workspace_size", "cast_par_params_default",
            "cast_block_step", "cast_block_workspace_size", "cast_status_string",
            "cast_last_error_detail", "cast_check_device", "cast_version",
            "cast_selftest_bounded_wait"]


class CastError(RuntimeError):
    def __init__(self, status, detail):
        self.status = status
        super().__init__(f"{_lib.cast_status_string(status).decode()}: {detail}")


def _check(status):
    if status != OK:
        raise CastError(status, _lib.cast_last_error_detail().decode())


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return C.c_void_p(s.cuda_stream)


def _dtype_code(t):
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def _host_i32(seq):
    arr = (_i32 * max(1, len(seq)))(*[int(v) for v in seq])
    return arr


def _row_stride(t):
    """Token row stride (elements) of a [frames|blocks, tokens, H, d] tensor whose H, d are
    contiguous and whose tokens of a frame are evenly spaced."""
    if t.dim() != 4 or t.stride(3) != 1 or t.stride(2) != t.shape[3]:
        raise ValueError("expected [N, T, H, d] with contiguous (H, d)")
    if t.shape[0] > 1 and t.stride(0) != t.stride(1) * t.shape[1]:
        raise ValueError("frames must be consecutive token rows")
    return t.stride(1)


def _history(k_hist, H, d):
    """(M, B_v, row stride, HistLayout) of the history tensor: [M, B_v, H, d] blocks, or
    [frames, Hg, Wg, H, d] frames cut into (1, 8, 8) blocks (M = frames ceil(Hg/8) ceil(Wg/8),
    nominal B_v = 64); None means no history."""
    lay = HistLayout()
    if k_hist is None or k_hist.shape[0] == 0:
        return 0, 0, H * d, lay
    if k_hist.dim() == 5:
        F, Hg, Wg = k_hist.shape[:3]
        if Hg > 1 and k_hist.stride(1) != k_hist.stride(2) * Wg:
            raise ValueError("history frames must hold consecutive token rows")
        rs = _row_stride(k_hist.flatten(1, 2))
        lay.kind, lay.frames, lay.Hg, lay.Wg = HIST_FRAMES, F, Hg, Wg
        return F * (-(-Hg // 8)) * (-(-Wg // 8)), 64, rs, lay
    return k_hist.shape[0], k_hist.shape[1], _row_stride(k_hist), lay


def _workspace(nbytes, device):
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


# --------------------------------------------------------------------------- params
def par_params(tile=(8, 8), tau_low=0.25, tau_high=0.75, q=2.0, T=0.10, eps=1e-8, eta_rel=1e-6,
               eta_abs=1e-8, band_radius=-1.0, gate_mode=GATE_PAPER):
    p = ParParams()
    _lib.cast_par_params_default(C.byref(p))
    p.tile_h, p.tile_w = tile
    p.tau_low, p.tau_high, p.q, p.T = tau_low, tau_high, q, T
    p.eps, p.eta_rel, p.eta_abs, p.band_radius, p.gate_mode = eps, eta_rel, eta_abs, band_radius, gate_mode
    return p


def default_par_params():
    p = ParParams()
    _lib.cast_par_params_default(C.byref(p))
    return p


# --------------------------------------------------------------------------- routing
REFINE_PAPER = dict(passes=2, lambda_anc=1.0, lambda_rec=1.0, tol=1e-6)   # Tab. config_cast


def _candidates(candidates):
    """Device int32 [K_f, H, M_c] candidate sets (App. B.3) -> (pointer, M_c)."""
    if candidates is None:
        return None, 0
    if candidates.dtype != torch.int32 or candidates.dim() != 3 or not candidates.is_contiguous():
        raise ValueError("candidates must be a contiguous int32 [K_f, H, M_c] tensor")
    return _ptr(candidates), candidates.shape[2]


def _route_args(q, anchors, k_hist, v_hist, K, gram=None, eps=1e-8, mode=ROUTE_OMISSION,
                refine=None, candidates=None):
    N, S, H, d = q.shape
    M, B_v, rs, lay = _history(k_hist, H, d)
    a = RouteArgs()
    a.q, a.q_row_stride = _ptr(q), _row_stride(q)
    a.n_frames, a.S, a.H, a.d = N, S, H, d
    a.dtype = _dtype_code(q)
    a._anchors = _host_i32(anchors)
    a.anchors = C.cast(a._anchors, C.POINTER(_i32))
    a.n_anchors = len(anchors)
    a.k_hist, a.v_hist = _ptr(k_hist), _ptr(v_hist)
    a.hist_row_stride = rs
    a.M, a.B_v, a.hist = M, B_v if M > 0 else k_hist.shape[1], lay
    a.gram = _ptr(gram)
    a.K, a.eps, a.mode = K, eps, mode
    a.candidates, a.M_c = _candidates(candidates)
    if refine:
        a.refine_passes, a.lambda_anc = refine["passes"], refine["lambda_anc"]
        a.lambda_rec, a.refine_tol = refine["lambda_rec"], refine["tol"]
    return a


def route_workspace_size(q, anchors, k_hist, v_hist, K, refine=None, candidates=None):
    a = _route_args(q, anchors, k_hist, v_hist, K, refine=refine, candidates=candidates)
    return _lib.cast_route_topk and _lib.cast_route_workspace_size(C.byref(a))


def cast_route_topk(q, anchors, k_hist, v_hist, K, gram=None, eps=1e-8, mode=ROUTE_OMISSION,
                    want_u=False, want_pooled=False, workspace=None, stream=None, refine=None,
                    candidates=None):
    """Returns idx [K_f, H, K_eff] int32 (and u, (qbar, kbar, vbar) when asked).  refine: None
    (independent TopK) or a dict like REFINE_PAPER (coupled refinement, Alg. routing);
    candidates: None (every block) or device int32 [K_f, H, M_c] fixed candidate sets."""
    a = _route_args(q, anchors, k_hist, v_hist, K, gram, eps, mode, refine, candidates)
    Kf, H, d, M = len(anchors), q.shape[2], q.shape[3], a.M
    keff = min(K, M)
    dev = q.device
    idx = torch.empty((Kf, H, keff), dtype=torch.int32, device=dev)
    u = torch.empty((Kf, H, M), dtype=torch.float32, device=dev) if want_u else None
    qb = kb = vb = None
    if want_pooled:
        qb = torch.empty((Kf, H, d), dtype=torch.float32, device=dev)
        kb = torch.empty((M, H, d), dtype=torch.float32, device=dev)
        vb = torch.empty((M, H, d), dtype=torch.float32, device=dev)
    a.idx, a.u, a.qbar, a.kbar, a.vbar = _ptr(idx), _ptr(u), _ptr(qb), _ptr(kb), _ptr(vb)
    keff_out = _i32(0)
    a.k_eff = C.pointer(keff_out)
    need = _lib.cast_route_workspace_size(C.byref(a))
    ws = workspace if workspace is not None else _workspace(need, dev)
    _check(_lib.cast_route_topk(C.byref(a), _ptr(ws), ws.numel(), _stream(stream)))
    out = [idx]
    if want_u:
        out.append(u)
    if want_pooled:
        out.append((qb, kb, vb))
    return out[0] if len(out) == 1 else tuple(out)


def cast_route_topk_noalloc(q, anchors, k_hist, v_hist, K, gram=None, eps=1e-8,
                            mode=ROUTE_OMISSION, want_u=False, stream=None):
    """As cast_route_topk, with the library's fixed 16 MiB device scratch instead of a
    caller workspace (for callers that cannot allocate); returns idx (and u)."""
    a = _route_args(q, anchors, k_hist, v_hist, K, gram, eps, mode)
    Kf, H, M = len(anchors), q.shape[2], a.M
    idx = torch.empty((Kf, H, min(K, M)), dtype=torch.int32, device=q.device)
    u = torch.empty((Kf, H, M), dtype=torch.float32, device=q.device) if want_u else None
    a.idx, a.u = _ptr(idx), _ptr(u)
    _check(_lib.cast_route_topk_noalloc(C.byref(a), _stream(stream)))
    return (idx, u) if want_u else idx


# --------------------------------------------------------------------------- attention
def _attn_args(q, k_cur, v_cur, anchors, k_hist, v_hist, idx, scale=0.0):
    N, S, H, d = q.shape
    M, B_v, rs, lay = _history(k_hist, H, d)
    a = AttnArgs()
    a.q, a.k_cur, a.v_cur = _ptr(q), _ptr(k_cur), _ptr(v_cur)
    a.q_row_stride, a.cur_row_stride = _row_stride(q), _row_stride(k_cur)
    a.n_frames, a.S, a.H, a.d = N, S, H, d
    a._anchors = _host_i32(anchors)
    a.anchors = C.cast(a._anchors, C.POINTER(_i32))
    a.n_anchors = len(anchors)
    a.k_hist, a.v_hist = _ptr(k_hist), _ptr(v_hist)
    a.hist_row_stride = rs
    a.M, a.B_v, a.hist = M, B_v, lay
    a.idx = _ptr(idx)
    a.K_eff = idx.shape[-1] if idx is not None else 0
    a.scale = scale
    return a


def attention_workspace_size(q, k_cur, v_cur, anchors, k_hist, v_hist, idx):
    a = _attn_args(q, k_cur, v_cur, anchors, k_hist, v_hist, idx)
    return _lib.cast_attention_workspace_size(C.byref(a))


def cast_anchor_attention(q, k_cur, v_cur, anchors, k_hist, v_hist, idx, scale=0.0,
                          out_dtype=torch.bfloat16, want_lse=False, out=None, workspace=None,
                          stream=None):
    """Returns O [K_f, S, H*d] (and lse [K_f, H, S])."""
    N, S, H, d = q.shape
    Kf = len(anchors)
    a = _attn_args(q, k_cur, v_cur, anchors, k_hist, v_hist, idx, scale)
    o = out if out is not None else torch.empty((Kf, S, H * d), dtype=out_dtype, device=q.device)
    a.o, a.o_dtype = _ptr(o), _dtype_code(o)
    lse = torch.empty((Kf, H, S), dtype=torch.float32, device=q.device) if want_lse else None
    a.lse = _ptr(lse)
    need = _lib.cast_attention_workspace_size(C.byref(a))
    ws = workspace if workspace is not None else _workspace(need, q.device)
    _check(_lib.cast_anchor_attention(C.byref(a), _ptr(ws), ws.numel(), _stream(stream)))
    return (o, lse) if want_lse else o


# --------------------------------------------------------------------------- PAR
def _par_args(r, anchor_mask, channel_weight=None, params=None):
    F, Hg, Wg, Cc = r.shape
    a = ParArgs()
    a.r, a.dtype = _ptr(r), _dtype_code(r)
    a.F, a.Hg, a.Wg, a.C = F, Hg, Wg, Cc
    a._mask = (C.c_uint8 * F)(*[1 if m else 0 for m in anchor_mask])
    a.anchor_mask = C.cast(a._mask, C.POINTER(C.c_uint8))
    a.channel_weight = _ptr(channel_weight)
    a.params = params if params is not None else default_par_params()
    return a


def par_workspace_size(r, anchor_mask, params=None):
    a = _par_args(r, anchor_mask, None, params)
    return _lib.cast_par_workspace_size(C.byref(a))


def cast_par_reconstruct(r, anchor_mask, channel_weight=None, params=None, workspace=None,
                         stream=None):
    """In place on r [F, Hg, Wg, C] (f32 or bf16): skipped frames are overwritten."""
    if not r.is_contiguous():
        raise ValueError("r must be contiguous [F, Hg, Wg, C]")
    a = _par_args(r, anchor_mask, channel_weight, params)
    need = _lib.cast_par_workspace_size(C.byref(a))
    ws = workspace if workspace is not None else _workspace(need, r.device)
    _check(_lib.cast_par_reconstruct(C.byref(a), _ptr(ws), ws.numel(), _stream(stream)))
    return r


# --------------------------------------------------------------------------- block step
def block_args(q, k_cur, v_cur, anchors, k_hist, v_hist, K, grid, r_out, x=None, idx_out=None,
               gram=None, route_eps=1e-8, route_mode=ROUTE_OMISSION, scale=0.0,
               channel_weight=None, params=None, refine=None, w_o=None, b_o=None, candidates=None):
    N, S, H, d = q.shape
    M, B_v, rs, lay = _history(k_hist, H, d)
    a = BlockArgs()
    a.q, a.k_cur, a.v_cur = _ptr(q), _ptr(k_cur), _ptr(v_cur)
    a.q_row_stride, a.cur_row_stride = _row_stride(q), _row_stride(k_cur)
    a.n_frames, a.Hg, a.Wg, a.H, a.d = N, grid[0], grid[1], H, d
    a._anchors = _host_i32(anchors)
    a.anchors = C.cast(a._anchors, C.POINTER(_i32))
    a.n_anchors = len(anchors)
    a.k_hist, a.v_hist = _ptr(k_hist), _ptr(v_hist)
    a.hist_row_stride = rs
    a.M, a.B_v, a.hist = M, B_v if M > 0 else k_hist.shape[1], lay
    a.gram, a.K, a.route_eps, a.route_mode, a.scale = _ptr(gram), K, route_eps, route_mode, scale
    if refine:
        a.route_refine_passes, a.route_lambda_anc = refine["passes"], refine["lambda_anc"]
        a.route_lambda_rec, a.route_refine_tol = refine["lambda_rec"], refine["tol"]
    a.r_out, a.r_dtype = _ptr(r_out), _dtype_code(r_out)
    a.x = _ptr(x)
    a.idx_out = _ptr(idx_out)
    a.channel_weight = _ptr(channel_weight)
    a.par = params if params is not None else default_par_params()
    a.w_o, a.b_o = _ptr(w_o), _ptr(b_o)
    a.route_candidates, a.route_M_c = _candidates(candidates)
    a._keep = (candidates,)
    return a


def block_workspace_size(args):
    return _lib.cast_block_workspace_size(C.byref(args))


def cast_block_step_args(args, workspace, stream=None):
    _check(_lib.cast_block_step(C.byref(args), _ptr(workspace), workspace.numel(), _stream(stream)))


def cast_block_step(q, k_cur, v_cur, anchors, k_hist, v_hist, K, grid, r_out, x=None,
                    idx_out=None, workspace=None, stream=None, **kw):
    """route -> attention -> PAR at one attention residual site; fills r_out [N, S, H*d]."""
    a = block_args(q, k_cur, v_cur, anchors, k_hist, v_hist, K, grid, r_out, x, idx_out, **kw)
    need = block_workspace_size(a)
    ws = workspace if workspace is not None else _workspace(need, q.device)
    cast_block_step_args(a, ws, stream)
    return r_out


def cast_check_device(stream=None):
    _check(_lib.cast_check_device(_stream(stream)))


def cast_selftest_bounded_wait(limit_ns, stream=None):
    """Enqueue a wait that can only end by its deadline (see include/cast.h)."""
    _check(_lib.cast_selftest_bounded_wait(int(limit_ns), _stream(stream)))


def version():
    return _lib.cast_version().decode()


def library():
    return _lib


# --------------------------------------------------------------------------- frame selection
def select_args(deltas, ages, anchor_mask, K_f, lambda_cov=0.5, eps=1e-8):
    """deltas: list of 0..2 device tensors [N_cur, ...] (same dtype, contiguous); ages int32 and
    anchor_mask uint8 device tensors [N_cur]."""
    a = SelectArgs()
    N = ages.shape[0]
    a.n_branch = len(deltas)
    for k, dk in enumerate(deltas):
        if not dk.is_contiguous():
            raise ValueError("control updates must be contiguous")
        a.delta[k] = dk.data_ptr()
    a.dtype = (F32 if deltas[0].dtype == torch.float32 else BF16) if deltas else F32
    a.n_frames = N
    a.frame_elems = deltas[0][0].numel() if deltas else 0
    a.ages, a.anchor_mask = _ptr(ages), _ptr(anchor_mask)
    a.K_f, a.lambda_cov, a.eps = K_f, lambda_cov, eps
    return a


def cast_select_frames(deltas, ages, anchor_mask, K_f, lambda_cov=0.5, eps=1e-8, want_rms=False,
                       want_score=False, workspace=None, stream=None):
    """Anchors of the next block (Eqs. sensitivity, normalization, debt, score).  Returns
    (anchors int32 [min(K_f, N)] ascending, ages int32 [N], mask uint8 [N]) plus the RMS
    [n_branch, N] and the scores [N] when asked; all on the device."""
    a = select_args(deltas, ages, anchor_mask, K_f, lambda_cov, eps)
    N, dev = ages.shape[0], ages.device
    anchors = torch.empty(min(K_f, N), dtype=torch.int32, device=dev)
    ages_out = torch.empty(N, dtype=torch.int32, device=dev)
    mask = torch.empty(N, dtype=torch.uint8, device=dev)
    rms = torch.empty((len(deltas), N), dtype=torch.float32, device=dev) if want_rms else None
    score = torch.empty(N, dtype=torch.float32, device=dev) if want_score else None
    a.ages_out, a.anchors_out, a.mask_out = _ptr(ages_out), _ptr(anchors), _ptr(mask)
    a.rms_out, a.score_out = _ptr(rms), _ptr(score)
    need = _lib.cast_select_workspace_size(C.byref(a))
    ws = workspace if workspace is not None else _workspace(need, dev)
    _check(_lib.cast_select_frames(C.byref(a), _ptr(ws), ws.numel(), _stream(stream)))
    out = [anchors, ages_out, mask]
    if want_rms:
        out.append(rms)
    if want_score:
        out.append(score)
    return tuple(out)


def select_workspace_size(deltas, ages, anchor_mask, K_f):
    return _lib.cast_select_workspace_size(C.byref(select_args(deltas, ages, anchor_mask, K_f)))


# --------------------------------------------------------------------------- FFN site
def ffn_args(x, anchors, w1, b1, w2, b2, grid, r_out, channel_weight=None, params=None):
    """x bf16 [F, S, D] (token rows contiguous per frame); w1 bf16 [D_ff, D], w2 bf16 [D, D_ff];
    b1 bf16 [D_ff] or None; b2 [D] of r_out's dtype or None; r_out [F, S, D] f32 or bf16."""
    F, S, D = x.shape[0], x.shape[1], x.shape[-1]
    a = FfnArgs()
    a.x, a.x_row_stride = _ptr(x), x.stride(1) if x.dim() == 3 else D
    a.n_frames, a.Hg, a.Wg, a.D, a.D_ff = F, grid[0], grid[1], D, w1.shape[0]
    a._anchors = _host_i32(anchors)
    a.anchors = C.cast(a._anchors, C.POINTER(_i32))
    a.n_anchors = len(anchors)
    a.w1, a.b1, a.w2, a.b2 = _ptr(w1), _ptr(b1), _ptr(w2), _ptr(b2)
    a.r_out = _ptr(r_out)
    a.r_dtype = F32 if r_out.dtype == torch.float32 else BF16
    a.channel_weight = _ptr(channel_weight)
    a.par = params if params is not None else default_par_params()
    return a


def cast_ffn_step(x, anchors, w1, b1, w2, b2, grid, r_out, channel_weight=None, params=None,
                  workspace=None, stream=None):
    """Anchor FFN residuals into r_out's anchor rows, PAR for the skipped rows."""
    a = ffn_args(x, anchors, w1, b1, w2, b2, grid, r_out, channel_weight, params)
    need = _lib.cast_ffn_workspace_size(C.byref(a))
    ws = workspace if workspace is not None else _workspace(need, x.device)
    _check(_lib.cast_ffn_step(C.byref(a), _ptr(ws), ws.numel(), _stream(stream)))
    return r_out


def ffn_workspace_size(x, anchors, w1, b1, w2, b2, grid, r_out):
    return _lib.cast_ffn_workspace_size(C.byref(ffn_args(x, anchors, w1, b1, w2, b2, grid, r_out)))

