"""The C ABI on the CPU: the library loads, exports every function include/cast.h declares, and
rejects bad arguments with the documented status before any CUDA call (no GPU needed)."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "cast.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"\b(cast_[a-z_]+)\s*\(", src)
    return sorted(set(names))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_34144_gb300 import native
    return native


def test_header_declares_the_entry_points():
    d = _declared()
    for n in ("cast_route_topk", "cast_anchor_attention", "cast_par_reconstruct", "cast_block_step"):
        assert n in d


def test_every_declared_symbol_is_exported(lib):
    so = lib.library()
    for name in _declared():
        assert hasattr(so, name), name
    assert set(_declared()) <= set(lib.EXPORTED) | {"cast_version"}


def test_status_strings(lib):
    so = lib.library()
    assert so.cast_status_string(0) == b"CAST_OK"
    assert so.cast_status_string(4) == b"CAST_ERR_DEVICE_TIMEOUT"


def test_default_params_are_the_papers(lib):
    p = lib.default_par_params()
    assert (p.tile_h, p.tile_w) == (8, 8)
    assert abs(p.tau_low - 0.25) < 1e-7 and abs(p.tau_high - 0.75) < 1e-7
    assert abs(p.q - 2.0) < 1e-7 and abs(p.T - 0.10) < 1e-7
    assert abs(p.eta_rel - 1e-6) < 1e-12 and abs(p.eta_abs - 1e-8) < 1e-14
    assert p.band_radius < 0 and p.gate_mode == lib.GATE_PAPER


def _fake(addr=0x10000):
    return C.c_void_p(addr)


def _route(lib, **kw):
    a = lib.RouteArgs()
    a.q = _fake()
    a.q_row_stride = 256
    a.n_frames, a.S, a.H, a.d = 3, 16, 2, 128
    a.dtype = lib.BF16
    anchors = kw.pop("anchors", [0, 2])
    a._an = (C.c_int32 * len(anchors))(*anchors)
    a.anchors = C.cast(a._an, C.POINTER(C.c_int32))
    a.n_anchors = len(anchors)
    a.k_hist, a.v_hist = _fake(0x20000), _fake(0x30000)
    a.hist_row_stride = 256
    a.M, a.B_v, a.K, a.eps, a.mode = 4, 8, 2, 1e-8, 0
    a.idx = _fake(0x40000)
    for k, v in kw.items():
        setattr(a, k, v)
    return a


@pytest.mark.parametrize("bad,status", [
    ({"anchors": [2, 0]}, 1),
    ({"anchors": [0, 5]}, 1),
    ({"d": 96}, 2),
    ({"q_row_stride": 100}, 1),
    ({"q": _fake(0x10008)}, 1),
    ({"K": -1}, 1),
    ({"mode": 7}, 1),
    ({"refine_passes": -1}, 1),
    ({"refine_passes": 2, "mode": 1}, 1),            # refinement needs the omission score
    ({"refine_passes": 2, "lambda_rec": -1.0}, 1),
    ({"refine_passes": 2, "M": 10000}, 2),           # u and masks exceed shared memory
])
def test_route_validation(lib, bad, status):
    a = _route(lib, **bad)
    ws = C.create_string_buffer(16)
    assert lib.library().cast_route_topk(C.byref(a), ws, 0, None) == status
    assert lib.library().cast_last_error_detail() != b""


def test_route_short_workspace_is_rejected(lib):
    a = _route(lib)
    need = lib.library().cast_route_workspace_size(C.byref(a))
    assert need > 0
    assert lib.library().cast_route_topk(C.byref(a), _fake(0x100000), need - 1, None) == 1


def _par(lib, mask, **kw):
    a = lib.ParArgs()
    a.r = _fake()
    a.dtype = lib.F32
    a.F, a.Hg, a.Wg, a.C = len(mask), 16, 16, 64
    a._m = (C.c_uint8 * len(mask))(*mask)
    a.anchor_mask = C.cast(a._m, C.POINTER(C.c_uint8))
    a.params = lib.default_par_params()
    for k, v in kw.items():
        if k.startswith("p_"):
            setattr(a.params, k[2:], v)
        else:
            setattr(a, k, v)
    return a


@pytest.mark.parametrize("mask,kw,status", [
    ([1, 0, 0], {}, 1),                   # one anchor with skipped frames (Eq. block needs two)
    ([1, 0, 1], {"C": 60}, 2),            # channels not a multiple of 8
    ([1, 0, 1], {"p_tile_h": 9}, 2),      # tile side above 8
    ([1, 0, 1], {"p_T": 0.0}, 1),         # gate temperature must be positive
    ([1, 0, 1], {"p_gate_mode": 5}, 1),
    ([1, 0, 1], {"dtype": 9}, 1),
])
def test_par_validation(lib, mask, kw, status):
    a = _par(lib, mask, **kw)
    assert lib.library().cast_par_reconstruct(C.byref(a), _fake(0x100000), 1 << 30, None) == status


def test_par_all_anchors_needs_nothing(lib):
    a = _par(lib, [1, 1, 1])
    # nothing to reconstruct: returns OK before touching the device
    assert lib.library().cast_par_reconstruct(C.byref(a), None, 0, None) == 0


def test_par_workspace_size(lib):
    # chunk records (120 floats per 128-channel chunk) and theta, g (80 floats) per tile and anchor
    def up(x):
        return (x + 255) // 256 * 256
    so = lib.library()
    for ch in (64, 512, 3072):
        a = _par(lib, [1, 0, 1], C=ch)
        tiles, na, chunks = 4, 2, -(-ch // 128)      # 16 x 16 grid of 8x8 tiles, 2 anchors
        want = up(tiles * na * chunks * 120 * 4) + up(tiles * na * 80 * 4)
        assert so.cast_par_workspace_size(C.byref(a)) == want
        assert so.cast_par_reconstruct(C.byref(a), _fake(0x100000), want - 1, None) == 1
    assert so.cast_par_workspace_size(C.byref(_par(lib, [1, 1, 1]))) == 0   # nothing to reconstruct


def test_attention_validation(lib):
    a = lib.AttnArgs()
    a.q = a.k_cur = a.v_cur = _fake()
    a.q_row_stride = a.cur_row_stride = 256
    a.n_frames, a.S, a.H, a.d = 2, 16, 2, 128
    an = (C.c_int32 * 1)(1)
    a.anchors = C.cast(an, C.POINTER(C.c_int32))
    a.n_anchors = 1
    a.M, a.B_v, a.K_eff = 0, 1, 1          # routed blocks without history
    a.o, a.o_dtype = _fake(), lib.BF16
    assert lib.library().cast_anchor_attention(C.byref(a), None, 0, None) == 1
    a.K_eff, a.d = 0, 80
    assert lib.library().cast_anchor_attention(C.byref(a), None, 0, None) == 2


def _select(lib, **kw):
    a = lib.SelectArgs()
    a.delta[0], a.delta[1] = 0x10000, 0x20000
    a.n_branch, a.dtype, a.n_frames, a.frame_elems = 2, lib.BF16, 8, 1560 * 1536
    a.ages, a.anchor_mask = 0x30000, 0x40000
    a.K_f, a.lambda_cov, a.eps = 4, 0.5, 1e-8
    a.ages_out, a.anchors_out = 0x50000, 0x60000
    for k, v in kw.items():
        setattr(a, k, v)
    return a


@pytest.mark.parametrize("bad,status", [
    ({"K_f": 0}, 1),
    ({"n_frames": 0}, 1),
    ({"n_frames": 257}, 1),
    ({"n_branch": 3}, 1),
    ({"frame_elems": 7}, 1),             # 14 bytes per frame: not a multiple of 16
    ({"lambda_cov": -1.0}, 1),
    ({"anchors_out": None}, 1),
])
def test_select_validation(lib, bad, status):
    a = _select(lib, **bad)
    assert lib.library().cast_select_frames(C.byref(a), _fake(0x100000), 1 << 20, None) == status
    assert lib.library().cast_last_error_detail() != b""


def test_select_misaligned_update_rejected(lib):
    a = _select(lib)
    a.delta[1] = 0x20008
    assert lib.library().cast_select_frames(C.byref(a), _fake(0x100000), 1 << 20, None) == 1


def test_select_workspace(lib):
    assert lib.library().cast_select_workspace_size(C.byref(_select(lib, n_branch=0))) == 0
    assert lib.library().cast_select_workspace_size(C.byref(_select(lib))) > 0


def test_ffn_validation(lib):
    a = lib.FfnArgs()
    a.x, a.x_row_stride = _fake(), 64
    a.n_frames, a.Hg, a.Wg, a.D, a.D_ff = 3, 4, 4, 64, 256
    an = (C.c_int32 * 2)(0, 2)
    a.anchors, a.n_anchors = C.cast(an, C.POINTER(C.c_int32)), 2
    a.w1, a.w2, a.r_out, a.r_dtype = _fake(0x20000), _fake(0x30000), _fake(0x40000), lib.F32
    a.par = lib.default_par_params()
    so = lib.library()
    need = so.cast_ffn_workspace_size(C.byref(a))
    # hidden activations [2 anchors, 16 rows, 256] bf16, then PAR's records and theta / g of the
    # single (4x4) tile: 2 anchors x 1 chunk x 120 floats and 2 x 80 floats, each 256-B aligned
    assert need == 2 * 16 * 256 * 2 + 1024 + 768
    assert so.cast_ffn_step(C.byref(a), _fake(0x100000), need - 1, None) == 1      # short workspace
    a.D = 60
    assert so.cast_ffn_step(C.byref(a), _fake(0x100000), need, None) == 1          # D not a multiple of 8
    a.D, a.w1 = 64, _fake(0x20004)
    assert so.cast_ffn_step(C.byref(a), _fake(0x100000), need, None) == 1          # misaligned weight



@pytest.mark.parametrize("hist,M,B_v,status", [
    ((5, 0, 0, 0), 4, 8, 1),                 # unknown layout kind
    ((1, 0, 16, 16), 4, 64, 1),              # no history frames
    ((1, 1, 16, 16), 4, 64, 0),              # 1 frame of 16x16 tokens = 4 (1,8,8) blocks
    ((1, 1, 17, 16), 4, 64, 1),              # 17 rows: 3 x 2 = 6 blocks, not 4
    ((1, 2, 9, 20), 12, 64, 0),              # truncated edge blocks: 2 x 2 x 3
    ((1, 1, 16, 16), 4, 8, 1),               # B_v must be the nominal 64
])
def test_route_history_layout_validation(lib, hist, M, B_v, status):
    a = _route(lib, M=M, B_v=B_v)
    a.hist.kind, a.hist.frames, a.hist.Hg, a.hist.Wg = hist
    so = lib.library()
    if status:
        assert so.cast_route_topk(C.byref(a), _fake(0x100000), 1 << 30, None) == status
        assert so.cast_last_error_detail() != b""
    else:
        # valid layouts pass validation: the call only fails later for the missing workspace
        assert so.cast_route_topk(C.byref(a), None, 0, None) == 1
        assert b"workspace" in so.cast_last_error_detail()


def test_attention_history_layout_validation(lib):
    a = lib.AttnArgs()
    a.q = a.k_cur = a.v_cur = _fake()
    a.k_hist, a.v_hist = _fake(0x20000), _fake(0x30000)
    a.q_row_stride = a.cur_row_stride = a.hist_row_stride = 256
    a.n_frames, a.S, a.H, a.d = 2, 16, 2, 128
    an = (C.c_int32 * 1)(1)
    a.anchors = C.cast(an, C.POINTER(C.c_int32))
    a.n_anchors = 1
    a.idx = _fake(0x40000)
    a.M, a.B_v, a.K_eff = 6, 64, 3
    a.o, a.o_dtype = _fake(), lib.BF16
    a.hist.kind, a.hist.frames, a.hist.Hg, a.hist.Wg = lib.HIST_FRAMES, 1, 16, 16   # 4 blocks
    so = lib.library()
    assert so.cast_anchor_attention(C.byref(a), None, 1 << 30, None) == 1
    assert b"(1,8,8)" in so.cast_last_error_detail()


def test_struct_layouts_match_the_header(lib, tmp_path):
    """Every ctypes argument struct has the size and field offsets that a C compiler gives
    the header's struct (compiled with gcc on the host)."""
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        pytest.skip("no gcc")
    structs = {"cast_route_args": lib.RouteArgs, "cast_attn_args": lib.AttnArgs,
               "cast_par_params": lib.ParParams, "cast_par_args": lib.ParArgs,
               "cast_block_args": lib.BlockArgs, "cast_ffn_args": lib.FfnArgs,
               "cast_select_args": lib.SelectArgs, "cast_hist_layout": lib.HistLayout}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "cast.h"', "int main(void) {"]
    for cname, py in structs.items():
        lines.append(f'printf("{cname} sizeof %zu\\n", sizeof({cname}));')
        for fname, _ in py._fields_:
            lines.append(f'printf("{cname} {fname} %zu\\n", offsetof({cname}, {fname}));')
    lines += ["return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)],
                   check=True, capture_output=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout
    for line in out.splitlines():
        cname, fname, val = line.split()
        py = structs[cname]
        got = C.sizeof(py) if fname == "sizeof" else getattr(py, fname).offset
        assert got == int(val), (cname, fname, got, int(val))


@pytest.mark.parametrize("M_c,status", [(1, 1), (2, 0), (4, 0), (5, 1)])
def test_route_candidate_set_size_validation(lib, M_c, status):
    a = _route(lib)                  # M = 4, K = 2
    a.candidates, a.M_c = _fake(0x50000), M_c
    so = lib.library()
    assert so.cast_route_topk(C.byref(a), None, 0, None) == 1
    msg = so.cast_last_error_detail()
    assert (b"M_c" in msg) == bool(status), msg


def test_selftest_limit_validated_on_the_host(lib):
    so = lib.library()
    assert so.cast_selftest_bounded_wait(10, None) == 1            # below 1 us
    assert so.cast_selftest_bounded_wait(3_000_000_000, None) == 1  # above 2 s
    assert so.cast_last_error_detail() != b""


def _block(lib, **kw):
    a = lib.BlockArgs()
    a.q, a.k_cur, a.v_cur = _fake(), _fake(0x20000), _fake(0x30000)
    a.q_row_stride = a.cur_row_stride = 256
    a.n_frames, a.Hg, a.Wg, a.H, a.d = 4, 4, 4, 2, 128
    anchors = kw.pop("anchors", [0, 3])
    a._an = (C.c_int32 * len(anchors))(*anchors)
    a.anchors = C.cast(a._an, C.POINTER(C.c_int32))
    a.n_anchors = len(anchors)
    a.k_hist, a.v_hist = _fake(0x40000), _fake(0x50000)
    a.hist_row_stride = 256
    a.M, a.B_v, a.K, a.route_eps = 4, 8, 2, 1e-8
    a.r_out, a.r_dtype = _fake(0x60000), lib.BF16
    a.par = lib.default_par_params()
    for k, v in kw.items():
        if k.startswith("p_"):
            setattr(a.par, k[2:], v)
        else:
            setattr(a, k, v)
    return a


@pytest.mark.parametrize("bad,status", [
    ({"anchors": [3, 0]}, 1),                 # anchors must ascend
    ({"anchors": [1]}, 1),                    # skipped frames need two anchors (Eq. block)
    ({"d": 96}, 2),                           # head dim outside {64, 128}
    ({"K": -1}, 1),
    ({"r_dtype": 7}, 1),
    ({"r_out": None}, 1),
    ({"route_refine_passes": -1}, 1),
    ({"p_T": 0.0}, 1),                        # PAR gate temperature
    ({"w_o": _fake(0x70008)}, 1),             # misaligned output projection
])
def test_block_step_validation(lib, bad, status):
    """Validation runs on the host before any launch, so these need no GPU."""
    a = _block(lib, **bad)
    assert lib.library().cast_block_step(C.byref(a), _fake(0x100000), 1 << 30, None) == status
    assert lib.library().cast_last_error_detail() != b""


def test_block_step_short_workspace_is_rejected(lib):
    a = _block(lib)
    need = lib.library().cast_block_workspace_size(C.byref(a))
    assert need > 0
    assert lib.library().cast_block_step(C.byref(a), _fake(0x100000), need - 1, None) == 1
