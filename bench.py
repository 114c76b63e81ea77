"""Benchmark of the CAST block step on GB300: prints one JSON line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Workload: the Matrix-Game-3.0-shaped bf16 block step (8 current latent frames of 30x52 tokens,
12 heads x 128, 16 history blocks of 1560 tokens, K = 4, anchors every second frame).
A step is cast_block_step: routing (pooled scores, TopK, then the reconstruction-coupled
refinement with the paper's L_s = 2 passes and (lambda_anc, lambda_rec) = (1, 1)) -> routed
anchor attention -> PAR.
  value   frames/s with inputs resident in HBM (CUDA events around each step, L2 flushed
          between steps outside the timed events)
  e2e     frames/s through the same C call with the inputs copied from pinned host memory
          and r_out copied back, copies inside the timed region (double-buffered: step k+1's
          upload and step k-1's read-back overlap step k's compute)
  roofline  the dominant kernel (routed attention): algorithmic FLOP per launch / its average
          CUDA-event duration (stages launched through their own entry points, same kernels
          and launch configuration as inside the block step) against the measured bf16 peak
  cpu_baseline  the CPU oracle timed on a bounded sample of the same workload
Under torchrun each rank runs its own block step (independent chunks, no collective): weak
scaling, value = frames of all ranks / max over ranks of the timed region.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from synthetic import generators as G  # noqa: E402
from synthetic import workloads as W  # noqa: E402

METRIC = "block-step frames/s; routed-attn TFLOP/s & PAR GB/s as % of GB300 peak"
WL = W.MG


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d.get("hbm_gbs", 6800.0), d.get("bf16_tflops", 1900.0), "measured"
    return 6800.0, 1900.0, "fallback"


def algorithmic_work(wl):
    S, D = wl.S, wl.H * wl.d
    keff = min(wl.K, wl.M)
    Kf = len(wl.anchors)
    attn_flop = 4.0 * Kf * S * (wl.n_cur * S + keff * wl.B_v) * wl.d * wl.H
    route_bytes = (Kf * S + 2 * wl.M * wl.B_v) * D * 2.0
    par_bytes = wl.n_cur * S * D * 2.0   # anchors read once + skipped frames written once (bf16)
    return attn_flop, route_bytes, par_bytes


# ------------------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, dev_index):
        self.proc = None
        self.dev = dev_index

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.dev)], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[3:7]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ------------------------------------------------------------------------------ GPU arm
def reduce_max_ms(total_ms, world, device):
    """The job's time is the slowest rank's: max over ranks (all-reduce; identity on one rank)."""
    if world <= 1:
        return total_ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([total_ms], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_value(world, frames_per_rank, steps, max_ms):
    """Frames of all ranks (each runs its own chunk: weak scaling) per second of the slowest."""
    return world * frames_per_rank * steps / (max_ms / 1e3)


def run_gpu(args):
    import torch
    import torch.distributed as dist

    from paper_2609_34144_gb300 import native as lib

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    wl = WL
    inp = W.block_step_inputs(wl)

    def to_bf16_host(x):
        return torch.from_numpy(G.bf16_bits(x).view(np.int16)).view(torch.bfloat16)

    names = ("q", "k_cur", "v_cur", "k_hist", "v_hist")
    host = {k: to_bf16_host(inp[k]).pin_memory() for k in names}
    d = {k: host[k].to(dev) for k in names}
    N, S, H, dh = inp["q"].shape
    anchors = list(wl.anchors)
    keff = min(wl.K, wl.M)
    r_out = torch.empty((N, S, H * dh), dtype=torch.bfloat16, device=dev)
    idx = torch.empty((len(anchors), H, keff), dtype=torch.int32, device=dev)
    params = lib.par_params(band_radius=wl.band_radius)
    bargs = lib.block_args(d["q"], d["k_cur"], d["v_cur"], anchors, d["k_hist"], d["v_hist"],
                           wl.K, wl.grid, r_out, idx_out=idx, params=params,
                           refine=lib.REFINE_PAPER)
    ws = torch.empty(max(lib.block_workspace_size(bargs), 256), dtype=torch.uint8, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        lib.cast_block_step_args(bargs, ws)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    lib.cast_check_device()

    # ---------------- timed region: device-resident inputs
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    clocks = ClockSampler(local)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.25)
    for k in range(args.steps):
        flush.fill_(k & 0xFF)   # L2 flush, outside the step's events
        ev[k][0].record(stream)
        step()
        ev[k][1].record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    if world > 1:
        dist.barrier()
    lib.cast_check_device()
    ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = reduce_max_ms(sum(ms), world, dev)
    value = whole_job_value(world, N, args.steps, total_ms)

    # ---------------- per-stage breakdown (same kernels through the stage entry points)
    o_att = torch.empty((len(anchors), S, H * dh), dtype=torch.bfloat16, device=dev)
    r_par = torch.empty_like(r_out)
    r_par.copy_(r_out)
    mask = W.anchor_mask(N, anchors)
    rws = torch.empty(max(lib.route_workspace_size(d["q"], anchors, d["k_hist"], d["v_hist"], wl.K,
                                                   refine=lib.REFINE_PAPER), 256),
                      dtype=torch.uint8, device=dev)
    pws = torch.empty(max(lib.par_workspace_size(r_par.view(N, wl.grid[0], wl.grid[1], H * dh), mask,
                                                 params), 256), dtype=torch.uint8, device=dev)
    aws = torch.empty(max(lib.attention_workspace_size(d["q"], d["k_cur"], d["v_cur"], anchors,
                                                      d["k_hist"], d["v_hist"], idx), 256),
                      dtype=torch.uint8, device=dev)
    nb = max(20, args.steps // 4)
    st_ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(nb)]
    rp = r_par.view(N, wl.grid[0], wl.grid[1], H * dh)
    for k in range(nb + 3):
        flush.fill_(k & 0xFF)
        e = st_ev[k - 3] if k >= 3 else None
        if e:
            e[0].record(stream)
        lib.cast_route_topk(d["q"], anchors, d["k_hist"], d["v_hist"], wl.K, workspace=rws,
                            refine=lib.REFINE_PAPER)
        if e:
            e[1].record(stream)
        lib.cast_anchor_attention(d["q"], d["k_cur"], d["v_cur"], anchors, d["k_hist"], d["v_hist"],
                                  idx, out=o_att, workspace=aws)
        if e:
            e[2].record(stream)
        lib.cast_par_reconstruct(rp, mask, None, params, workspace=pws)
        if e:
            e[3].record(stream)
    torch.cuda.synchronize()
    t_route = statistics.mean(e[0].elapsed_time(e[1]) for e in st_ev)
    t_attn = statistics.mean(e[1].elapsed_time(e[2]) for e in st_ev)
    t_par = statistics.mean(e[2].elapsed_time(e[3]) for e in st_ev)

    # ---------------- end to end through the C call with host buffers
    # Double-buffered, as a serving loop runs it: the inputs of step k+1 travel host -> device on
    # a copy stream while step k computes, and each step's result goes device -> host on a second
    # copy stream.  Every step's copies are inside the timed region (first upload to last read).
    h_out = [torch.empty((N, S, H * dh), dtype=torch.bfloat16).pin_memory() for _ in range(2)]
    sets = [(d, r_out, bargs, ws)]
    d1 = {k: torch.empty_like(d[k]) for k in names}
    r1 = torch.empty_like(r_out)
    idx1 = torch.empty_like(idx)
    b1 = lib.block_args(d1["q"], d1["k_cur"], d1["v_cur"], anchors, d1["k_hist"], d1["v_hist"],
                        wl.K, wl.grid, r1, idx_out=idx1, params=params, refine=lib.REFINE_PAPER)
    sets.append((d1, r1, b1, torch.empty_like(ws)))
    up, down = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    uploaded = [torch.cuda.Event() for _ in range(2)]
    computed = [torch.cuda.Event() for _ in range(2)]
    read = [torch.cuda.Event() for _ in range(2)]
    ne = max(10, args.steps // 4)

    def e2e_run(n):
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        t0.record(stream)
        up.wait_stream(stream)
        down.wait_stream(stream)
        for k in range(n):
            sb = k % 2
            dk, rk, ak, wk = sets[sb]
            if k >= 2:
                up.wait_event(computed[sb])       # step k-2 has finished reading this input set
            with torch.cuda.stream(up):
                for nm in names:
                    dk[nm].copy_(host[nm], non_blocking=True)
                uploaded[sb].record(up)
            stream.wait_event(uploaded[sb])
            if k >= 2:
                stream.wait_event(read[sb])       # step k-2's result has been read back
            lib.cast_block_step_args(ak, wk)
            computed[sb].record(stream)
            down.wait_event(computed[sb])
            with torch.cuda.stream(down):
                h_out[sb].copy_(rk, non_blocking=True)
                read[sb].record(down)
        stream.wait_stream(down)
        t1.record(stream)
        torch.cuda.synchronize()
        return t0.elapsed_time(t1) / n

    e2e_run(2)
    e2e_ms = e2e_run(ne)
    lib.cast_check_device()
    h2d = sum(host[nm].numel() * host[nm].element_size() for nm in names)
    d2h = h_out[0].numel() * h_out[0].element_size()

    if rank == 0:
        hbm, bf16, src = _peaks()
        attn_flop, route_bytes, par_bytes = algorithmic_work(wl)
        achieved = attn_flop / (t_attn / 1e3) / 1e12
        traffic = _captured_traffic()
        line = {
            "metric": METRIC, "value": round(value, 3), "unit": "frames/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(total_ms / args.steps, 5), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": wl.name, "frames_per_step": N, "grid": list(wl.grid),
                       "heads": H, "head_dim": dh, "history_blocks": wl.M, "block_tokens": wl.B_v,
                       "K": wl.K, "anchors": anchors, "global_batch": world,
                       "routing": "coupled refinement, 2 passes, lambda (1, 1), tol 1e-6",
                       "l2": "flushed (256 MiB write) between timed steps, outside the events",
                       "parallelism": f"replicas x{world} (independent chunks, no collective)"},
            "roofline": {"bound": "tensor", "kernel": "k_attn<128> (routed anchor attention)",
                         "achieved": round(achieved, 2), "peak": bf16, "unit": "TFLOP/s",
                         "frac": round(achieved / bf16, 4), "peak_source": f"{src} bf16 burst",
                         "traffic": traffic, "flop_per_launch": attn_flop,
                         "launch_ms": round(t_attn, 5)},
            "breakdown": {
                "route": {"ms": round(t_route, 5), "GB/s": round(route_bytes / t_route / 1e6, 1),
                          "frac_hbm": round(route_bytes / t_route / 1e6 / hbm, 4),
                          "bytes": route_bytes, "kernels": 3},
                "attention": {"ms": round(t_attn, 5), "TFLOP/s": round(achieved, 2),
                              "frac_bf16": round(achieved / bf16, 4)},
                "par": {"ms": round(t_par, 5), "GB/s": round(par_bytes / t_par / 1e6, 1),
                        "frac_hbm": round(par_bytes / t_par / 1e6 / hbm, 4), "bytes": par_bytes},
                "hbm_peak_gbs": hbm},
            "e2e": {"value": round(N / (e2e_ms / 1e3) * world, 3), "unit": "frames/s",
                    "ms_per_step": round(e2e_ms, 4), "h2d_bytes_per_step": int(h2d),
                    "d2h_bytes_per_step": int(d2h),
                    "pipeline": "double-buffered: upload of step k+1 and read-back of step k-1 "
                                "overlap step k (host link ~210 GB/s measured)"},
            "gpu_launches": launches_per_step(wl) * args.steps,
            "clocks": clk,
        }
        if not args.no_scale_points:
            line["scale_points"] = scale_points(lib, torch, dev, flush)
        if not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline(wl)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ------------------------------------------------------------------------------ scale points
SCALE_POINTS = ("par_sweep_f32", "par_sweep_bf16", "route_stress", "attn_hy", "select_mg", "ffn_mg",
                "route_mg64", "attn_mg64", "attn_hy64", "block_mg64", "block_hy", "block_hy64")


def _block_tokens(wl):
    """Tokens of each (1, 8, 8) block of the workload's history frames (edge blocks truncated)."""
    hg, wg = wl.grid
    ys = [min(8, hg - 8 * by) for by in range(-(-hg // 8))]
    xs = [min(8, wg - 8 * bx) for bx in range(-(-wg // 8))]
    per_frame = [h * w for h in ys for w in xs]
    return per_frame * wl.hist_frames


def _scale_setup(name, lib, torch, dev):
    """Inputs (seeded, generated on the device) and the call for one full-size stage run.
    Returns (fn, work, unit): work is algorithmic bytes or FLOP per call."""
    g = torch.Generator(device=dev).manual_seed(0)

    def rnd(*shape, dtype=torch.bfloat16):
        return torch.randn(*shape, generator=g, device=dev, dtype=torch.float32).to(dtype)

    if name.startswith("par_sweep"):
        w = W.PAR_SWEEP
        dt = torch.float32 if name.endswith("f32") else torch.bfloat16
        r = rnd(w.F, w.grid[0], w.grid[1], w.C, dtype=dt)
        wc = torch.rand(w.C, generator=g, device=dev)
        mask = W.anchor_mask(w.F, w.anchors(2))
        p = lib.par_params(band_radius=w.band_radius)
        ws = torch.empty(lib.par_workspace_size(r, mask, p), dtype=torch.uint8, device=dev)
        return (lambda: lib.cast_par_reconstruct(r, mask, wc, p, workspace=ws),
                r.numel() * r.element_size(), "B")
    if name == "route_stress":
        s = W.STRESS
        q = rnd(s.n_cur, s.S, s.H, s.d)
        kh, vh = rnd(s.M, s.B_v, s.H, s.d), rnd(s.M, s.B_v, s.H, s.d)
        an = list(range(s.n_cur))
        ws = torch.empty(lib.route_workspace_size(q, an, kh, vh, 8), dtype=torch.uint8, device=dev)
        return (lambda: lib.cast_route_topk(q, an, kh, vh, 8, workspace=ws),
                (s.n_cur * s.S + 2 * s.M * s.B_v) * s.H * s.d * 2, "B")
    if name == "attn_hy":
        wl = W.HY
        N, S = wl.n_cur, wl.S
        q, kc, vc = rnd(N, S, wl.H, wl.d), rnd(N, S, wl.H, wl.d), rnd(N, S, wl.H, wl.d)
        kh, vh = rnd(wl.M, wl.B_v, wl.H, wl.d), rnd(wl.M, wl.B_v, wl.H, wl.d)
        Kf = len(wl.anchors)
        perm = torch.stack([torch.randperm(wl.M, generator=torch.Generator().manual_seed(k))[:wl.K]
                            for k in range(Kf * wl.H)]).view(Kf, wl.H, wl.K)
        idx = perm.int().to(dev)
        o = torch.empty((Kf, S, wl.H * wl.d), dtype=torch.bfloat16, device=dev)
        flop = 4.0 * Kf * S * (N * S + wl.K * wl.B_v) * wl.d * wl.H
        aws = torch.empty(max(lib.attention_workspace_size(q, kc, vc, list(wl.anchors), kh, vh, idx), 256),
                          dtype=torch.uint8, device=dev)
        return (lambda: lib.cast_anchor_attention(q, kc, vc, list(wl.anchors), kh, vh, idx, out=o,
                                                  workspace=aws),
                flop, "FLOP")
    if name == "select_mg":
        w = W.SELECT_MG
        S = w.grid[0] * w.grid[1]
        deltas = [rnd(w.n_cur, S, w.D) for _ in range(w.n_branch)]
        ages = torch.zeros(w.n_cur, dtype=torch.int32, device=dev)
        mask = torch.zeros(w.n_cur, dtype=torch.uint8, device=dev)
        mask[::2] = 1
        ws = torch.empty(max(lib.select_workspace_size(deltas, ages, mask, w.K_f), 256),
                         dtype=torch.uint8, device=dev)
        return (lambda: lib.cast_select_frames(deltas, ages, mask, w.K_f, workspace=ws),
                w.n_branch * w.n_cur * S * w.D * 2, "B")
    if name == "ffn_mg":
        wl = W.MG
        N, S, D = wl.n_cur, wl.S, wl.H * wl.d
        Dff = 4 * D
        x = rnd(N, S, D)
        w1, w2 = rnd(Dff, D) * (D ** -0.5), rnd(D, Dff) * (Dff ** -0.5)
        b1, b2 = rnd(Dff), rnd(D)
        r = torch.zeros((N, S, D), dtype=torch.bfloat16, device=dev)
        an = list(wl.anchors)
        ws = torch.empty(lib.ffn_workspace_size(x, an, w1, b1, w2, b2, wl.grid, r), dtype=torch.uint8,
                         device=dev)
        return (lambda: lib.cast_ffn_step(x, an, w1, b1, w2, b2, wl.grid, r, workspace=ws),
                4.0 * len(an) * S * D * Dff, "FLOP")
    if name == "block_hy":
        wl = W.HY
        N, S, H, d = wl.n_cur, wl.S, wl.H, wl.d
        q, kc, vc = rnd(N, S, H, d), rnd(N, S, H, d), rnd(N, S, H, d)
        kh, vh = rnd(wl.M, wl.B_v, H, d), rnd(wl.M, wl.B_v, H, d)
        r = torch.zeros((N, S, H * d), dtype=torch.bfloat16, device=dev)
        a = lib.block_args(q, kc, vc, list(wl.anchors), kh, vh, wl.K, wl.grid, r,
                           params=lib.par_params(band_radius=wl.band_radius), refine=lib.REFINE_PAPER)
        ws = torch.empty(lib.block_workspace_size(a), dtype=torch.uint8, device=dev)
        return (lambda: lib.cast_block_step_args(a, ws), N, "frames")
    if name in ("route_mg64", "attn_mg64", "attn_hy64", "block_mg64", "block_hy64"):
        wl = W.HY64 if name in ("attn_hy64", "block_hy64") else W.MG64
        N, S, H, d = wl.n_cur, wl.S, wl.H, wl.d
        an = list(wl.anchors)
        Kf = len(an)
        hist = (wl.hist_frames, wl.grid[0], wl.grid[1], H, d)
        q, kc, vc = rnd(N, S, H, d), rnd(N, S, H, d), rnd(N, S, H, d)
        kh, vh = rnd(*hist), rnd(*hist)
        if name == "route_mg64":
            ws = torch.empty(lib.route_workspace_size(q, an, kh, vh, wl.K), dtype=torch.uint8, device=dev)
            return (lambda: lib.cast_route_topk(q, an, kh, vh, wl.K, workspace=ws),
                    (Kf * S + 2 * wl.hist_frames * S) * H * d * 2, "B")
        if name in ("block_mg64", "block_hy64"):
            r = torch.zeros((N, S, H * d), dtype=torch.bfloat16, device=dev)
            a = lib.block_args(q, kc, vc, an, kh, vh, wl.K, wl.grid, r, refine=lib.REFINE_PAPER)
            ws = torch.empty(lib.block_workspace_size(a), dtype=torch.uint8, device=dev)
            return (lambda: lib.cast_block_step_args(a, ws), N, "frames")
        perm = torch.stack([torch.randperm(wl.M, generator=torch.Generator().manual_seed(k))[:wl.K]
                            for k in range(Kf * H)]).view(Kf, H, wl.K)
        sizes = torch.tensor(_block_tokens(wl), dtype=torch.float64)
        routed_tokens = float(sizes[perm].sum())          # keys of the routed blocks, all (i, h)
        flop = 4.0 * S * d * (Kf * H * N * S + routed_tokens)
        idx = perm.int().to(dev)
        o = torch.empty((Kf, S, H * d), dtype=torch.bfloat16, device=dev)
        aws = torch.empty(max(lib.attention_workspace_size(q, kc, vc, an, kh, vh, idx), 256),
                          dtype=torch.uint8, device=dev)
        return (lambda: lib.cast_anchor_attention(q, kc, vc, an, kh, vh, idx, out=o, workspace=aws),
                flop, "FLOP")
    raise ValueError(name)


def scale_points(lib, torch, dev, flush, reps=10):
    """Each stage at the full size of its own workload (device-resident inputs, L2 flushed
    between launches, CUDA events on the launching stream)."""
    hbm, bf16, _ = _peaks()
    out = {}
    stream = torch.cuda.current_stream(dev)
    for name in SCALE_POINTS:
        fn, work, unit = _scale_setup(name, lib, torch, dev)
        for _ in range(3):
            fn()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(reps)]
        for k in range(reps):
            flush.fill_(k & 0xFF)
            ev[k][0].record(stream)
            fn()
            ev[k][1].record(stream)
        torch.cuda.synchronize()
        ms = statistics.median(a.elapsed_time(b) for a, b in ev)
        if unit == "B":
            rate = work / ms / 1e6
            out[name] = {"ms": round(ms, 4), "GB/s": round(rate, 1), "frac_hbm": round(rate / hbm, 4),
                         "bytes": work}
        elif unit == "frames":
            out[name] = {"ms": round(ms, 4), "frames/s": round(work / ms * 1e3, 1)}
        else:
            rate = work / ms / 1e9
            out[name] = {"ms": round(ms, 4), "TFLOP/s": round(rate, 1),
                         "frac_bf16": round(rate / bf16, 4), "flop": work}
        del fn
        torch.cuda.empty_cache()
    return out


def run_profile(name):
    """A few launches of one stage at full size, for an ncu capture."""
    import torch

    from paper_2609_34144_gb300 import native as lib
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    fn, _, _ = _scale_setup(name, lib, torch, dev)
    for _ in range(3):
        fn()
    torch.cuda.synchronize()
    lib.cast_check_device()
    print(f"profiled {name}")


def _captured_traffic():
    """DRAM bytes per attention launch from the committed ncu summary, or None when the
    kernel sources changed since that capture (hash of attention.cu + ptx.cuh)."""
    import hashlib
    import re
    prof = os.path.join(ROOT, "profiles", "k_attn_mg_block_step.md")
    if not os.path.exists(prof):
        return None
    m = re.search(r"dram_bytes_per_launch=(\d+) source_sha256_16=([0-9a-f]+)", open(prof).read())
    if not m:
        return None
    csrc = os.path.join(ROOT, "paper_2609_34144_gb300", "csrc")
    h = hashlib.sha256()
    for f in ("attention.cu", "ptx.cuh"):
        h.update(open(os.path.join(csrc, f), "rb").read())
    return int(m.group(1)) if h.hexdigest()[:16] == m.group(2) else None


# ------------------------------------------------------------------------------ CPU oracle
def launches_per_step(wl):
    """Library kernels one block step launches: pooling (anchor frames, history blocks) and
    the per-head routing kernel, attention, and PAR (statistics, transport and blend passes
    for the full 8x8 tiles and for the truncated edge tiles when the grid has both)."""
    hg, wg = wl.grid
    full = (hg // 8) * (wg // 8) > 0
    edge = hg % 8 != 0 or wg % 8 != 0
    return 3 + 1 + 3 * (int(full) + int(edge))


def _oracle_sample(wl, inp, R, heads, row_stride, tiles):
    """One bounded sample of the block step in the CPU oracle: routing and attention on the
    first `heads` heads (attention on every `row_stride`-th query row), PAR on the first
    `tiles` tiles (pooled over every channel).  Returns (seconds for the whole workload
    scaled from the sample, description of the sample)."""
    import oracle.cast_oracle as O
    anchors = list(wl.anchors)
    hs = slice(0, heads)
    t0 = time.perf_counter()
    rt = O.pooled_routing(inp["q"][:, :, hs], anchors, inp["k_hist"][:, :, hs],
                          inp["v_hist"][:, :, hs])
    idx = np.stack([O.coupled_routing(rt.u[:, h], anchors, wl.n_cur, wl.K)
                    for h in range(rt.u.shape[1])], axis=1)
    t1 = time.perf_counter()
    rows = np.arange(0, wl.S, row_stride)
    O.routed_attention(inp["q"][:, :, hs], inp["k_cur"][:, :, hs], inp["v_cur"][:, :, hs],
                       inp["k_hist"][:, :, hs], inp["v_hist"][:, :, hs], anchors, idx, rows=rows)
    t2 = time.perf_counter()
    n_tiles = len(O.tiles_of(wl.grid[0], wl.grid[1], 8, 8))
    O.par_reconstruct(R, W.anchor_mask(wl.n_cur, anchors), None,
                      O.ParParams(band_radius=wl.band_radius), tiles=range(tiles))
    t3 = time.perf_counter()
    hf = wl.H / heads
    est = (t1 - t0) * hf + (t2 - t1) * hf * (wl.S / len(rows)) + (t3 - t2) * (n_tiles / tiles)
    desc = (f"routing with 2-pass refinement on {heads}/{wl.H} heads (all tokens, all blocks), "
            f"attention on those heads "
            f"for {len(rows)}/{wl.S} query rows of every anchor, PAR on {tiles}/{n_tiles} tiles; "
            f"each stage scaled to the full workload by its share of the work")
    return est, desc


def _par_input(wl):
    return np.random.default_rng(0).standard_normal(
        (wl.n_cur, wl.grid[0], wl.grid[1], wl.H * wl.d)).astype(np.float32)


def cpu_baseline(wl):
    inp = W.block_step_inputs(wl)
    R = _par_input(wl)
    cores = len(os.sched_getaffinity(0))
    n_tiles = (wl.grid[0] + 7) // 8 * ((wl.grid[1] + 7) // 8)
    est, desc = _oracle_sample(wl, inp, R, heads=wl.H, row_stride=16, tiles=n_tiles)
    return {"value": round(wl.n_cur / est, 6), "unit": "frames/s", "cores": cores, "kind": "oracle",
            "sample": desc, "est_seconds_per_step": round(est, 3)}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = WL
    inp = W.block_step_inputs(wl)
    R = _par_input(wl)
    cores = len(os.sched_getaffinity(0))
    for _ in range(args.warmup):
        _oracle_sample(wl, inp, R, heads=1, row_stride=wl.S // 8, tiles=1)
    total, desc = 0.0, ""
    for _ in range(args.steps):
        est, desc = _oracle_sample(wl, inp, R, heads=1, row_stride=wl.S // 8, tiles=1)
        total += est
    value = wl.n_cur * args.steps / total
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "frames/s",
            "n_gpus": int(os.environ.get("WORLD_SIZE", "1")), "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(total / args.steps * 1e3, 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": wl.name},
            "cpu_baseline": {"value": round(value, 6), "unit": "frames/s", "cores": cores,
                             "kind": "oracle", "sample": desc},
            "e2e": {"value": round(value, 6), "unit": "frames/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-scale-points", action="store_true")
    ap.add_argument("--profile", default=None, choices=SCALE_POINTS,
                    help="run only a few launches of one full-size stage (for ncu) and exit")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.profile:
        run_profile(args.profile)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
