"""Benchmark of the CAST block step on GB300: prints one JSON line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Workload: the HY-World-1.5-shaped bf16 block step, the largest block-step configuration (16
current latent frames of 44x80 tokens, 24 heads x 128, 32 history blocks of 3520 tokens, K = 8,
anchors {0, 3, 7, 12, 15}), on its seeded synthetic inputs.
A step is cast_block_step: routing (pooled scores, TopK, then the reconstruction-coupled
refinement with the paper's L_s = 2 passes and (lambda_anc, lambda_rec) = (1, 1)) -> routed
anchor attention -> PAR.
  value   frames/s with inputs resident in HBM (CUDA events around each step, L2 flushed
          between steps outside the timed events)
  e2e     frames/s through the same C call with the inputs copied from pinned host memory
          (current K/V and history K/V whole, the queries of the anchor frames: the step reads
          no other query frame) and r_out copied back, copies inside the timed region
          (double-buffered: step k+1's upload and step k-1's read-back overlap step k's compute)
  roofline  the dominant kernel (routed attention): algorithmic FLOP per launch / its average
          CUDA-event duration (stages launched through their own entry points, same kernels
          and launch configuration as inside the block step) against the measured bf16 peak
  cpu_baseline  the CPU oracle timed on a bounded sample of the same workload (the same sample
          and scaling model as `--impl reference`)
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
WL = W.HY


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


def bench_config(wl, world):
    """The workload description both arms print."""
    return {"workload": wl.name, "frames_per_step": wl.n_cur, "grid": list(wl.grid),
            "heads": wl.H, "head_dim": wl.d, "history_blocks": wl.M, "block_tokens": wl.B_v,
            "K": wl.K, "anchors": list(wl.anchors), "global_batch": world,
            "routing": "coupled refinement, 2 passes, lambda (1, 1), tol 1e-6",
            "l2": "flushed (256 MiB write) between timed steps, outside the events",
            "parallelism": f"replicas x{world} (independent chunks, no collective)"}


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
                    if nm == "q":   # routing and attention read the anchor frames' queries only
                        for f in anchors:
                            dk[nm][f].copy_(host[nm][f], non_blocking=True)
                    else:
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
    h2d = sum(host[nm][0].numel() * host[nm].element_size() * (len(anchors) if nm == "q" else host[nm].shape[0])
              for nm in names)
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
            "config": bench_config(wl, world),
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
                    "pipeline": "double-buffered: upload of step k+1 (the anchor frames' queries, "
                                "current and history K/V) and read-back of step k-1 overlap step k "
                                "(host link ~210 GB/s measured)"},
            "gpu_launches": launches_per_step(wl) * args.steps,
            "clocks": clk,
        }
        if not args.no_scale_points:
            line["scale_points"] = scale_points(lib, torch, dev, flush)
        if not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline(wl, inp)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ------------------------------------------------------------------------------ scale points
SCALE_POINTS = ("block_mg", "route_mg", "attn_mg", "par_mg",
                "par_sweep_f32_s2", "par_sweep_f32_s3", "par_sweep_f32_s4",
                "par_sweep_bf16_s2", "par_sweep_bf16_s3", "par_sweep_bf16_s4",
                "route_stress_k4", "route_stress_k8", "route_stress_k16", "route_stress_k32",
                "route_stress_k8_refine", "route_stress_k32_refine",
                "attn_stress_k4", "attn_stress_k8", "attn_stress_k16", "attn_stress_k32",
                "select_mg", "ffn_mg", "route_mg64", "attn_mg64", "attn_hy64", "block_mg64",
                "block_hy64")


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
        dt = torch.float32 if "_f32_" in name else torch.bfloat16
        r = rnd(w.F, w.grid[0], w.grid[1], w.C, dtype=dt)
        wc = torch.rand(w.C, generator=g, device=dev)
        mask = W.anchor_mask(w.F, w.anchors(int(name.rsplit("_s", 1)[1])))
        p = lib.par_params(band_radius=w.band_radius)
        ws = torch.empty(lib.par_workspace_size(r, mask, p), dtype=torch.uint8, device=dev)
        return (lambda: lib.cast_par_reconstruct(r, mask, wc, p, workspace=ws),
                r.numel() * r.element_size(), "B")
    if name.startswith("route_stress"):
        s = W.STRESS
        K = int(name.split("_k")[1].split("_")[0])
        refine = lib.REFINE_PAPER if name.endswith("_refine") else None
        q = rnd(s.n_cur, s.S, s.H, s.d)
        kh, vh = rnd(s.M, s.B_v, s.H, s.d), rnd(s.M, s.B_v, s.H, s.d)
        an = list(range(s.n_cur))
        ws = torch.empty(lib.route_workspace_size(q, an, kh, vh, K, refine=refine), dtype=torch.uint8,
                         device=dev)
        return (lambda: lib.cast_route_topk(q, an, kh, vh, K, workspace=ws, refine=refine),
                (s.n_cur * s.S + 2 * s.M * s.B_v) * s.H * s.d * 2, "B")
    if name.startswith("attn_stress"):
        s = W.STRESS
        K = int(name.split("_k")[1])
        N, S = s.n_cur, s.S
        q, kc, vc = rnd(N, S, s.H, s.d), rnd(N, S, s.H, s.d), rnd(N, S, s.H, s.d)
        kh, vh = rnd(s.M, s.B_v, s.H, s.d), rnd(s.M, s.B_v, s.H, s.d)
        an = list(range(N))
        idx = lib.cast_route_topk(q, an, kh, vh, K)   # the kernel's own routing of these inputs
        o = torch.empty((N, S, s.H * s.d), dtype=torch.bfloat16, device=dev)
        flop = 4.0 * N * S * (N * S + K * s.B_v) * s.d * s.H
        aws = torch.empty(max(lib.attention_workspace_size(q, kc, vc, an, kh, vh, idx), 256),
                          dtype=torch.uint8, device=dev)
        return (lambda: lib.cast_anchor_attention(q, kc, vc, an, kh, vh, idx, out=o, workspace=aws),
                flop, "FLOP")
    if name in ("block_mg", "route_mg", "attn_mg", "par_mg"):
        # the Matrix-Game-shaped chunk on its seeded inputs
        wl = W.MG
        inp = W.block_step_inputs(wl)
        t = {k: torch.from_numpy(G.bf16_bits(inp[k]).view(np.int16)).to(dev).view(torch.bfloat16)
             for k in ("q", "k_cur", "v_cur", "k_hist", "v_hist")}
        N, S, H, d = inp["q"].shape
        an = list(wl.anchors)
        attn_flop, route_bytes, par_bytes = algorithmic_work(wl)
        if name == "block_mg":
            r = torch.zeros((N, S, H * d), dtype=torch.bfloat16, device=dev)
            a = lib.block_args(t["q"], t["k_cur"], t["v_cur"], an, t["k_hist"], t["v_hist"], wl.K,
                               wl.grid, r, params=lib.par_params(band_radius=wl.band_radius),
                               refine=lib.REFINE_PAPER)
            ws = torch.empty(lib.block_workspace_size(a), dtype=torch.uint8, device=dev)
            return (lambda: lib.cast_block_step_args(a, ws), N, "frames")
        if name == "route_mg":
            ws = torch.empty(lib.route_workspace_size(t["q"], an, t["k_hist"], t["v_hist"], wl.K,
                                                      refine=lib.REFINE_PAPER),
                             dtype=torch.uint8, device=dev)
            return (lambda: lib.cast_route_topk(t["q"], an, t["k_hist"], t["v_hist"], wl.K, workspace=ws,
                                                refine=lib.REFINE_PAPER), route_bytes, "B")
        if name == "attn_mg":
            idx = lib.cast_route_topk(t["q"], an, t["k_hist"], t["v_hist"], wl.K, refine=lib.REFINE_PAPER)
            o = torch.empty((len(an), S, H * d), dtype=torch.bfloat16, device=dev)
            aws = torch.empty(max(lib.attention_workspace_size(t["q"], t["k_cur"], t["v_cur"], an,
                                                               t["k_hist"], t["v_hist"], idx), 256),
                              dtype=torch.uint8, device=dev)
            return (lambda: lib.cast_anchor_attention(t["q"], t["k_cur"], t["v_cur"], an, t["k_hist"],
                                                      t["v_hist"], idx, out=o, workspace=aws),
                    attn_flop, "FLOP")
        # par_mg: PAR of the chunk's attention output (the block step's residual site)
        idx = lib.cast_route_topk(t["q"], an, t["k_hist"], t["v_hist"], wl.K, refine=lib.REFINE_PAPER)
        r = torch.zeros((N, S, H * d), dtype=torch.bfloat16, device=dev)
        o = lib.cast_anchor_attention(t["q"], t["k_cur"], t["v_cur"], an, t["k_hist"], t["v_hist"], idx)
        r[an] = o
        rp = r.view(N, wl.grid[0], wl.grid[1], H * d)
        mask = W.anchor_mask(N, an)
        p = lib.par_params(band_radius=wl.band_radius)
        ws = torch.empty(max(lib.par_workspace_size(rp, mask, p), 256), dtype=torch.uint8, device=dev)
        return (lambda: lib.cast_par_reconstruct(rp, mask, None, p, workspace=ws), par_bytes, "B")
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
    """DRAM bytes per attention launch at the bench workload from the committed ncu summary, or
    None when the kernel sources changed since that capture (hash of attention.cu + ptx.cuh)."""
    import hashlib
    import re
    prof = os.path.join(ROOT, "profiles", "k_attn_hy_block_step.md")
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


# One bounded sample of the block step, the same for the `cpu_baseline` leg and for `--impl
# reference`: routing (pooled scores, omission, TopK and the 2-pass refinement) on the first
# `route_heads` heads with every token and block; routed attention on the first `attn_heads`
# heads for `attn_rows` evenly spaced query rows of every anchor; PAR on `par_tiles` tiles
# spread over the grid (pooled over every channel).
SAMPLE_PLAN = {"route_heads": 4, "attn_heads": 1, "attn_rows": 128, "par_tiles": 3}


def _oracle_sample(wl, inp, R, plan=SAMPLE_PLAN):
    """Runs the sample in the CPU oracle.  Returns (estimated seconds of the whole block step,
    measured seconds of the sample, description).  Scaling model: each stage's sample time
    times the stage's share of the full work (routing heads H / route_heads; attention
    (H / attn_heads) * (S / attn_rows); PAR n_tiles / par_tiles)."""
    import oracle.cast_oracle as O
    anchors = list(wl.anchors)
    hr, ha = slice(0, plan["route_heads"]), slice(0, plan["attn_heads"])
    t0 = time.perf_counter()
    rt = O.pooled_routing(inp["q"][:, :, hr], anchors, inp["k_hist"][:, :, hr],
                          inp["v_hist"][:, :, hr])
    idx = np.stack([O.coupled_routing(rt.u[:, h], anchors, wl.n_cur, wl.K)
                    for h in range(rt.u.shape[1])], axis=1)
    t1 = time.perf_counter()
    rows = np.linspace(0, wl.S - 1, plan["attn_rows"]).astype(np.int64)
    O.routed_attention(inp["q"][:, :, ha], inp["k_cur"][:, :, ha], inp["v_cur"][:, :, ha],
                       inp["k_hist"][:, :, ha], inp["v_hist"][:, :, ha], anchors,
                       idx[:, :plan["attn_heads"]], rows=rows)
    t2 = time.perf_counter()
    n_tiles = len(O.tiles_of(wl.grid[0], wl.grid[1], 8, 8))
    tiles = sorted({int(v) for v in np.linspace(0, n_tiles - 1, plan["par_tiles"])})
    O.par_reconstruct(R, W.anchor_mask(wl.n_cur, anchors), None,
                      O.ParParams(band_radius=wl.band_radius), tiles=tiles)
    t3 = time.perf_counter()
    est = ((t1 - t0) * wl.H / plan["route_heads"]
           + (t2 - t1) * (wl.H / plan["attn_heads"]) * (wl.S / len(rows))
           + (t3 - t2) * (n_tiles / len(tiles)))
    desc = (f"routing with 2-pass refinement on {plan['route_heads']}/{wl.H} heads (all tokens, all "
            f"blocks); attention on {plan['attn_heads']}/{wl.H} heads for {len(rows)}/{wl.S} query "
            f"rows of every anchor; PAR on {len(tiles)}/{n_tiles} tiles (all channels); whole-step "
            f"time = sum of each stage's sample time x its share of the full work")
    return est, t3 - t0, desc


def _par_input(wl):
    return np.random.default_rng(0).standard_normal(
        (wl.n_cur, wl.grid[0], wl.grid[1], wl.H * wl.d)).astype(np.float32)


def cpu_baseline(wl, inp):
    R = _par_input(wl)
    cores = len(os.sched_getaffinity(0))
    est, took, desc = _oracle_sample(wl, inp, R)
    return {"value": round(wl.n_cur / est, 6), "unit": "frames/s", "cores": cores, "kind": "oracle",
            "sample": desc, "est_seconds_per_step": round(est, 3), "sample_seconds": round(took, 3)}


def run_reference(args):
    """The reference arm: the CPU oracle as it stands, one bounded sample per step (the
    sample and scaling model of `cpu_baseline`).  value = frames of the whole workload per
    second of estimated full-step time; ms_per_step is the measured time of one sample."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = WL
    inp = W.block_step_inputs(wl)
    R = _par_input(wl)
    cores = len(os.sched_getaffinity(0))
    for _ in range(args.warmup):
        _oracle_sample(wl, inp, R)
    est_total, took_total, desc = 0.0, 0.0, ""
    for _ in range(args.steps):
        est, took, desc = _oracle_sample(wl, inp, R)
        est_total += est
        took_total += took
    value = wl.n_cur * args.steps / est_total
    world = int(os.environ.get("WORLD_SIZE", "1"))
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "frames/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(took_total / args.steps * 1e3, 2),
            "est_full_step_ms": round(est_total / args.steps * 1e3, 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": bench_config(wl, 1),
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
