"""Benchmark of the foreground-only block-sparse attention hot path on GB300.

One step = one pass of the whole path over one synthetic 2048-canvas batch:
compaction of Q, K, V, dO -> Top-K block lists (+ transpose) -> block-sparse
attention forward -> backward -> scatter of O, dQ, dK, dV to the canvas.

value  = retained-block attention FLOPs of the step (forward + backward,
         4*|Q_i|*|K_j|*d per retained pair per head for the forward and 2.5x
         that for the backward) / device time of the whole step, summed over
         ranks (replicas).
e2e    = the same FLOPs / time of the step through the public API with the
         canvas inputs in pinned host memory: host->device copies of the
         mask and Q, K, V, dO, the step, and device->host copies of O, dQ,
         dK, dV canvases inside the timed region.
The reference arm (--impl reference) times the fp64 CPU oracle on a bounded
sample of the same workload (this build has no reference implementation).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

FALLBACK_PEAKS = dict(hbm_gbs=6800.0, bf16_tflops=1900.0, bf16_tflops_sustained=1700.0)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="c2048")
    ap.add_argument("--heads", type=int, default=0, help="override the head count (small profiling cases)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--sweep", action="store_true",
                    help="2048-canvas sweep: one JSON line per (foreground, rho, block) point instead of the bench line")
    return ap.parse_args()


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            import tempfile
            fd, self.path = tempfile.mkstemp(prefix=f"clocks_gpu{self.gpu}_", suffix=".csv")
            self.f = os.fdopen(fd, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        try:
            os.remove(self.path)
        except OSError:
            pass
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": float(max(mx)), "reasons": sorted(reasons),
                "samples": len(sm)}


# --------------------------------------------------------------- workload
def make_inputs(w, device, seed_note=True):
    import torch
    mask = w.canvas_mask()
    q, k, v, do = w.q(), w.k(), w.v(), w.dout()
    return mask, q, k, v, do


def retained_flops(row_ptr, col_idx, N, b, d):
    """Forward FLOPs 4*|Q_i|*|K_j|*d per retained pair, from the device lists (host copy)."""
    nq = -(-N // b)
    sizes = np.full(nq, b, dtype=np.float64)
    if N % b:
        sizes[-1] = N % b
    rp = row_ptr.astype(np.int64)
    rows = np.repeat(np.arange(len(rp) - 1), np.diff(rp))
    qsz = sizes[rows % nq]
    ksz = sizes[col_idx[:rp[-1]]]
    return 4.0 * d * float((qsz * ksz).sum())


def whole_job(ms_local: float, flops_local: float, world: int, device=None):
    """Whole-job figures of a multi-rank run: the slowest rank's time (max over
    ranks) and the work of all ranks (sum over ranks; replicas may process
    different sequence lengths).  world == 1 returns the inputs."""
    if world <= 1:
        return float(ms_local), float(flops_local)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(ms_local)], dtype=torch.float64, device=device)
    f = torch.tensor([float(flops_local)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(f, op=dist.ReduceOp.SUM)
    return float(t.item()), float(f.item())


def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist
    import __graft_entry__ as g
    from paper_2609_23169_gb300 import path as P
    from paper_2609_23169_gb300 import ultratex as u
    from synth import CONFIGS

    if rank == 0:
        g.build()
    if world > 1:
        dist.barrier()
    g.build()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    w = CONFIGS[args.workload]
    if args.heads:
        w = w.with_(heads=args.heads)
    assert w.mask_mode == "topk", "the benchmark workload uses the Top-K rule"
    mask_np, q, k, v, do = make_inputs(w, dev)
    mask = torch.from_numpy(mask_np).to(dev)
    tq, tk, tv, tdo = (x.to(dev) for x in (q, k, v, do))
    hp = P.HotPath(w.T, w.heads, w.head_dim, w.block, torch.bfloat16, u.UT_MASK_TOPK, rho=w.rho, device=dev)
    stream = torch.cuda.current_stream()

    ev = {}

    def timed(name, fn):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        r = fn()
        b.record(stream)
        ev.setdefault(name, []).append((a, b))
        return r

    def step(record):
        if not record:
            return hp.step(mask, tq, tk, tv, tdo)
        N = timed("compact", lambda: hp.compact(mask, [tq, tk, tv, tdo]))
        timed("block_mask", lambda: hp.block_lists(N))
        timed("bsattn_fwd", lambda: hp.forward(N))
        timed("bsattn_bwd", lambda: hp.backward_pass(N))
        timed("scatter", lambda: hp.scatter(N))
        return N

    for _ in range(args.warmup):
        N = step(False)
    torch.cuda.synchronize()
    u.check_status(hp.status)
    rp = hp.row_ptr[:w.heads * hp.nq_cap + 1].cpu().numpy()
    nq = -(-N // w.block)
    rp = rp[:w.heads * nq + 1]
    ci = hp.col_idx[:int(rp[-1])].cpu().numpy()
    f_fwd = retained_flops(rp, ci, N, w.block, w.head_dim)
    f_step = 3.5 * f_fwd
    density = float(rp[-1]) / (w.heads * nq * nq)

    clocks = ClockSampler(local_rank)
    clocks.start()
    time.sleep(0.3)
    ev.clear()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        step(True)
    t1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    ms_total = t0.elapsed_time(t1)
    clk = clocks.stop()
    u.check_status(hp.status)
    kern_ms = {n: sum(a.elapsed_time(b) for a, b in l) / len(l) for n, l in ev.items()}

    # whole-job: max time over ranks, FLOPs summed over ranks (replicas)
    ms_total, flops_total = whole_job(ms_total, f_step * args.steps, world, dev)
    ms_step = ms_total / args.steps
    value = flops_total / (ms_total * 1e-3) / 1e12

    # ---- e2e through host buffers: every step copies its canvas inputs from
    # pinned host memory and its canvas results back.  The copies of
    # neighbouring steps overlap the compute of the current one (three sets
    # of device inputs and outputs).  Whether uploads and downloads should
    # run at the same time depends on the host link (full duplex on some
    # hosts, less total bandwidth with both directions at once on others), so
    # the warm-up times both arrangements -- one copy stream for both
    # directions, or one per direction -- and the timed steps use the faster.
    e2e = None
    if not args.no_e2e:
        pin_in = [x.pin_memory() for x in (torch.from_numpy(mask_np), q, k, v, do)]
        NB = 3  # buffer sets: a step's outputs stay untouched until its download ends two steps later
        pin_out = [[torch.empty((w.T, w.heads, w.head_dim), dtype=torch.bfloat16).pin_memory() for _ in range(4)]
                   for _ in range(NB)]
        h2d = sum(x.numel() * x.element_size() for x in pin_in)
        d2h = sum(x.numel() * x.element_size() for x in pin_out[0])
        dev_in = [[mask, tq, tk, tv, tdo]] + [[torch.empty_like(x) for x in (mask, tq, tk, tv, tdo)]
                                              for _ in range(NB - 1)]
        paths = [hp] + [P.HotPath(w.T, w.heads, w.head_dim, w.block, torch.bfloat16, u.UT_MASK_TOPK, rho=w.rho,
                                  device=dev) for _ in range(NB - 1)]
        s_cmp = torch.cuda.Stream(dev)
        s_copy = [torch.cuda.Stream(dev), torch.cuda.Stream(dev)]
        mode = {"split": False}   # False: uploads and downloads share s_copy[0]
        up_s = lambda: s_copy[0]  # noqa: E731
        dn_s = lambda: s_copy[1] if mode["split"] else s_copy[0]  # noqa: E731
        ev = lambda: torch.cuda.Event(enable_timing=False)  # noqa: E731
        in_ready = [ev() for _ in range(NB)]
        in_free = [None] * NB
        out_free = [None] * NB

        def upload(k_):
            b = k_ % NB
            s_up = up_s()
            with torch.cuda.stream(s_up):
                if in_free[b] is not None:
                    s_up.wait_event(in_free[b])
                for hst, dvc in zip(pin_in, dev_in[b]):
                    dvc.copy_(hst, non_blocking=True)
                in_ready[b].record(s_up)

        def compute(k_):
            b = k_ % NB
            with torch.cuda.stream(s_cmp):
                s_cmp.wait_event(in_ready[b])
                if out_free[b] is not None:
                    s_cmp.wait_event(out_free[b])
                m_, q_, k2, v_, d_ = dev_in[b]
                paths[b].step(m_, q_, k2, v_, d_)
                done = ev()
                done.record(s_cmp)
                in_free[b] = done

        def download(k_):
            b = k_ % NB
            s_dn = dn_s()
            with torch.cuda.stream(s_dn):
                s_dn.wait_event(in_free[b])
                for hst, dvc in zip(pin_out[b], [paths[b].o_canvas] + paths[b].g_canvas):
                    hst.copy_(dvc, non_blocking=True)
                fin = ev()
                fin.record(s_dn)
                out_free[b] = fin

        def run(n_steps):
            # step k's results are downloaded while step k+1 computes, queued
            # only after step k+1 has read its token count N (a 4-byte read
            # that would otherwise wait behind a whole download)
            upload(0)
            for k_ in range(n_steps):
                if k_ + 1 < n_steps:
                    upload(k_ + 1)
                compute(k_)
                if k_ >= 1:
                    download(k_ - 1)
            download(n_steps - 1)

        def time_e2e(n_steps):
            torch.cuda.synchronize()
            s_up, s_dn = up_s(), dn_s()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(s_up)
            s_cmp.wait_stream(s_up)
            s_dn.wait_stream(s_up)
            run(n_steps)
            s_dn.wait_stream(s_cmp)
            s_dn.wait_stream(s_up)
            e1.record(s_dn)
            torch.cuda.synchronize()
            return e0.elapsed_time(e1) / n_steps

        run(2)
        trial = {}
        for split in (False, True):
            mode["split"] = split
            trial[split] = time_e2e(max(3, args.warmup))
        if world > 1:   # every rank takes the arrangement that is faster on the slowest rank
            t = torch.tensor([trial[False], trial[True]], device=dev)
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            trial = {False: float(t[0]), True: float(t[1])}
        mode["split"] = trial[True] < trial[False]
        if world > 1:
            dist.barrier()
        e_ms = time_e2e(args.steps)
        for x in paths:
            u.check_status(x.status)
        if world > 1:
            t = torch.tensor([e_ms], device=dev)
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            e_ms = float(t.item())
        e2e = {"value": round(world * f_step / (e_ms * 1e-3) / 1e12, 3), "unit": "TFLOP/s",
               "ms_per_step": round(e_ms, 3), "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "pipeline": ("3 streams (uploads | downloads | compute)" if mode["split"] else
                            "2 streams (uploads and downloads, one at a time | compute)") +
                           ", 3 sets of device inputs and outputs; warm-up ms/step with one copy stream "
                           f"{trial[False]:.1f}, with one per direction {trial[True]:.1f}"}

    peaks, peak_src = load_peaks()
    # DRAM bytes per launch of each entry point from the last ncu capture of the
    # current kernels (summarised under profiles/), taken at 8 heads and scaled
    # to 24 (each head is an independent problem of the same size); only valid
    # for the 24-head 2048 workload.  Backward: fused kernel 6.08 GB + dQ
    # finalize 0.49 GB + D/LSE pre-pass 0.36 GB + accumulator clear 0.35 GB.
    traffic_24h = {"bsattn_fwd": 2.60e9, "bsattn_bwd": 21.8e9}
    # dominant kernel by measured time
    dom = max(("bsattn_fwd", "bsattn_bwd"), key=lambda n: kern_ms.get(n, 0))
    dom_flops = f_fwd if dom == "bsattn_fwd" else 2.5 * f_fwd
    achieved = dom_flops / (kern_ms[dom] * 1e-3) / 1e12
    peak = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    bytes_tensor = 2 * N * w.heads * w.head_dim * 2 + w.T + 4 * N   # per tensor, compaction
    kernels = {
        n: {"ms": round(kern_ms[n], 4)} for n in kern_ms
    }
    kernels["bsattn_fwd"]["tflops"] = round(f_fwd / (kern_ms["bsattn_fwd"] * 1e-3) / 1e12, 2)
    kernels["bsattn_bwd"]["tflops"] = round(2.5 * f_fwd / (kern_ms["bsattn_bwd"] * 1e-3) / 1e12, 2)
    kernels["compact"]["gbs"] = round(4 * bytes_tensor / (kern_ms["compact"] * 1e-3) / 1e9, 1)
    sc_bytes = 2 * N * w.heads * w.head_dim * 2 + 3 * (2 * N * w.heads * w.head_dim * 2 +
                                                      (w.T - N) * w.heads * w.head_dim * 2)
    kernels["scatter"]["gbs"] = round(sc_bytes / (kern_ms["scatter"] * 1e-3) / 1e9, 1)

    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    sampler = time_sampler_steps(w, dev, hbm_peak) if rank == 0 else None
    rope = time_rope(w, dev, hbm_peak) if rank == 0 else None
    alpha_mask = time_mask_from_alpha(w, dev, hbm_peak) if rank == 0 else None
    line = {
        "metric": "retained-block attention TFLOP/s and % of GB300 bf16 peak at 2048 canvas (~213K tokens)",
        "value": round(value, 3),
        "unit": "TFLOP/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_step, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": f"{w.name}: 13 images x {w.side}x{w.side} tokens (T={w.T}), "
                               f"{int(w.fg_frac*100)}% blob foreground (N={N}), H={w.heads}, d={w.head_dim}, "
                               f"b={w.block}, Top-K rho={w.rho} (density {density:.4f}), forward+backward",
                   "N": N, "T": w.T, "heads": w.heads, "head_dim": w.head_dim, "block": w.block, "rho": w.rho,
                   "retained_fwd_tflop": round(f_fwd / 1e12, 4), "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (each canvas tensor 1.31 GB > 129 MB)"},
        "pct_of_peak": round(100 * value / world / peak, 2),
        "roofline": {"bound": "tensor", "kernel": dom, "achieved": round(achieved, 2), "peak": peak,
                     "unit": "TFLOP/s", "frac": round(achieved / peak, 4),
                     "traffic": traffic_24h.get(dom) if (w.heads == 24 and w.name == "c2048") else None,
                     "peak_source": f"{peak_src} bf16 sustained"},
        "kernels": kernels,
        "e2e": e2e,
        "gpu_launches": args.steps * hp_launches(hp),
        "clocks": clk,
    }
    if sampler is not None:
        line["sampler_steps"] = sampler
    if rope is not None:
        line["rope_fused"] = rope
    if alpha_mask is not None:
        line["mask_from_alpha"] = alpha_mask
    return line, w


def time_sampler_steps(w, dev, hbm_peak: float, reps: int = 20) -> dict:
    """The sampler steps around the model call (sparse Euler update, Eq. euler;
    composite latent, Eq. mixed_latent), timed alone on the workload's target
    canvas (bf16, 64 latent channels per token), L2 flushed (by a read) before
    each call.
    Not part of the attention step's time."""
    import torch
    from paper_2609_23169_gb300 import ultratex as u
    x = w.sampler_inputs()
    mask_np = x["mask"]
    idx = torch.from_numpy(np.flatnonzero(mask_np).astype(np.int32)).to(dev)
    n, T = int(idx.numel()), int(mask_np.size)
    mask = torch.from_numpy(mask_np).to(dev)
    z, v, tile = x["z"].to(dev), x["v"].to(dev), x["tile"].to(dev)
    row = z[0].numel() * z.element_size()
    # L2 is flushed by reading a buffer twice its size: the lines left behind
    # are clean, so the timed call pays no write-back of someone else's data
    flush = torch.ones(64 << 20, dtype=torch.float32, device=dev)
    st = u.status_word(dev)

    def timed(fn):
        fn()
        tot = 0.0
        for _ in range(reps):
            flush.sum()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize()
            tot += e0.elapsed_time(e1)
        return tot / reps

    ms_e = timed(lambda: u.ut_fg_euler_update(idx, n, z, v, x["dt"], status=st))
    ms_c = timed(lambda: u.ut_fg_composite(mask, z, tile))
    u.check_status(st)
    b_e = n * (4 + 3 * row)            # idx, v read, z read + write (foreground rows)
    b_c = T + (T - n) * row            # mask read, background rows written
    out = {"workload": f"{w.name} target canvas: {T} tokens, {n} foreground, 64 channels bf16, "
                       f"tile of {x['period']} rows", "l2": "flushed before each call by reading 256 MB"}
    for name, ms, b in (("euler_update", ms_e, b_e), ("composite", ms_c, b_c)):
        gbs = b / (ms * 1e-3) / 1e9
        out[name] = {"ms": round(ms, 5), "bytes": int(b), "gbs": round(gbs, 1), "frac_hbm": round(gbs / hbm_peak, 4)}
    return out


def time_rope(w, dev, hbm_peak: float, reps: int = 10) -> dict:
    """RoPE fused with the gather of Q and K (and, inverted, with the ZERO
    scatter of dQ and dK) on the workload's canvas; inputs larger than L2.
    Not part of the attention step's time."""
    import torch
    from paper_2609_23169_gb300 import ultratex as u
    mask = w.canvas_mask()
    idx = torch.from_numpy(np.flatnonzero(mask).astype(np.int32)).to(dev)
    N, T = int(idx.numel()), int(mask.size)
    q, k = w.q().to(dev), w.k().to(dev)
    cfg = u.rope_config(w.side, prefix=w.text_prefix)
    qc, kc = (torch.empty((N, w.heads, w.head_dim), dtype=q.dtype, device=dev) for _ in range(2))
    dq, dk = torch.empty_like(q), torch.empty_like(k)
    row = w.heads * w.head_dim * q.element_size()

    def timed(fn):
        fn()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    ms_g = timed(lambda: u.ut_fg_gather_rope(idx, N, [q, k], cfg, dsts=[qc, kc]))
    ms_s = timed(lambda: u.ut_fg_scatter_rope(idx, N, [qc, kc], [dq, dk], cfg, u.UT_BG_ZERO))
    b_g = 2 * 2 * N * row + 4 * N          # read N canvas rows, write N rows, per tensor; idx once
    b_s = 2 * (N * row + T * row) + 4 * N  # read N rows, write all T canvas rows, per tensor
    out = {"workload": f"{w.name}: Q and K (H={w.heads}, d={w.head_dim}, bf16), N={N} of T={T} rows, "
                       f"axes 16/56/56, theta 1e4", "l2": "inputs larger than L2 (1.31 GB per canvas tensor)"}
    for name, ms, b in (("gather_rope", ms_g, b_g), ("scatter_rope_zero", ms_s, b_s)):
        gbs = b / (ms * 1e-3) / 1e9
        out[name] = {"ms": round(ms, 4), "bytes": int(b), "gbs": round(gbs, 1), "frac_hbm": round(gbs / hbm_peak, 4)}
    del q, k, qc, kc, dq, dk
    torch.cuda.empty_cache()
    return out


def time_mask_from_alpha(w, dev, hbm_peak: float, reps: int = 20) -> dict:
    """Canvas mask from the renders' alpha channels (Sec. 3.2), timed alone on
    the workload's alpha images (V + 1 images of side*16 pixels), L2 flushed
    (by a read) before each call.  Not part of the attention step's time."""
    import torch
    from paper_2609_23169_gb300 import ultratex as u
    alpha = torch.from_numpy(w.alpha_images()).to(dev)
    out = u.ut_fg_mask_from_alpha(alpha)
    flush = torch.ones(64 << 20, dtype=torch.float32, device=dev)
    tot = 0.0
    for _ in range(reps):
        flush.sum()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        u.ut_fg_mask_from_alpha(alpha, out=out)
        e1.record()
        torch.cuda.synchronize()
        tot += e0.elapsed_time(e1)
    ms = tot / reps
    b = alpha.numel() + out.numel()
    gbs = b / (ms * 1e-3) / 1e9
    return {"workload": f"{w.name}: {alpha.shape[0]} alpha images of {alpha.shape[1]}x{alpha.shape[2]} px, factor 16, "
                        f"radius 1, threshold 0 -> {out.numel()} tokens ({float(out.float().mean()):.3f} foreground)",
            "ms": round(ms, 5), "bytes": int(b), "gbs": round(gbs, 1), "frac_hbm": round(gbs / hbm_peak, 4),
            "l2": "flushed before each call by reading 256 MB"}


def hp_launches(hp) -> int:
    """Kernel launches of one HotPath.step (compaction 3, Top-K lists 3 + transpose 3,
    forward 1, backward 3 (preprocess, fused dK/dV/dQ, dQ finalize), scatter 2)."""
    return 3 + 6 + 1 + 3 + 2


# ------------------------------------------------------------------- oracle
def oracle_sample(w, seconds: float):
    """Time the fp64 oracle on a bounded sample: whole query blocks of head 0,
    forward and dQ rows, until `seconds` have passed.  Returns (TFLOP/s, desc)."""
    import torch
    import oracle.ultratex_oracle as o
    mask = w.canvas_mask()
    idx = np.flatnonzero(mask)
    t = torch.from_numpy(idx)
    h = 0
    qc, kc, vc, dc = (x[t][:, h:h + 1].float().numpy().astype(np.float64) for x in (w.q(), w.k(), w.v(), w.dout()))
    N = len(idx)
    b = w.block
    rp, ci, _, kr = o.topk_block_mask(qc, kc, b, w.rho)
    nq = -(-N // b)
    t0 = time.perf_counter()
    flops = 0.0
    done = 0
    for i in range(nq):
        rows = np.arange(i * b, min(N, (i + 1) * b))
        o.bsattn_fwd_rows(qc, kc, vc, rp, ci, b, 0, rows)
        o.bsattn_bwd_dq_rows(qc, kc, vc, dc, rp, ci, b, 0, rows)
        keys = sum(min(b, N - j * b) for j in ci[rp[i]:rp[i + 1]])
        # forward (4 d per pair) + dQ part of the backward (dP, dS, dQ: 4 d per pair)
        flops += 8.0 * w.head_dim * len(rows) * keys
        done += 1
        if time.perf_counter() - t0 > seconds:
            break
    dt = time.perf_counter() - t0
    desc = (f"fp64 numpy oracle, head 0, {done} of {nq} query blocks (x{len(rows)} rows) of {w.name}: "
            f"forward + dQ rows against their {kr} Top-K key blocks; mask/pool/Top-K excluded")
    return flops / dt / 1e12, desc, dt


def run_sweep(args):
    """One line per point of the 2048-canvas sweep (foreground x rho x block):
    device time of forward and backward, their TFLOP/s and % of the measured
    peak, and the ratio to the same foreground's rho = 1 (dense-foreground)
    point.  Not the benchmark line; the points are parity-test shapes."""
    import torch
    import __graft_entry__ as g
    from paper_2609_23169_gb300 import path as P
    from paper_2609_23169_gb300 import ultratex as u
    from synth.workloads import SWEEP_BLOCK, SWEEP_FG, SWEEP_RHO, sweep2048

    g.build()
    dev = torch.device("cuda", 0)
    peaks, src = load_peaks()
    peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    steps = max(1, args.steps if args.steps != 10 else 2)
    for fg in SWEEP_FG:
        base = sweep2048(fg, 1.0, 128)
        q, k, v, do = (x.to(dev) for x in (base.q(), base.k(), base.v(), base.dout()))
        mask = torch.from_numpy(base.canvas_mask()).to(dev)
        dense_ms = {}
        for block in sorted(SWEEP_BLOCK, reverse=True):
            for rho in sorted(SWEEP_RHO, reverse=True):
                w = sweep2048(fg, rho, block)
                line = {"sweep": True, "workload": w.name, "fg": fg, "rho": rho, "block": block, "N": w.N}
                hp = P.HotPath(w.T, w.heads, w.head_dim, block, torch.bfloat16, u.UT_MASK_TOPK, rho=rho, device=dev)
                N = hp.step(mask, q, k, v, do)
                torch.cuda.synchronize()
                nq = -(-N // block)
                rp = hp.row_ptr[:w.heads * nq + 1].cpu().numpy()
                ci = hp.col_idx[:int(rp[-1])].cpu().numpy()
                f_fwd = retained_flops(rp, ci, N, block, w.head_dim)
                ev = []
                for _ in range(steps):
                    Nn = hp.compact(mask, [q, k, v, do])
                    hp.block_lists(Nn)
                    a, b_, c_ = (torch.cuda.Event(enable_timing=True) for _ in range(3))
                    a.record()
                    hp.forward(Nn)
                    b_.record()
                    hp.backward_pass(Nn)
                    c_.record()
                    hp.scatter(Nn)
                    ev.append((a, b_, c_))
                torch.cuda.synchronize()
                u.check_status(hp.status)
                fwd_ms = sum(a.elapsed_time(b_) for a, b_, _ in ev) / steps
                bwd_ms = sum(b_.elapsed_time(c_) for _, b_, c_ in ev) / steps
                if rho == 1.0:
                    dense_ms[block] = (fwd_ms, bwd_ms)
                d_f, d_b = dense_ms.get(block, (None, None))
                line.update({"density": round(float(rp[-1]) / (w.heads * nq * nq), 4),
                             "fwd_ms": round(fwd_ms, 3), "bwd_ms": round(bwd_ms, 3),
                             "fwd_tflops": round(f_fwd / fwd_ms / 1e9, 1),
                             "bwd_tflops": round(2.5 * f_fwd / bwd_ms / 1e9, 1),
                             "fwd_pct_peak": round(100 * f_fwd / fwd_ms / 1e9 / peak, 1),
                             "speedup_vs_dense_fg": {"fwd": round(d_f / fwd_ms, 2) if d_f else None,
                                                     "bwd": round(d_b / bwd_ms, 2) if d_b else None},
                             "peak": f"{peak} TFLOP/s ({src} bf16 burst)"})
                print(json.dumps(line), flush=True)
                del hp
                torch.cuda.empty_cache()
    return 0


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    from synth import CONFIGS
    if args.sweep:
        return run_sweep(args)
    if args.impl == "reference":
        if rank != 0:
            return 0
        w = CONFIGS[args.workload]
        per = max(2.0, 60.0 / max(1, args.steps + args.warmup))
        vals = []
        for s in range(args.warmup + args.steps):
            v, desc, dt = oracle_sample(w, per)
            if s >= args.warmup:
                vals.append(v)
        val = float(np.mean(vals))
        line = {"impl": "reference", "metric": "retained-block attention TFLOP/s and % of GB300 bf16 peak at 2048 canvas (~213K tokens)",
                "value": round(val, 6), "unit": "TFLOP/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": {"workload": w.name}, "ms_per_step": None,
                "cpu_baseline": {"value": round(val, 6), "unit": "TFLOP/s", "cores": cpu_cores(), "kind": "oracle",
                                 "sample": desc},
                "e2e": {"value": round(val, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return 0
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    line, w = run_ours(args, rank, world, local_rank)
    if rank == 0:
        if not args.no_cpu_baseline and world == 1:
            v, desc, dt = oracle_sample(w, args.cpu_seconds)
            line["cpu_baseline"] = {"value": round(v, 6), "unit": "TFLOP/s", "cores": cpu_cores(), "kind": "oracle",
                                    "sample": desc + f" ({dt:.1f} s)"}
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
