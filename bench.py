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
per_config  the same step on the 512 and 1024 canvases (structured block
         lists), L2 flushed before each step.
The reference arm (--impl reference) and cpu_baseline time the fp64 CPU
oracle on a bounded sample of the same workload, counting the same work per
retained pair as the GPU value (forward + full backward, 14*d FLOP per
query-key row pair); oracle_times records the oracle's wall time on whole
configurations (this build has no reference implementation).
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
    ap.add_argument("--no-per-config", action="store_true", help="skip the 512 / 1024 canvas steps")
    ap.add_argument("--no-oracle-times", action="store_true", help="skip the whole-config oracle wall times")
    ap.add_argument("--oracle-time", default="", help=argparse.SUPPRESS)  # internal: one oracle timing run
    ap.add_argument("--oracle-parts", default="fwd,bwd", help=argparse.SUPPRESS)
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


METRIC = "retained-block attention TFLOP/s and % of GB300 bf16 peak at 2048 canvas (~213K tokens)"


def workload_config(w, N: int, density: float, world: int) -> dict:
    """config object of the JSON line; both arms build it from here so that
    the same workload gives the same object."""
    rule = (f"Top-K rho={w.rho}" if w.mask_mode == "topk" else "structured lists (own view, partner view, reference)")
    return {"workload": f"{w.name}: {w.n_images} images x {w.side}x{w.side} tokens (T={w.T}), "
                        f"{int(round(w.fg_frac * 100))}% {w.shape} foreground (N={N}), H={w.heads}, d={w.head_dim}, "
                        f"b={w.block}, {rule} (density {density:.4f}), forward+backward",
            "N": N, "T": w.T, "heads": w.heads, "head_dim": w.head_dim, "block": w.block,
            "rho": w.rho if w.mask_mode == "topk" else None, "parallelism": f"replicas x{world}",
            "l2": l2_note(w)}


def l2_note(w) -> str:
    gb = w.T * w.heads * w.head_dim * 2 / 1e9
    if gb > 0.129:
        return "inputs larger than L2 (each canvas tensor %.2f GB > 129 MB)" % gb
    return "L2 flushed before each step by a 256 MB write (each canvas tensor %.3f GB < 129 MB)" % gb


def list_density(w, N: int) -> float:
    """Retained fraction of the block pairs; for Top-K it is K_rho / N_k in every head."""
    nq = -(-N // w.block)
    if w.mask_mode == "topk":
        return max(1, int(math.floor(w.rho * nq))) / nq
    return float(w.block_bitmap().mean())


class StepRunner:
    """One HotPath on one workload with resident inputs; times whole steps and
    the entry points inside them with CUDA events on the launching stream."""

    def __init__(self, w, dev):
        import torch
        from paper_2609_23169_gb300 import path as P
        from paper_2609_23169_gb300 import ultratex as u
        self.w, self.dev, self.u = w, dev, u
        self.mask_np, q, k, v, do = make_inputs(w, dev)
        self.host = (q, k, v, do)
        self.mask = torch.from_numpy(self.mask_np).to(dev)
        self.tq, self.tk, self.tv, self.tdo = (x.to(dev) for x in (q, k, v, do))
        topk = w.mask_mode == "topk"
        self.mode = u.UT_MASK_TOPK if topk else u.UT_MASK_BITMAP
        self.bitmap = None if topk else torch.from_numpy(w.block_bitmap()).to(dev)
        self.hp = P.HotPath(w.T, w.heads, w.head_dim, w.block, torch.bfloat16, self.mode,
                            rho=w.rho if topk else 0.0, device=dev)
        self.stream = torch.cuda.current_stream()
        self.ev = {}

    def timed(self, name, fn):
        import torch
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(self.stream)
        r = fn()
        b.record(self.stream)
        self.ev.setdefault(name, []).append((a, b))
        return r

    def step(self, record: bool) -> int:
        hp = self.hp
        inputs = [self.tq, self.tk, self.tv, self.tdo]
        if not record:
            return hp.step(self.mask, *inputs, bitmap=self.bitmap)
        N = self.timed("compact", lambda: hp.compact(self.mask, inputs))
        self.timed("block_mask", lambda: hp.block_lists(N, self.bitmap))
        self.timed("bsattn_fwd", lambda: hp.forward(N))
        self.timed("bsattn_bwd", lambda: hp.backward_pass(N))
        self.timed("scatter", lambda: hp.scatter(N))
        return N

    def lists_flops(self, N: int):
        w, hp = self.w, self.hp
        nq = -(-N // w.block)
        rp = hp.row_ptr[:w.heads * nq + 1].cpu().numpy()
        ci = hp.col_idx[:int(rp[-1])].cpu().numpy()
        f_fwd = retained_flops(rp, ci, N, w.block, w.head_dim)
        density = float(rp[-1]) / (w.heads * nq * nq)
        return f_fwd, density

    def kernel_ms(self) -> dict:
        return {n: sum(a.elapsed_time(b) for a, b in l) / len(l) for n, l in self.ev.items()}


def time_per_config(names, dev, steps: int, warmup: int, peak: float) -> dict:
    """The whole step on the smaller canvases (structured block lists), timed
    step by step with the L2 flushed (a 256 MB write) before each step: the
    512 canvas's tensors are smaller than L2."""
    import torch
    from synth import CONFIGS
    out = {}
    flush = torch.empty(64 << 20, dtype=torch.float32, device=dev)
    for name in names:
        w = CONFIGS[name]
        r = StepRunner(w, dev)
        for _ in range(warmup):
            N = r.step(False)
        torch.cuda.synchronize()
        r.u.check_status(r.hp.status)
        f_fwd, density = r.lists_flops(N)
        tot = 0.0
        for _ in range(steps):
            flush.fill_(1.0)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(r.stream)
            r.step(True)
            e1.record(r.stream)
            torch.cuda.synchronize()
            tot += e0.elapsed_time(e1)
        r.u.check_status(r.hp.status)
        ms = tot / steps
        km = r.kernel_ms()
        tf = 3.5 * f_fwd / (ms * 1e-3) / 1e12
        out[name] = {"workload": workload_config(w, N, density, 1)["workload"], "N": N,
                     "ms_per_step": round(ms, 4), "tflops": round(tf, 2), "pct_of_burst_peak": round(100 * tf / peak, 2),
                     "retained_fwd_tflop": round(f_fwd / 1e12, 4),
                     "bsattn_fwd": {"ms": round(km["bsattn_fwd"], 4),
                                    "tflops": round(f_fwd / (km["bsattn_fwd"] * 1e-3) / 1e12, 2)},
                     "bsattn_bwd": {"ms": round(km["bsattn_bwd"], 4),
                                    "tflops": round(2.5 * f_fwd / (km["bsattn_bwd"] * 1e-3) / 1e12, 2)},
                     "l2": "flushed before each step (256 MB write)", "steps": steps}
        del r
        torch.cuda.empty_cache()
    return out


def load_traffic_record():
    """DRAM bytes per launch of the attention entry points from the committed
    ncu summary (profiles/dram_traffic.txt): one line per entry point with the
    workload and head count it was captured on, the bytes, and the SHA-256 of
    the kernel sources at capture time."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    rec = {}
    if not os.path.exists(path):
        return rec
    with open(path) as f:
        for line in f:
            parts = line.split()
            if len(parts) >= 5 and parts[0] in ("bsattn_fwd", "bsattn_bwd") and not line.startswith("#"):
                rec[parts[0]] = {"workload": parts[1], "heads": int(parts[2]), "bytes": float(parts[3]),
                                 "sha256": parts[4]}
    return rec


KERNEL_SOURCES = {"bsattn_fwd": ["attn_fwd_tc.cu", "common.cuh"],
                  "bsattn_bwd": ["attn_bwd_tc.cu", "common.cuh"]}


def kernel_source_hash(entry: str) -> str:
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[entry]:
        with open(os.path.join(ROOT, "paper_2609_23169_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def traffic_for(entry: str, w) -> tuple:
    """(bytes per launch or None, note).  The recorded capture is scaled by the
    head count (each head is an independent problem of the same size); it is
    withheld when the kernel sources changed since the capture or the
    workload differs."""
    rec = load_traffic_record().get(entry)
    if rec is None:
        return None, "no ncu record"
    if rec["sha256"] != kernel_source_hash(entry):
        return None, "kernel sources changed since the ncu capture"
    if rec["workload"] != w.name:
        return None, f"ncu capture is of {rec['workload']}, not {w.name}"
    return rec["bytes"] * w.heads / rec["heads"], f"ncu, {rec['heads']}-head capture scaled to {w.heads} heads"


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
    r = StepRunner(w, dev)
    hp, stream, mask_np, mask = r.hp, r.stream, r.mask_np, r.mask
    q, k, v, do = r.host
    tq, tk, tv, tdo = r.tq, r.tk, r.tv, r.tdo

    for _ in range(args.warmup):
        N = r.step(False)
    torch.cuda.synchronize()
    u.check_status(hp.status)
    f_fwd, density = r.lists_flops(N)
    f_step = 3.5 * f_fwd

    clocks = ClockSampler(local_rank)
    clocks.start()
    time.sleep(0.3)
    r.ev.clear()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        r.step(True)
    t1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    ms_total = t0.elapsed_time(t1)
    clk = clocks.stop()
    u.check_status(hp.status)
    kern_ms = r.kernel_ms()

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
        paths = [hp] + [P.HotPath(w.T, w.heads, w.head_dim, w.block, torch.bfloat16, r.mode,
                                  rho=w.rho if w.mask_mode == "topk" else 0.0, device=dev) for _ in range(NB - 1)]
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
                paths[b].step(m_, q_, k2, v_, d_, bitmap=r.bitmap)
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
    # dominant entry point by measured time
    dom = max(("bsattn_fwd", "bsattn_bwd"), key=lambda n: kern_ms.get(n, 0))
    dom_flops = f_fwd if dom == "bsattn_fwd" else 2.5 * f_fwd
    achieved = dom_flops / (kern_ms[dom] * 1e-3) / 1e12
    # the step runs for seconds under the power cap, so the dominant kernel is
    # held against the sustained peak; the burst fraction is reported beside it
    peak = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    burst = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    traffic, traffic_note = traffic_for(dom, w)
    # algorithmic bytes of the dominant entry point: forward reads Q, K, V once
    # and writes O, LSE; backward reads Q, K, V, O, dO, LSE and writes dQ, dK, dV
    row = N * w.heads * w.head_dim * 2
    alg_bytes = (4 * row + 4 * w.heads * N) if dom == "bsattn_fwd" else (8 * row + 4 * w.heads * N)
    bytes_tensor = 2 * N * w.heads * w.head_dim * 2 + w.T + 4 * N   # per tensor, compaction
    kernels = {
        n: {"ms": round(kern_ms[n], 4)} for n in kern_ms
    }
    kernels["bsattn_fwd"]["tflops"] = round(f_fwd / (kern_ms["bsattn_fwd"] * 1e-3) / 1e12, 2)
    kernels["bsattn_bwd"]["tflops"] = round(2.5 * f_fwd / (kern_ms["bsattn_bwd"] * 1e-3) / 1e12, 2)
    for n in ("bsattn_fwd", "bsattn_bwd"):
        kernels[n]["frac_burst"] = round(kernels[n]["tflops"] / burst, 4)
    kernels["compact"]["gbs"] = round(4 * bytes_tensor / (kern_ms["compact"] * 1e-3) / 1e9, 1)
    sc_bytes = 2 * N * w.heads * w.head_dim * 2 + 3 * (2 * N * w.heads * w.head_dim * 2 +
                                                      (w.T - N) * w.heads * w.head_dim * 2)
    kernels["scatter"]["gbs"] = round(sc_bytes / (kern_ms["scatter"] * 1e-3) / 1e9, 1)

    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    for n, b_ in (("compact", 4 * bytes_tensor), ("scatter", sc_bytes)):
        kernels[n]["frac_hbm"] = round(kernels[n]["gbs"] / hbm_peak, 4)
    per_config = None
    if rank == 0 and not args.no_per_config and w.name == "c2048" and not args.heads:
        per_config = time_per_config(("c512", "c1024"), dev, max(3, min(args.steps, 10)), 3, burst)
    sampler = time_sampler_steps(w, dev, hbm_peak) if rank == 0 else None
    rope = time_rope(w, dev, hbm_peak) if rank == 0 else None
    alpha_mask = time_mask_from_alpha(w, dev, hbm_peak) if rank == 0 else None
    line = {
        "metric": METRIC,
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
        "config": workload_config(w, N, density, world),
        "retained_fwd_tflop": round(f_fwd / 1e12, 4),
        "pct_of_peak": round(100 * value / world / peak, 2),
        "pct_of_burst_peak": round(100 * value / world / burst, 2),
        "roofline": {"bound": "tensor", "kernel": dom, "achieved": round(achieved, 2), "peak": peak,
                     "unit": "TFLOP/s", "frac": round(achieved / peak, 4), "frac_burst": round(achieved / burst, 4),
                     "traffic": traffic, "traffic_note": traffic_note, "algorithmic_bytes": int(alg_bytes),
                     "peak_source": f"{peak_src} bf16 sustained (burst {burst})"},
        "kernels": kernels,
        "e2e": e2e,
        "gpu_launches": args.steps * hp_launches(hp),
        "clocks": clk,
    }
    if per_config is not None:
        line["per_config"] = per_config
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

    zc = torch.empty_like(v)
    ms_e = timed(lambda: u.ut_fg_euler_update(idx, n, z, v, x["dt"], status=st))
    ms_g = timed(lambda: u.ut_fg_euler_update_gather(idx, n, z, v, x["dt"], zc=zc, status=st))
    ms_c = timed(lambda: u.ut_fg_composite(mask, z, tile))
    u.check_status(st)
    b_e = n * (4 + 3 * row)            # idx, v read, z read + write (foreground rows)
    b_g = n * (4 + 4 * row)            # the same and the compacted rows written for the next step
    b_c = T + (T - n) * row            # mask read, background rows written
    out = {"workload": f"{w.name} target canvas: {T} tokens, {n} foreground, 64 channels bf16, "
                       f"tile of {x['period']} rows", "l2": "flushed before each call by reading 256 MB"}
    for name, ms, b in (("euler_update", ms_e, b_e), ("euler_update_gather", ms_g, b_g), ("composite", ms_c, b_c)):
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
def oracle_inputs(w, head: int = 0):
    """Compacted inputs of one head (fp64, the exact bf16 values) and that
    head's block lists: the oracle's own Top-K lists, or the bitmap's CSR."""
    import torch
    import oracle.ultratex_oracle as o
    idx = np.flatnonzero(w.canvas_mask())
    t = torch.from_numpy(idx)
    xs = [x[t][:, head:head + 1].float().numpy().astype(np.float64) for x in (w.q(), w.k(), w.v(), w.dout())]
    N = len(idx)
    if w.mask_mode == "topk":
        rp, ci, _, _ = o.topk_block_mask(xs[0], xs[1], w.block, w.rho)
    else:
        rp, ci = o.bitmap_to_csr(w.block_bitmap()[head:head + 1])
    return xs, np.asarray(rp, np.int64), np.asarray(ci, np.int64), N


def oracle_sample(w, seconds: float, prepared=None):
    """Time the fp64 oracle, as it stands, on a bounded sample of the workload:
    the forward and the full backward (dQ, dK, dV) of a seeded set of whole
    query blocks of head 0 over their own key-block lists, sized to take about
    `seconds`.  The work is counted as the GPU value counts it: 14*d FLOP per
    retained query-key row pair (forward 4*d, backward 2.5x).  Returns
    (TFLOP/s, description, seconds)."""
    import oracle.ultratex_oracle as o
    (qc, kc, vc, dc), rp, ci, N = prepared if prepared is not None else oracle_inputs(w)
    b = w.block
    nq = -(-N // b)
    sizes = np.array([len(o.tile_rows(j, N, b)) for j in range(nq)], dtype=np.float64)
    order = np.random.Generator(np.random.PCG64([w.seed, 6])).permutation(nq)

    def run(blocks):
        keep = np.zeros(nq, dtype=bool)
        keep[blocks] = True
        lens = np.where(keep, np.diff(rp), 0)
        rps = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
        cis = np.concatenate([ci[rp[i]:rp[i + 1]] for i in sorted(blocks)]).astype(np.int64)
        t0 = time.perf_counter()
        o.bsattn_fwd(qc, kc, vc, rps, cis, b)
        o.bsattn_bwd(qc, kc, vc, dc, rps, cis, b)
        dt = time.perf_counter() - t0
        pairs = sum(sizes[i] * sizes[ci[rp[i]:rp[i + 1]]].sum() for i in blocks)
        return dt, 14.0 * w.head_dim * pairs

    dt1, _ = run(order[:1])
    m = int(max(1, min(nq, seconds / max(dt1, 1e-3))))
    dt, flops = run(order[:m])
    kr = int(np.diff(rp).max()) if len(rp) > 1 else 0
    desc = (f"fp64 numpy oracle (bsattn_fwd + bsattn_bwd as they stand), head 0, {m} seeded query blocks of "
            f"{nq} of {w.name} with their lists (up to {kr} key blocks each); 14*d FLOP per retained row pair, "
            f"as the GPU value counts; lists built beforehand, not timed")
    return flops / dt / 1e12, desc, dt


def cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.machine()


def oracle_time_config(name: str, parts: str) -> dict:
    """Wall time of the oracle on a whole configuration (all heads): the
    forward, then the backward (which recomputes its softmax rows).  Lists
    come from the bitmap (structured configs); compacted inputs in fp64."""
    import torch
    import oracle.ultratex_oracle as o
    from synth import CONFIGS
    w = CONFIGS[name]
    idx = np.flatnonzero(w.canvas_mask())
    t = torch.from_numpy(idx)
    qc, kc, vc, dc = (x[t].double().numpy() for x in (w.q(), w.k(), w.v(), w.dout()))
    rp, ci = o.bitmap_to_csr(w.block_bitmap())
    out = {"N": len(idx), "heads": w.heads}
    if "fwd" in parts:
        t0 = time.perf_counter()
        o.bsattn_fwd(qc, kc, vc, rp, ci, w.block)
        out["fwd_s"] = round(time.perf_counter() - t0, 3)
    if "bwd" in parts:
        t0 = time.perf_counter()
        o.bsattn_bwd(qc, kc, vc, dc, rp, ci, w.block)
        out["bwd_s"] = round(time.perf_counter() - t0, 3)
    return out


def oracle_wall_times(cores: int) -> dict:
    """The oracle's wall time on the tiny, 512 and 1024 configurations in full
    with every host core, and on tiny and 512 with one thread, each in a fresh
    interpreter whose BLAS / OpenMP thread count is set before numpy loads."""
    runs = [("tiny", cores), ("c512", cores), ("c1024", cores), ("tiny", 1), ("c512", 1)]
    out = {"cores": cores, "cpu_model": cpu_model(), "note": "fp64 numpy oracle, forward then full backward"}
    for name, threads in runs:
        env = dict(os.environ)
        for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS"):
            env[var] = str(threads)
        cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--oracle-time", name]
        try:
            r = subprocess.run(cmd, capture_output=True, text=True, env=env, timeout=900)
            rec = json.loads(r.stdout.strip().splitlines()[-1])
        except Exception as e:  # noqa: BLE001  (a timing that failed is reported as such)
            rec = {"error": str(e)[:200]}
        rec["threads"] = threads
        out[f"{name}_{threads}t"] = rec
    return out


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
    if args.oracle_time:
        print(json.dumps(oracle_time_config(args.oracle_time, args.oracle_parts)))
        return 0
    if args.impl == "reference":
        if rank != 0:
            return 0
        w = CONFIGS[args.workload]
        prepared = oracle_inputs(w)
        N = prepared[3]
        per = max(2.0, min(10.0, 100.0 / max(1, args.steps + args.warmup)))
        vals, secs = [], []
        for s in range(args.warmup + args.steps):
            v, desc, dt = oracle_sample(w, per, prepared)
            if s >= args.warmup:
                vals.append(v)
                secs.append(dt)
        val = float(np.mean(vals))
        line = {"impl": "reference", "metric": METRIC,
                "value": round(val, 6), "unit": "TFLOP/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": workload_config(w, N, list_density(w, N), 1),
                "ms_per_step": round(1e3 * float(np.mean(secs)), 1),
                "cpu_baseline": {"value": round(val, 6), "unit": "TFLOP/s", "cores": cpu_cores(), "kind": "oracle",
                                 "sample": desc + f"; one sample per step, ~{per:.0f} s each"},
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
            step_tflop = 3.5 * line["retained_fwd_tflop"]
            line["cpu_baseline"] = {"value": round(v, 6), "unit": "TFLOP/s", "cores": cpu_cores(), "kind": "oracle",
                                    "sample": desc + f" ({dt:.1f} s)",
                                    "extrapolated_step_s": round(step_tflop / v, 1),
                                    "extrapolation": "the whole step's retained-pair work (forward + backward, "
                                                     f"{step_tflop:.2f} TFLOP) at the sample's rate; not measured"}
        if not args.no_oracle_times and world == 1:
            line["oracle_times"] = oracle_wall_times(cpu_cores())
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
