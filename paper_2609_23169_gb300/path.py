"""The hot path end to end: compaction -> block lists -> attention fwd/bwd -> scatter.

``HotPath`` owns every device buffer for one canvas size, so a step launches
only the library's kernels (plus one 4-byte device-to-host read of N, the
number of retained tokens, which sizes the compacted problem).
"""
from __future__ import annotations

import math
from typing import Optional

import numpy as np
import torch

from . import ultratex as u


class HotPath:
    def __init__(self, T: int, H: int, d: int, block: int, dtype: torch.dtype, mode: int, rho: float = 0.0,
                 device="cuda", backward: bool = True):
        self.T, self.H, self.d, self.block, self.dtype = T, H, d, block, dtype
        self.mode, self.rho, self.backward = mode, rho, backward
        self.dev = torch.device(device)
        cap = T
        e = dict(dtype=dtype, device=self.dev)
        n_in = 4 if backward else 3
        self.xc = [torch.empty((cap, H, d), **e) for _ in range(n_in)]          # Qc, Kc, Vc, dOc
        self.idx = torch.empty(max(cap, 1), dtype=torch.int32, device=self.dev)
        self.n_dev = torch.empty(1, dtype=torch.int32, device=self.dev)
        # N is read by the host once per step.  Where the device can address
        # pinned host memory, the compaction kernel writes N there and the host
        # waits on an event: a device-to-host copy of 4 bytes would queue on
        # the copy engine behind any large transfer already in flight.
        self.n_host = torch.zeros(1, dtype=torch.int32).pin_memory()
        self.n_zero_copy = u.device_accessible(self.n_host)
        self.status = torch.zeros(1, dtype=torch.int32, device=self.dev)
        self.ws_compact = torch.empty(max(u.lib().ut_fg_compact_workspace_size(T), 16), dtype=torch.uint8,
                                      device=self.dev)
        nq = -(-cap // block)
        self.nq_cap = nq
        kr_cap = nq if mode == u.UT_MASK_BITMAP else u.ut_topk_count(rho, nq)
        self.col_cap = H * nq * kr_cap
        self.row_ptr = torch.empty(H * nq + 1, dtype=torch.int32, device=self.dev)
        self.col_idx = torch.empty(max(self.col_cap, 1), dtype=torch.int32, device=self.dev)
        self.col_ptr = torch.empty(H * nq + 1, dtype=torch.int32, device=self.dev)
        self.row_idx = torch.empty(max(self.col_cap, 1), dtype=torch.int32, device=self.dev)
        shape_cap = u.AttnShape(cap, H, d, block, u._dtype_code(self.xc[0]), H * d)
        import ctypes
        self.ws_mask = torch.empty(max(u.lib().ut_block_mask_workspace_size(ctypes.byref(shape_cap), mode), 16),
                                   dtype=torch.uint8, device=self.dev)
        self.ws_bwd = torch.empty(max(u.lib().ut_bsattn_bwd_workspace_size(ctypes.byref(shape_cap)), 16),
                                  dtype=torch.uint8, device=self.dev)
        self.oc = torch.empty((cap, H, d), **e)
        self.lse = torch.empty(H * cap, dtype=torch.float32, device=self.dev)
        self.gc = [torch.empty((cap, H, d), **e) for _ in range(3)] if backward else []
        self.o_canvas = torch.zeros((T, H, d), **e)
        self.g_canvas = [torch.zeros((T, H, d), **e) for _ in range(3)] if backward else []
        self.scale = 1.0 / math.sqrt(d)
        self.N: Optional[int] = None

    def compact(self, mask: torch.Tensor, canvas: list[torch.Tensor]) -> int:
        if self.n_zero_copy:
            u.ut_fg_compact(mask, canvas, capacity=self.T, outs=self.xc[:len(canvas)], idx=self.idx,
                            n_out=self.n_host, ws=self.ws_compact, status=self.status)
            done = torch.cuda.Event()
            done.record()
            done.synchronize()
            self.N = int(self.n_host[0])  # the one device-to-host read of a step
        else:
            u.ut_fg_compact(mask, canvas, capacity=self.T, outs=self.xc[:len(canvas)], idx=self.idx,
                            n_out=self.n_dev, ws=self.ws_compact, status=self.status)
            self.N = int(self.n_dev.item())  # the one device-to-host read of a step
        return self.N

    def views(self, N: int):
        return [x[:N] for x in self.xc]

    def block_lists(self, N: int, bitmap: Optional[torch.Tensor] = None):
        shape = u.AttnShape(N, self.H, self.d, self.block, u._dtype_code(self.xc[0]), self.H * self.d)
        qc, kc = self.xc[0][:N], self.xc[1][:N]
        u.ut_block_mask(shape, self.mode, qc, kc, self.rho, bitmap, col_cap=self.col_cap,
                        with_transpose=self.backward, status=self.status, ws=self.ws_mask,
                        out=(self.row_ptr, self.col_idx, self.col_ptr if self.backward else None,
                             self.row_idx if self.backward else None))

    def forward(self, N: int):
        qc, kc, vc = (x[:N] for x in self.xc[:3])
        lse = self.lse[:self.H * N].view(self.H, N)
        u.ut_bsattn_fwd(qc, kc, vc, self.row_ptr, self.col_idx, self.block, self.scale, o=self.oc[:N], lse=lse,
                        status=self.status)
        return self.oc[:N], lse

    def backward_pass(self, N: int):
        qc, kc, vc, doc = (x[:N] for x in self.xc)
        lse = self.lse[:self.H * N].view(self.H, N)
        u.ut_bsattn_bwd(qc, kc, vc, self.oc[:N], lse, doc, self.row_ptr, self.col_idx, self.col_ptr, self.row_idx,
                        self.block, self.scale, dq=self.gc[0][:N], dk=self.gc[1][:N], dv=self.gc[2][:N],
                        ws=self.ws_bwd, status=self.status)

    def scatter(self, N: int):
        u.ut_fg_scatter(self.idx, N, [self.oc[:N]], [self.o_canvas], u.UT_BG_KEEP)
        if self.backward:
            u.ut_fg_scatter(self.idx, N, [g[:N] for g in self.gc], self.g_canvas, u.UT_BG_ZERO)

    def step(self, mask: torch.Tensor, q, k, v, dout=None, bitmap: Optional[torch.Tensor] = None) -> int:
        canvas = [q, k, v] + ([dout] if self.backward else [])
        N = self.compact(mask, canvas)
        self.block_lists(N, bitmap)
        self.forward(N)
        if self.backward:
            self.backward_pass(N)
        self.scatter(N)
        return N


def run_path(w, mask: np.ndarray, q, k, v, dout=None, bitmap: Optional[np.ndarray] = None, device="cuda"):
    """One pass of the hot path for a synthetic workload; returns the device results."""
    dev = torch.device(device)
    dtype = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    mode = u.UT_MASK_BITMAP if bitmap is not None else u.UT_MASK_TOPK
    hp = HotPath(w.T, w.heads, w.head_dim, w.block, dtype, mode, rho=(w.density if mode == u.UT_MASK_TOPK else 0.0),
                 device=dev, backward=dout is not None)
    m = torch.from_numpy(np.ascontiguousarray(mask)).to(dev)
    tq, tk, tv = (x.to(dev) for x in (q, k, v))
    tdo = dout.to(dev) if dout is not None else None
    bm = torch.from_numpy(np.ascontiguousarray(bitmap)).to(dev) if bitmap is not None else None
    N = hp.step(m, tq, tk, tv, tdo, bm)
    torch.cuda.synchronize(dev)
    u.check_status(hp.status)
    out = dict(N=N, idx=hp.idx[:N], o_canvas=hp.o_canvas, oc=hp.oc[:N],
               lse=hp.lse[:w.heads * N].view(w.heads, N), row_ptr=hp.row_ptr, col_idx=hp.col_idx,
               col_ptr=hp.col_ptr, row_idx=hp.row_idx, path=hp)
    if dout is not None:
        out.update(dq_canvas=hp.g_canvas[0], dk_canvas=hp.g_canvas[1], dv_canvas=hp.g_canvas[2],
                   dqc=hp.gc[0][:N], dkc=hp.gc[1][:N], dvc=hp.gc[2][:N])
    return out
