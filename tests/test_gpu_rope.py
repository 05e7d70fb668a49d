"""GPU parity of the rotary embedding fused with the gather of Q / K and with
the scatter of dQ / dK (Sec. 3.2: every retained token keeps its original
canvas position as its RoPE index), against the fp64 oracle, through the C ABI.

Tolerance: the kernel forms each angle in fp32 from a frequency rounded to
fp32 (angle error <= 127 * 2^-23 rad for canvas coordinates below 128),
evaluates sin/cos in fp32 and rounds the rotated pair once to the storage
type.  Against the exact rotation, element e of pair (x0, x1) may therefore
be off by half an ulp of the storage type plus 3e-5 * (|x0| + |x1|):
|gpu - exact| <= 2^-8 |exact| + 3e-5 (|x0| + |x1|) for bf16 and
<= 2^-23 |exact| + 3e-5 (|x0| + |x1|) for fp32.  Rows the call must not touch
(KEEP) or must zero (ZERO) are compared bit for bit."""
import numpy as np
import pytest
import torch

import oracle.ultratex_oracle as o
from gpu_util import bits, need_gpu
from synth import CONFIGS

pytestmark = pytest.mark.gpu

REL = {torch.bfloat16: 2.0 ** -8, torch.float32: 2.0 ** -23}
ABS_PER_PAIR = 3e-5


def _axes(d):
    return {128: (16, 56, 56), 64: (8, 28, 28)}[d]


def _assert_rotation_close(got, exact, x_in, dtype, what):
    got = np.asarray(got, np.float64)
    x = np.asarray(x_in, np.float64)
    pair = np.abs(x[..., 0::2]) + np.abs(x[..., 1::2])
    pair = np.repeat(pair, 2, axis=-1)
    bound = REL[dtype] * np.abs(exact) + ABS_PER_PAIR * pair
    err = np.abs(got - exact)
    assert np.all(err <= bound), (what, float((err - bound).max()))


def _canvas(cfg, dtype, heads=None):
    w = CONFIGS[cfg]
    if heads:
        w = w.with_(heads=heads)
    mask = w.canvas_mask()
    idx = np.flatnonzero(mask).astype(np.int32)
    q, k = w.q().to(dtype), w.k().to(dtype)
    return w, mask, idx, q, k


@pytest.mark.parametrize("cfg,heads,dtype", [("tiny", None, torch.float32), ("c512", 4, torch.bfloat16),
                                             ("c512", 2, torch.float32), ("c1024", 2, torch.bfloat16)])
def test_gather_rope_matches_oracle(cfg, heads, dtype):
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    w, mask, idx, q, k = _canvas(cfg, dtype, heads)
    d = q.shape[2]
    cfg_r = u.rope_config(w.side, _axes(d))
    qg, kg = u.ut_fg_gather_rope(torch.from_numpy(idx).cuda(), len(idx), [q.cuda(), k.cuda()], cfg_r)
    torch.cuda.synchronize()
    for name, x, g in (("Q", q, qg), ("K", k, kg)):
        xn = x.double().numpy()
        i2, ref = o.fg_compact_rope(mask, xn, w.side, _axes(d))
        assert np.array_equal(i2, idx)
        _assert_rotation_close(g.cpu().double().numpy(), ref, xn[idx], dtype, name)


def test_gather_rope_c2048_sampled_rows():
    """Full 2048 canvas (24 heads, d = 128, bf16) in the launch the sampled rows
    are checked from: 1% of the retained rows, seeded."""
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    w, mask, idx, q, _ = _canvas("c2048", torch.bfloat16)
    cfg_r = u.rope_config(w.side)
    (qg,) = u.ut_fg_gather_rope(torch.from_numpy(idx).cuda(), len(idx), [q.cuda()], cfg_r)
    torch.cuda.synchronize()
    rows = w.row_subsample(len(idx), 0.01)
    x = q[torch.from_numpy(idx[rows]).long()].double().numpy()
    ang = o.rope_angles(o.rope_positions(idx[rows], w.side), 128)
    ref = o.rope_rotate(x, ang)
    _assert_rotation_close(qg[torch.from_numpy(rows).cuda()].cpu().double().numpy(), ref, x, torch.bfloat16, "Q")


@pytest.mark.parametrize("mode", ["keep", "zero"])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_scatter_rope_matches_oracle(mode, dtype):
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    w = CONFIGS["c512"].with_(heads=3)
    mask = w.canvas_mask()
    idx = np.flatnonzero(mask).astype(np.int32)
    T, N = len(mask), len(idx)
    g = np.random.Generator(np.random.PCG64(21))
    src = torch.from_numpy(g.standard_normal((N, 3, 128)).astype(np.float32)).to(dtype)
    dst0 = torch.from_numpy(g.standard_normal((T, 3, 128)).astype(np.float32)).to(dtype)
    dst = dst0.cuda()
    bg = u.UT_BG_KEEP if mode == "keep" else u.UT_BG_ZERO
    u.ut_fg_scatter_rope(torch.from_numpy(idx).cuda(), N, [src.cuda()], [dst], u.rope_config(w.side), bg)
    torch.cuda.synchronize()
    ref = o.fg_scatter_rope(idx, src.double().numpy(), dst0.double().numpy(), w.side,
                            o.BG_KEEP if mode == "keep" else o.BG_ZERO)
    got = dst.cpu()
    bgm = torch.from_numpy(mask == 0)
    if mode == "keep":
        assert np.array_equal(bits(got[bgm]), bits(dst0[bgm]))
    else:
        assert not got[bgm].float().abs().any()
    _assert_rotation_close(got.double().numpy()[idx], ref[idx], src.double().numpy(), dtype, "scatter")


def test_gather_then_scatter_round_trip_and_empty():
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    w, mask, idx, q, _ = _canvas("c512", torch.float32, heads=2)
    cfg_r = u.rope_config(w.side)
    ic = torch.from_numpy(idx).cuda()
    (qg,) = u.ut_fg_gather_rope(ic, len(idx), [q.cuda()], cfg_r)
    back = torch.zeros_like(q).cuda()
    u.ut_fg_scatter_rope(ic, len(idx), [qg], [back], cfg_r, u.UT_BG_ZERO)
    torch.cuda.synchronize()
    fg = torch.from_numpy(idx).long()
    assert torch.allclose(back.cpu()[fg], q[fg], rtol=0, atol=1e-4)
    assert not back.cpu()[torch.from_numpy(mask == 0)].abs().any()
    # n = 0: nothing is written
    out = torch.full((4, 2, 128), 7.0).cuda()
    u.ut_fg_gather_rope(ic, 0, [q.cuda()], cfg_r, dsts=[out])
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())
