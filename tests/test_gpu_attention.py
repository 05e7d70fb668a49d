"""GPU parity: block-sparse attention forward and backward against the fp64 oracle.

Small configurations are compared element by element in full; the 1024 and
2048 canvases, in the launch configuration the benchmark times, are compared
on seeded row samples that the oracle computes one by one.
"""
import math

import numpy as np
import pytest
import torch

import oracle.ultratex_oracle as o
from gpu_util import assert_bf16_close, assert_f32_close, need_gpu, to_np
from synth import CONFIGS

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    need_gpu()


def _lists_from_bitmap(bm, N, H, d, b, dtype_code):
    from paper_2609_23169_gb300 import ultratex as u
    shape = u.AttnShape(N, H, d, b, dtype_code, H * d)
    st = u.status_word()
    out = u.ut_block_mask(shape, u.UT_MASK_BITMAP, bitmap=torch.from_numpy(bm).cuda(), status=st,
                          col_cap=max(1, int((bm != 0).sum())))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return out


def _random_problem(N, H, d, b, density, seed, dtype=torch.bfloat16, empty_rows=()):
    g = np.random.Generator(np.random.PCG64([77, seed]))
    q, k, v, do = (torch.from_numpy(g.standard_normal((N, H, d)).astype(np.float32)).to(dtype) for _ in range(4))
    nq = -(-N // b)
    bm = (g.random((H, nq, nq)) < density).astype(np.uint8)
    for h in range(H):
        for i in range(nq):
            if not bm[h, i].any():
                bm[h, i, g.integers(nq)] = 1
    for (h, i) in empty_rows:
        bm[h, i] = 0
    return q, k, v, do, bm


def _run_fwd(q, k, v, bm, b):
    from paper_2609_23169_gb300 import ultratex as u
    N, H, d = q.shape
    code = u.UT_BF16 if q.dtype == torch.bfloat16 else u.UT_F32
    rp, ci, cp, ri = _lists_from_bitmap(bm, N, H, d, b, code)
    st = u.status_word()
    O, L = u.ut_bsattn_fwd(q.cuda(), k.cuda(), v.cuda(), rp, ci, b, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return O, L, (rp, ci, cp, ri)


# ------------------------------------------------------------------ forward
def test_fwd_fp32_tiny_full():
    w = CONFIGS["tiny"]
    mask = w.canvas_mask()
    idx = np.flatnonzero(mask)
    q, k, v = (x[torch.from_numpy(idx)] for x in (w.q(), w.k(), w.v()))
    bm = w.block_bitmap()
    O, L, _ = _run_fwd(q, k, v, bm, w.block)
    rp, ci = o.bitmap_to_csr(bm)
    rO, rL = o.bsattn_fwd(q.double().numpy(), k.double().numpy(), v.double().numpy(), rp, ci, w.block)
    assert_f32_close(to_np(O), rO, "O")
    assert_f32_close(to_np(L), rL, "LSE")


@pytest.mark.parametrize("N,H,b,dens,seed", [(300, 2, 128, 0.6, 1), (128, 1, 128, 1.0, 2), (1, 1, 128, 1.0, 3),
                                             (129, 3, 128, 0.5, 4), (1000, 2, 128, 0.3, 5), (2049, 1, 128, 1.0, 6)])
def test_fwd_bf16_small_full(N, H, b, dens, seed):
    q, k, v, _, bm = _random_problem(N, H, 128, b, dens, seed)
    O, L, _ = _run_fwd(q, k, v, bm, b)
    rp, ci = o.bitmap_to_csr(bm)
    rO, rL = o.bsattn_fwd(q.double().numpy(), k.double().numpy(), v.double().numpy(), rp, ci, b)
    assert_bf16_close(to_np(O), rO, "O")
    assert np.abs(to_np(L) - rL).max() < 1e-3


def test_fwd_bf16_head_dim_64():
    q, k, v, _, bm = _random_problem(700, 3, 64, 128, 0.5, 9)
    O, L, _ = _run_fwd(q, k, v, bm, 128)
    rp, ci = o.bitmap_to_csr(bm)
    rO, rL = o.bsattn_fwd(q.double().numpy(), k.double().numpy(), v.double().numpy(), rp, ci, 128)
    assert_bf16_close(to_np(O), rO, "O d=64")


def test_fwd_bf16_empty_rows_and_large_logits():
    # empty lists give O = 0 and LSE = -inf; scaled inputs exercise the running-max rescale
    q, k, v, _, bm = _random_problem(1100, 2, 128, 128, 0.7, 10, empty_rows=[(0, 3), (1, 8)])
    q = (q.float() * 6).to(torch.bfloat16)
    O, L, _ = _run_fwd(q, k, v, bm, 128)
    rp, ci = o.bitmap_to_csr(bm)
    rO, rL = o.bsattn_fwd(q.double().numpy(), k.double().numpy(), v.double().numpy(), rp, ci, 128)
    Og, Lg = to_np(O), to_np(L)
    assert np.all(Og[384:512, 0] == 0) and np.all(np.isneginf(Lg[0, 384:512]))
    assert np.all(Og[1024:1100, 1] == 0)
    assert not np.isnan(Og).any()
    assert_bf16_close(Og, rO, "O")
    fin = np.isfinite(rL)
    assert np.abs(Lg[fin] - rL[fin]).max() < 2e-3


def test_fwd_bf16_c512_full():
    w = CONFIGS["c512"]
    idx = np.flatnonzero(w.canvas_mask())
    t = torch.from_numpy(idx)
    q, k, v = (x[t] for x in (w.q(), w.k(), w.v()))
    bm = w.block_bitmap()
    O, L, _ = _run_fwd(q, k, v, bm, w.block)
    rp, ci = o.bitmap_to_csr(bm)
    rO, rL = o.bsattn_fwd(q.double().numpy(), k.double().numpy(), v.double().numpy(), rp, ci, w.block)
    s = assert_bf16_close(to_np(O), rO, "O c512")
    print("c512 O error", s)
    assert np.abs(to_np(L) - rL).max() < 1e-3


def _sampled_fwd_check(w, mode):
    """Full-size problem through the bench's path; the oracle checks sampled rows."""
    from paper_2609_23169_gb300 import path as P
    mask = w.canvas_mask()
    q, k, v = w.q(), w.k(), w.v()
    bm = w.block_bitmap() if mode == "bitmap" else None
    out = P.run_path(w, mask, q, k, v, None, bitmap=bm)
    idx = np.flatnonzero(mask)
    t = torch.from_numpy(idx)
    qc, kc, vc = (x[t].float().numpy() for x in (q, k, v))
    nq = -(-w.N // w.block)
    rp = out["row_ptr"][:w.heads * nq + 1].cpu().numpy()
    ci = out["col_idx"][:int(rp[-1])].cpu().numpy()
    if mode == "bitmap":
        rrp, rci = o.bitmap_to_csr(bm)
        assert np.array_equal(rp, rrp) and np.array_equal(ci[:len(rci)], rci)
    rows = w.row_subsample(w.N, 0.01)
    O = out["oc"].float().cpu().numpy()
    L = out["lse"].cpu().numpy()
    errs = []
    for h in range(w.heads):
        rO, rL = o.bsattn_fwd_rows(qc, kc, vc, rp, ci, w.block, h, rows)
        errs.append((O[rows, h], rO))
        assert np.abs(L[h, rows] - rL).max() < 1e-3
    got = np.concatenate([e[0] for e in errs])
    ref = np.concatenate([e[1] for e in errs])
    s = assert_bf16_close(got, ref, w.name)
    # scatter put the compacted rows at their canvas positions
    oc = out["o_canvas"][torch.from_numpy(idx[rows]).cuda()].float().cpu().numpy()
    assert np.array_equal(oc, O[rows])
    return s


def test_fwd_c1024_sampled():
    print(_sampled_fwd_check(CONFIGS["c1024"], "bitmap"))


def test_fwd_c2048_sampled():
    print(_sampled_fwd_check(CONFIGS["c2048"], "topk"))


# ----------------------------------------------------------------- backward
def _run_bwd(q, k, v, do, bm, b):
    from paper_2609_23169_gb300 import ultratex as u
    O, L, (rp, ci, cp, ri) = _run_fwd(q, k, v, bm, b)
    st = u.status_word()
    dq, dk, dv = u.ut_bsattn_bwd(q.cuda(), k.cuda(), v.cuda(), O, L, do.cuda(), rp, ci, cp, ri, b, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return dq, dk, dv


def test_bwd_fp32_tiny_full():
    w = CONFIGS["tiny"]
    idx = torch.from_numpy(np.flatnonzero(w.canvas_mask()))
    q, k, v, do = (x[idx] for x in (w.q(), w.k(), w.v(), w.dout()))
    bm = w.block_bitmap()
    dq, dk, dv = _run_bwd(q, k, v, do, bm, w.block)
    rp, ci = o.bitmap_to_csr(bm)
    rq, rk, rv = o.bsattn_bwd(*(x.double().numpy() for x in (q, k, v, do)), rp, ci, w.block)
    for name, g, r in (("dQ", dq, rq), ("dK", dk, rk), ("dV", dv, rv)):
        assert_f32_close(to_np(g), r, name)


@pytest.mark.parametrize("N,H,d,dens,seed", [(300, 2, 128, 0.6, 21), (1000, 2, 128, 0.3, 22), (700, 2, 64, 0.5, 23),
                                             (129, 1, 128, 1.0, 24)])
def test_bwd_bf16_small_full(N, H, d, dens, seed):
    q, k, v, do, bm = _random_problem(N, H, d, 128, dens, seed, empty_rows=[(0, 0)] if N > 256 else ())
    dq, dk, dv = _run_bwd(q, k, v, do, bm, 128)
    rp, ci = o.bitmap_to_csr(bm)
    rq, rk, rv = o.bsattn_bwd(*(x.double().numpy() for x in (q, k, v, do)), rp, ci, 128)
    for name, g, r in (("dQ", dq, rq), ("dK", dk, rk), ("dV", dv, rv)):
        assert_bf16_close(to_np(g), r, name)


def test_bwd_c512_four_heads_full():
    w = CONFIGS["c512"].with_(heads=4)
    idx = torch.from_numpy(np.flatnonzero(w.canvas_mask()))
    q, k, v, do = (x[idx] for x in (w.q(), w.k(), w.v(), w.dout()))
    bm = w.block_bitmap()
    dq, dk, dv = _run_bwd(q, k, v, do, bm, w.block)
    rp, ci = o.bitmap_to_csr(bm)
    rq, rk, rv = o.bsattn_bwd(*(x.double().numpy() for x in (q, k, v, do)), rp, ci, w.block)
    for name, g, r in (("dQ", dq, rq), ("dK", dk, rk), ("dV", dv, rv)):
        print(name, assert_bf16_close(to_np(g), r, name))


def _sampled_bwd_check(w, mode, key_heads=(0, 7)):
    """Full-size forward + backward through the bench's path; sampled dQ rows in
    every head and sampled dK/dV rows in two heads against the oracle."""
    from paper_2609_23169_gb300 import path as P
    mask = w.canvas_mask()
    q, k, v, do = w.q(), w.k(), w.v(), w.dout()
    bm = w.block_bitmap() if mode == "bitmap" else None
    out = P.run_path(w, mask, q, k, v, do, bitmap=bm)
    idx = np.flatnonzero(mask)
    t = torch.from_numpy(idx)
    qc, kc, vc, dc = (x[t].float().numpy() for x in (q, k, v, do))
    nq = -(-w.N // w.block)
    rp = out["row_ptr"][:w.heads * nq + 1].cpu().numpy()
    ci = out["col_idx"][:int(rp[-1])].cpu().numpy()
    rows = w.row_subsample(w.N, 0.005)
    dq = out["dqc"].float().cpu().numpy()
    dk = out["dkc"].float().cpu().numpy()
    dv = out["dvc"].float().cpu().numpy()
    got, ref = [], []
    for h in range(w.heads):
        got.append(dq[rows, h])
        ref.append(o.bsattn_bwd_dq_rows(qc, kc, vc, dc, rp, ci, w.block, h, rows))
    sq = assert_bf16_close(np.concatenate(got), np.concatenate(ref), "dQ " + w.name)
    krows = rows[:24]
    gk, gv, rk, rv = [], [], [], []
    for h in key_heads:
        a, b = o.bsattn_bwd_dkdv_rows(qc, kc, vc, dc, rp, ci, w.block, h, krows)
        gk.append(dk[krows, h]); gv.append(dv[krows, h]); rk.append(a); rv.append(b)
    sk = assert_bf16_close(np.concatenate(gk), np.concatenate(rk), "dK " + w.name)
    sv = assert_bf16_close(np.concatenate(gv), np.concatenate(rv), "dV " + w.name)
    # scatter (ZERO mode) put gradients at canvas positions and zeros elsewhere
    gq = out["dq_canvas"]
    assert torch.equal(gq[torch.from_numpy(idx[rows]).cuda()].float().cpu(), torch.from_numpy(dq[rows]))
    bg = torch.from_numpy(np.flatnonzero(mask == 0)[:1000]).cuda()
    assert torch.all(gq[bg] == 0)
    return sq, sk, sv


def test_bwd_c1024_sampled():
    print(_sampled_bwd_check(CONFIGS["c1024"], "bitmap"))


def test_bwd_c2048_sampled():
    print(_sampled_bwd_check(CONFIGS["c2048"], "topk"))


def test_hot_path_count_in_pinned_or_device_memory():
    """The step reads N either from pinned host memory the device writes (after
    an event) or by a device-to-host copy; both give the same N and the same
    canvas results: bit for bit for O, dK and dV, and for dQ up to the order
    of its fp32 reductions."""
    from paper_2609_23169_gb300 import path as P
    from paper_2609_23169_gb300 import ultratex as u
    w = CONFIGS["c512"].with_(heads=2)
    m = torch.from_numpy(w.canvas_mask()).cuda()
    q, k, v, do = (x.cuda() for x in (w.q(), w.k(), w.v(), w.dout()))
    bm = torch.from_numpy(w.block_bitmap()).cuda()
    outs = []
    for zero_copy in (True, False):
        hp = P.HotPath(w.T, w.heads, w.head_dim, w.block, torch.bfloat16, u.UT_MASK_BITMAP, device="cuda")
        assert hp.n_zero_copy   # pinned host memory is device-accessible on this system
        hp.n_zero_copy = zero_copy
        N = hp.step(m, q, k, v, do, bm)
        torch.cuda.synchronize()
        u.check_status(hp.status)
        outs.append((N, [t.cpu() for t in [hp.o_canvas] + hp.g_canvas]))
    assert outs[0][0] == outs[1][0] == w.N
    (o0, dq0, dk0, dv0), (o1, dq1, dk1, dv1) = outs[0][1], outs[1][1]
    for a, b in ((o0, o1), (dk0, dk1), (dv0, dv1)):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    assert torch.allclose(dq0.float(), dq1.float(), rtol=1e-2, atol=1e-4)
