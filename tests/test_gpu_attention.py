"""GPU parity: block-sparse attention forward and backward against the fp64 oracle.

Small configurations, the 512 canvas and the whole 1024 canvas (24 heads,
forward and backward, through the benchmark's path) are compared element by
element in full.  The 2048 canvas, in the launch configuration the benchmark
times, is compared on seeded row samples in every head plus two whole heads
(dQ, dK, dV of every row); its Top-K lists are first checked against the
oracle's own, and the oracle reference is computed from the oracle's lists.
"""
import math

import numpy as np
import pytest
import torch

import oracle.ultratex_oracle as o
from gpu_util import assert_bf16_close, assert_f32_close, compare_topk_lists, head_lists, need_gpu, to_np
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


def _chain(w, mode, backward):
    """One pass of the whole hot path (compaction, lists, forward, backward,
    scatter) through the benchmark's HotPath on the full-size canvas.  Returns
    the device results, the canvas positions, the compacted inputs (fp32, the
    exact bf16 values) and the block lists the oracle reference uses: the
    bitmap's CSR, or the oracle's own Top-K lists after checking that the
    GPU's lists equal them (rows with an A16 near tie may swap near-tied
    blocks; if any such row exists the reference follows the GPU's lists)."""
    from paper_2609_23169_gb300 import path as P
    mask = w.canvas_mask()
    q, k, v = w.q(), w.k(), w.v()
    do = w.dout() if backward else None
    bm = w.block_bitmap() if mode == "bitmap" else None
    out = P.run_path(w, mask, q, k, v, do, bitmap=bm)
    idx = np.flatnonzero(mask)
    assert out["N"] == len(idx) == w.N
    assert np.array_equal(out["idx"].cpu().numpy(), idx)
    t = torch.from_numpy(idx)
    xs = [x[t].float().numpy() for x in ((q, k, v, do) if backward else (q, k, v))]
    nq = -(-w.N // w.block)
    rp = out["row_ptr"][:w.heads * nq + 1].cpu().numpy()
    ci = out["col_idx"][:int(rp[-1])].cpu().numpy()
    if mode == "bitmap":
        rrp, rci = o.bitmap_to_csr(bm)
        assert np.array_equal(rp, rrp) and np.array_equal(ci, rci)
        n_ties = 0
    else:
        rrp, rci, scores, kr = o.topk_block_mask(xs[0], xs[1], w.block, w.rho)
        n_ties = compare_topk_lists(rp, ci, rrp, rci, scores, kr)
        print(f"{w.name}: Top-K near-tie rows {n_ties} of {w.heads * nq}")
        if n_ties:
            rrp, rci = rp, ci
    return out, idx, xs, rrp, rci


def test_fwd_c2048_sampled():
    """2048 canvas, Top-K rho = 0.12: the lists against the oracle's, then O and
    LSE of a seeded 1% of query rows in every head against the oracle computed
    from the oracle's lists; the scatter put those rows at their positions."""
    w = CONFIGS["c2048"]
    out, idx, (qc, kc, vc), rp, ci = _chain(w, "topk", backward=False)
    rows = w.row_subsample(w.N, 0.01)
    O = out["oc"].float().cpu().numpy()
    L = out["lse"].cpu().numpy()
    got, ref = [], []
    for h in range(w.heads):
        rO, rL = o.bsattn_fwd_rows(qc, kc, vc, rp, ci, w.block, h, rows)
        got.append(O[rows, h])
        ref.append(rO)
        assert np.abs(L[h, rows] - rL).max() < 1e-3
    print(assert_bf16_close(np.concatenate(got), np.concatenate(ref), w.name))
    oc = out["o_canvas"][torch.from_numpy(idx[rows]).cuda()].float().cpu().numpy()
    assert np.array_equal(oc, O[rows])


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


def test_bwd_c512_full():
    """The 512 canvas, all 24 heads, forward and backward in full."""
    w = CONFIGS["c512"]
    idx = torch.from_numpy(np.flatnonzero(w.canvas_mask()))
    q, k, v, do = (x[idx] for x in (w.q(), w.k(), w.v(), w.dout()))
    bm = w.block_bitmap()
    dq, dk, dv = _run_bwd(q, k, v, do, bm, w.block)
    rp, ci = o.bitmap_to_csr(bm)
    rq, rk, rv = o.bsattn_bwd(*(x.double().numpy() for x in (q, k, v, do)), rp, ci, w.block)
    for name, g, r in (("dQ", dq, rq), ("dK", dk, rk), ("dV", dv, rv)):
        print(name, assert_bf16_close(to_np(g), r, name))


def _check_scatter(out, idx, mask, rows):
    """KEEP put O at the canvas positions; ZERO put the gradients there and
    zeros on every background row."""
    at = torch.from_numpy(idx[rows]).cuda()
    assert torch.equal(out["o_canvas"][at], out["oc"][torch.from_numpy(rows).cuda()])
    bg = torch.from_numpy(np.flatnonzero(mask == 0)).cuda()
    for name, comp in (("dq_canvas", "dqc"), ("dk_canvas", "dkc"), ("dv_canvas", "dvc")):
        g = out[name]
        assert torch.equal(g[at], out[comp][torch.from_numpy(rows).cuda()])
        assert torch.all(g[bg] == 0)


def test_fwd_bwd_c1024_full():
    """The whole 1024 canvas (N = 23,959, 24 heads, structured lists, density
    ~0.24) through the benchmark's path: O, LSE, dQ, dK and dV of every row and
    head against the full oracle, element by element."""
    w = CONFIGS["c1024"]
    out, idx, (qc, kc, vc, dc), rp, ci = _chain(w, "bitmap", backward=True)
    rO, rL = o.bsattn_fwd(qc, kc, vc, rp, ci, w.block)
    print("O c1024", assert_bf16_close(to_np(out["oc"]), rO, "O c1024"))
    L = out["lse"].cpu().numpy()
    fin = np.isfinite(rL)
    assert np.array_equal(np.isfinite(L), fin)
    assert np.abs(L[fin] - rL[fin]).max() < 1e-3
    rq, rk, rv = o.bsattn_bwd(qc, kc, vc, dc, rp, ci, w.block)
    for name, comp, r in (("dQ", "dqc", rq), ("dK", "dkc", rk), ("dV", "dvc", rv)):
        print(name, "c1024", assert_bf16_close(to_np(out[comp]), r, name + " c1024"))
    _check_scatter(out, idx, w.canvas_mask(), np.arange(0, w.N, 37))


def test_bwd_c2048():
    """2048 canvas, Top-K rho = 0.12, forward + backward through the
    benchmark's path: dQ of a seeded 0.5% of query rows in every head, and
    dQ, dK, dV of every row of two whole heads (the first and the last, which
    the backward hands out first and last), against the oracle computed from
    the oracle's own lists."""
    w = CONFIGS["c2048"]
    out, idx, (qc, kc, vc, dc), rp, ci = _chain(w, "topk", backward=True)
    nq = -(-w.N // w.block)
    rows = w.row_subsample(w.N, 0.005)
    dq = out["dqc"].float().cpu().numpy()
    dk = out["dkc"].float().cpu().numpy()
    dv = out["dvc"].float().cpu().numpy()
    got, ref = [], []
    for h in range(w.heads):
        got.append(dq[rows, h])
        ref.append(o.bsattn_bwd_dq_rows(qc, kc, vc, dc, rp, ci, w.block, h, rows))
    print("dQ rows c2048", assert_bf16_close(np.concatenate(got), np.concatenate(ref), "dQ rows c2048"))
    for h in (0, w.heads - 1):
        hr, hc = head_lists(rp, ci, h, nq)
        sl = slice(h, h + 1)
        rq, rk, rv = o.bsattn_bwd(qc[:, sl], kc[:, sl], vc[:, sl], dc[:, sl], hr, hc, w.block)
        for name, g, r in (("dQ", dq, rq), ("dK", dk, rk), ("dV", dv, rv)):
            print(name, "c2048 head", h, assert_bf16_close(g[:, sl], r, f"{name} c2048 head {h}"))
    _check_scatter(out, idx, w.canvas_mask(), rows)


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
