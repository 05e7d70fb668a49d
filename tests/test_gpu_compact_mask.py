"""GPU parity: compaction, scatter and block lists are bit-exact against the oracle."""
import numpy as np
import pytest
import torch

import oracle.ultratex_oracle as o
from gpu_util import bits, compare_topk_lists, need_gpu
from synth import CONFIGS

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    need_gpu()


def _compact_check(mask, tensors, capacity=None):
    from paper_2609_23169_gb300 import ultratex as u
    dev = torch.device("cuda")
    st = u.status_word()
    m = torch.from_numpy(mask).to(dev)
    ts = [t.to(dev) for t in tensors]
    idx, n_out, outs = u.ut_fg_compact(m, ts, capacity=capacity, status=st)
    torch.cuda.synchronize()
    ref_idx, ref_rows = o.fg_compact(mask, [bits(t) for t in tensors])
    N = int(n_out.item())
    assert N == len(ref_idx)
    cap = len(mask) if capacity is None else capacity
    n_w = min(N, cap)
    assert np.array_equal(idx[:n_w].cpu().numpy(), ref_idx[:n_w])
    for out, ref in zip(outs, ref_rows):
        assert np.array_equal(bits(out[:n_w]), ref[:n_w])
    return int(st.item()), idx, N, ts


@pytest.mark.parametrize("name", ["tiny", "c512", "c1024"])
def test_compaction_configs(name):
    w = CONFIGS[name]
    if w.heads > 4:
        w = w.with_(heads=4)
    st, _, N, _ = _compact_check(w.canvas_mask(), [w.q(), w.k(), w.v()])
    assert st == 0 and N == w.N


def test_compaction_full_2048_canvas():
    w = CONFIGS["c2048"]
    mask = w.canvas_mask()
    g = np.random.Generator(np.random.PCG64(3))
    x = torch.from_numpy(g.integers(-30000, 30000, size=(w.T, 24 * 128), dtype=np.int16)).view(torch.bfloat16)
    st, _, N, _ = _compact_check(mask, [x])
    assert st == 0 and N == 85202


@pytest.mark.parametrize("T,frac,row", [(1, 1.0, 16), (37, 0.5, 48), (4096 * 3 + 37, 0.3, 256), (5000, 0.0, 32),
                                        (9000, 1.0, 32), (70001, 0.9, 16)])
def test_compaction_ragged_and_degenerate(T, frac, row):
    g = np.random.Generator(np.random.PCG64(T))
    mask = (g.random(T) < frac).astype(np.uint8)
    if frac == 1.0:
        mask[:] = 1
    mask = mask * g.integers(1, 255, size=T).astype(np.uint8)   # any nonzero byte is foreground
    x = torch.from_numpy(g.integers(-2 ** 31, 2 ** 31 - 1, size=(T, row // 4), dtype=np.int32)).view(torch.float32)
    st, _, N, _ = _compact_check(mask, [x])
    assert st == 0 and N == int((mask != 0).sum())


def test_device_accessible_query():
    from paper_2609_23169_gb300 import ultratex as u
    assert u.device_accessible(torch.zeros(4, device="cuda"))
    assert u.device_accessible(torch.zeros(4).pin_memory())


@pytest.mark.parametrize("T,frac", [(37, 0.5), (70001, 0.3), (5000, 0.0)])
def test_compaction_count_in_pinned_host_memory(T, frac):
    """N written straight into pinned host memory matches the device count and
    the oracle; the gather that reads N back from there copies the same rows."""
    from paper_2609_23169_gb300 import ultratex as u
    g = np.random.Generator(np.random.PCG64([5, T]))
    mask = (g.random(T) < frac).astype(np.uint8)
    x = torch.from_numpy(g.integers(-2 ** 31, 2 ** 31 - 1, size=(T, 8), dtype=np.int32)).view(torch.float32)
    m, xd = torch.from_numpy(mask).cuda(), x.cuda()
    n_host = torch.full((1,), -1, dtype=torch.int32).pin_memory()
    assert u.device_accessible(n_host)
    st = u.status_word()
    idx, _, (out,) = u.ut_fg_compact(m, [xd], n_out=n_host, status=st)
    done = torch.cuda.Event()
    done.record()
    done.synchronize()
    ref_idx, (ref_rows,) = o.fg_compact(mask, [bits(x)])
    assert int(n_host[0]) == len(ref_idx) and int(st.item()) == 0
    assert np.array_equal(idx[:len(ref_idx)].cpu().numpy(), ref_idx)
    assert np.array_equal(bits(out[:len(ref_idx)]), ref_rows)


def test_compaction_capacity_overflow_reports_status():
    from paper_2609_23169_gb300 import ultratex as u
    g = np.random.Generator(np.random.PCG64(9))
    mask = (g.random(10000) < 0.5).astype(np.uint8)
    x = torch.from_numpy(g.standard_normal((10000, 8)).astype(np.float32))
    st, _, N, _ = _compact_check(mask, [x], capacity=1000)
    assert st == u.UT_ERR_CAPACITY and N == int(mask.sum())


@pytest.mark.parametrize("mode", ["keep", "zero", "fill"])
def test_scatter_modes(mode):
    from paper_2609_23169_gb300 import ultratex as u
    w = CONFIGS["c512"].with_(heads=2)
    mask = w.canvas_mask()
    dev = torch.device("cuda")
    idx_np = np.flatnonzero(mask).astype(np.int32)
    N = len(idx_np)
    g = np.random.Generator(np.random.PCG64(4))
    src = torch.from_numpy(g.integers(-30000, 30000, size=(N, 2, 128), dtype=np.int16)).view(torch.bfloat16)
    base = torch.from_numpy(g.integers(-30000, 30000, size=(w.T, 2, 128), dtype=np.int16)).view(torch.bfloat16)
    fill = torch.from_numpy(g.integers(-30000, 30000, size=(2, 128), dtype=np.int16)).view(torch.bfloat16)
    dst = base.clone().to(dev)
    code = dict(keep=u.UT_BG_KEEP, zero=u.UT_BG_ZERO, fill=u.UT_BG_FILL)[mode]
    u.ut_fg_scatter(torch.from_numpy(idx_np).to(dev), N, [src.to(dev)], [dst], code, fill.to(dev))
    torch.cuda.synchronize()
    ref = o.fg_scatter(idx_np, bits(src), bits(base), code, bits(fill))
    assert np.array_equal(bits(dst), ref)


def test_scatter_inverts_compaction_on_foreground():
    from paper_2609_23169_gb300 import ultratex as u
    w = CONFIGS["tiny"]
    mask = w.canvas_mask()
    q = w.q()
    st, idx, N, ts = _compact_check(mask, [q])
    _, _, outs = u.ut_fg_compact(torch.from_numpy(mask).cuda(), ts)
    y = torch.zeros_like(ts[0])
    u.ut_fg_scatter(idx, N, [outs[0][:N]], [y], u.UT_BG_KEEP)
    torch.cuda.synchronize()
    m = torch.from_numpy(mask.astype(bool)).cuda()
    assert torch.equal(y[m], ts[0][m]) and torch.all(y[~m] == 0)


# --------------------------------------------------------------- block lists
def _bitmap_lists(bm, H, N, b):
    from paper_2609_23169_gb300 import ultratex as u
    shape = u.AttnShape(N, H, 64, b, u.UT_F32, H * 64)
    st = u.status_word()
    rp, ci, cp, ri = u.ut_block_mask(shape, u.UT_MASK_BITMAP, bitmap=torch.from_numpy(bm).cuda(), status=st,
                                     col_cap=int((bm != 0).sum()))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return [x.cpu().numpy() for x in (rp, ci, cp, ri)]


@pytest.mark.parametrize("name", ["tiny", "c512", "c1024"])
def test_bitmap_lists_exact(name):
    w = CONFIGS[name]
    bm = w.block_bitmap()
    H, nq, _ = bm.shape
    rp, ci, cp, ri = _bitmap_lists(bm, H, w.N, w.block)
    rrp, rci = o.bitmap_to_csr(bm)
    rcp, rri = o.csr_to_csc(rrp, rci, H, nq, nq)
    assert np.array_equal(rp, rrp) and np.array_equal(ci[:len(rci)], rci)
    assert np.array_equal(cp, rcp) and np.array_equal(ri[:len(rri)], rri)


def test_bitmap_lists_with_empty_rows_and_overflow():
    from paper_2609_23169_gb300 import ultratex as u
    g = np.random.Generator(np.random.PCG64(12))
    H, nq = 3, 37
    bm = (g.random((H, nq, nq)) < 0.3).astype(np.uint8)
    bm[1, 5] = 0
    bm[2, :, 7] = 0
    rp, ci, cp, ri = _bitmap_lists(bm, H, nq * 64 - 5, 64)
    rrp, rci = o.bitmap_to_csr(bm)
    rcp, rri = o.csr_to_csc(rrp, rci, H, nq, nq)
    assert np.array_equal(rp, rrp) and np.array_equal(ci[:len(rci)], rci)
    assert np.array_equal(cp, rcp) and np.array_equal(ri[:len(rri)], rri)
    # too small a capacity is reported on the device
    shape = u.AttnShape(nq * 64, H, 64, 64, u.UT_F32, H * 64)
    st = u.status_word()
    u.ut_block_mask(shape, u.UT_MASK_BITMAP, bitmap=torch.from_numpy(bm).cuda(), status=st, col_cap=10)
    torch.cuda.synchronize()
    assert int(st.item()) == u.UT_ERR_CAPACITY


def _topk_gpu(qc: torch.Tensor, kc: torch.Tensor, b: int, rho: float):
    from paper_2609_23169_gb300 import ultratex as u
    shape = u.attn_shape(qc, b)
    rp, ci, cp, ri = u.ut_block_mask(shape, u.UT_MASK_TOPK, qc.cuda(), kc.cuda(), rho)
    torch.cuda.synchronize()
    return [x.cpu().numpy() for x in (rp, ci, cp, ri)]


def _check_topk(qc_np, kc_np, rp, ci, cp, ri, b, rho, allow_near_ties=False):
    """Exact list match; with allow_near_ties, rows whose K-th/(K+1)-th oracle
    scores are within 1e-4*max|s| may differ, but only by swapping near-tied blocks."""
    rrp, rci, scores, kr = o.topk_block_mask(qc_np, kc_np, b, rho)
    H, nq, _ = scores.shape
    n_tie_rows = compare_topk_lists(rp, ci, rrp, rci, scores, kr)
    assert allow_near_ties or n_tie_rows == 0
    rcp, rri = o.csr_to_csc(rp, ci, H, nq, nq)   # transpose of the GPU's own lists
    assert np.array_equal(cp, rcp) and np.array_equal(ri[:len(rri)], rri)
    return n_tie_rows


def test_topk_hand_fixture(golden_dir):
    import json, os
    with open(os.path.join(golden_dir, "topk_hand.json")) as f:
        gd = json.load(f)
    q = np.zeros((7, 1, 64), np.float32)
    k = np.zeros((7, 1, 64), np.float32)
    q[:, 0, :2] = gd["q"]
    k[:, 0, :2] = gd["k"]
    for rho, want in gd["expected"].items():
        rp, ci, cp, ri = _topk_gpu(torch.from_numpy(q), torch.from_numpy(k), gd["block"], float(rho))
        got = [list(ci[rp[r]:rp[r + 1]]) for r in range(4)]
        assert got == want, (rho, got)


@pytest.mark.parametrize("N,H,d,b,rho", [(1000, 3, 64, 64, 0.2), (4000, 2, 128, 128, 0.12), (777, 4, 128, 32, 0.5),
                                         (300, 1, 64, 128, 1.0)])
def test_topk_random_exact(N, H, d, b, rho):
    g = np.random.Generator(np.random.PCG64(N))
    q = g.standard_normal((N, H, d)).astype(np.float32)
    k = g.standard_normal((N, H, d)).astype(np.float32)
    qb = torch.from_numpy(q).to(torch.bfloat16)
    kb = torch.from_numpy(k).to(torch.bfloat16)
    rp, ci, cp, ri = _topk_gpu(qb, kb, b, rho)
    _check_topk(qb.double().numpy(), kb.double().numpy(), rp, ci, cp, ri, b, rho, allow_near_ties=True)


def test_topk_full_2048():
    w = CONFIGS["c2048"]
    mask = w.canvas_mask()
    idx = np.flatnonzero(mask)
    qc = w.q()[torch.from_numpy(idx)]
    kc = w.k()[torch.from_numpy(idx)]
    rp, ci, cp, ri = _topk_gpu(qc, kc, w.block, w.rho)
    assert rp[-1] == 24 * 666 * 79
    n_ties = _check_topk(qc.double().numpy(), kc.double().numpy(), rp, ci, cp, ri, w.block, w.rho,
                         allow_near_ties=True)
    print(f"near-tie rows at 2048: {n_ties} of {24 * 666}")
