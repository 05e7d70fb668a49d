"""GPU parity with 64-row blocks on either side (Sec. 3.3 sizes query blocks
b_q and key blocks b_kv separately): bf16 tensor-core forward and backward
against the fp64 oracle, in full on small problems and the 512 canvas, and on
the 2048 canvas at b = 64 on seeded row samples in every head plus two whole
heads.  The kernels work on 128 x 128 tiles and mask the 64 x 64 sub-blocks a
tile pair does not list."""
import numpy as np
import pytest
import torch

import oracle.ultratex_oracle as o
from gpu_util import assert_bf16_close, compare_topk_lists, head_lists, need_gpu, to_np
from synth import CONFIGS

pytestmark = pytest.mark.gpu

COMBOS = [(64, 64), (128, 64), (64, 128)]


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    need_gpu()


def _lists(q, bq, bk, bitmap):
    from paper_2609_23169_gb300 import ultratex as u
    shape = u.attn_shape(q, bq, bk)
    st = u.status_word()
    out = u.ut_block_mask(shape, u.UT_MASK_BITMAP, bitmap=torch.from_numpy(bitmap).cuda(), status=st,
                          col_cap=max(1, int(bitmap.sum())))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return out


def _bitmap_problem(N, H, d, bq, bk, density, seed, empty=()):
    g = np.random.Generator(np.random.PCG64([91, seed]))
    q, k, v, do = (torch.from_numpy(g.standard_normal((N, H, d)).astype(np.float32)).to(torch.bfloat16)
                   for _ in range(4))
    nq, nk = -(-N // bq), -(-N // bk)
    bm = (g.random((H, nq, nk)) < density).astype(np.uint8)
    for h in range(H):
        for i in range(nq):
            if not bm[h, i].any():
                bm[h, i, g.integers(nk)] = 1
    for (h, i) in empty:
        bm[h, i] = 0
    return q, k, v, do, bm


def _gpu_fwd_bwd(q, k, v, do, lists, bq, bk):
    from paper_2609_23169_gb300 import ultratex as u
    rp, ci, cp, ri = lists
    st = u.status_word()
    qd, kd, vd, dd = (x.cuda() for x in (q, k, v, do))
    O, L = u.ut_bsattn_fwd(qd, kd, vd, rp, ci, bq, status=st, block_k=bk)
    dq, dk, dv = u.ut_bsattn_bwd(qd, kd, vd, O, L, dd, rp, ci, cp, ri, bq, status=st, block_k=bk)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return O, L, dq, dk, dv


@pytest.mark.parametrize("bq,bk", COMBOS)
@pytest.mark.parametrize("N,H,d,dens,seed", [(300, 2, 128, 0.5, 1), (1000, 2, 128, 0.25, 2), (700, 1, 64, 0.4, 3),
                                             (1500, 2, 128, 0.9, 4), (2100, 2, 128, 0.06, 5)])
def test_bitmap_lists_full(bq, bk, N, H, d, dens, seed):
    # dense (0.9) and sparse (0.06) lists take both forms of the 64-row
    # handling (merged tiles, paired blocks); lists of unequal lengths leave
    # one half of some paired tiles empty.
    # one 64-row query block with an empty list: its rows see nothing (O = 0, LSE = -inf)
    empty = [(0, 1)] if bq == 64 else [(0, 0)]
    q, k, v, do, bm = _bitmap_problem(N, H, d, bq, bk, dens, seed, empty)
    lists = _lists(q, bq, bk, bm)
    O, L, dq, dk, dv = _gpu_fwd_bwd(q, k, v, do, lists, bq, bk)
    rp, ci = o.bitmap_to_csr(bm)
    qn, kn, vn, dn = (x.double().numpy() for x in (q, k, v, do))
    rO, rL = o.bsattn_fwd(qn, kn, vn, rp, ci, bq, b_kv=bk)
    assert_bf16_close(to_np(O), rO, "O")
    Lg = L.cpu().numpy()
    fin = np.isfinite(rL)
    assert np.array_equal(np.isfinite(Lg), fin) and np.all(np.isneginf(Lg[~fin]))
    assert np.allclose(Lg[fin], rL[fin], rtol=0, atol=2e-2)
    rq, rk, rv = o.bsattn_bwd(qn, kn, vn, dn, rp, ci, bq, b_kv=bk)
    for name, g, r in (("dQ", dq, rq), ("dK", dk, rk), ("dV", dv, rv)):
        assert_bf16_close(to_np(g), r, name)


@pytest.mark.parametrize("bq,bk", COMBOS)
def test_topk_c512_four_heads_full(bq, bk):
    from paper_2609_23169_gb300 import ultratex as u
    w = CONFIGS["c512"].with_(heads=4)
    idx = torch.from_numpy(np.flatnonzero(w.canvas_mask()))
    q, k, v, do = (x[idx] for x in (w.q(), w.k(), w.v(), w.dout()))
    qd, kd = q.cuda(), k.cuda()
    lists = u.ut_block_mask(u.attn_shape(qd, bq, bk), u.UT_MASK_TOPK, qd, kd, 0.3)
    qn, kn, vn, dn = (x.double().numpy() for x in (q, k, v, do))
    rp, ci, _, _ = o.topk_block_mask(qn, kn, bq, 0.3, b_kv=bk)
    assert np.array_equal(lists[0].cpu().numpy()[:len(rp)], rp)
    assert np.array_equal(lists[1].cpu().numpy()[:len(ci)], ci)
    O, L, dq, dk, dv = _gpu_fwd_bwd(q, k, v, do, lists, bq, bk)
    rO, _ = o.bsattn_fwd(qn, kn, vn, rp, ci, bq, b_kv=bk)
    assert_bf16_close(to_np(O), rO, "O")
    rq, rk, rv = o.bsattn_bwd(qn, kn, vn, dn, rp, ci, bq, b_kv=bk)
    for name, g, r in (("dQ", dq, rq), ("dK", dk, rk), ("dV", dv, rv)):
        assert_bf16_close(to_np(g), r, name)


def test_c2048_block64():
    """The 2048 canvas at b_q = b_kv = 64 (the sweep's small block), 24 heads,
    Top-K rho = 0.12: the GPU lists against the oracle's own, then sampled
    forward and dQ rows in every head and dQ, dK, dV of every row of two whole
    heads, against the oracle computed from the oracle's lists."""
    from paper_2609_23169_gb300 import ultratex as u
    w = CONFIGS["c2048"]
    mask = w.canvas_mask()
    idx = np.flatnonzero(mask)
    t = torch.from_numpy(idx)
    q, k, v, do = (x[t] for x in (w.q(), w.k(), w.v(), w.dout()))
    qd, kd = q.cuda(), k.cuda()
    lists = u.ut_block_mask(u.attn_shape(qd, 64, 64), u.UT_MASK_TOPK, qd, kd, w.rho)
    O, L, dq, dk, dv = _gpu_fwd_bwd(q, k, v, do, lists, 64, 64)
    N = len(idx)
    nq = -(-N // 64)
    rp = lists[0][:w.heads * nq + 1].cpu().numpy()
    ci = lists[1][:int(rp[-1])].cpu().numpy()
    qn, kn, vn, dn = (x.float().numpy() for x in (q, k, v, do))
    rrp, rci, scores, kr = o.topk_block_mask(qn, kn, 64, w.rho)
    n_ties = compare_topk_lists(rp, ci, rrp, rci, scores, kr)
    print(f"c2048 b64: Top-K near-tie rows {n_ties} of {w.heads * nq}")
    if n_ties == 0:
        rp, ci = rrp, rci
    rows = w.row_subsample(N, 0.003)
    Og, dqg = O.float().cpu().numpy(), dq.float().cpu().numpy()
    go, ro, gq, rq = [], [], [], []
    for h in range(w.heads):
        go.append(Og[rows, h])
        ro.append(o.bsattn_fwd_rows(qn, kn, vn, rp, ci, 64, h, rows)[0])
        gq.append(dqg[rows, h])
        rq.append(o.bsattn_bwd_dq_rows(qn, kn, vn, dn, rp, ci, 64, h, rows))
    print(assert_bf16_close(np.concatenate(go), np.concatenate(ro), "O c2048 b64"))
    print(assert_bf16_close(np.concatenate(gq), np.concatenate(rq), "dQ c2048 b64"))
    dkg, dvg = dk.float().cpu().numpy(), dv.float().cpu().numpy()
    for h in (0, w.heads - 1):
        hr, hc = head_lists(rp, ci, h, nq)
        sl = slice(h, h + 1)
        a, b, c = o.bsattn_bwd(qn[:, sl], kn[:, sl], vn[:, sl], dn[:, sl], hr, hc, 64)
        for name, g, r in (("dQ", dqg, a), ("dK", dkg, b), ("dV", dvg, c)):
            print(name, "c2048 b64 head", h, assert_bf16_close(g[:, sl], r, f"{name} c2048 b64 head {h}"))
