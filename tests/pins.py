"""Checks that pin the fp64 oracle to facts outside itself.

Each ``check_*`` function takes the oracle functions it exercises as
arguments and returns a list of failure messages (empty = pinned).  The pin
tests call them with the real oracle; the planted-mistake tests call them
with deliberately broken copies and require a failure, so a plausible slip
anywhere in the oracle (a dropped scale, a wrong sign, a transposed operand,
an off-by-one tile, a reversed tie-break) is shown to be caught.

Independent sources used: hand-worked fixtures under tests/golden/, torch's
CPU scaled_dot_product_attention and autograd in float64, brute-force Python
loops, closed forms and central finite differences.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np
import torch
import torch.nn.functional as F

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _close(a, b, tol=1e-10):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return a.shape == b.shape and bool(np.all(np.abs(a - b) <= tol * (1.0 + np.abs(b))))


# ------------------------------------------------------------ small inputs
def random_case(seed=0, N=13, H=2, d=8, b=4, density=0.5, force_nonempty=True):
    g = np.random.Generator(np.random.PCG64([1234, seed]))
    q = g.standard_normal((N, H, d))
    k = g.standard_normal((N, H, d))
    v = g.standard_normal((N, H, d))
    do = g.standard_normal((N, H, d))
    nq = -(-N // b)
    bm = (g.random((H, nq, nq)) < density).astype(np.uint8)
    if force_nonempty:
        for h in range(H):
            for i in range(nq):
                if not bm[h, i].any():
                    bm[h, i, g.integers(nq)] = 1
    return q, k, v, do, bm


def token_mask(bm: np.ndarray, N: int, b: int) -> np.ndarray:
    """[H, N, N] bool: query token r may see key token c (brute-force expansion)."""
    H = bm.shape[0]
    m = np.zeros((H, N, N), dtype=bool)
    for h in range(H):
        for r in range(N):
            for c in range(N):
                m[h, r, c] = bool(bm[h, r // b, c // b])
    return m


def sdpa_reference(q, k, v, tok_mask, scale, need_grad=False, do=None):
    """torch SDPA in float64 on CPU; heads as the batch dim."""
    Q = torch.tensor(q.transpose(1, 0, 2), dtype=torch.float64, requires_grad=need_grad)
    K = torch.tensor(k.transpose(1, 0, 2), dtype=torch.float64, requires_grad=need_grad)
    V = torch.tensor(v.transpose(1, 0, 2), dtype=torch.float64, requires_grad=need_grad)
    M = None if tok_mask is None else torch.tensor(tok_mask)
    O = F.scaled_dot_product_attention(Q, K, V, attn_mask=M, scale=scale)
    if not need_grad:
        return O.detach().numpy().transpose(1, 0, 2)
    O.backward(torch.tensor(do.transpose(1, 0, 2)))
    return (O.detach().numpy().transpose(1, 0, 2),
            Q.grad.numpy().transpose(1, 0, 2), K.grad.numpy().transpose(1, 0, 2),
            V.grad.numpy().transpose(1, 0, 2))


# ---------------------------------------------------------------- compaction
def check_compaction(fg_compact, fg_scatter, BG_KEEP=0, BG_ZERO=1, BG_FILL=2):
    bad = []
    gd = _load("compaction_hand.json")
    mask = np.array(gd["mask"], np.uint8)
    rows = np.array(gd["rows"], np.float64)
    idx, (xc,) = fg_compact(mask, [rows])
    if list(idx) != gd["idx"]:
        bad.append(f"hand idx {list(idx)} != {gd['idx']}")
    if not _close(xc, gd["compacted"]):
        bad.append("hand compacted rows")
    src = np.array(gd["scatter_src"], np.float64)
    for mode, key in ((BG_KEEP, "scatter_keep"), (BG_ZERO, "scatter_zero"), (BG_FILL, "scatter_fill")):
        y = fg_scatter(np.array(gd["idx"], np.int32), src, rows, mode, np.array(gd["fill_row"], np.float64))
        if not _close(y, gd[key]):
            bad.append(f"hand {key}")
    g = np.random.Generator(np.random.PCG64(7))
    T = 257
    x = g.standard_normal((T, 3, 4))
    # all-foreground: identity
    idx, (xc,) = fg_compact(np.ones(T, np.uint8), [x])
    if not (np.array_equal(idx, np.arange(T)) and np.array_equal(xc, x)):
        bad.append("all-foreground is not the identity")
    # all-background: empty
    idx, (xc,) = fg_compact(np.zeros(T, np.uint8), [x])
    if len(idx) != 0 or xc.shape[0] != 0:
        bad.append("all-background is not empty")
    # random: N = popcount, strictly increasing, rows gathered, scatter o gather
    m = (g.random(T) < 0.37).astype(np.uint8)
    idx, (xc,) = fg_compact(m, [x])
    if len(idx) != int(m.sum()):
        bad.append("N != popcount")
    if len(idx) > 1 and not np.all(np.diff(idx) > 0):
        bad.append("idx not strictly increasing")
    if not all(m[t] for t in idx):
        bad.append("idx holds a background position")
    if not all(np.array_equal(xc[n], x[idx[n]]) for n in range(len(idx))):
        bad.append("compacted row is not the canvas row")
    y0 = g.standard_normal(x.shape)
    y = fg_scatter(idx, xc, y0, BG_KEEP)
    if not (np.array_equal(y[m == 1], x[m == 1]) and np.array_equal(y[m == 0], y0[m == 0])):
        bad.append("scatter o gather is not identity on fg / untouched on bg")
    return bad


# -------------------------------------------------------------- block lists
def check_block_lists(bitmap_to_csr, csr_to_csc):
    bad = []
    g = np.random.Generator(np.random.PCG64(11))
    H, nq, nk = 3, 7, 7
    bm = (g.random((H, nq, nk)) < 0.4).astype(np.uint8)
    bm[1, 2, :] = 0                                   # an empty row
    row_ptr, col_idx = bitmap_to_csr(bm)
    # brute force: Python loops
    rp, ci = [0], []
    for h in range(H):
        for i in range(nq):
            for j in range(nk):
                if bm[h, i, j]:
                    ci.append(j)
            rp.append(len(ci))
    if list(row_ptr) != rp or list(col_idx) != ci:
        bad.append("CSR differs from brute force")
    col_ptr, row_idx = csr_to_csc(row_ptr, col_idx, H, nq, nk)
    cp, ri = [0], []
    for h in range(H):
        for j in range(nk):
            for i in range(nq):
                if bm[h, i, j]:
                    ri.append(i)
            cp.append(len(ri))
    if list(col_ptr) != cp or list(row_idx) != ri:
        bad.append("CSC differs from brute-force transpose")
    return bad


# ------------------------------------------------------------------- Top-K
def check_topk(topk_block_mask, block_pool, k_rho):
    bad = []
    gd = _load("topk_hand.json")
    q = np.array(gd["q"], np.float64)[:, None, :]
    k = np.array(gd["k"], np.float64)[:, None, :]
    b = gd["block"]
    pq = block_pool(q[:, 0], b)
    pk = block_pool(k[:, 0], b)
    if not _close(pq @ pk.T, gd["scores"]):
        bad.append("hand S_c")
    for rho, want in gd["expected"].items():
        rp, ci, _, kr = topk_block_mask(q, k, b, float(rho))
        got = [list(ci[rp[r]:rp[r + 1]]) for r in range(len(rp) - 1)]
        if got != want:
            bad.append(f"hand Top-K rho={rho}: {got} != {want}")
    # brute force on random inputs (Python sort on (-score, j))
    g = np.random.Generator(np.random.PCG64(5))
    N, H, d, b = 45, 2, 6, 4
    q = g.standard_normal((N, H, d))
    k = g.standard_normal((N, H, d))
    nk = -(-N // b)
    for rho in (0.05, 0.2, 0.5, 1.0):
        rp, ci, _, kr = topk_block_mask(q, k, b, rho)
        if kr != max(1, math.floor(rho * nk)):
            bad.append(f"K_rho for rho={rho}")
        for h in range(H):
            means_q = [q[i * b:min(N, i * b + b), h].sum(0) / len(range(i * b, min(N, i * b + b))) for i in range(nk)]
            means_k = [k[j * b:min(N, j * b + b), h].sum(0) / len(range(j * b, min(N, j * b + b))) for j in range(nk)]
            for i in range(nk):
                s = [float(np.dot(means_q[i], means_k[j])) for j in range(nk)]
                want = sorted(sorted(range(nk), key=lambda j: (-s[j], j))[:kr])
                r = h * nk + i
                if list(ci[rp[r]:rp[r + 1]]) != want:
                    bad.append(f"brute-force Top-K rho={rho} h={h} i={i}")
                    break
    # rho = 1 keeps every block; constant scores keep the first K_rho blocks
    rp, ci, _, kr = topk_block_mask(q, k, b, 1.0)
    if kr != nk or not all(list(ci[rp[r]:rp[r + 1]]) == list(range(nk)) for r in range(len(rp) - 1)):
        bad.append("rho = 1 does not keep every block")
    z = np.zeros((N, H, d))
    rp, ci, _, kr = topk_block_mask(z, k, b, 0.3)
    if not all(list(ci[rp[r]:rp[r + 1]]) == list(range(kr)) for r in range(len(rp) - 1)):
        bad.append("all-tied scores do not keep the smallest indices")
    return bad


# ---------------------------------------------------------- attention forward
def check_forward(bsattn_fwd, bitmap_to_csr):
    bad = []
    gd = _load("attention_hand.json")
    q = np.array(gd["q"], np.float64).reshape(-1, 1, 1)
    k = np.array(gd["k"], np.float64).reshape(-1, 1, 1)
    v = np.array(gd["v"], np.float64).reshape(-1, 1, 1)
    b = gd["block"]
    row_ptr = np.array([0] + list(np.cumsum([len(x) for x in gd["lists"]])), np.int32)
    col_idx = np.array(sum(gd["lists"], []), np.int32)
    O, LSE = bsattn_fwd(q, k, v, row_ptr, col_idx, b, gd["scale"])
    if not _close(O[:, 0, 0], gd["o"]):
        bad.append(f"hand O {O[:, 0, 0]} != {gd['o']}")
    if not _close(LSE[0], gd["lse"]):
        bad.append(f"hand LSE {LSE[0]} != {gd['lse']}")

    for seed, (N, H, d, b, dens) in enumerate([(13, 2, 8, 4, 0.5), (32, 1, 16, 8, 0.3), (9, 3, 4, 3, 0.7)]):
        q, k, v, _, bm = random_case(seed, N, H, d, b, dens)
        scale = 1.0 / math.sqrt(d)
        rp, ci = bitmap_to_csr(bm)
        O, LSE = bsattn_fwd(q, k, v, rp, ci, b)
        tm = token_mask(bm, N, b)
        ref = sdpa_reference(q, k, v, tm, scale)
        if not _close(O, ref, 1e-10):
            bad.append(f"masked SDPA mismatch (case {seed})")
        # rows sum to one: sum_k exp(s - LSE) over the visible keys
        for h in range(H):
            s = (q[:, h] @ k[:, h].T) * scale
            tot = np.where(tm[h], np.exp(s - LSE[h][:, None]), 0.0).sum(1)
            if not _close(tot, np.ones(N), 1e-12):
                bad.append(f"softmax rows do not sum to 1 (case {seed})")
                break
        # all-ones mask equals dense attention
        ones = np.ones_like(bm)
        rp1, ci1 = bitmap_to_csr(ones)
        O1, _ = bsattn_fwd(q, k, v, rp1, ci1, b)
        if not _close(O1, sdpa_reference(q, k, v, None, scale), 1e-10):
            bad.append(f"all-ones mask != dense SDPA (case {seed})")
        # constant V rows -> O equals the constant
        cv = np.broadcast_to(np.arange(d, dtype=np.float64), (N, H, d)).copy()
        Oc, _ = bsattn_fwd(q, k, cv, rp, ci, b)
        if not _close(Oc, cv, 1e-12):
            bad.append(f"constant V closed form (case {seed})")
        # identical K rows (or Q = 0) -> mean of the selected V rows
        kk = np.broadcast_to(k[:1], k.shape).copy()
        for qq, kk_, name in ((q, kk, "identical K"), (np.zeros_like(q), k, "Q = 0")):
            Om, _ = bsattn_fwd(qq, kk_, v, rp, ci, b)
            want = np.zeros_like(Om)
            for h in range(H):
                for r in range(N):
                    want[r, h] = v[tm[h, r], h].mean(0)
            if not _close(Om, want, 1e-12):
                bad.append(f"{name} closed form (case {seed})")
    # an empty list: O = 0, LSE = -inf, no NaN
    q, k, v, _, bm = random_case(3, 8, 1, 4, 4, 0.5)
    bm[0, 1, :] = 0
    rp, ci = bitmap_to_csr(bm)
    O, LSE = bsattn_fwd(q, k, v, rp, ci, 4)
    if not (np.all(O[4:8] == 0) and np.all(np.isneginf(LSE[0, 4:8])) and not np.isnan(O).any()):
        bad.append("empty key list is not O = 0, LSE = -inf")
    return bad


# --------------------------------------------------------- attention backward
def check_backward(bsattn_fwd, bsattn_bwd, bitmap_to_csr):
    bad = []
    for seed, (N, H, d, b, dens) in enumerate([(13, 2, 8, 4, 0.5), (10, 1, 4, 5, 0.6)]):
        q, k, v, do, bm = random_case(10 + seed, N, H, d, b, dens)
        scale = 1.0 / math.sqrt(d)
        rp, ci = bitmap_to_csr(bm)
        dQ, dK, dV = bsattn_bwd(q, k, v, do, rp, ci, b)
        _, gq, gk, gv = sdpa_reference(q, k, v, token_mask(bm, N, b), scale, True, do)
        for name, a, r in (("dQ", dQ, gq), ("dK", dK, gk), ("dV", dV, gv)):
            if not _close(a, r, 1e-9):
                bad.append(f"{name} != torch autograd (case {seed})")
        # invariants: sum over keys of dK is 0, sum over keys of dV = sum over queries of dO
        if not _close(dK.sum(0), np.zeros((H, d)), 1e-9):
            bad.append(f"sum of dK over keys is not 0 (case {seed})")
        if not _close(dV.sum(0), do.sum(0), 1e-9):
            bad.append(f"sum of dV over keys != sum of dO (case {seed})")
    # central finite differences of L = <O, dO> against the oracle's own forward
    q, k, v, do, bm = random_case(20, 7, 1, 3, 3, 0.6)
    rp, ci = bitmap_to_csr(bm)
    dQ, dK, dV = bsattn_bwd(q, k, v, do, rp, ci, 3)
    eps = 1e-6

    def loss(qq, kk, vv):
        return float((bsattn_fwd(qq, kk, vv, rp, ci, 3)[0] * do).sum())

    for name, which, grad in (("dQ", 0, dQ), ("dK", 1, dK), ("dV", 2, dV)):
        fd = np.zeros_like(grad)
        for pos in np.ndindex(grad.shape):
            args_p = [q.copy(), k.copy(), v.copy()]
            args_m = [q.copy(), k.copy(), v.copy()]
            args_p[which][pos] += eps
            args_m[which][pos] -= eps
            fd[pos] = (loss(*args_p) - loss(*args_m)) / (2 * eps)
        if not np.allclose(fd, grad, atol=1e-7, rtol=1e-6):
            bad.append(f"{name} != finite differences")
    return bad


def check_subsample_consistency(o, bitmap_to_csr):
    """Row-subset helpers agree with the full oracle functions."""
    bad = []
    q, k, v, do, bm = random_case(30, 21, 2, 4, 4, 0.5)
    rp, ci = bitmap_to_csr(bm)
    O, LSE = o.bsattn_fwd(q, k, v, rp, ci, 4)
    dQ, dK, dV = o.bsattn_bwd(q, k, v, do, rp, ci, 4)
    rows = np.array([0, 3, 4, 9, 20])
    for h in range(2):
        Or, Lr = o.bsattn_fwd_rows(q, k, v, rp, ci, 4, h, rows)
        if not (_close(Or, O[rows, h]) and _close(Lr, LSE[h, rows])):
            bad.append("bsattn_fwd_rows")
        if not _close(o.bsattn_bwd_dq_rows(q, k, v, do, rp, ci, 4, h, rows), dQ[rows, h]):
            bad.append("bsattn_bwd_dq_rows")
        dk, dv = o.bsattn_bwd_dkdv_rows(q, k, v, do, rp, ci, 4, h, rows)
        if not (_close(dk, dK[rows, h]) and _close(dv, dV[rows, h])):
            bad.append("bsattn_bwd_dkdv_rows")
    return bad


# ------------------------------------------------------------ sampler steps
def check_sampler(fg_euler_update, fg_composite, fg_scatter, BG_FILL=2):
    """Pins of the sparse Euler step (Sec. 3.2, Eq. euler) and the composite
    latent (Sec. 3.4, Eq. mixed_latent)."""
    bad = []
    gd = _load("sampler_hand.json")
    z = np.array(gd["z"], np.float64)
    dt = gd["t_prev"] - gd["t_curr"]
    y = fg_euler_update(z, np.array(gd["idx"], np.int32), np.array(gd["v"], np.float64), dt)
    if not _close(y, gd["euler"]):
        bad.append("hand Euler step")
    y = fg_composite(z, np.array(gd["mask"], np.uint8), np.array(gd["tile"], np.float64))
    if not _close(y, gd["composite"]):
        bad.append("hand composite")
    g = np.random.Generator(np.random.PCG64(11))
    T, C = 203, 6
    m = (g.random(T) < 0.45).astype(np.uint8)
    idx = np.nonzero(m)[0].astype(np.int32)
    z = g.standard_normal((T, C))
    v = g.standard_normal((len(idx), C))
    # dt = 0 and v = 0 leave z unchanged
    if not np.array_equal(fg_euler_update(z, idx, v, 0.0), z):
        bad.append("Euler with dt = 0 changed z")
    if not np.array_equal(fg_euler_update(z, idx, np.zeros_like(v), -0.3), z):
        bad.append("Euler with v = 0 changed z")
    # background rows are never updated (bit for bit)
    y = fg_euler_update(z, idx, v, -0.125)
    if not np.array_equal(y[m == 0], z[m == 0]):
        bad.append("Euler touched a background row")
    # a constant velocity field is integrated exactly by Euler: after steps
    # whose sizes sum to t_end - t_start the foreground moved by that times v
    steps = [0.25, 0.125, 0.375, 0.25]                       # t: 1 -> 0 (dyadic sizes)
    y = z.copy()
    for h in steps:
        y = fg_euler_update(y, idx, v, -h)
    if not (np.allclose(y[idx], z[idx] - v, rtol=0, atol=1e-12) and np.array_equal(y[m == 0], z[m == 0])):
        bad.append("Euler does not integrate a constant velocity exactly")
    # composite: all-foreground keeps z, all-background is the tile repeated,
    # foreground rows are bit-exact copies, period 1 equals the FILL scatter
    P = 17
    tile = g.standard_normal((P, C))
    if not np.array_equal(fg_composite(z, np.ones(T, np.uint8), tile), z):
        bad.append("composite with all foreground is not the identity")
    allbg = fg_composite(z, np.zeros(T, np.uint8), tile)
    if not np.array_equal(allbg, np.tile(tile, (-(-T // P), 1))[:T]):
        bad.append("composite with all background is not the repeated tile")
    y = fg_composite(z, m, tile)
    if not np.array_equal(y[m == 1], z[m == 1]):
        bad.append("composite changed a foreground row")
    y1 = fg_composite(z, m, tile[:1])
    yf = fg_scatter(idx, z[idx], z, BG_FILL, tile[0])
    if not np.array_equal(y1, yf):
        bad.append("composite with a one-row tile differs from the FILL scatter")
    return bad


# --------------------------------------------------------------------- RoPE
def check_rope(o):
    """Pins of the rotary embedding at original canvas positions (Sec. 3.2)."""
    bad = []
    gd = _load("rope_hand.json")
    for c in gd["cases"]:
        pos = o.rope_positions(np.array([c["t"]]), c["side"])
        if list(pos[0]) != c["pos"]:
            bad.append(f"hand position of t={c['t']}")
        ang = o.rope_angles(pos, len(c["x"]), tuple(c["axes"]), c["theta"])
        if not _close(ang[0], c["angles"]):
            bad.append(f"hand angles of t={c['t']}")
        y = o.rope_rotate(np.array(c["x"], np.float64)[None, None, :], ang)[0, 0]
        if not _close(y, c["y"]):
            bad.append(f"hand rotation of t={c['t']}")
    g = np.random.Generator(np.random.PCG64(13))
    side, H, d = 8, 3, 128
    T = 5 * side * side
    idx = np.sort(g.choice(T, size=70, replace=False)).astype(np.int32)
    x = g.standard_normal((len(idx), H, d))
    ang = o.rope_angles(o.rope_positions(idx, side), d)
    y = o.rope_rotate(x, ang)
    # a rotation keeps every pair's length; the inverse undoes it
    if not np.allclose(np.hypot(y[..., 0::2], y[..., 1::2]), np.hypot(x[..., 0::2], x[..., 1::2]), atol=1e-12):
        bad.append("rotation changes a pair's length")
    if not np.allclose(o.rope_rotate(y, ang, inverse=True), x, atol=1e-12):
        bad.append("inverse rotation does not undo the rotation")
    # position (0, 0, 0) is the identity
    if not np.array_equal(o.rope_rotate(x[:1], o.rope_angles(np.zeros((1, 3)), d)), x[:1]):
        bad.append("position 0 is not the identity")
    # the same rotation as complex multiplication (x0 + i x1) e^{i phi}
    zc = (x[..., 0::2] + 1j * x[..., 1::2]) * np.exp(1j * ang)[:, None, :]
    if not (np.allclose(y[..., 0::2], zc.real, atol=1e-12) and np.allclose(y[..., 1::2], zc.imag, atol=1e-12)):
        bad.append("rotation differs from the complex-number form")
    # the defining RoPE property: q.k after rotation depends only on the
    # position difference, axis by axis
    q, k = g.standard_normal(d), g.standard_normal(d)
    for shift in ([1, 0, 0], [0, 3, 0], [0, 0, 5], [2, 1, 4]):
        pm, pn = np.array([[1, 2, 3]]), np.array([[4, 6, 1]])
        s_ = np.array([shift])
        dots = []
        for a, b in ((pm, pn), (pm + s_, pn + s_)):
            rq = o.rope_rotate(q[None, None], o.rope_angles(a, d))[0, 0]
            rk = o.rope_rotate(k[None, None], o.rope_angles(b, d))[0, 0]
            dots.append(float(rq @ rk))
        if abs(dots[0] - dots[1]) > 1e-9 * (1 + abs(dots[0])):
            bad.append(f"q.k not shift-invariant for shift {shift}")
    # the gather applies the rotation of each token's own canvas position;
    # the scatter of the gathered rows through the inverse returns the canvas
    xt = g.standard_normal((T, H, d))
    m = np.zeros(T, np.uint8)
    m[idx] = 1
    i2, xr = o.fg_compact_rope(m, xt, side)
    if not (np.array_equal(i2, idx) and np.allclose(xr, o.rope_rotate(xt[idx], ang), atol=1e-12)):
        bad.append("rope gather is not gather + rotation")
    back = o.fg_scatter_rope(idx, xr, np.zeros_like(xt), side, o.BG_ZERO)
    if not (np.allclose(back[idx], xt[idx], atol=1e-12) and not back[m == 0].any()):
        bad.append("rope scatter is not the inverse of the rope gather")
    # a text prefix: its tokens are not rotated, image tokens keep the
    # coordinates they have without the prefix
    pre = 7
    tp = np.concatenate([np.arange(pre), pre + idx]).astype(np.int64)
    pp = o.rope_positions(tp, side, prefix=pre)
    if pp[:pre].any() or not np.array_equal(pp[pre:], o.rope_positions(idx, side)):
        bad.append("text prefix positions")
    return bad


# --------------------------------------------------------- mask from alpha
def check_alpha_mask(token_mask_from_alpha, canvas_mask_from_alpha):
    """Pins of the mask construction (Sec. 3.2)."""
    import scipy.ndimage as ndi
    bad = []
    gd = _load("alpha_mask_hand.json")
    a = np.array(gd["alpha"], np.uint8)
    if token_mask_from_alpha(a, gd["factor"], 0, gd["threshold"]).tolist() != gd["pooled"]:
        bad.append("hand pooled mask")
    if token_mask_from_alpha(a, gd["factor"], gd["radius"], gd["threshold"]).tolist() != gd["dilated"]:
        bad.append("hand dilated mask")
    g = np.random.Generator(np.random.PCG64(17))
    f, H, W = 4, 48, 40
    alpha = (g.random((H, W)) < 0.02).astype(np.uint8) * g.integers(1, 256, size=(H, W), dtype=np.uint8)
    # library routines: block any-pool by reshape, square dilation by scipy
    for thr in (0, 100):
        pooled = (alpha.reshape(H // f, f, W // f, f) > thr).any(axis=(1, 3))
        for r in (0, 1, 2):
            ref = ndi.binary_dilation(pooled, structure=np.ones((2 * r + 1, 2 * r + 1), bool)) if r else pooled
            if not np.array_equal(token_mask_from_alpha(alpha, f, r, thr), ref.astype(np.uint8)):
                bad.append(f"differs from pool + scipy dilation (threshold {thr}, radius {r})")
    # a single lit pixel lights a (2r+1)^2 square of tokens, clipped at the border
    one = np.zeros((H, W), np.uint8)
    one[f * 5 + 1, f * 0 + 2] = 255
    m = token_mask_from_alpha(one, f, 2, 0)
    sq = np.zeros_like(m)
    sq[3:8, 0:3] = 1
    if not np.array_equal(m, sq):
        bad.append("single pixel is not a clipped square")
    # empty and full alpha; monotone in the alpha
    if token_mask_from_alpha(np.zeros((H, W), np.uint8), f, 1, 0).any():
        bad.append("empty alpha gives foreground")
    if not token_mask_from_alpha(np.full((H, W), 255, np.uint8), f, 1, 0).all():
        bad.append("full alpha is not all foreground")
    more = np.maximum(alpha, (g.random((H, W)) < 0.01).astype(np.uint8) * 255)
    if np.any(token_mask_from_alpha(alpha, f, 1, 0) > token_mask_from_alpha(more, f, 1, 0)):
        bad.append("more alpha gives less foreground")
    # canvas: V targets, the same V masks for the conditions, then the reference
    V = 3
    stack = (g.random((V + 1, H, W)) < 0.01).astype(np.uint8) * 255
    cm = canvas_mask_from_alpha(stack, f, 1, 0)
    n_tok = (H // f) * (W // f)
    if cm.size != (2 * V + 1) * n_tok:
        bad.append("canvas mask size")
    else:
        blocks = cm.reshape(2 * V + 1, n_tok)
        for v in range(V):
            mv = token_mask_from_alpha(stack[v], f, 1, 0).ravel()
            if not (np.array_equal(blocks[v], mv) and np.array_equal(blocks[V + v], mv)):
                bad.append(f"view {v}: target / condition masks")
        if not np.array_equal(blocks[2 * V], token_mask_from_alpha(stack[V], f, 1, 0).ravel()):
            bad.append("reference mask")
    return bad


# --------------------------------------------------- unequal block sizes
def check_unequal_blocks(o):
    """Query blocks of b_q rows and key blocks of b_kv rows (Sec. 3.3 defines
    both sizes): Top-K by brute force, forward and backward against masked
    SDPA, FLOPs against the expanded token mask."""
    bad = []
    g = np.random.Generator(np.random.PCG64(29))
    for N, H, d, bq, bk in ((23, 2, 6, 4, 2), (23, 2, 6, 2, 5), (16, 1, 4, 8, 4)):
        q, k, v, do = (g.standard_normal((N, H, d)) for _ in range(4))
        nq, nk = -(-N // bq), -(-N // bk)
        # Top-K over N_k key blocks of b_kv rows
        for rho in (0.2, 0.5):
            rp, ci, _, kr = o.topk_block_mask(q, k, bq, rho, b_kv=bk)
            if kr != max(1, math.floor(rho * nk)) or len(rp) != H * nq + 1:
                bad.append(f"K_rho / list count for b_q={bq}, b_kv={bk}")
                continue
            for h in range(H):
                mq = [q[i * bq:min(N, i * bq + bq), h].mean(0) for i in range(nq)]
                mk = [k[j * bk:min(N, j * bk + bk), h].mean(0) for j in range(nk)]
                for i in range(nq):
                    s = [float(np.dot(mq[i], mk[j])) for j in range(nk)]
                    want = sorted(sorted(range(nk), key=lambda j: (-s[j], j))[:kr])
                    r = h * nq + i
                    if list(ci[rp[r]:rp[r + 1]]) != want:
                        bad.append(f"brute-force Top-K b_q={bq} b_kv={bk} rho={rho}")
                        break
        # forward / backward against SDPA with the token mask bm[h, r // b_q, c // b_kv]
        bm = (g.random((H, nq, nk)) < 0.5).astype(np.uint8)
        for h in range(H):
            for i in range(nq):
                if not bm[h, i].any():
                    bm[h, i, g.integers(nk)] = 1
        rp, ci = o.bitmap_to_csr(bm)
        tm = np.zeros((H, N, N), dtype=bool)
        for h in range(H):
            for r in range(N):
                for c in range(N):
                    tm[h, r, c] = bool(bm[h, r // bq, c // bk])
        scale = 1.0 / math.sqrt(d)
        O, _ = o.bsattn_fwd(q, k, v, rp, ci, bq, b_kv=bk)
        _, gq, gk, gv = sdpa_reference(q, k, v, tm, scale, True, do)
        if not _close(O, sdpa_reference(q, k, v, tm, scale), 1e-10):
            bad.append(f"forward b_q={bq} b_kv={bk} != masked SDPA")
        dQ, dK, dV = o.bsattn_bwd(q, k, v, do, rp, ci, bq, b_kv=bk)
        for name, a, r_ in (("dQ", dQ, gq), ("dK", dK, gk), ("dV", dV, gv)):
            if not _close(a, r_, 1e-9):
                bad.append(f"{name} b_q={bq} b_kv={bk} != autograd")
        if not np.isclose(o.retained_flops_fwd(rp, ci, N, bq, d, b_kv=bk), 4.0 * d * tm.sum()):
            bad.append(f"FLOPs b_q={bq} b_kv={bk}")
    return bad
