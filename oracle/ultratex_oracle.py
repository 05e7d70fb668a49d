"""fp64 CPU oracle for UltraTex's foreground-only block-sparse attention path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports, calls or
executes this module: only the tests, ``__graft_entry__.smoke()`` and the CPU
baseline legs of ``bench.py`` use it.  It shares no code with the CUDA path.

Every function is the plain definition from the paper, in float64 numpy, with
no blocking, fusion or reordering beyond what the definition states:

* Background Token Dropping (Sec. 3.2): ``z~ = Gather_{M_fg}(z)``; each
  retained token keeps its canvas position (its RoPE index).
* Block partition (Sec. 3.3): Q into query blocks of b_q rows, K/V into key
  blocks of b_kv rows (the functions take b = b_q and an optional b_kv,
  equal to b when not given).
* Compressed scores and Top-K (Sec. 3.3, the equation for S_c and the one
  for M_c): ``S_c = pool(Q) pool(K)^T`` with mean pooling per block, and per
  head and query block the K_rho = floor(rho * N_k) key blocks of largest score.
* Block-sparse attention (Sec. 3.3, the equation for O_i):
  ``O_i = softmax(Q_i K_{S_i}^T / sqrt(d)) V_{S_i}``.
* Its gradient (implied by that equation; the paper trains stage 3 with it,
  Sec. 4.1): the standard softmax-attention backward.
* Scatter back to canvas positions: background rows are "not updated"
  (Sec. 3.2, "Efficient Inference"); ``z_mix`` places foreground latents at
  their positions and a fill elsewhere (Sec. 3.4, the z_mix equation).
* Mask construction (Sec. 3.2): a token is foreground when any alpha pixel of
  its factor x factor block exceeds the threshold (the 1/16 downsampling of
  the alpha channel), then the token mask is dilated by a square of radius r
  (the slight dilation); the six view masks serve both the noisy targets and
  the conditions, the reference image has its own.
* Rotary position embedding at the retained tokens' original canvas positions
  (Sec. 3.2: each retained token carries its original RoPE index).  The paper
  does not print the formula; the reading used: canvas position t of images of
  side S maps to (image, y, x) = (t // S^2, (t mod S^2) // S, t mod S); the
  head dimension is split into three axes (default 16/56/56 of 128); within
  axis a of d_a dimensions, pair k = (x[2k], x[2k+1]) is rotated by the angle
  pos_a * theta^(-2k/d_a) (theta = 10000).  Gathering Q and K applies the
  rotation; scattering their gradients back applies its inverse.  Text tokens
  placed before the images (the joint sequence's 512-token prefix of Table
  S1) sit at position (0, 0, 0).
* Sampler steps on the canvas latent: the sparse Euler update (Sec. 3.2,
  Eq. euler) moves only the retained positions by (t_prev - t_curr) times
  their predicted velocity; the composite latent (Sec. 3.4, Eq. mixed_latent)
  keeps the denoised foreground and takes the canonical background latent,
  tile-repeated over the canvas, everywhere else.

Readings where the paper is silent (listed with the design notes):
* tiles are ceil-sized; the last tile may be partial (N is rarely a multiple of b);
* pooling over a partial tile averages its valid rows only;
* S_c carries no 1/sqrt(d) and no softmax (ranking is unaffected);
* K_rho = max(1, floor(rho * N_k)) evaluated in float64; equal scores are
  broken toward the smaller key-block index;
* a query block with an empty key-block list gets O = 0 and LSE = -inf.

Parity status: every function here is pinned by the ``-m "not gpu"`` tests in
tests/test_oracle_pins.py (brute force, closed forms, library routines,
finite differences and hand-worked fixtures).  The choice of blocks on real
model activations cannot be pinned (no weights, no printed example); only
the rule is.
"""
from __future__ import annotations

import math
from typing import Optional, Sequence

import numpy as np

BG_KEEP, BG_ZERO, BG_FILL = 0, 1, 2


# ---------------------------------------------------------------- compaction
def fg_compact(mask: np.ndarray, xs: Sequence[np.ndarray]):
    """Background Token Dropping (Sec. 3.2): Gather_{M_fg}.

    ``mask``: [T] of 0/1.  Returns (idx, [X[idx] for X in xs]) where idx is the
    ascending list of retained canvas positions (int32), i.e. the RoPE indices
    the retained tokens carry.
    """
    mask = np.asarray(mask)
    idx = np.flatnonzero(mask != 0).astype(np.int32)
    return idx, [np.asarray(x)[idx] for x in xs]


def fg_scatter(idx: np.ndarray, src: np.ndarray, dst_in: np.ndarray,
               mode: int = BG_KEEP, fill_row: Optional[np.ndarray] = None) -> np.ndarray:
    """Scatter compacted rows back to canvas positions (Sec. 3.2 / Sec. 3.4).

    KEEP: background rows of ``dst_in`` are not updated.  ZERO: they become 0
    (the adjoint of the gather).  FILL: they become ``fill_row`` (z_bg).
    """
    y = np.array(dst_in, copy=True)
    if mode == BG_ZERO:
        y[...] = 0
    elif mode == BG_FILL:
        y[...] = np.asarray(fill_row).reshape(y.shape[1:])
    y[np.asarray(idx, dtype=np.int64)] = src
    return y


# ----------------------------------------------------------- mask from alpha
def token_mask_from_alpha(alpha: np.ndarray, factor: int = 16, radius: int = 1, threshold: int = 0) -> np.ndarray:
    """One image's token mask (Sec. 3.2): [H_px, W_px] alpha -> [H_px/factor, W_px/factor] uint8.

    Token (y, x) is foreground before dilation when some pixel of its block
    alpha[y*f:(y+1)*f, x*f:(x+1)*f] exceeds ``threshold``; after dilation when
    some token within Chebyshev distance ``radius`` (inside the image) is.
    """
    a = np.asarray(alpha)
    h, w = a.shape[0] // factor, a.shape[1] // factor
    pooled = np.zeros((h, w), dtype=bool)
    for y in range(h):
        for x in range(w):
            pooled[y, x] = bool((a[y * factor:(y + 1) * factor, x * factor:(x + 1) * factor] > threshold).any())
    out = np.zeros((h, w), dtype=bool)
    for y in range(h):
        for x in range(w):
            out[y, x] = pooled[max(0, y - radius):y + radius + 1, max(0, x - radius):x + radius + 1].any()
    return out.astype(np.uint8)


def canvas_mask_from_alpha(alpha: np.ndarray, factor: int = 16, radius: int = 1, threshold: int = 0) -> np.ndarray:
    """Canvas mask of the multi-view sequence (Sec. 3.2): alpha [V + 1, H_px, W_px]
    (V view renders, then the reference) -> [(2V + 1) * h * w] uint8 laid out as
    the V target images, the V condition images (view v's mask again) and the
    reference image, raster order inside each."""
    a = np.asarray(alpha)
    V = a.shape[0] - 1
    views = [token_mask_from_alpha(a[v], factor, radius, threshold).ravel() for v in range(V)]
    ref = token_mask_from_alpha(a[V], factor, radius, threshold).ravel()
    return np.concatenate(views + views + [ref]).astype(np.uint8)


# --------------------------------------------------------------------- RoPE
def rope_positions(idx: np.ndarray, side: int, prefix: int = 0) -> np.ndarray:
    """Canvas positions -> (image, y, x) of images of side x side tokens, stored
    one after another in raster order.  [n] -> [n, 3] int64.

    With a text prefix (the joint sequence of the MM-DiT carries its text
    tokens before the images), positions t < prefix are text tokens at
    (0, 0, 0) and image coordinates count from t - prefix."""
    t = np.asarray(idx, dtype=np.int64)
    s2 = int(side) * int(side)
    ti = t - int(prefix)
    pos = np.stack([ti // s2, (ti % s2) // side, ti % side], axis=1)
    pos[t < int(prefix)] = 0
    return pos


def rope_angles(pos: np.ndarray, head_dim: int, axes=(16, 56, 56), theta: float = 10000.0) -> np.ndarray:
    """Rotation angle of every pair: [n, 3] positions -> [n, head_dim // 2].

    Pairs are taken axis by axis: the first axes[0] / 2 pairs use the image
    index, the next axes[1] / 2 the row y, the last axes[2] / 2 the column x;
    pair k of axis a (d_a = axes[a] dimensions) turns by pos_a * theta^(-2k/d_a).
    """
    assert sum(axes) == head_dim and all(a % 2 == 0 for a in axes)
    pos = np.asarray(pos, dtype=np.float64)
    cols = []
    for a, d_a in enumerate(axes):
        k = np.arange(d_a // 2, dtype=np.float64)
        freq = float(theta) ** (-2.0 * k / d_a)
        cols.append(pos[:, a:a + 1] * freq[None, :])
    return np.concatenate(cols, axis=1)


def rope_rotate(x: np.ndarray, angles: np.ndarray, inverse: bool = False) -> np.ndarray:
    """Rotate each consecutive pair (x[..., 2k], x[..., 2k+1]) of every row by
    angles[row, k] (by -angles[row, k] if ``inverse``).  x: [n, H, d]."""
    x = np.asarray(x, dtype=np.float64)
    a = -angles if inverse else angles
    c = np.cos(a)[:, None, :]
    s = np.sin(a)[:, None, :]
    x0, x1 = x[..., 0::2], x[..., 1::2]
    y = np.empty_like(x)
    y[..., 0::2] = x0 * c - x1 * s
    y[..., 1::2] = x0 * s + x1 * c
    return y


def fg_compact_rope(mask: np.ndarray, x: np.ndarray, side: int, axes=(16, 56, 56), theta: float = 10000.0,
                    prefix: int = 0):
    """Gather of Q or K (Sec. 3.2) with the rotary embedding of each retained
    token's original canvas position applied.  Returns (idx, rotated rows)."""
    idx, (xc,) = fg_compact(mask, [x])
    ang = rope_angles(rope_positions(idx, side, prefix), np.asarray(x).shape[-1], axes, theta)
    return idx, rope_rotate(xc, ang)


def fg_scatter_rope(idx: np.ndarray, src: np.ndarray, dst_in: np.ndarray, side: int, mode: int = BG_ZERO,
                    axes=(16, 56, 56), theta: float = 10000.0, prefix: int = 0) -> np.ndarray:
    """Scatter of dQ or dK back to the canvas through the inverse rotation (the
    gradient of the rotated gather); background rows per ``mode``."""
    ang = rope_angles(rope_positions(idx, side, prefix), np.asarray(src).shape[-1], axes, theta)
    return fg_scatter(idx, rope_rotate(src, ang, inverse=True), dst_in, mode)


# ----------------------------------------------------------- sampler steps
def fg_euler_update(z: np.ndarray, idx: np.ndarray, v: np.ndarray, dt: float) -> np.ndarray:
    """Sparse Euler step (Sec. 3.2, Eq. euler), in float64.

    ``z``: canvas latent [T, ...]; ``idx``: the retained positions M_fg
    (distinct); ``v``: predicted velocities of the retained tokens, row n for
    position idx[n]; ``dt`` = t_prev - t_curr.  z_i <- z_i + dt * v_i for
    i in M_fg; every other row keeps its value (the background stays at its
    initial noise).
    """
    y = np.array(z, dtype=np.float64, copy=True)
    ii = np.asarray(idx, dtype=np.int64)
    y[ii] = y[ii] + float(dt) * np.asarray(v, dtype=np.float64)[: len(ii)]
    return y


def fg_composite(z: np.ndarray, mask: np.ndarray, z_bg_tile: np.ndarray) -> np.ndarray:
    """Composite latent z_mix (Sec. 3.4, Eq. mixed_latent).

    Foreground rows (mask = 1) keep the denoised latent; background row t takes
    the canonical background latent tile-repeated over the canvas,
    ``z_bg_tile[t mod P]`` with P = len(z_bg_tile) rows per tile (one image's
    latent when P = side^2 and the images are stored one after another).
    """
    y = np.array(z, copy=True)
    tile = np.asarray(z_bg_tile)
    P = tile.shape[0]
    for t in range(y.shape[0]):
        if not mask[t]:
            y[t] = tile[t % P]
    return y


# -------------------------------------------------------------------- tiles
def n_blocks(n: int, b: int) -> int:
    return -(-int(n) // int(b))


def tile_rows(i: int, n: int, b: int) -> np.ndarray:
    """Rows of block i: [i*b, min((i+1)*b, n))."""
    return np.arange(i * b, min((i + 1) * b, n))


# ------------------------------------------------------------- block lists
def bitmap_to_csr(bitmap: np.ndarray):
    """Block mask M_c -> per-query-block key lists S_i = {j | M_c[i,j] = 1}.

    ``bitmap``: [H, N_q, N_k].  Rows are (h, i) in head-major order; each list
    ascending.  Returns (row_ptr [H*N_q+1] int32, col_idx int32).
    """
    bm = np.asarray(bitmap)
    H, nq, nk = bm.shape
    lists = [np.flatnonzero(bm[h, i]) for h in range(H) for i in range(nq)]
    row_ptr = np.zeros(H * nq + 1, dtype=np.int64)
    row_ptr[1:] = np.cumsum([len(x) for x in lists])
    col_idx = np.concatenate(lists) if lists else np.zeros(0, np.int64)
    return row_ptr.astype(np.int32), col_idx.astype(np.int32)


def csr_to_bitmap(row_ptr: np.ndarray, col_idx: np.ndarray, H: int, nq: int, nk: int) -> np.ndarray:
    bm = np.zeros((H, nq, nk), dtype=np.uint8)
    for r in range(H * nq):
        h, i = divmod(r, nq)
        bm[h, i, col_idx[row_ptr[r]:row_ptr[r + 1]]] = 1
    return bm


def csr_to_csc(row_ptr: np.ndarray, col_idx: np.ndarray, H: int, nq: int, nk: int):
    """Transpose of the block lists: per (h, j) the ascending query blocks i with j in S_i."""
    bm = csr_to_bitmap(row_ptr, col_idx, H, nq, nk)
    return bitmap_to_csr(np.ascontiguousarray(bm.transpose(0, 2, 1)))


# ------------------------------------------------------- pooled Top-K mask
def block_pool(x: np.ndarray, b: int) -> np.ndarray:
    """pool(.) of Sec. 3.3: mean over the (valid) tokens of each block. x: [N, d]."""
    x = np.asarray(x, dtype=np.float64)
    n = x.shape[0]
    return np.stack([x[tile_rows(i, n, b)].mean(axis=0) for i in range(n_blocks(n, b))]) \
        if n else np.zeros((0, x.shape[1]))


def k_rho(rho: float, nk: int) -> int:
    """K_rho = floor(rho * N_k) (Sec. 3.3), at least one block."""
    return max(1, int(math.floor(float(rho) * int(nk))))


def compressed_scores(qc_h: np.ndarray, kc_h: np.ndarray, b: int, b_kv: Optional[int] = None) -> np.ndarray:
    """S_c = pool(Q) pool(K)^T for one head (Sec. 3.3); Q pooled over b_q = b rows,
    K over b_kv rows (b_kv = b when not given)."""
    return block_pool(qc_h, b) @ block_pool(kc_h, b if b_kv is None else b_kv).T


def topk_block_mask(qc: np.ndarray, kc: np.ndarray, b: int, rho: float, b_kv: Optional[int] = None):
    """Per head and query block, the K_rho key blocks with the largest S_c (Sec. 3.3).

    qc, kc: [N, H, d]; query blocks of b rows, key blocks of b_kv rows (b when
    not given), K_rho = max(1, floor(rho N_k)).  Returns (row_ptr, col_idx,
    scores [H, N_q, N_k], K_rho); lists ascending, ties toward the smaller
    key-block index.
    """
    N, H, _ = qc.shape
    bk = b if b_kv is None else b_kv
    nq, nk = n_blocks(N, b), n_blocks(N, bk)
    kr = k_rho(rho, nk)
    scores = np.zeros((H, nq, nk))
    lists = []
    for h in range(H):
        sc = compressed_scores(qc[:, h], kc[:, h], b, bk)
        scores[h] = sc
        for i in range(nq):
            order = np.lexsort((np.arange(nk), -sc[i]))   # score desc, index asc
            lists.append(np.sort(order[:kr]))
    row_ptr = np.arange(H * nq + 1, dtype=np.int64) * kr
    col_idx = np.concatenate(lists) if lists else np.zeros(0, np.int64)
    return row_ptr.astype(np.int32), col_idx.astype(np.int32), scores, kr


# ------------------------------------------------------ attention forward
def _keys(row_ptr, col_idx, r: int, n: int, b: int) -> np.ndarray:
    tiles = col_idx[row_ptr[r]:row_ptr[r + 1]]
    if len(tiles) == 0:
        return np.zeros(0, dtype=np.int64)
    return np.concatenate([tile_rows(int(j), n, b) for j in tiles])


def _row_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float):
    """softmax(q k^T * scale) v for a set of query rows against one key set."""
    if k.shape[0] == 0:
        return np.zeros((q.shape[0], v.shape[1])), np.full(q.shape[0], -np.inf), None
    s = (q @ k.T) * scale
    m = s.max(axis=1, keepdims=True)
    e = np.exp(s - m)
    l = e.sum(axis=1, keepdims=True)
    p = e / l
    return p @ v, (m + np.log(l))[:, 0], p


def bsattn_fwd(qc, kc, vc, row_ptr, col_idx, b: int, scale: Optional[float] = None, b_kv: Optional[int] = None):
    """Block-sparse attention forward (Sec. 3.3): O_i = softmax(Q_i K_{S_i}^T/sqrt d) V_{S_i}.

    qc, kc, vc: [N, H, d]; query blocks of b rows, key blocks of b_kv rows (b
    when not given).  Returns O [N, H, d] and LSE [H, N] (natural log).
    """
    qc, kc, vc = (np.asarray(a, dtype=np.float64) for a in (qc, kc, vc))
    N, H, d = qc.shape
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    bk = b if b_kv is None else b_kv
    nq = n_blocks(N, b)
    O = np.zeros((N, H, d))
    LSE = np.full((H, N), -np.inf)
    for h in range(H):
        for i in range(nq):
            rows = tile_rows(i, N, b)
            keys = _keys(row_ptr, col_idx, h * nq + i, N, bk)
            o, lse, _ = _row_attention(qc[rows, h], kc[keys, h], vc[keys, h], scale)
            O[rows, h] = o
            LSE[h, rows] = lse
    return O, LSE


def bsattn_fwd_rows(qc, kc, vc, row_ptr, col_idx, b: int, h: int, rows: np.ndarray,
                    scale: Optional[float] = None, b_kv: Optional[int] = None):
    """The forward for a subset of query rows of head h (spot checks at full size)."""
    N, H, d = qc.shape
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    bk = b if b_kv is None else b_kv
    nq = n_blocks(N, b)
    rows = np.asarray(rows, dtype=np.int64)
    O = np.zeros((len(rows), d))
    LSE = np.full(len(rows), -np.inf)
    for t in np.unique(rows // b):
        sel = np.flatnonzero(rows // b == t)
        keys = _keys(row_ptr, col_idx, h * nq + int(t), N, bk)
        q = np.asarray(qc[rows[sel], h], dtype=np.float64)
        o, lse, _ = _row_attention(q, np.asarray(kc[keys, h], np.float64),
                                   np.asarray(vc[keys, h], np.float64), scale)
        O[sel] = o
        LSE[sel] = lse
    return O, LSE


# ----------------------------------------------------- attention backward
def bsattn_bwd(qc, kc, vc, dout, row_ptr, col_idx, b: int, scale: Optional[float] = None,
               b_kv: Optional[int] = None):
    """Gradients of the block-sparse forward w.r.t. Q, K, V.

    Per retained (query row r, key row k): P = softmax row, D_r = dO_r . O_r,
    dV_k += P_rk dO_r, dP_rk = dO_r . V_k, dS_rk = P_rk (dP_rk - D_r),
    dQ_r += dS_rk K_k * scale, dK_k += dS_rk Q_r * scale.
    """
    qc, kc, vc, dout = (np.asarray(a, dtype=np.float64) for a in (qc, kc, vc, dout))
    N, H, d = qc.shape
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    bk = b if b_kv is None else b_kv
    nq = n_blocks(N, b)
    dQ = np.zeros_like(qc)
    dK = np.zeros_like(kc)
    dV = np.zeros_like(vc)
    for h in range(H):
        for i in range(nq):
            rows = tile_rows(i, N, b)
            keys = _keys(row_ptr, col_idx, h * nq + i, N, bk)
            if len(keys) == 0:
                continue
            q, k, v, do = qc[rows, h], kc[keys, h], vc[keys, h], dout[rows, h]
            o, _, p = _row_attention(q, k, v, scale)
            D = (do * o).sum(axis=1, keepdims=True)
            dV[keys, h] += p.T @ do
            dP = do @ v.T
            dS = p * (dP - D)
            dQ[rows, h] += (dS @ k) * scale
            dK[keys, h] += (dS.T @ q) * scale
    return dQ, dK, dV


def bsattn_bwd_dq_rows(qc, kc, vc, dout, row_ptr, col_idx, b: int, h: int, rows: np.ndarray,
                       scale: Optional[float] = None, b_kv: Optional[int] = None):
    """dQ for a subset of query rows of head h."""
    N, H, d = qc.shape
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    bk = b if b_kv is None else b_kv
    nq = n_blocks(N, b)
    rows = np.asarray(rows, dtype=np.int64)
    dQ = np.zeros((len(rows), d))
    for t in np.unique(rows // b):
        sel = np.flatnonzero(rows // b == t)
        keys = _keys(row_ptr, col_idx, h * nq + int(t), N, bk)
        if len(keys) == 0:
            continue
        q = np.asarray(qc[rows[sel], h], np.float64)
        k = np.asarray(kc[keys, h], np.float64)
        v = np.asarray(vc[keys, h], np.float64)
        do = np.asarray(dout[rows[sel], h], np.float64)
        o, _, p = _row_attention(q, k, v, scale)
        D = (do * o).sum(axis=1, keepdims=True)
        dQ[sel] = ((p * (do @ v.T - D)) @ k) * scale
    return dQ


def bsattn_bwd_dkdv_rows(qc, kc, vc, dout, row_ptr, col_idx, b: int, h: int,
                         key_rows: np.ndarray, scale: Optional[float] = None, b_kv: Optional[int] = None):
    """dK, dV for a subset of key rows of head h.

    A key row in block j gathers contributions from every query block i whose
    list S_i holds j; each such query row needs its full softmax row (its own
    O and normaliser), which is recomputed here.
    """
    N, H, d = qc.shape
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    bk = b if b_kv is None else b_kv
    nq = n_blocks(N, b)
    key_rows = np.asarray(key_rows, dtype=np.int64)
    dK = np.zeros((len(key_rows), d))
    dV = np.zeros((len(key_rows), d))
    want = set(int(x) // bk for x in key_rows)
    for i in range(nq):
        r = h * nq + i
        tiles = set(int(x) for x in col_idx[row_ptr[r]:row_ptr[r + 1]])
        hit = tiles & want
        if not hit:
            continue
        rows = tile_rows(i, N, b)
        keys = _keys(row_ptr, col_idx, r, N, bk)
        q = np.asarray(qc[rows, h], np.float64)
        k = np.asarray(kc[keys, h], np.float64)
        v = np.asarray(vc[keys, h], np.float64)
        do = np.asarray(dout[rows, h], np.float64)
        o, _, p = _row_attention(q, k, v, scale)
        D = (do * o).sum(axis=1, keepdims=True)
        dS = p * (do @ v.T - D)
        pos = {int(kk): c for c, kk in enumerate(keys)}
        for s_, kr in enumerate(key_rows):
            c = pos.get(int(kr))
            if c is None:
                continue
            dV[s_] += p[:, c] @ do
            dK[s_] += (dS[:, c] @ q) * scale
    return dK, dV


# ------------------------------------------------------------------ FLOPs
def retained_flops_fwd(row_ptr, col_idx, n: int, b: int, d: int, b_kv: Optional[int] = None) -> float:
    """4 * |Q_i| * |K_j| * d per retained (head, i, j) pair, actual tail sizes."""
    bk = b if b_kv is None else b_kv
    nq, nk = n_blocks(n, b), n_blocks(n, bk)
    qs = np.array([len(tile_rows(i, n, b)) for i in range(nq)], dtype=np.float64)
    ks = np.array([len(tile_rows(j, n, bk)) for j in range(nk)], dtype=np.float64)
    total = 0.0
    for r in range(len(row_ptr) - 1):
        i = r % nq
        total += qs[i] * ks[col_idx[row_ptr[r]:row_ptr[r + 1]]].sum()
    return 4.0 * d * total
