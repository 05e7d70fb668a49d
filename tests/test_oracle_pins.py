"""Pins of the fp64 oracle (CPU only) and planted-mistake checks that show the pins bite."""
import json
import math
import os

import numpy as np
import pytest

import oracle.ultratex_oracle as o
import pins
from synth import CONFIGS


def test_compaction_and_scatter_pinned():
    assert pins.check_compaction(o.fg_compact, o.fg_scatter) == []


def test_block_lists_pinned():
    assert pins.check_block_lists(o.bitmap_to_csr, o.csr_to_csc) == []


def test_topk_pinned():
    assert pins.check_topk(o.topk_block_mask, o.block_pool, o.k_rho) == []


def test_forward_pinned():
    assert pins.check_forward(o.bsattn_fwd, o.bitmap_to_csr) == []


def test_backward_pinned():
    assert pins.check_backward(o.bsattn_fwd, o.bsattn_bwd, o.bitmap_to_csr) == []


def test_sampler_steps_pinned():
    assert pins.check_sampler(o.fg_euler_update, o.fg_composite, o.fg_scatter) == []


def test_unequal_blocks_pinned():
    assert pins.check_unequal_blocks(o) == []


def test_alpha_mask_pinned():
    assert pins.check_alpha_mask(o.token_mask_from_alpha, o.canvas_mask_from_alpha) == []


def test_rope_pinned():
    assert pins.check_rope(o) == []


def test_row_subset_helpers_agree():
    assert pins.check_subsample_consistency(o, o.bitmap_to_csr) == []


def test_canvas_arithmetic(golden_dir):
    """Sec. 3.1 token counts and the Table S1 length column pin the canvas generator."""
    with open(os.path.join(golden_dir, "token_counts.json")) as f:
        g = json.load(f)
    w = CONFIGS["c2048"]
    assert w.tokens_per_image == g["tokens_per_image_2048"]
    assert w.n_images == sum(g["images"].values())
    assert w.T == g["canvas_tokens_2048"]
    for f_str, length in g["table_s1_token_length"].items():
        n = w.with_(fg_frac=float(f_str)).N
        assert abs(n - (length - g["text_prefix_tokens_reading"])) <= 12, (f_str, n, length)


def test_flop_count_matches_definition():
    rp = np.array([0, 2, 3], np.int32)
    ci = np.array([0, 1, 1], np.int32)
    # N = 6, b = 4: tiles of 4 and 2 rows.  pairs (0,0):4*4, (0,1):4*2, (1,1):2*2
    assert o.retained_flops_fwd(rp, ci, 6, 4, 8) == 4 * 8 * (16 + 8 + 4)


# ------------------------------------------------------------ planted mistakes
def _fwd_no_scale(q, k, v, rp, ci, b, scale=None):
    return o.bsattn_fwd(q, k, v, rp, ci, b, 1.0 if scale is None else scale)


def _fwd_transposed_lists(q, k, v, rp, ci, b, scale=None):
    N, H, _ = q.shape
    nq = o.n_blocks(N, b)
    bm = o.csr_to_bitmap(rp, ci, H, nq, nq).transpose(0, 2, 1)
    rp2, ci2 = o.bitmap_to_csr(np.ascontiguousarray(bm))
    return o.bsattn_fwd(q, k, v, rp2, ci2, b, scale)


def _fwd_drop_tail(q, k, v, rp, ci, b, scale=None):
    N = q.shape[0]
    O, L = o.bsattn_fwd(q, k, v, rp, ci, b, scale)
    if N % b:
        O[N - (N % b):] = 0
    return O, L


def _fwd_lse_log2(q, k, v, rp, ci, b, scale=None):
    O, L = o.bsattn_fwd(q, k, v, rp, ci, b, scale)
    return O, L / math.log(2)


def _bwd_sign(q, k, v, do, rp, ci, b, scale=None):
    dQ, dK, dV = o.bsattn_bwd(q, k, v, do, rp, ci, b, scale)
    return -dQ, dK, dV


def _bwd_no_D(q, k, v, do, rp, ci, b, scale=None):
    # dS = P * dP, forgetting the D_r term
    N, H, d = q.shape
    scale = 1.0 / math.sqrt(d) if scale is None else scale
    dQ, dK, dV = o.bsattn_bwd(q, k, v, do, rp, ci, b, scale)
    nq = o.n_blocks(N, b)
    for h in range(H):
        for i in range(nq):
            rows = o.tile_rows(i, N, b)
            keys = o._keys(rp, ci, h * nq + i, N, b)
            if len(keys) == 0:
                continue
            _, _, p = o._row_attention(q[rows, h], k[keys, h], v[keys, h], scale)
            dS = p * (do[rows, h] @ v[keys, h].T)
            dQ[rows, h] = (dS @ k[keys, h]) * scale
    return dQ, dK, dV


def _bwd_dv_transposed(q, k, v, do, rp, ci, b, scale=None):
    dQ, dK, dV = o.bsattn_bwd(q, k, v, do, rp, ci, b, scale)
    return dQ, dV, dK


def _topk_smallest(qc, kc, b, rho):
    return o.topk_block_mask(-qc, kc, b, rho)


def _topk_tie_high(qc, kc, b, rho):
    N, H, _ = qc.shape
    nq = o.n_blocks(N, b)
    kr = o.k_rho(rho, nq)
    lists = []
    for h in range(H):
        sc = o.compressed_scores(qc[:, h], kc[:, h], b)
        for i in range(nq):
            order = np.lexsort((-np.arange(nq), -sc[i]))
            lists.append(np.sort(order[:kr]))
    return (np.arange(H * nq + 1) * kr).astype(np.int32), np.concatenate(lists).astype(np.int32), None, kr


def _pool_sum(x, b):
    x = np.asarray(x, np.float64)
    return np.stack([x[o.tile_rows(i, x.shape[0], b)].sum(0) for i in range(o.n_blocks(x.shape[0], b))])


def _topk_pool_sum(qc, kc, b, rho):
    N, H, _ = qc.shape
    nq = o.n_blocks(N, b)
    kr = o.k_rho(rho, nq)
    lists = []
    for h in range(H):
        sc = _pool_sum(qc[:, h], b) @ _pool_sum(kc[:, h], b).T
        for i in range(nq):
            lists.append(np.sort(np.lexsort((np.arange(nq), -sc[i]))[:kr]))
    return (np.arange(H * nq + 1) * kr).astype(np.int32), np.concatenate(lists).astype(np.int32), None, kr


def _krho_ceil(rho, nk):
    return max(1, int(math.ceil(rho * nk)))


def _topk_krho_ceil(qc, kc, b, rho):
    N, H, _ = qc.shape
    nq = o.n_blocks(N, b)
    kr = _krho_ceil(rho, nq)
    lists = []
    for h in range(H):
        sc = o.compressed_scores(qc[:, h], kc[:, h], b)
        for i in range(nq):
            lists.append(np.sort(np.lexsort((np.arange(nq), -sc[i]))[:kr]))
    return (np.arange(H * nq + 1) * kr).astype(np.int32), np.concatenate(lists).astype(np.int32), None, kr


def _compact_off_by_one(mask, xs):
    idx, out = o.fg_compact(mask, xs)
    idx = np.minimum(idx + 1, len(mask) - 1).astype(np.int32)
    return idx, [np.asarray(x)[idx] for x in xs]


def _scatter_zero_everything(idx, src, dst_in, mode=0, fill_row=None):
    return o.fg_scatter(idx, src, dst_in, o.BG_ZERO, fill_row)


def _euler_sign_flipped(z, idx, v, dt):
    return o.fg_euler_update(z, idx, v, -dt)


def _euler_rows_in_order(z, idx, v, dt):
    return o.fg_euler_update(z, np.arange(len(idx)), v, dt)


def _composite_tile_by_block(z, mask, tile):
    y = np.array(z, copy=True)
    P = len(tile)
    for t in range(len(y)):
        if not mask[t]:
            y[t] = tile[(t // P) % P]
    return y


def _composite_overwrites_all(z, mask, tile):
    return o.fg_composite(z, np.zeros_like(mask), tile)


class _OracleWith:
    """The oracle module with one function replaced (a planted mistake)."""
    def __init__(self, **kw):
        self.__dict__.update(kw)

    def __getattr__(self, name):
        return getattr(o, name)


def _rope_sin_sign(x, angles, inverse=False):
    return o.rope_rotate(x, -angles, inverse)


def _rope_half_split(x, angles, inverse=False):
    x = np.asarray(x, dtype=np.float64)
    h = x.shape[-1] // 2
    a = -angles if inverse else angles
    c, s_ = np.cos(a)[:, None, :], np.sin(a)[:, None, :]
    y = np.empty_like(x)
    y[..., :h] = x[..., :h] * c - x[..., h:] * s_
    y[..., h:] = x[..., :h] * s_ + x[..., h:] * c
    return y


def _rope_freq_k_over_d(pos, head_dim, axes=(16, 56, 56), theta=10000.0):
    pos = np.asarray(pos, dtype=np.float64)
    cols = []
    for a, d_a in enumerate(axes):
        k = np.arange(d_a // 2, dtype=np.float64)
        cols.append(pos[:, a:a + 1] * (float(theta) ** (-k / d_a))[None, :])
    return np.concatenate(cols, axis=1)


def _rope_xy_swapped(idx, side, prefix=0):
    p = o.rope_positions(idx, side, prefix)
    return p[:, [0, 2, 1]]


def _rope_prefix_rotated(idx, side, prefix=0):
    t = np.asarray(idx, dtype=np.int64) - prefix   # text tokens treated as images at negative positions
    s2 = side * side
    return np.stack([t // s2, (t % s2) // side, t % side], axis=1)


def _alpha_all_pixels(alpha, factor=16, radius=1, threshold=0):
    a = np.asarray(alpha)
    h, w = a.shape[0] // factor, a.shape[1] // factor
    pooled = (a.reshape(h, factor, w, factor) > threshold).all(axis=(1, 3))
    return o.token_mask_from_alpha(pooled.astype(np.uint8) * 255, 1, radius, 0)


def _alpha_radius_plus_one(alpha, factor=16, radius=1, threshold=0):
    return o.token_mask_from_alpha(alpha, factor, radius + 1, threshold)


def _alpha_at_least(alpha, factor=16, radius=1, threshold=0):
    return o.token_mask_from_alpha(alpha, factor, radius, max(threshold - 1, -1))


def _canvas_conditions_use_reference(alpha, factor=16, radius=1, threshold=0):
    a = np.asarray(alpha)
    V = a.shape[0] - 1
    views = [o.token_mask_from_alpha(a[v], factor, radius, threshold).ravel() for v in range(V)]
    ref = o.token_mask_from_alpha(a[V], factor, radius, threshold).ravel()
    return np.concatenate(views + [ref] * V + [ref]).astype(np.uint8)


def _fwd_keys_at_query_size(q, k, v, rp, ci, b, scale=None, b_kv=None):
    return o.bsattn_fwd(q, k, v, rp, ci, b, scale)


def _topk_pool_k_at_query_size(qc, kc, b, rho, b_kv=None):
    return o.topk_block_mask(qc, kc, b, rho)


def _csr_descending(bm):
    rp, ci = o.bitmap_to_csr(bm)
    ci = ci.copy()
    for r in range(len(rp) - 1):
        ci[rp[r]:rp[r + 1]] = ci[rp[r]:rp[r + 1]][::-1]
    return rp, ci


@pytest.mark.parametrize("name,check", [
    ("fwd without 1/sqrt(d)", lambda: pins.check_forward(_fwd_no_scale, o.bitmap_to_csr)),
    ("fwd with transposed block lists", lambda: pins.check_forward(_fwd_transposed_lists, o.bitmap_to_csr)),
    ("fwd dropping the partial tile", lambda: pins.check_forward(_fwd_drop_tail, o.bitmap_to_csr)),
    ("fwd LSE in log2", lambda: pins.check_forward(_fwd_lse_log2, o.bitmap_to_csr)),
    ("bwd dQ sign", lambda: pins.check_backward(o.bsattn_fwd, _bwd_sign, o.bitmap_to_csr)),
    ("bwd without the D term", lambda: pins.check_backward(o.bsattn_fwd, _bwd_no_D, o.bitmap_to_csr)),
    ("bwd dK/dV swapped", lambda: pins.check_backward(o.bsattn_fwd, _bwd_dv_transposed, o.bitmap_to_csr)),
    ("Top-K keeps smallest", lambda: pins.check_topk(_topk_smallest, o.block_pool, o.k_rho)),
    ("Top-K tie toward larger index", lambda: pins.check_topk(_topk_tie_high, o.block_pool, o.k_rho)),
    ("Top-K sum pooling", lambda: pins.check_topk(_topk_pool_sum, _pool_sum, o.k_rho)),
    ("Top-K ceil(rho N_k)", lambda: pins.check_topk(_topk_krho_ceil, o.block_pool, _krho_ceil)),
    ("compaction off by one", lambda: pins.check_compaction(_compact_off_by_one, o.fg_scatter)),
    ("scatter ignores the mode", lambda: pins.check_compaction(o.fg_compact, _scatter_zero_everything)),
    ("CSR lists descending", lambda: pins.check_block_lists(_csr_descending, o.csr_to_csc)),
    ("b_kv ignored by the forward", lambda: pins.check_unequal_blocks(_OracleWith(bsattn_fwd=_fwd_keys_at_query_size))),
    ("b_kv ignored by Top-K", lambda: pins.check_unequal_blocks(_OracleWith(topk_block_mask=_topk_pool_k_at_query_size))),
    ("alpha pooled with all() instead of any()", lambda: pins.check_alpha_mask(_alpha_all_pixels,
                                                                               o.canvas_mask_from_alpha)),
    ("alpha dilation one token too wide", lambda: pins.check_alpha_mask(_alpha_radius_plus_one,
                                                                        o.canvas_mask_from_alpha)),
    ("alpha compared with >= instead of >", lambda: pins.check_alpha_mask(_alpha_at_least,
                                                                          o.canvas_mask_from_alpha)),
    ("conditions take the reference mask", lambda: pins.check_alpha_mask(o.token_mask_from_alpha,
                                                                         _canvas_conditions_use_reference)),
    ("RoPE with the sine's sign flipped", lambda: pins.check_rope(_OracleWith(rope_rotate=_rope_sin_sign))),
    ("RoPE pairing halves instead of neighbours", lambda: pins.check_rope(_OracleWith(rope_rotate=_rope_half_split))),
    ("RoPE frequencies theta^(-k/d)", lambda: pins.check_rope(_OracleWith(rope_angles=_rope_freq_k_over_d))),
    ("RoPE with x and y swapped", lambda: pins.check_rope(_OracleWith(rope_positions=_rope_xy_swapped))),
    ("RoPE rotating the text prefix", lambda: pins.check_rope(_OracleWith(rope_positions=_rope_prefix_rotated))),
    ("Euler step with t_curr - t_prev", lambda: pins.check_sampler(_euler_sign_flipped, o.fg_composite, o.fg_scatter)),
    ("Euler step on rows 0..n-1", lambda: pins.check_sampler(_euler_rows_in_order, o.fg_composite, o.fg_scatter)),
    ("composite tile indexed by t // P", lambda: pins.check_sampler(o.fg_euler_update, _composite_tile_by_block,
                                                                    o.fg_scatter)),
    ("composite overwrites the foreground", lambda: pins.check_sampler(o.fg_euler_update, _composite_overwrites_all,
                                                                       o.fg_scatter)),
])
def test_planted_mistake_is_caught(name, check):
    assert check() != [], f"the pins did not catch: {name}"
