"""Helpers for the GPU parity tests (comparison metrics, device setup)."""
import numpy as np
import pytest
import torch

BF16_MAX_ABS, BF16_MEAN_ABS = 2e-2, 5e-3   # stated tolerance for bf16 attention outputs
F32_MAX_ABS = 1e-5                          # stated tolerance for the fp32 configuration
# Stricter sanity bound used alongside: error RMS relative to the reference RMS.
# bf16 rounding of P (2^-9 relative) and of the outputs keeps this near 4e-3.
BF16_REL_RMS = 2e-2


def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()


def err_stats(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    d = np.abs(got - ref)
    rms = float(np.sqrt((ref ** 2).mean())) if ref.size else 0.0
    return dict(max_abs=float(d.max()) if d.size else 0.0, mean_abs=float(d.mean()) if d.size else 0.0,
                rel_rms=float(np.sqrt((d ** 2).mean()) / rms) if rms > 0 else 0.0)


def assert_bf16_close(got, ref, what=""):
    s = err_stats(got, ref)
    assert s["max_abs"] <= BF16_MAX_ABS, (what, s)
    assert s["mean_abs"] <= BF16_MEAN_ABS, (what, s)
    assert s["rel_rms"] <= BF16_REL_RMS, (what, s)
    return s


def assert_f32_close(got, ref, what=""):
    s = err_stats(got, ref)
    assert s["max_abs"] <= F32_MAX_ABS, (what, s)
    return s


def to_np(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def bits(t: torch.Tensor) -> np.ndarray:
    """Raw bit pattern (bit-exact comparisons of bf16 / fp32 rows)."""
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy()
    if t.dtype == torch.float32:
        return t.view(torch.int32).numpy()
    return t.numpy()


def compare_topk_lists(rp, ci, rrp, rci, scores, kr):
    """GPU Top-K lists (rp, ci) against the oracle's (rrp, rci): equal row
    pointers; every row equal, except rows whose oracle K-th and (K+1)-th
    scores lie within 1e-4 * max|s| (reading A16), where only near-tied blocks
    may differ.  Returns the number of such near-tie rows."""
    H, nq, nk = scores.shape
    rp = np.asarray(rp)[:H * nq + 1]
    assert np.array_equal(rp, rrp)
    n_tie_rows = 0
    for r in range(H * nq):
        got = np.asarray(ci[rp[r]:rp[r + 1]])
        want = rci[rrp[r]:rrp[r + 1]]
        assert np.all(np.diff(got) > 0)
        if np.array_equal(got, want):
            continue
        h, i = divmod(r, nq)
        s = scores[h, i]
        srt = np.sort(s)[::-1]
        kth = srt[kr - 1]
        eps = 1e-4 * np.abs(s).max()
        assert kr < nk and srt[kr - 1] - srt[kr] < eps, f"row {r} differs without a near tie"
        assert np.all(s[got] >= kth - eps)
        n_tie_rows += 1
    return n_tie_rows


def head_lists(rp, ci, h, nq):
    """The CSR rows of head h alone (row pointers rebased to 0)."""
    rp = np.asarray(rp)
    base = int(rp[h * nq])
    end = int(rp[(h + 1) * nq])
    return (rp[h * nq:(h + 1) * nq + 1] - base).astype(np.int64), np.asarray(ci[base:end])
