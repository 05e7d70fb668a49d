"""Host-side checks of the C ABI (no GPU needed): the library loads, exports
every declared entry point, and rejects bad arguments before launching."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    import __graft_entry__ as g
    g.build()
    from paper_2609_23169_gb300 import ultratex
    return ultratex.lib()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "ultratex.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ut_[a-z0-9_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(L):
    names = declared_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(L, n), n
    from paper_2609_23169_gb300 import ultratex
    assert sorted(ultratex.EXPORTS) == sorted(names)


def test_strerror_and_topk_count(L):
    from paper_2609_23169_gb300 import ultratex as u
    assert L.ut_strerror(u.UT_ERR_TIMEOUT) == b"device wait timed out"
    import oracle.ultratex_oracle as o
    for rho in (0.05, 0.1, 0.12, 0.2, 0.25, 0.3, 0.5, 0.7, 1.0):
        for nk in (1, 3, 8, 10, 61, 188, 666, 1332):
            assert u.ut_topk_count(rho, nk) == o.k_rho(rho, nk), (rho, nk)


def _shape(u, N=256, H=2, d=64, b=32, dtype=1, rs=None):
    return u.AttnShape(N, H, d, b, dtype, H * d if rs is None else rs)


def test_argument_errors_are_caught_on_host(L):
    from paper_2609_23169_gb300 import ultratex as u
    bogus = ctypes.c_void_p(16 * 1024)   # never dereferenced: every call must fail validation first
    S = ctypes.byref
    # unsupported head dim / dtype / block
    assert L.ut_bsattn_fwd(S(_shape(u, d=96)), bogus, bogus, bogus, bogus, bogus, 0.1, bogus, bogus, None, None) \
        == u.UT_ERR_UNSUPPORTED
    assert L.ut_bsattn_fwd(S(_shape(u, dtype=7)), bogus, bogus, bogus, bogus, bogus, 0.1, bogus, bogus, None, None) \
        == u.UT_ERR_INVALID_ARG
    assert L.ut_bsattn_fwd(S(_shape(u, dtype=0, b=32)), bogus, bogus, bogus, bogus, bogus, 0.1, bogus, bogus, None,
                           None) == u.UT_ERR_UNSUPPORTED
    # unequal blocks: bf16 only, each 64 or 128
    sh = _shape(u, dtype=1, b=64)
    sh.block_k = 128
    assert L.ut_bsattn_fwd(S(sh), bogus, bogus, bogus, bogus, bogus, 0.1, bogus, bogus, None, None) \
        == u.UT_ERR_UNSUPPORTED
    sh = _shape(u, dtype=0, b=128)
    sh.block_k = 32
    assert L.ut_bsattn_fwd(S(sh), bogus, bogus, bogus, bogus, bogus, 0.1, bogus, bogus, None, None) \
        == u.UT_ERR_UNSUPPORTED
    sh.block_k = -1
    assert L.ut_bsattn_fwd(S(sh), bogus, bogus, bogus, bogus, bogus, 0.1, bogus, bogus, None, None) \
        == u.UT_ERR_INVALID_ARG
    # bad row stride, null pointers, bad scale, misalignment
    assert L.ut_bsattn_fwd(S(_shape(u, rs=100)), bogus, bogus, bogus, bogus, bogus, 0.1, bogus, bogus, None, None) \
        == u.UT_ERR_INVALID_ARG
    assert L.ut_bsattn_fwd(S(_shape(u)), None, bogus, bogus, bogus, bogus, 0.1, bogus, bogus, None, None) \
        == u.UT_ERR_INVALID_ARG
    assert L.ut_bsattn_fwd(S(_shape(u)), bogus, bogus, bogus, bogus, bogus, -1.0, bogus, bogus, None, None) \
        == u.UT_ERR_INVALID_ARG
    odd = ctypes.c_void_p(16 * 1024 + 4)
    assert L.ut_bsattn_fwd(S(_shape(u)), odd, bogus, bogus, bogus, bogus, 0.1, bogus, bogus, None, None) \
        == u.UT_ERR_INVALID_ARG
    # N = 0 is a no-op
    assert L.ut_bsattn_fwd(S(_shape(u, N=0)), None, None, None, None, None, 0.1, None, None, None, None) == u.UT_OK
    # compaction: row bytes not a multiple of 16, too many tensors, no workspace
    arr = (ctypes.c_void_p * 1)(bogus.value)
    assert L.ut_fg_compact(bogus, 100, 1, arr, arr, 24, 100, bogus, bogus, bogus, 64, None, None) \
        == u.UT_ERR_INVALID_ARG
    assert L.ut_fg_compact(bogus, 100, 9, arr, arr, 32, 100, bogus, bogus, bogus, 64, None, None) \
        == u.UT_ERR_INVALID_ARG
    assert L.ut_fg_compact(bogus, 100, 1, arr, arr, 32, 100, bogus, bogus, None, 0, None, None) \
        == u.UT_ERR_INVALID_ARG
    # scatter: n > T, unknown mode, FILL without a row
    assert L.ut_fg_scatter(bogus, 10, 1, arr, arr, 32, u.UT_BG_KEEP, None, 5, None) == u.UT_ERR_INVALID_ARG
    assert L.ut_fg_scatter(bogus, 1, 1, arr, arr, 32, 9, None, 5, None) == u.UT_ERR_INVALID_ARG
    assert L.ut_fg_scatter(bogus, 1, 1, arr, arr, 32, u.UT_BG_FILL, None, 5, None) == u.UT_ERR_INVALID_ARG
    # block mask: rho out of range, capacity too small for Top-K, bitmap mode without a status word
    sh = _shape(u, N=256, b=32)
    wsb = L.ut_block_mask_workspace_size(S(sh), u.UT_MASK_TOPK)
    assert wsb > 0
    assert L.ut_block_mask(S(sh), u.UT_MASK_TOPK, bogus, bogus, 0.0, None, bogus, bogus, 100, None, None, bogus, wsb,
                           None, None) == u.UT_ERR_INVALID_ARG
    assert L.ut_block_mask(S(sh), u.UT_MASK_TOPK, bogus, bogus, 0.5, None, bogus, bogus, 3, None, None, bogus, wsb,
                           None, None) == u.UT_ERR_CAPACITY
    assert L.ut_block_mask(S(sh), u.UT_MASK_BITMAP, None, None, 0.0, bogus, bogus, bogus, 100, None, None, bogus,
                           wsb, None, None) == u.UT_ERR_INVALID_ARG
    # backward needs the transposed lists
    assert L.ut_bsattn_bwd(S(_shape(u)), bogus, bogus, bogus, bogus, bogus, bogus, bogus, bogus, None, None, 0.1,
                           bogus, bogus, bogus, bogus, 1 << 20, None, None) == u.UT_ERR_INVALID_ARG


def test_backward_workspace_holds_accumulator_and_counter(L):
    """The bf16 backward's workspace covers D and LSE*log2e per padded row, the
    fp32 dQ accumulator and the key-block counter after it; one byte less is
    refused before any launch (the pointers are also misaligned, a second
    reason to refuse)."""
    from paper_2609_23169_gb300 import ultratex as u
    S = ctypes.byref
    N, H, d = 1000, 2, 128
    sh = _shape(u, N=N, H=H, d=d, b=128, dtype=u.UT_BF16)
    Np = -(-N // 128) * 128
    need = 2 * H * Np * 4 + H * Np * d * 4 + 16
    wsb = L.ut_bsattn_bwd_workspace_size(S(sh))
    assert wsb >= need
    bad = ctypes.c_void_p(16 * 1024 + 8)
    assert L.ut_bsattn_bwd(S(sh), bad, bad, bad, bad, bad, bad, bad, bad, bad, bad, 0.1, bad, bad, bad,
                           ctypes.c_void_p(16 * 1024), need - 1, None, None) == u.UT_ERR_INVALID_ARG


def test_sampler_argument_errors_are_caught_on_host(L):
    from paper_2609_23169_gb300 import ultratex as u
    bogus = ctypes.c_void_p(16 * 1024)   # never dereferenced: every call must fail validation first
    odd = ctypes.c_void_p(16 * 1024 + 4)
    f = L.ut_fg_euler_update
    # n > T, negative sizes, unknown dtype, rows not a multiple of 16 bytes, non-finite dt, misaligned z
    assert f(bogus, 11, bogus, bogus, 10, 64, u.UT_BF16, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    assert f(bogus, -1, bogus, bogus, 10, 64, u.UT_BF16, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    assert f(bogus, 5, bogus, bogus, 10, 64, 7, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    assert f(bogus, 5, bogus, bogus, 10, 12, u.UT_BF16, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    assert f(bogus, 5, bogus, bogus, 10, 6, u.UT_F32, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    assert f(bogus, 5, bogus, bogus, 10, 64, u.UT_F32, float("nan"), None, None) == u.UT_ERR_INVALID_ARG
    assert f(bogus, 5, odd, bogus, 10, 64, u.UT_F32, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    assert f(None, 5, bogus, bogus, 10, 64, u.UT_F32, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    # n = 0 is a no-op (nothing is dereferenced)
    assert f(None, 0, None, None, 10, 64, u.UT_BF16, 0.5, None, None) == u.UT_OK
    fg = L.ut_fg_euler_update_gather
    # the fused gather: same checks, plus a missing or misaligned zc
    assert fg(bogus, 11, bogus, bogus, bogus, 10, 64, u.UT_BF16, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    assert fg(bogus, 5, bogus, bogus, None, 10, 64, u.UT_BF16, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    assert fg(bogus, 5, bogus, bogus, odd, 10, 64, u.UT_BF16, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    assert fg(bogus, 5, bogus, bogus, bogus, 10, 12, u.UT_BF16, 0.5, None, None) == u.UT_ERR_INVALID_ARG
    assert fg(None, 0, None, None, None, 10, 64, u.UT_BF16, 0.5, None, None) == u.UT_OK
    g = L.ut_fg_composite
    assert g(bogus, 10, bogus, bogus, 0, 128, None) == u.UT_ERR_INVALID_ARG      # empty tile
    assert g(bogus, 10, bogus, bogus, 4, 100, None) == u.UT_ERR_INVALID_ARG      # row not 16-byte multiple
    assert g(bogus, 10, odd, bogus, 4, 128, None) == u.UT_ERR_INVALID_ARG        # misaligned z
    assert g(None, 10, bogus, bogus, 4, 128, None) == u.UT_ERR_INVALID_ARG       # no mask
    assert g(None, 0, None, None, 4, 128, None) == u.UT_OK                       # T = 0 is a no-op


def test_rope_argument_errors_are_caught_on_host(L):
    from paper_2609_23169_gb300 import ultratex as u
    bogus = ctypes.c_void_p(16 * 1024)   # never dereferenced: every call must fail validation first
    arr = (ctypes.c_void_p * 2)(bogus.value, bogus.value)
    S = ctypes.byref
    ok = u.rope_config(16)
    g, sc = L.ut_fg_gather_rope, L.ut_fg_scatter_rope
    assert g(bogus, 11, 1, arr, arr, 10, 2, 128, u.UT_BF16, S(ok), None) == u.UT_ERR_INVALID_ARG        # n > T
    assert g(bogus, 5, 9, arr, arr, 10, 2, 128, u.UT_BF16, S(ok), None) == u.UT_ERR_INVALID_ARG         # 9 tensors
    assert g(bogus, 5, 1, arr, arr, 10, 2, 128, 5, S(ok), None) == u.UT_ERR_INVALID_ARG                 # dtype
    assert g(bogus, 5, 1, arr, arr, 10, 2, 128, u.UT_BF16, None, None) == u.UT_ERR_INVALID_ARG          # no config
    assert g(bogus, 5, 1, arr, arr, 10, 2, 120, u.UT_BF16, S(ok), None) == u.UT_ERR_INVALID_ARG         # axes != d
    assert g(bogus, 5, 1, arr, arr, 10, 2, 128, u.UT_BF16, S(u.rope_config(16, (15, 57, 56))), None) \
        == u.UT_ERR_INVALID_ARG                                                                         # odd axis
    assert g(bogus, 5, 1, arr, arr, 10, 2, 128, u.UT_BF16, S(u.rope_config(0)), None) == u.UT_ERR_INVALID_ARG
    assert g(bogus, 5, 1, arr, arr, 10, 2, 128, u.UT_BF16, S(u.rope_config(16, theta=-1.0)), None) \
        == u.UT_ERR_INVALID_ARG
    assert g(bogus, 5, 1, arr, arr, 10, 2, 12, u.UT_BF16, S(u.rope_config(16, (4, 4, 4))), None) \
        == u.UT_ERR_UNSUPPORTED                                                                         # 24-byte heads
    assert g(bogus, 5, 1, arr, arr, 10, 2, 96, u.UT_BF16, S(u.rope_config(16, (16, 40, 40))), None) \
        == u.UT_ERR_UNSUPPORTED                                                                         # 192 B !| 512
    assert sc(bogus, 5, 1, arr, arr, 10, 2, 128, u.UT_BF16, S(ok), u.UT_BG_FILL, None) == u.UT_ERR_INVALID_ARG
    assert g(None, 0, 1, arr, arr, 10, 2, 128, u.UT_BF16, S(ok), None) == u.UT_OK                       # n = 0


def test_alpha_mask_argument_errors_are_caught_on_host(L):
    from paper_2609_23169_gb300 import ultratex as u
    bogus = ctypes.c_void_p(16 * 1024)   # never dereferenced: every call must fail validation first
    f = L.ut_fg_mask_from_alpha
    assert f(bogus, 6, 2048, 2048, 0, 1, 0, bogus, None) == u.UT_ERR_INVALID_ARG       # factor 0
    assert f(bogus, 6, 2040, 2048, 16, 1, 0, bogus, None) == u.UT_ERR_INVALID_ARG      # height not divisible
    assert f(bogus, 6, 2048, 2048, 16, 17, 0, bogus, None) == u.UT_ERR_INVALID_ARG     # radius too large
    assert f(bogus, 6, 2048, 2048, 16, 1, 256, bogus, None) == u.UT_ERR_INVALID_ARG    # threshold
    assert f(bogus, -1, 2048, 2048, 16, 1, 0, bogus, None) == u.UT_ERR_INVALID_ARG     # views
    assert f(None, 6, 2048, 2048, 16, 1, 0, bogus, None) == u.UT_ERR_INVALID_ARG       # no alpha
    assert f(None, 6, 0, 2048, 16, 1, 0, None, None) == u.UT_OK                        # empty image


def test_device_accessible_without_device(L):
    """Null and plain host pointers are never reported as device-accessible;
    on a machine without a GPU every pointer reads 0 (the query only asks the
    runtime and never launches)."""
    import torch
    from paper_2609_23169_gb300 import ultratex as u
    assert L.ut_device_accessible(None) == 0
    assert u.device_accessible(torch.zeros(4, dtype=torch.int32)) is False
    with pytest.raises(ValueError, match="n_out"):
        u.ut_fg_compact(torch.ones(4, dtype=torch.uint8), [torch.zeros(4, 4)], n_out=torch.zeros(1, dtype=torch.int32))


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    from paper_2609_23169_gb300 import ultratex as u
    monkeypatch.setattr(u, "_lib", None)
    monkeypatch.setattr(u, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="missing"):
        u.lib()


def test_binding_rejects_mixed_row_sizes():
    """One row size per call: a list mixing row sizes never reaches a kernel."""
    import torch
    from paper_2609_23169_gb300 import ultratex as u
    m = torch.ones(10, dtype=torch.uint8)
    a = torch.zeros(10, 2, 128, dtype=torch.bfloat16)
    b = torch.zeros(10, 8, dtype=torch.float32)
    with pytest.raises(ValueError, match="row size"):
        u.ut_fg_compact(m, [a, b])
    with pytest.raises(ValueError, match="rows"):
        u.ut_fg_compact(m, [a[:5]])
    idx = torch.zeros(10, dtype=torch.int32)
    with pytest.raises(ValueError):
        u.ut_fg_scatter(idx, 10, [a], [b])
