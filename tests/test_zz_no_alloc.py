"""ut_fg_compact_noalloc: the compaction entry point for callers that cannot
allocate device memory (its scratch is a fixed array inside the library).

Collected last on purpose.  Checked through the C ABI against ut_fg_compact on
two calls in a row (the second call reuses the scratch the first one left)."""
import ctypes

import numpy as np
import pytest
import torch

from gpu_util import bits, need_gpu

pytestmark = pytest.mark.gpu


def _noalloc(L):
    f = L.ut_fg_compact_noalloc
    f.restype = ctypes.c_int32
    vp = ctypes.c_void_p
    f.argtypes = [vp, ctypes.c_int64, ctypes.c_int32, ctypes.POINTER(vp), ctypes.POINTER(vp), ctypes.c_int64,
                  ctypes.c_int64, vp, vp, vp, vp]
    return f


def _arr(ts):
    return (ctypes.c_void_p * len(ts))(*[t.data_ptr() for t in ts])


def test_noalloc_compaction_matches_workspace_entry_point():
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    L = u.lib()
    f = _noalloc(L)
    dev = torch.device("cuda")
    stream = torch.cuda.current_stream().cuda_stream
    g = np.random.Generator(np.random.PCG64(2024))
    for call, (T, frac) in enumerate([(212992, 0.4), (53248 + 77, 0.45)]):
        mask = torch.from_numpy((g.random(T) < frac).astype(np.uint8)).to(dev)
        x = torch.from_numpy(g.integers(-30000, 30000, size=(T, 2, 128), dtype=np.int16)).view(torch.bfloat16).to(dev)
        y = torch.from_numpy(g.standard_normal((T, 8)).astype(np.float32)).to(dev)
        # existing entry point (caller workspace); one call per row size
        idx_ref, n_ref, (xr,) = u.ut_fg_compact(mask, [x])
        _, _, (yr,) = u.ut_fg_compact(mask, [y])
        # no-allocation entry point, same inputs, two outputs of the same sizes
        idx = torch.full((T,), -1, dtype=torch.int32, device=dev)
        n = torch.zeros(1, dtype=torch.int32, device=dev)
        st = torch.zeros(1, dtype=torch.int32, device=dev)
        xo, yo = torch.zeros_like(x), torch.zeros_like(y)
        # row_bytes is per tensor; x and y have different rows, so one call each
        for src, dst in ((x, xo), (y, yo)):
            rb = src[0].numel() * src.element_size()
            rc = f(mask.data_ptr(), T, 1, _arr([src]), _arr([dst]), rb, T, idx.data_ptr(), n.data_ptr(),
                   st.data_ptr(), stream)
            assert rc == u.UT_OK, (call, rc)
        torch.cuda.synchronize()
        assert int(st.item()) == 0
        N = int(n_ref.item())
        assert int(n.item()) == N
        assert torch.equal(idx[:N], idx_ref[:N])
        assert np.array_equal(bits(xo[:N]), bits(xr[:N]))
        assert np.array_equal(bits(yo[:N]), bits(yr[:N]))


def test_noalloc_rejects_canvas_beyond_its_scratch():
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    f = _noalloc(u.lib())
    dummy = ctypes.c_void_p(1 << 20)
    arr = (ctypes.c_void_p * 1)(1 << 20)
    rc = f(dummy, 4096 * 1024 + 1, 1, arr, arr, 16, 10, dummy, dummy, None, None)
    assert rc == u.UT_ERR_UNSUPPORTED


def test_noalloc_empty_canvas_and_capacity_overflow():
    """T = 0 writes N = 0 and launches nothing else; N > capacity writes the
    first `capacity` rows, keeps N in n_out and reports UT_ERR_CAPACITY in the
    status word, exactly like the workspace entry point with the same capacity."""
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    L = u.lib()
    f = _noalloc(L)
    dev = torch.device("cuda")
    stream = torch.cuda.current_stream().cuda_stream
    # empty canvas
    n = torch.full((1,), 123, dtype=torch.int32, device=dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    src = torch.zeros((1, 16), dtype=torch.uint8, device=dev)
    rc = f(None, 0, 1, _arr([src]), _arr([src]), 16, 0, None, n.data_ptr(), st.data_ptr(), stream)
    assert rc == u.UT_OK
    torch.cuda.synchronize()
    assert int(n.item()) == 0 and int(st.item()) == 0
    # more foreground tokens than capacity
    g = np.random.Generator(np.random.PCG64(77))
    T, cap = 50000 + 3, 9000
    mask = torch.from_numpy((g.random(T) < 0.5).astype(np.uint8)).to(dev)
    x = torch.from_numpy(g.integers(-30000, 30000, size=(T, 64), dtype=np.int16)).view(torch.bfloat16).to(dev)
    N = int(mask.sum().item())
    assert N > cap
    outs = []
    for use_noalloc in (True, False):
        idx = torch.full((cap,), -1, dtype=torch.int32, device=dev)
        n = torch.zeros(1, dtype=torch.int32, device=dev)
        st = torch.zeros(1, dtype=torch.int32, device=dev)
        xo = torch.zeros((cap, 64), dtype=torch.bfloat16, device=dev)
        if use_noalloc:
            rc = f(mask.data_ptr(), T, 1, _arr([x]), _arr([xo]), 128, cap, idx.data_ptr(), n.data_ptr(),
                   st.data_ptr(), stream)
            assert rc == u.UT_OK
        else:
            u.ut_fg_compact(mask, [x], capacity=cap, outs=[xo], idx=idx, n_out=n, status=st)
        torch.cuda.synchronize()
        assert int(n.item()) == N
        assert int(st.item()) == u.UT_ERR_CAPACITY
        outs.append((idx.cpu(), bits(xo)))
    ref = np.flatnonzero(mask.cpu().numpy())[:cap]
    assert np.array_equal(outs[0][0].numpy(), ref)
    assert torch.equal(outs[0][0], outs[1][0])
    assert np.array_equal(outs[0][1], outs[1][1])
    assert np.array_equal(outs[0][1], bits(x[torch.from_numpy(ref).to(dev)]))
