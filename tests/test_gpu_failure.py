"""Failure detection on the GPU without a fault: every device wait in the
tensor-core kernels is bounded.  With the limit forced to 0 (give up at the
first wait that is not already satisfied) the waits run out, the kernels record UT_ERR_TIMEOUT in the status word, drain their own
copies and MMAs, free TMEM and return; the next normal call on the same
context must succeed and be correct."""
import numpy as np
import pytest
import torch

import oracle.ultratex_oracle as o
from gpu_util import assert_bf16_close, need_gpu, to_np

pytestmark = pytest.mark.gpu


def _problem(seed=3, N=1500, H=2):
    g = np.random.Generator(np.random.PCG64([99, seed]))
    q, k, v, do = (torch.from_numpy(g.standard_normal((N, H, 128)).astype(np.float32)).to(torch.bfloat16)
                   for _ in range(4))
    nq = -(-N // 128)
    bm = (g.random((H, nq, nq)) < 0.5).astype(np.uint8)
    bm[:, np.arange(nq), np.arange(nq)] = 1
    return q, k, v, do, bm


def test_expired_waits_report_timeout_and_context_survives(monkeypatch):
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    q, k, v, do, bm = _problem()
    N, H, _ = q.shape
    shape = u.AttnShape(N, H, 128, 128, u.UT_BF16, H * 128)
    st0 = u.status_word()
    rp, ci, cp, ri = u.ut_block_mask(shape, u.UT_MASK_BITMAP, bitmap=torch.from_numpy(bm).cuda(), status=st0,
                                     col_cap=int(bm.sum()))
    qd, kd, vd, dd = (x.cuda() for x in (q, k, v, do))

    monkeypatch.setenv("UT_WAIT_TIMEOUT_NS", "0")
    st = u.status_word()
    O, L = u.ut_bsattn_fwd(qd, kd, vd, rp, ci, 128, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == u.UT_ERR_TIMEOUT
    st = u.status_word()
    u.ut_bsattn_bwd(qd, kd, vd, O, L, dd, rp, ci, cp, ri, 128, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == u.UT_ERR_TIMEOUT

    monkeypatch.delenv("UT_WAIT_TIMEOUT_NS")
    st = u.status_word()
    O, L = u.ut_bsattn_fwd(qd, kd, vd, rp, ci, 128, status=st)
    dq, dk, dv = u.ut_bsattn_bwd(qd, kd, vd, O, L, dd, rp, ci, cp, ri, 128, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    rrp, rci = o.bitmap_to_csr(bm)
    qn, kn, vn, dn = (x.double().numpy() for x in (q, k, v, do))
    rO, _ = o.bsattn_fwd(qn, kn, vn, rrp, rci, 128)
    assert_bf16_close(to_np(O), rO, "O after recovery")
    rq, rk, rv = o.bsattn_bwd(qn, kn, vn, dn, rrp, rci, 128)
    for name, g_, r_ in (("dQ", dq, rq), ("dK", dk, rk), ("dV", dv, rv)):
        assert_bf16_close(to_np(g_), r_, name + " after recovery")
