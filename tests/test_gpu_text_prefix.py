"""The joint sequence's text tokens in front of the images (the token lengths
of Table S1 include 512 of them): always kept by the mask, unrotated by RoPE,
and carried through compaction, Top-K block lists and attention like any
other retained token.  GPU against the oracle, through the C ABI."""
import numpy as np
import pytest
import torch

import oracle.ultratex_oracle as o
from gpu_util import assert_bf16_close, need_gpu, to_np
from synth import CONFIGS
from test_gpu_rope import _assert_rotation_close

pytestmark = pytest.mark.gpu


def _workload():
    return CONFIGS["c512"].with_(name="c512t", mask_mode="topk", density=0.3, text_prefix=512, heads=2)


def test_text_prefix_is_kept_and_unrotated():
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    w = _workload()
    mask = w.canvas_mask()
    assert mask[:512].all() and len(mask) == w.T
    q = w.q()
    idx, n, (qc,) = u.ut_fg_compact(torch.from_numpy(mask).cuda(), [q.cuda()])
    N = int(n.item())
    assert N == w.N and np.array_equal(idx[:512].cpu().numpy(), np.arange(512))
    cfg = u.rope_config(w.side, prefix=512)
    (qr,) = u.ut_fg_gather_rope(idx[:N], N, [q.cuda()], cfg)
    torch.cuda.synchronize()
    xn = q.double().numpy()
    i2, ref = o.fg_compact_rope(mask, xn, w.side, prefix=512)
    _assert_rotation_close(qr.cpu().double().numpy(), ref, xn[i2], torch.bfloat16, "Q with text prefix")
    # the text rows come out exactly as they went in (rotation by 0)
    assert torch.equal(qr[:512].cpu(), q[:512])


def test_attention_path_with_text_prefix():
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    w = _workload()
    mask = w.canvas_mask()
    q, k, v = w.q(), w.k(), w.v()
    idx, n, (qc, kc, vc) = u.ut_fg_compact(torch.from_numpy(mask).cuda(), [q.cuda(), k.cuda(), v.cuda()])
    N = int(n.item())
    qc, kc, vc = qc[:N], kc[:N], vc[:N]
    rp, ci, _, _ = u.ut_block_mask(u.attn_shape(qc, 128), u.UT_MASK_TOPK, qc, kc, w.rho, with_transpose=False)
    O, L = u.ut_bsattn_fwd(qc, kc, vc, rp, ci, 128)
    torch.cuda.synchronize()
    idx_ref, (qn, kn, vn) = o.fg_compact(mask, [x.double().numpy() for x in (q, k, v)])
    rrp, rci, _, _ = o.topk_block_mask(qn, kn, 128, w.rho)
    assert np.array_equal(rp.cpu().numpy()[:len(rrp)], rrp)
    assert np.array_equal(ci.cpu().numpy()[:len(rci)], rci)
    rO, _ = o.bsattn_fwd(qn, kn, vn, rrp, rci, 128)
    assert_bf16_close(to_np(O), rO, "O with text prefix")
