"""GPU parity of the canvas mask built from alpha channels (Sec. 3.2, mask
construction) against the oracle, through the C ABI: integer work, compared
bit for bit."""
import numpy as np
import pytest
import torch

import oracle.ultratex_oracle as o
from gpu_util import need_gpu
from synth import CONFIGS

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("cfg", ["c512", "c2048"])
@pytest.mark.parametrize("radius,threshold", [(1, 0), (0, 0), (2, 64)])
def test_mask_from_alpha_matches_oracle(cfg, radius, threshold):
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    alpha = CONFIGS[cfg].alpha_images()
    got = u.ut_fg_mask_from_alpha(torch.from_numpy(alpha).cuda(), 16, radius, threshold)
    torch.cuda.synchronize()
    ref = o.canvas_mask_from_alpha(alpha, 16, radius, threshold)
    assert np.array_equal(got.cpu().numpy(), ref)


@pytest.mark.parametrize("V,H,W,factor,radius", [(2, 48, 80, 16, 1),    # partial tiles (3 x 5 tokens)
                                                 (1, 40, 56, 8, 2),     # byte path (factor not a multiple of 16)
                                                 (0, 64, 64, 16, 3),    # reference only
                                                 (3, 272, 16, 16, 16)])  # one token column, widest dilation
def test_mask_from_alpha_shapes(V, H, W, factor, radius):
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    g = np.random.Generator(np.random.PCG64(V * 1000 + H))
    alpha = ((g.random((V + 1, H, W)) < 0.01) * g.integers(1, 256, size=(V + 1, H, W))).astype(np.uint8)
    got = u.ut_fg_mask_from_alpha(torch.from_numpy(alpha).cuda(), factor, radius, 0)
    torch.cuda.synchronize()
    assert np.array_equal(got.cpu().numpy(), o.canvas_mask_from_alpha(alpha, factor, radius, 0))


def test_mask_from_alpha_empty_and_full():
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    for fill, want in ((0, 0), (255, 1)):
        alpha = np.full((7, 64, 64), fill, np.uint8)
        got = u.ut_fg_mask_from_alpha(torch.from_numpy(alpha).cuda(), 16, 1, 0)
        torch.cuda.synchronize()
        assert got.numel() == 13 * 16 and bool((got.cpu() == want).all())
