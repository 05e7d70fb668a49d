"""The seeded generator: exact counts, shared view masks, reproducibility, densities."""
import numpy as np
import torch

from synth import CONFIGS, sweep2048


def test_exact_counts_and_shared_view_masks():
    for name in ("tiny", "c512", "c1024", "c2048"):
        w = CONFIGS[name]
        masks = w.image_masks()
        assert masks.shape == (w.n_images, w.side * w.side)
        assert list(masks.sum(1)) == list(w.image_counts())
        assert int(w.canvas_mask().sum()) == w.N
        if w.multiview:
            for v in range(6):
                assert np.array_equal(masks[v], masks[6 + v])
    assert CONFIGS["c512"].image_masks()[-1].all()
    assert CONFIGS["c512"].N == 7780
    assert CONFIGS["c1024"].N == 23959
    assert CONFIGS["c2048"].N == 85202
    assert [sweep2048(f, 0.1).N for f in (0.2, 0.4, 0.6, 0.8)] == [42601, 85202, 127790, 170391]


def test_reproducible_and_rounded():
    w = CONFIGS["c512"].with_(heads=2)
    a, b = w.q(), w.q()
    assert a.dtype == torch.bfloat16 and torch.equal(a, b)
    assert not torch.equal(w.q(), w.k())
    t = CONFIGS["tiny"]
    assert t.q().dtype == torch.float32 and t.q().shape == (512, 1, 64)


def test_structured_densities():
    t = CONFIGS["tiny"]
    bm = t.block_bitmap()
    base = t.structural_bitmap()
    assert bm.shape == (1, 8, 8)
    assert np.all(bm[:, base == 1] == 1)
    for name in ("c512", "c1024"):
        w = CONFIGS[name]
        bm = w.block_bitmap()
        assert bm.shape == (w.heads, w.n_tiles, w.n_tiles)
        assert 0.15 <= bm.mean() <= 0.40
        assert np.all(bm.diagonal(axis1=1, axis2=2) == 1)   # own-view always kept
