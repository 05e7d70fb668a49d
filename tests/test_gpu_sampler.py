"""GPU parity of the sampler steps on the canvas latent against the fp64 oracle:
the sparse Euler update (Sec. 3.2, Eq. euler) and the composite latent
(Sec. 3.4, Eq. mixed_latent), through the C ABI.

Tolerance of the Euler step: the kernel computes one fp32 fused multiply-add
per element and rounds it once to the storage type, so against the exact
(fp64) value the error is at most half an ulp of the fp32 result, plus, for
bf16 storage, half an ulp of the bf16 result: |gpu - exact| <= 2^-23 |exact|
for fp32 and <= (2^-8 + 2^-22) |exact| for bf16 (each bound with a factor-2
margin on the fp32 part).  Background rows and the composite are bit copies
and must match bit for bit."""
import numpy as np
import pytest
import torch

import oracle.ultratex_oracle as o
from gpu_util import bits, need_gpu
from synth import CONFIGS

pytestmark = pytest.mark.gpu

REL_BOUND = {torch.float32: 2.0 ** -23, torch.bfloat16: 2.0 ** -8 + 2.0 ** -22}


def _inputs(cfg, dtype, channels=64):
    return CONFIGS[cfg].sampler_inputs(channels=channels, dtype=dtype)


def _check_euler(z0, z_gpu, idx, v, dt, dtype):
    mask = np.zeros(z0.shape[0], bool)
    mask[idx] = True
    exact = o.fg_euler_update(z0.double().numpy(), idx, v.double().numpy(), dt)
    got = z_gpu.cpu().double().numpy()
    # background rows: not touched, bit for bit
    assert np.array_equal(bits(z_gpu.cpu()[torch.from_numpy(~mask)]), bits(z0[torch.from_numpy(~mask)]))
    err = np.abs(got[mask] - exact[mask])
    assert np.all(err <= REL_BOUND[dtype] * np.abs(exact[mask])), float((err / (np.abs(exact[mask]) + 1e-30)).max())
    return exact


@pytest.mark.parametrize("cfg", ["tiny", "c512", "c2048"])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_euler_update_matches_oracle(cfg, dtype):
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    x = _inputs(cfg, dtype)
    idx = np.nonzero(x["mask"])[0].astype(np.int32)
    n = len(idx)
    dt = float(np.float32(x["dt"]))
    z0, v = x["z"], x["v"]
    z = z0.cuda()
    st = u.status_word()
    u.ut_fg_euler_update(torch.from_numpy(idx).cuda(), n, z, v.cuda(), dt, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    _check_euler(z0, z, idx, v, dt, dtype)


def test_euler_two_steps_in_a_row_ragged_channels():
    """Two consecutive steps on the same buffer (the second reads the first's
    output), fp32 with 12 channels (48-byte rows) and an odd foreground."""
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    g = np.random.Generator(np.random.PCG64(5))
    T, C = 4099, 12
    mask = g.random(T) < 0.31
    idx = np.nonzero(mask)[0].astype(np.int32)
    z0 = torch.from_numpy(g.standard_normal((T, C)).astype(np.float32))
    v1 = torch.from_numpy(g.standard_normal((len(idx), C)).astype(np.float32))
    v2 = torch.from_numpy(g.standard_normal((len(idx), C)).astype(np.float32))
    z = z0.cuda()
    ic = torch.from_numpy(idx).cuda()
    u.ut_fg_euler_update(ic, len(idx), z, v1.cuda(), -0.25)
    z1 = z.cpu().clone()
    u.ut_fg_euler_update(ic, len(idx), z, v2.cuda(), -0.125)
    torch.cuda.synchronize()
    _check_euler(z0, z1, idx, v1, -0.25, torch.float32)
    _check_euler(z1, z, idx, v2, -0.125, torch.float32)


def test_euler_edge_cases():
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    g = np.random.Generator(np.random.PCG64(6))
    T, C = 1000, 64
    z0 = torch.from_numpy(g.standard_normal((T, C)).astype(np.float32)).to(torch.bfloat16)
    v = torch.from_numpy(g.standard_normal((T, C)).astype(np.float32)).to(torch.bfloat16)
    # n = 0: nothing changes
    z = z0.cuda()
    u.ut_fg_euler_update(torch.zeros(1, dtype=torch.int32).cuda(), 0, z, v.cuda(), -0.5)
    torch.cuda.synchronize()
    assert np.array_equal(bits(z.cpu()), bits(z0))
    # all foreground: every row moves
    idx = np.arange(T, dtype=np.int32)
    z = z0.cuda()
    u.ut_fg_euler_update(torch.from_numpy(idx).cuda(), T, z, v.cuda(), -0.5)
    torch.cuda.synchronize()
    _check_euler(z0, z, idx, v, -0.5, torch.bfloat16)
    # an index outside the canvas: that row is skipped and the status word says so
    idx = np.array([3, 7, T + 5, 11], dtype=np.int32)
    z = z0.cuda()
    st = u.status_word()
    u.ut_fg_euler_update(torch.from_numpy(idx).cuda(), 4, z, v[:4].cuda(), -0.5, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == u.UT_ERR_INVALID_ARG
    ok_rows = np.array([0, 1, 3])
    exact = o.fg_euler_update(z0.double().numpy(), idx[ok_rows], v[:4].double().numpy()[ok_rows], -0.5)
    got = z.cpu().double().numpy()
    sel = idx[ok_rows]
    assert np.all(np.abs(got[sel] - exact[sel]) <= REL_BOUND[torch.bfloat16] * np.abs(exact[sel]))
    others = np.setdiff1d(np.arange(T), sel)
    assert np.array_equal(bits(z.cpu()[torch.from_numpy(others)]), bits(z0[torch.from_numpy(others)]))


@pytest.mark.parametrize("cfg,period", [("c512", None), ("c2048", None), ("c512", 1), ("c512", 17)])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_composite_matches_oracle(cfg, period, dtype):
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    x = _inputs(cfg, dtype)
    tile = x["tile"] if period is None else x["tile"][:period].contiguous()
    z0 = x["z"]
    z = z0.cuda()
    u.ut_fg_composite(torch.from_numpy(x["mask"]).cuda(), z, tile.cuda())
    torch.cuda.synchronize()
    ref = o.fg_composite(bits(z0), x["mask"], bits(tile))   # a copy: compared bit for bit
    assert np.array_equal(bits(z.cpu()), ref)


def test_composite_all_foreground_and_all_background():
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    x = _inputs("c512", torch.bfloat16)
    z0, tile = x["z"], x["tile"]
    T = z0.shape[0]
    for m in (np.ones(T, np.uint8), np.zeros(T, np.uint8)):
        z = z0.cuda()
        u.ut_fg_composite(torch.from_numpy(m).cuda(), z, tile.cuda())
        torch.cuda.synchronize()
        assert np.array_equal(bits(z.cpu()), o.fg_composite(bits(z0), m, bits(tile)))


@pytest.mark.parametrize("cfg", ["c512", "c2048"])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_euler_update_gather_matches_oracle(cfg, dtype):
    """The Euler step fused with the next step's gather: the canvas rows as in
    ut_fg_euler_update (within the rounding bound of the oracle, background
    untouched) and zc[n] = the updated z[idx[n]] bit for bit."""
    need_gpu()
    from paper_2609_23169_gb300 import ultratex as u
    x = _inputs(cfg, dtype)
    idx = np.nonzero(x["mask"])[0].astype(np.int32)
    n = len(idx)
    dt = float(np.float32(x["dt"]))
    z0, v = x["z"], x["v"]
    z = z0.cuda()
    z_ref = z0.cuda()
    ti = torch.from_numpy(idx).cuda()
    st = u.status_word()
    zc = u.ut_fg_euler_update_gather(ti, n, z, v.cuda(), dt, status=st)
    u.ut_fg_euler_update(ti, n, z_ref, v.cuda(), dt, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    _check_euler(z0, z, idx, v, dt, dtype)
    assert np.array_equal(bits(z), bits(z_ref))            # same canvas as the unfused step
    assert np.array_equal(bits(zc[:n]), bits(z[ti]))       # the gather of the updated rows
