"""The synthetic input recipe, checked on the CPU.

Shapes and bytes per history slot of the five workloads, their schedules'
full/skipped step counts, and the statistical structure of the generated
trajectories: a Chebyshev series of the stated degree whose d-th coefficient
has standard deviation 1/(d+1)^2, additive N(0, 0.1^2) noise per node, and
(DiT-XL/2 512^2) per-channel LogNormal(0, 1) scales. Same seed, same bytes.
Also the window of each schedule that bench.py times.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2608_23429_gb300 import workloads as wl

# (preset, tensors, bytes per slot, full steps, skipped steps)
SLOTS = [
    ("tiny", 4, 4_718_592, None, None),
    ("dit256-k3", 56, 264_241_152, 15, 35),
    ("dit256", 56, 264_241_152, 16, 34),
    ("dit512", 56, 528_482_304, 13, 37),
    ("pixart", 84, 1_585_446_912, 9, 11),
    ("flux", 114, 2_151_677_952, 13, 37),
]


@pytest.fixture(scope="module", autouse=True)
def _built():
    orc.build()


@pytest.mark.parametrize("name,n,slot,n_full,n_skip", SLOTS)
def test_shapes_slots_and_schedules(name, n, slot, n_full, n_skip):
    w = wl.PRESETS[name]()
    assert len(w.tensors) == n
    assert w.slot_elems * w.esize() == slot
    for t in w.tensors:  # members of a residual group share one hidden-state shape
        assert t.shape == w.group_shape(t.group)
    if n_full is not None:
        full = orc.full_schedule(w.T, w.r, w.s0, w.s1, w.K)
        assert (int(full.sum()), int((~full).sum())) == (n_full, n_skip)
        assert len(w.timesteps) == w.T and w.timesteps[0] == w.t_max and w.timesteps[-1] == w.t_min


def test_same_seed_same_bytes():
    w = wl.scaled(wl.dit256(), 64)
    a = wl.trajectory(w, 3, 500.0, 2, "cpu")
    b = wl.trajectory(w, 3, 500.0, 2, "cpu")
    c = wl.trajectory(w, 3, 500.0, 3, "cpu")  # another node: other noise
    d = wl.trajectory(w, 4, 500.0, 2, "cpu")  # another tensor: other coefficients
    assert a.dtype == torch.bfloat16 and a.shape == w.tensors[3].shape
    assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    assert not torch.equal(a, c) and not torch.equal(a, d)


def test_trajectory_is_a_chebyshev_series_of_the_stated_degree():
    C = np.polynomial.chebyshev
    w = wl.scaled(wl.dit256(), 64)
    D = w.degree
    taus = np.cos(np.pi * (np.arange(D + 1) + 0.5) / (D + 1))  # D+1 Chebyshev points fix the series
    ts = [(tau + 1.0) / 2.0 * (w.t_max - w.t_min) + w.t_min for tau in taus]
    vals = np.stack([wl.trajectory(w, 0, t, 0, "cpu", exact=True).numpy().ravel() for t in ts])
    coef = C.chebfit(taus, vals, D)  # [D+1, n]
    # a further point lies on the same degree-D series
    t_extra = 0.37 * (w.t_max - w.t_min) + w.t_min
    extra = wl.trajectory(w, 0, t_extra, 0, "cpu", exact=True).numpy().ravel()
    tau_x = 2.0 * (t_extra - w.t_min) / (w.t_max - w.t_min) - 1.0
    assert np.max(np.abs(C.chebval(tau_x, coef) - extra)) < 1e-9
    # c_d ~ N(0, 1) / (d+1)^2
    for d in range(D + 1):
        sd = coef[d].std() * (d + 1) ** 2
        assert abs(sd - 1.0) < 0.05, (d, sd)


def test_noise_and_channel_scales():
    w = wl.scaled(wl.dit256(), 64)
    t = 640.0
    noisy = wl.trajectory(w, 1, t, 5, "cpu", out_dtype=torch.float32).double()
    exact = wl.trajectory(w, 1, t, 5, "cpu", exact=True)
    noise = (noisy - exact).numpy().ravel()
    assert abs(noise.std() - 0.1) < 0.005 and abs(noise.mean()) < 0.005
    # DiT-XL/2 512^2: the same series times a per-channel LogNormal(0, 1) scale
    w5 = wl.scaled(wl.dit512(), 64)
    ratio = (wl.trajectory(w5, 2, t, 0, "cpu", exact=True)
             / wl.trajectory(wl.scaled(_no_scale(wl.dit512()), 64), 2, t, 0, "cpu", exact=True))
    r = ratio.numpy().reshape(-1, w5.tensors[2].shape[-1])
    assert np.allclose(r, r[0:1], rtol=1e-12)  # shared over batch and tokens
    logs = np.log(r[0])
    assert abs(logs.std() - 1.0) < 0.1 and abs(logs.mean()) < 0.1
    # the tiny case has no noise and degree 3
    tw = wl.tiny()
    assert tw.noise == 0.0 and tw.degree == 3 and tw.cache_dtype == "fp32"


def _no_scale(w):
    w.lognormal = False
    return w


@pytest.mark.parametrize("name", ["dit256", "dit256-k3", "dit512", "pixart", "flux"])
def test_bench_timed_window(name):
    """The window bench.py times: the full steps pushed before it end with K
    equispaced full steps one refresh interval apart, past the warm-up, and
    the targets are the skipped steps right after the last of them."""
    import bench
    w = wl.PRESETS[name]()
    mask = orc.full_schedule(w.T, w.r, w.s0, w.s1, w.K)
    pushed, targets = bench.window_of(w, mask)
    win = pushed[-w.K:]
    assert len(set(b - a for a, b in zip(win, win[1:]))) == 1 and win[-1] - win[0] == w.r * (w.K - 1)
    assert all(mask[s] for s in pushed) and not any(mask[s] for s in targets)
    assert targets == list(range(win[-1] + 1, targets[-1] + 1)) and mask[targets[-1] + 1]
    assert pushed == [s for s in range(win[-1] + 1) if mask[s]]  # every full step up to the window, in order
