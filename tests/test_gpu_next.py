"""GPU parity for the widened rows: partial history during warm-up, caller-given
weights (other node families, truncated Taylor), and a non-affine schedule.

Same gates as test_gpu_parity.py: within one bf16 ulp of the oracle's fp64
result rounded to bf16 (exact cancellations below 2^-40 sum|w F| counted apart).
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2608_23429_gb300 import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cb():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_23429_gb300 import build
    build.build()
    from paper_2608_23429_gb300 import chebboost
    return chebboost


@pytest.fixture(scope="module")
def H(cb):
    import gpu_harness
    orc.build()
    return gpu_harness


def _ok(stats, what):
    assert stats is not None and stats["bad"] == 0, (what, stats)


@pytest.mark.parametrize("kernel", ["bulk", "direct"])
def test_partial_history_warmup(cb, H, kernel):
    """Alg. 1 read literally: with no warm-up full steps, the steps after the
    first full step extrapolate from the 1, 2, ... entries H holds."""
    w = workloads.scaled(workloads.pixart(), 32)
    mask = orc.full_schedule(w.T, w.r, 0, 0, 0)  # the set F alone
    node_t = [t for s, t in enumerate(w.timesteps) if mask[s]]
    walk = H.Walk(w, node_t=node_t, kernel=kernel)
    walk.push(w.timesteps[0], 0)
    with pytest.raises(cb.CbError) as e:  # default reading: |H| = K is required
        walk.extrapolate(w.timesteps[1])
    assert e.value.status == cb.CB_ERR_HISTORY_NOT_FULL
    cb.cb_plan_set_option(walk.plan, cb.CB_OPT_PARTIAL_HISTORY, 1)
    used = set()
    for s in range(1, w.T):
        t = w.timesteps[s]
        if mask[s]:
            walk.push(t, s)
            continue
        n = len(walk.H.entries())
        used.add(n)
        wl = cb.cb_weights(walk.plan, t, n)
        ref = orc.weights(walk.H.times(), t, w.t_min, w.t_max)
        assert np.max(np.abs(wl - ref)) <= 1e-12 * np.abs(ref).sum()
        outs, resid, rh = walk.extrapolate(t, fused=(s % 2 == 0), salt=s)
        so, sr, _ = walk.expected_and_compare(t, outs, resid, rh)
        _ok(so, ("partial", n, s))
        if resid is not None:
            _ok(sr, ("partial resid", n, s))
    assert used == {1, 2, 3, 4}
    walk.close()


def test_explicit_weights_and_taylor(cb, H):
    w = workloads.scaled(workloads.dit256(4), 16)
    nodes = [w.timesteps[s] for s in (4, 8, 12, 16)]  # equispaced, as Taylor needs
    walk = H.Walk(w, node_t=nodes)
    for k, t in enumerate(nodes):
        walk.push(t, k)
    t = w.timesteps[18]
    # the weights cb_extrapolate computes, passed explicitly: identical bits
    ref_outs, _, _ = walk.extrapolate(t)
    wl = cb.cb_weights(walk.plan, t, 4)
    outs, _, _ = walk.extrapolate(t, explicit=wl)
    for a, b in zip(ref_outs, outs):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    rng = np.random.default_rng(5)
    tw = cb.cb_taylor_weights(nodes, t)
    assert np.max(np.abs(tw - orc.taylor_weights(nodes, t))) <= 1e-12 * np.abs(tw).sum()
    for name, wts in (("taylor", tw), ("random", rng.standard_normal(4)),
                      ("reuse-newest", np.array([0.0, 0.0, 0.0, 1.0]))):
        for fused in (False, True):
            outs, resid, rh = walk.extrapolate(t, fused=fused, explicit=wts, salt=3)
            so, sr, _ = walk.expected_and_compare(t, outs, resid, rh, wts=np.asarray(wts, float))
            _ok(so, (name, fused))
            if fused:
                _ok(sr, (name, "resid"))
    with pytest.raises(cb.CbError):
        walk.extrapolate(t, explicit=np.array([1.0, np.nan, 0.0, 0.0]))
    walk.close()


def test_shifted_flow_schedule(cb, H):
    """A non-affine timestep schedule (flow matching with a time shift,
    t = a s / (1 + (a - 1) s), a = 3, on a uniform s grid): node times are not
    equispaced, so every window gets its own general rho."""
    base = workloads.scaled(workloads.flux(), 16)
    a = 3.0
    base.timesteps = [a * x / (1 + (a - 1) * x) for x in base.timesteps]
    walk = H.Walk(base, samples=None)
    mask, skipped = H.schedule_steps(base, base.K)
    stats = []
    for s in range(base.T):
        t = base.timesteps[s]
        if mask[s]:
            walk.push(t, s)
        elif s in skipped[::4]:
            outs, _, _ = walk.extrapolate(t)
            so, _, _ = walk.expected_and_compare(t, outs, None, None)
            _ok(so, ("shifted", s))
            stats.append(so)
    print("shifted schedule", H.merge(stats))
    walk.close()
