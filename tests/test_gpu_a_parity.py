"""GPU parity: the CUDA library, called through its C ABI, against the oracle.

Gates (element by element on the same seeded inputs):
  * cb_cache_push: bit-exact against the oracle's conversion of the inputs;
  * bf16 results: within one bf16 ulp of the oracle's fp64 result rounded to
    bf16 (exact cancellations below 2^-40 sum|w F| are counted apart);
  * fp32 results: max |err| <= 2e-6 * max|F| per tensor.
Small workloads are compared on every element; the full-size benchmark
shapes are compared on sampled elements, in the launch configuration the
benchmark times.
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


def _assert_ok(stats, what):
    assert stats is not None
    assert stats["bad"] == 0, (what, stats)


# ------------------------------------------------------------------ push
@pytest.mark.parametrize("src,dst", [("bf16", "bf16"), ("fp32", "bf16"), ("bf16", "fp32"), ("fp32", "fp32")])
def test_push_bit_exact(cb, H, src, dst):
    numels = [1, 7, 8, 9, 4095, 4097, 8192, 12345, 65536 + 3]
    K = 3
    tensors = [(i, 0, n, -1) for i, n in enumerate(numels)]
    plan = cb.cb_plan_create([900.0, 800.0, 700.0, 600.0, 500.0], K, tensors, H.CB[dst], 0.0, 1000.0)
    cache = torch.zeros(cb.cb_plan_cache_bytes(plan), dtype=torch.uint8, device="cuda")
    cb.cb_plan_bind_cache(plan, cache, cache.numel())
    es = 2 if dst == "bf16" else 4
    offs, slot = H.slot_layout(numels, es)
    g = torch.Generator(device="cuda").manual_seed(5)
    specials = torch.tensor([0.0, -0.0, 1e-40, -3e-39, 1.0039062, 1.01171875, 3.3895e38, -3.3895e38, 1e-45],
                            dtype=torch.float32, device="cuda")
    pushed = []
    for k, t in enumerate([900.0, 800.0, 700.0, 600.0, 500.0]):
        feats = []
        for i, n in enumerate(numels):
            x = torch.randn(n + 1, generator=g, device="cuda") * (10.0 ** (k - 2))
            m = min(n, specials.numel())
            x[1:1 + m] = specials[:m]
            x = x.to(H.TORCH[src])
            # odd tensors start one element past an aligned address (scalar path)
            feats.append(x[1:] if i % 2 else x[:n])
        cb.cb_cache_push(plan, feats, H.CB[src], t)
        pushed.append([H.host(f) for f in feats])
        torch.cuda.synchronize()
        raw = cache.cpu().numpy()
        for p in range(K):  # every slot holds the right push
            last = [q for q in range(k + 1) if q % K == p]
            if not last:
                continue
            q = last[-1]
            for i, n in enumerate(numels):
                b = raw[p * slot + offs[i]: p * slot + offs[i] + n * es]
                got = b.view(np.uint16) if dst == "bf16" else b.view(np.float32)
                ref = orc.convert(pushed[q][i], H.ORC[src], H.ORC[dst])
                assert np.array_equal(got.view(np.uint8), ref.view(np.uint8)), (src, dst, k, p, i)
    slot_t, head, count = cb.cb_plan_history(plan, K)
    assert count == K and head == 5 % K
    assert list(slot_t) == [600.0, 500.0, 700.0]
    # pushing against the sampling direction, or a live node time, is refused
    with pytest.raises(cb.CbError) as e:
        cb.cb_cache_push(plan, feats, H.CB[src], 650.0)
    assert e.value.status == cb.CB_ERR_ORDER
    cb.cb_plan_destroy(plan)


# ------------------------------------------------------------- tiny, fp32
def test_tiny_fp32_polynomial_exact(cb, H):
    w = workloads.tiny()
    walk = H.Walk(w, node_t=w.explicit_nodes)
    for k, t in enumerate(w.explicit_nodes):
        walk.push(t, k)
    for t in w.explicit_targets:
        outs, _, _ = walk.extrapolate(t, out_dtype="fp32")
        so, _, wts = walk.expected_and_compare(t, outs, None, None, out_dtype="fp32")
        _assert_ok(so, ("tiny", t))
        # degree 3 < K = 4: the extrapolation reproduces the trajectory itself, up
        # to the fp32 rounding of the generator's sums at the nodes
        for i in range(len(w.tensors)):
            exact = workloads.trajectory(w, i, t, 99, "cuda", exact=True)
            mag = max(float(workloads.trajectory(w, i, tn, 99, "cuda", exact=True, absolute=True).abs().max())
                      for tn in w.explicit_nodes)
            tol = np.abs(wts).sum() * (w.degree + 3) * 2.0 ** -24 * mag
            got = outs[i].double()
            assert float((got - exact).abs().max()) <= tol + so["tol"], (t, i)
    walk.close()


# ----------------------------------------- scaled schedules, every element
@pytest.mark.parametrize("K,kernel", [(3, "bulk"), (4, "bulk"), (4, "direct")])
def test_dit256_scaled_full_schedule_fused(cb, H, K, kernel):
    w = workloads.scaled(workloads.dit256(K), 8)
    walk = H.Walk(w, K=K, kernel=kernel)
    mask, skipped = H.schedule_steps(w, K)
    agg_o, agg_r = [], []
    for s in range(w.T):
        t = w.timesteps[s]
        if mask[s]:
            walk.push(t, s)
            continue
        outs, resid, rh = walk.extrapolate(t, fused=True, salt=s)
        so, sr, _ = walk.expected_and_compare(t, outs, resid, rh)
        _assert_ok(so, ("out", s))
        _assert_ok(sr, ("resid", s))
        agg_o.append(so)
        agg_r.append(sr)
    m = H.merge(agg_o)
    print("dit256/8 K=%d %s outs" % (K, kernel), m, "resid", H.merge(agg_r))
    # one-ulp differences arise where the exact sum of bf16 inputs with
    # near-dyadic weights lands on a bf16 rounding tie: the kernel breaks the
    # tie to even, the oracle by the ~1e-16 rounding noise of its fp64 weights
    assert m["exact"] >= 0.9 * m["n"]
    walk.close()


def test_pixart_scaled_outputs_and_fp32(cb, H):
    w = workloads.scaled(workloads.pixart(), 32)
    walk = H.Walk(w)
    mask, skipped = H.schedule_steps(w, w.K)
    for s in range(w.T):
        t = w.timesteps[s]
        if mask[s]:
            walk.push(t, s)
        elif s in (skipped[0], skipped[-1]):
            outs, _, _ = walk.extrapolate(t)
            _assert_ok(walk.expected_and_compare(t, outs, None, None)[0], ("bf16", s))
            outs, _, _ = walk.extrapolate(t, out_dtype="fp32")
            _assert_ok(walk.expected_and_compare(t, outs, None, None, out_dtype="fp32")[0], ("fp32", s))
            outs, resid, rh = walk.extrapolate(t, fused=True, resid_dtype="fp32", salt=s)
            so, sr, _ = walk.expected_and_compare(t, outs, resid, rh, resid_dtype="fp32")
            _assert_ok(so, ("fused-out", s))
            _assert_ok(sr, ("fused-fp32-resid", s))
    walk.close()


# ------------------------------------- repeated launches give the same bits
def _launch(cb, H, walk, t, kernel, resid0=None):
    """One skipped step into output buffers filled with NaN (an element the
    kernel fails to write cannot pass as a stale copy of an earlier launch);
    with resid0 the hidden states start from a copy of those tensors."""
    cb.cb_plan_set_option(walk.plan, cb.CB_OPT_KERNEL, H.KERNEL[kernel])
    outs = [torch.full(s.shape, float("nan"), dtype=torch.bfloat16, device="cuda") for s in walk.w.tensors]
    resid = None if resid0 is None else [r.clone() for r in resid0]
    cb.cb_extrapolate(walk.plan, t, outs, cb.CB_BF16, resid, cb.CB_BF16)
    torch.cuda.synchronize()
    assert cb.cb_plan_device_status(walk.plan) == 0
    return outs + (resid or [])


def _same_bits(a, b):
    return sum(int((x.view(torch.int16) != y.view(torch.int16)).sum()) for x, y in zip(a, b))


def _repeat(cb, H, walk, t, reps, fused=False, salt=0):
    """The oracle checks the first bulk launch; every further launch, and the
    direct kernel's, must write exactly the same bits."""
    resid0 = None
    rh = None
    if fused:
        resid0 = [workloads.hidden_state(walk.w, g, "cuda", salt=salt) for g in range(walk.n_groups)]
        rh = [H.host(resid0[g], walk._gidx(g)) for g in range(walk.n_groups)]
    first = _launch(cb, H, walk, t, "bulk", resid0)
    nt = len(walk.w.tensors)
    so, sr, _ = walk.expected_and_compare(t, first[:nt], first[nt:] if fused else None, rh)
    _assert_ok(so, ("repeat: first launch", t))
    if fused:
        _assert_ok(sr, ("repeat: first launch, hidden states", t))
    assert _same_bits(first, _launch(cb, H, walk, t, "direct", resid0)) == 0, "direct kernel differs"
    diffs = [_same_bits(first, _launch(cb, H, walk, t, "bulk", resid0)) for _ in range(reps)]
    assert not any(diffs), diffs
    cb.cb_plan_set_option(walk.plan, cb.CB_OPT_KERNEL, H.KERNEL["auto"])


def test_repeat_partial_history_step(cb, H):
    """PixArt/32 with no warm-up full steps, n = 2 live entries at step 5: a
    prediction-only launch of two CTAs per SM, 20 times over."""
    w = workloads.scaled(workloads.pixart(), 32)
    mask = H.library_schedule(w, 0)
    node_t = [t for s, t in enumerate(w.timesteps) if mask[s]]
    walk = H.Walk(w, node_t=node_t)
    cb.cb_plan_set_option(walk.plan, cb.CB_OPT_PARTIAL_HISTORY, 1)
    walk.push(w.timesteps[0], 0)
    walk.push(w.timesteps[3], 3)
    _repeat(cb, H, walk, w.timesteps[5], 20)
    walk.close()


@pytest.mark.parametrize("K", range(1, 9))
def test_repeat_prediction_only_shapes(cb, H, K):
    """Every prediction-only launch shape (K = 1..8) on PixArt/4 (48384 tiles,
    so every CTA cycles its stage ring many times), 20 launches each."""
    w = workloads.scaled(workloads.pixart(), 4)
    nodes = [999.0 - 45.0 * k for k in range(K)]
    walk = H.Walk(w, K=K, node_t=nodes, samples=4096, seed=K)
    for k, t in enumerate(nodes):
        walk.push(t, k)
    _repeat(cb, H, walk, nodes[-1] - 30.0, 20)
    walk.close()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("K,fused", [(1, False), (2, False), (3, True)])
def test_repeat_full_size_two_ctas_per_sm(cb, H, K, fused):
    """Full-size PixArt-Sigma 1024^2 shapes in the launches that run two CTAs
    per SM (K = 1 and 2 prediction-only; K = 3 with the hidden states fused),
    20 launches each."""
    w = workloads.pixart()
    nodes = [999.0 - 45.0 * k for k in range(K)]
    walk = H.Walk(w, K=K, node_t=nodes, samples=2048, seed=10 + K)
    for k, t in enumerate(nodes):
        walk.push(t, k)
        torch.cuda.empty_cache()
    _repeat(cb, H, walk, nodes[-1] - 30.0, 20, fused=fused, salt=K)
    walk.close()
    torch.cuda.empty_cache()


# --------------------------------------------- full-size, sampled outputs
FULL = {
    "dit256": (lambda: workloads.dit256(4), True),
    "dit256-k3": (lambda: workloads.dit256(3), True),
    "dit512": (workloads.dit512, False),
    "pixart": (workloads.pixart, False),
    "flux": (workloads.flux, False),
}


@pytest.mark.parametrize("name", list(FULL))
def test_full_size_sampled(cb, H, name):
    make, fused = FULL[name]
    w = make()
    walk = H.Walk(w, samples=2048, seed=len(name))
    mask, skipped = H.schedule_steps(w, w.K)
    full_steps = [s for s in range(w.T) if mask[s]]
    # every skipped step of the schedule (among them the first, one right after
    # the ring wraps, and the last)
    wrap = next(s for s in skipped if sum(1 for f in full_steps if f < s) > w.K)
    check = set(skipped)
    assert {skipped[0], wrap, skipped[-1]} <= check
    stats = []
    for s in range(w.T):
        t = w.timesteps[s]
        if mask[s]:
            walk.push(t, s)
        elif s in check:
            outs, resid, rh = walk.extrapolate(t, fused=fused, salt=s)
            so, sr, _ = walk.expected_and_compare(t, outs, resid, rh)
            _assert_ok(so, (name, "out", s))
            if fused:
                _assert_ok(sr, (name, "resid", s))
            stats.append(so)
            del outs, resid
    print(name, H.merge(stats))
    walk.close()
    torch.cuda.empty_cache()


# ------------------------------------------------------------ ring variant
def _odd_workload(K=4, cache="bf16"):
    numels = [1, 7, 8, 9, 4095, 4097, 8191, 12345, 40000]
    tensors = []
    for i, n in enumerate(numels):
        tensors.append(workloads.TensorSpec(i, 0, (1, 1, n), -1))
    # two residual groups of equal-sized members
    tensors += [workloads.TensorSpec(20, b, (2, 3, 1001), 0) for b in range(3)]
    tensors += [workloads.TensorSpec(21, b, (1, 16, 512), 1) for b in range(2)]
    return workloads.Workload(name="odd", tensors=tensors, K=K, cache_dtype=cache, T=0, r=0, t_min=0.0,
                              t_max=999.0, timesteps=[], degree=6, noise=0.1, seed=77)


def test_ring_variant_and_rotation_bit_exact(cb, H):
    w = _odd_workload()
    nodes = [980.0, 900.0, 820.0, 740.0]
    a = H.Walk(w, node_t=nodes)
    b = H.Walk(w, node_t=[999.0] + nodes)
    feats_extra = b.push(999.0, 0)
    for k, t in enumerate(nodes):
        f = a.push(t, k + 1)
        b.push(t, k + 1, feats=f)
    sa, ha, _ = cb.cb_plan_history(a.plan, 4)
    sb, hb, _ = cb.cb_plan_history(b.plan, 4)
    assert ha != hb  # the same logical history sits in rotated slots
    for t in (700.0, 655.5):
        oa, ra, _ = a.extrapolate(t, fused=True, salt=1)
        ob, rb, _ = b.extrapolate(t, fused=True, salt=1)
        oc, rc, _ = b.extrapolate(t, fused=True, salt=1, ring=(sb, hb))
        for x, y, z in zip(oa, ob, oc):
            assert torch.equal(x.view(torch.int16), y.view(torch.int16))
            assert torch.equal(x.view(torch.int16), z.view(torch.int16))
        for x, y, z in zip(ra, rb, rc):
            assert torch.equal(x.view(torch.int16), y.view(torch.int16))
            assert torch.equal(x.view(torch.int16), z.view(torch.int16))
    # a caller-described (shifted) history: relabel the slot times
    shifted = sb.copy()
    shifted[hb] = 1000.0  # the oldest entry now claims a different time
    oc, rc, rh = b.extrapolate(700.0, fused=True, salt=2, ring=(shifted, hb))
    times = [shifted[(hb + j) % 4] for j in range(4)]
    so, sr, _ = b.expected_and_compare(700.0, oc, rc, rh, times=times)
    _assert_ok(so, "ring-shifted out")
    _assert_ok(sr, "ring-shifted resid")
    a.close()
    b.close()
    del feats_extra


# ------------------------------------------------------------- edge cases
@pytest.mark.parametrize("kernel", ["direct", "bulk"])
@pytest.mark.parametrize("K,cache", [(1, "bf16"), (1, "fp32"), (2, "bf16"), (2, "fp32"), (3, "bf16"), (5, "bf16"),
                                     (6, "bf16"), (7, "fp32"), (8, "bf16"), (8, "fp32")])
def test_odd_sizes_every_element(cb, H, K, cache, kernel):
    w = _odd_workload(K, cache)
    nodes = [990.0 - 37.0 * k for k in range(K)]
    walk = H.Walk(w, node_t=nodes, kernel=kernel)
    for k, t in enumerate(nodes):
        walk.push(t, k)
    t = nodes[-1] - 20.0
    for out_dt in ("bf16", "fp32"):
        outs, _, _ = walk.extrapolate(t, out_dtype=out_dt)
        _assert_ok(walk.expected_and_compare(t, outs, None, None, out_dtype=out_dt)[0], (K, cache, out_dt))
    outs, resid, rh = walk.extrapolate(t, fused=True, salt=3)
    so, sr, _ = walk.expected_and_compare(t, outs, resid, rh)
    _assert_ok(so, "fused out")
    _assert_ok(sr, "fused resid")
    # hidden states only (no prediction outputs)
    _, resid, rh = walk.extrapolate(t, fused=True, outs=False, salt=4)
    _, sr, _ = walk.expected_and_compare(t, None, resid, rh)
    _assert_ok(sr, "resid only")
    walk.close()


@pytest.mark.parametrize("kernel", ["direct", "bulk"])
def test_misaligned_outputs_take_scalar_path(cb, H, kernel):
    w = _odd_workload(4)
    nodes = [950.0, 900.0, 850.0, 800.0]
    walk = H.Walk(w, node_t=nodes, kernel=kernel)
    for k, t in enumerate(nodes):
        walk.push(t, k)
    t = 760.0
    aligned, _, _ = walk.extrapolate(t)
    bufs = [torch.empty(s.numel + 1, dtype=torch.bfloat16, device="cuda") for s in w.tensors]
    outs = [b[1:] for b in bufs]  # 2-byte aligned, never 16-byte aligned
    cb.cb_extrapolate(walk.plan, t, outs, cb.CB_BF16)
    torch.cuda.synchronize()
    so, _, _ = walk.expected_and_compare(t, [o.view(s.shape) for o, s in zip(outs, w.tensors)], None, None)
    _assert_ok(so, "misaligned")
    with pytest.raises(cb.CbError) as e:
        cb.cb_extrapolate(walk.plan, t, [b.view(torch.uint8)[1:] for b in bufs], cb.CB_BF16)
    assert e.value.status == cb.CB_ERR_ALIGN
    walk.close()


def test_target_on_node_returns_cached_features(cb, H):
    w = _odd_workload(3)
    nodes = [900.0, 800.0, 700.0]
    walk = H.Walk(w, node_t=nodes)
    feats = [walk.push(t, k) for k, t in enumerate(nodes)]
    for k, t in enumerate(nodes):
        outs, _, _ = walk.extrapolate(t)
        for i in range(len(w.tensors)):
            assert torch.equal(outs[i].view(torch.int16), feats[k][i].view(torch.int16))
    walk.close()


@pytest.mark.parametrize("kernel", ["direct", "bulk"])
@pytest.mark.parametrize("cache", ["bf16", "fp32"])
def test_cancellation_stress(cb, H, cache, kernel):
    """Histories whose extrapolation nearly cancels (|P| << sum |w F|), which
    sends elements through the compensated fallback of the fast path.

    fp32 cache: the newest entry is solved for P ~ 0 and rounded to fp32, so
    |P| ~ 2^-24 sum|w F|. bf16 cache: the two newest entries are searched over
    neighbouring bf16 values for the smallest |P|. Only even elements are
    constructed this way; odd ones stay random."""
    K = 5
    n = 1 << 15
    tensors = [workloads.TensorSpec(0, 0, (1, 1, n), 0), workloads.TensorSpec(0, 1, (1, 1, n), 0)]
    w = workloads.Workload(name="cancel", tensors=tensors, K=K, cache_dtype=cache, T=0, r=0, t_min=0.0,
                           t_max=1.0, timesteps=[])
    nodes = [0.9, 0.8, 0.7, 0.6, 0.5]
    tq = 0.43
    wt = orc.weights(nodes, tq, 0.0, 1.0)
    rng = np.random.default_rng(31)
    walk = H.Walk(w, node_t=nodes, kernel=kernel)
    F = rng.standard_normal((2, K, n))
    if cache == "fp32":
        F = F.astype(np.float32).astype(np.float64)
        F[:, K - 1, 0::2] = (-(np.einsum("j,bjn->bn", wt[:K - 1], F[:, :K - 1, 0::2])) / wt[K - 1]).astype(np.float32)
        vals = F.astype(np.float32)
    else:
        Fb = H.bf16_to_f64(orc.convert(F.ravel(), orc.FP64, orc.BF16)).reshape(F.shape)
        base = np.einsum("j,bjn->bn", wt[:K - 2], Fb[:, :K - 2, 0::2])
        a_ideal = -(base + wt[K - 1] * Fb[:, K - 1, 0::2]) / wt[K - 2]
        Fb[:, K - 2, 0::2] = H.bf16_to_f64(orc.convert(a_ideal.ravel(), orc.FP64, orc.BF16)).reshape(a_ideal.shape)
        best = np.full(base.shape, np.inf)
        pick_a = Fb[:, K - 2, 0::2].copy()
        pick_b = Fb[:, K - 1, 0::2].copy()
        for da in range(-6, 7):
            ca = H.bf16_to_f64(H._step(orc.convert(Fb[:, K - 2, 0::2].ravel(), orc.FP64, orc.BF16), da)).reshape(base.shape)
            for db in range(-6, 7):
                cbv = H.bf16_to_f64(H._step(orc.convert(Fb[:, K - 1, 0::2].ravel(), orc.FP64, orc.BF16), db)).reshape(base.shape)
                r = np.abs(base + wt[K - 2] * ca + wt[K - 1] * cbv)
                better = r < best
                best = np.where(better, r, best)
                pick_a = np.where(better, ca, pick_a)
                pick_b = np.where(better, cbv, pick_b)
        Fb[:, K - 2, 0::2] = pick_a
        Fb[:, K - 1, 0::2] = pick_b
        vals = Fb
    tdt = torch.float32 if cache == "fp32" else torch.bfloat16
    for k in range(K):
        feats = [torch.from_numpy(np.ascontiguousarray(vals[b, k])).to(torch.float64).to(tdt).cuda().view(1, 1, n)
                 for b in range(2)]
        walk.push(nodes[k], k, feats=feats)
    Fd = vals.astype(np.float64)
    P = np.einsum("j,bjn->bn", wt, Fd)
    S = np.einsum("j,bjn->bn", np.abs(wt), np.abs(Fd))
    ratio = np.abs(P[:, 0::2]) / S[:, 0::2]
    assert np.median(ratio) < 2.0 ** -12  # the constructed elements really cancel
    for fused in (False, True):
        outs, resid, rh = walk.extrapolate(tq, fused=fused, salt=7)
        so, sr, _ = walk.expected_and_compare(tq, outs, resid, rh)
        _assert_ok(so, ("cancel out", cache, fused))
        if fused:
            _assert_ok(sr, ("cancel resid", cache))
        print("cancellation", cache, fused, so, sr)
    walk.close()


def test_nothing_requested_is_a_no_op(cb, H):
    w = _odd_workload(2)
    walk = H.Walk(w, node_t=[900.0, 800.0])
    walk.push(900.0, 0)
    walk.push(800.0, 1)
    cb.cb_extrapolate(walk.plan, 700.0, None, cb.CB_BF16)
    cb.cb_extrapolate(walk.plan, 700.0, [None] * len(w.tensors), cb.CB_BF16, [None, None], cb.CB_BF16)
    torch.cuda.synchronize()
    walk.close()


def test_side_stream_and_graph_replay(cb, H):
    w = _odd_workload(4)
    nodes = [950.0, 900.0, 850.0, 800.0]
    walk = H.Walk(w, node_t=nodes)
    for k, t in enumerate(nodes):
        walk.push(t, k)
    t = 740.0
    ref, _, _ = walk.extrapolate(t)
    s = torch.cuda.Stream()
    outs = [torch.zeros_like(o) for o in ref]
    with torch.cuda.stream(s):
        cb.cb_extrapolate(walk.plan, t, outs, cb.CB_BF16, stream=s)
    s.synchronize()
    for a, b in zip(ref, outs):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    # capture the skipped step in a CUDA graph and replay it
    outs2 = [torch.zeros_like(o) for o in ref]
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        cb.cb_extrapolate(walk.plan, t, outs2, cb.CB_BF16, stream=torch.cuda.current_stream())
    graph.replay()
    torch.cuda.synchronize()
    for a, b in zip(ref, outs2):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    walk.close()


def test_reset_and_history_errors(cb, H):
    w = _odd_workload(2)
    walk = H.Walk(w, node_t=[900.0, 800.0])
    walk.push(900.0, 0)
    with pytest.raises(cb.CbError) as e:
        walk.extrapolate(700.0)
    assert e.value.status == cb.CB_ERR_HISTORY_NOT_FULL
    walk.push(800.0, 1)
    walk.extrapolate(700.0)
    cb.cb_plan_reset(walk.plan)
    assert cb.cb_plan_history(walk.plan, 2)[2] == 0
    with pytest.raises(cb.CbError):
        cb.cb_weights(walk.plan, 700.0, 2)
    walk.close()


# ------------------------------------------------- kernel variants, wait limit
@pytest.mark.parametrize("name", ["flux", "dit256"])
def test_direct_and_bulk_kernels_bit_identical(cb, H, name):
    """Both skipped-step kernels run the same arithmetic: identical bits on a
    full-size workload (outputs, and the fused hidden states on DiT-256)."""
    w = workloads.flux() if name == "flux" else workloads.dit256(4)
    walk = H.Walk(w)
    mask, skipped = H.schedule_steps(w, w.K)
    s_stop = skipped[len(skipped) // 2]
    for s in range(s_stop):
        if mask[s]:
            walk.push(w.timesteps[s], s, )
    t = w.timesteps[s_stop]
    res = {}
    for kern in ("direct", "bulk"):
        cb.cb_plan_set_option(walk.plan, cb.CB_OPT_KERNEL, H.KERNEL[kern])
        outs, resid, _ = walk.extrapolate(t, fused=(name == "dit256"), salt=5)
        res[kern] = (outs, resid)
    for a, b in zip(res["direct"][0], res["bulk"][0]):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    if name == "dit256":
        for a, b in zip(res["direct"][1], res["bulk"][1]):
            assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    walk.close()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("K,fused", [(4, False), (2, False), (3, True)])
def test_bulk_wait_limit_reports_and_recovers(cb, H, K, fused):
    """The failure path of the bulk kernel's bounded waits, without a fault: the
    producer announces every CTA's first unit but never issues its copies (a
    flag that nothing sets), so the consumers' wait runs out after the limit.
    The kernel must record it in the status word and return; the context stays
    usable and the next launch is correct and clean. Shapes: predictions only
    with one CTA per SM (K = 4) and with two (K = 2), hidden states fused with
    two CTAs per SM (K = 3)."""
    import time
    w = workloads.scaled(workloads.pixart(), 16)
    nodes = [999.0 - 45.0 * k for k in range(K)]
    walk = H.Walk(w, K=K, node_t=nodes, kernel="bulk")
    for k, t in enumerate(nodes):
        walk.push(t, k)
    t = nodes[-1] - 30.0
    outs = [torch.empty(s.shape, dtype=torch.bfloat16, device="cuda") for s in w.tensors]
    resid = [workloads.hidden_state(w, g, "cuda") for g in range(walk.n_groups)] if fused else None
    cb.cb_plan_set_option(walk.plan, cb.CB_OPT_WAIT_NS, 20_000_000)  # 20 ms
    cb.cb_plan_set_option(walk.plan, cb.CB_OPT_TEST_WITHHOLD, 1)
    t0 = time.perf_counter()
    cb.cb_extrapolate(walk.plan, t, outs, cb.CB_BF16, resid, cb.CB_BF16)
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    st = cb.cb_plan_device_status(walk.plan)
    assert st & cb.CB_DEV_CONSUMER_TIMEOUT, st
    assert st & cb.CB_DEV_PRODUCER_TIMEOUT, st
    assert elapsed < 5.0
    assert cb.cb_plan_device_status(walk.plan) == 0  # the read cleared it
    cb.cb_plan_set_option(walk.plan, cb.CB_OPT_TEST_WITHHOLD, 0)
    cb.cb_plan_set_option(walk.plan, cb.CB_OPT_WAIT_NS, 10 ** 9)
    outs, resid, rh = walk.extrapolate(t, fused=fused, salt=K)
    so, sr, _ = walk.expected_and_compare(t, outs, resid, rh)
    _assert_ok(so, ("after timeout", K))
    if fused:
        _assert_ok(sr, ("after timeout, hidden states", K))
    walk.close()


def test_element_offsets_beyond_2_31(cb, H):
    """One tensor of 2^31 + 12345 elements (4.3 GB per slot in bf16, a ragged
    last tile): the kernels' 64-bit element offsets, checked on sampled
    elements including both ends and the 2^31 boundary, both kernels."""
    n = (1 << 31) + 12345
    w = workloads.Workload(name="huge", tensors=[workloads.TensorSpec(0, 0, (1, 1, n), -1)], K=2,
                           cache_dtype="bf16", T=0, r=0, t_min=0.0, t_max=999.0, timesteps=[], degree=1,
                           noise=0.0, seed=71)
    nodes = [900.0, 850.0]
    for kernel in ("bulk", "direct"):
        walk = H.Walk(w, node_t=nodes, kernel=kernel)
        g = torch.Generator().manual_seed(3)
        pick = torch.randint(0, n, (4096,), generator=g, dtype=torch.int64)
        extra = torch.tensor([0, 1, (1 << 31) - 9, (1 << 31) - 1, 1 << 31, (1 << 31) + 7, n - 12345, n - 4096,
                              n - 1], dtype=torch.int64)
        walk.idx = [torch.unique(torch.cat([pick, extra])).to("cuda")]
        for k, t in enumerate(nodes):
            walk.push(t, k)
            torch.cuda.empty_cache()
        outs, _, _ = walk.extrapolate(810.0)
        so, _, _ = walk.expected_and_compare(810.0, outs, None, None)
        _assert_ok(so, ("huge", kernel))
        del outs
        walk.close()
        del walk
        torch.cuda.empty_cache()
