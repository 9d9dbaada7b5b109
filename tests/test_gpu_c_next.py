"""GPU parity for the widened rows: partial history during warm-up, caller-given
weights (other node families, truncated Taylor), and a non-affine schedule.

Same gates as test_gpu_a_parity.py: within one bf16 ulp of the oracle's fp64
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
    mask = H.library_schedule(w, 0)  # the set F alone (no warm-up rule)
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
        if n < w.K:  # a count other than the live entries' is refused, not truncated or padded
            for call in (lambda: cb.cb_weights(walk.plan, t, n + 1),
                         lambda: cb.cb_extrapolate_weights(walk.plan, np.full(n + 1, 1.0 / (n + 1)), None,
                                                           cb.CB_BF16)):
                with pytest.raises(cb.CbError) as e:
                    call()
                assert e.value.status == cb.CB_ERR_ARG
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


def _gates(w, dtype, seed, skip=()):
    g = torch.Generator(device="cuda").manual_seed(seed)
    out = []
    for i, t in enumerate(w.tensors):
        if i in skip:
            out.append(None)
            continue
        b, _, h = t.shape
        out.append((0.5 * torch.randn(b, h, generator=g, device="cuda")).to(dtype))
    return out


@pytest.mark.parametrize("kernel", ["bulk", "direct"])
@pytest.mark.parametrize("resid_dtype", ["bf16", "fp32"])
def test_gated_residual(cb, H, kernel, resid_dtype):
    """x <- x + sum_b g_b * P_b with per-(batch, channel) gates broadcast over
    tokens (a DiT block's adaLN gates applied to the un-gated cached outputs)."""
    w = workloads.scaled(workloads.dit256(4), 8)
    nodes = [w.timesteps[s] for s in (4, 8, 12, 16)]
    walk = H.Walk(w, node_t=nodes, kernel=kernel)
    cb.cb_plan_set_shapes(walk.plan, [t.shape for t in w.tensors])
    for k, t in enumerate(nodes):
        walk.push(t, k)
    t = w.timesteps[18]
    gates = _gates(w, torch.bfloat16, 11, skip={3, 10})
    outs, resid, rh = walk.extrapolate(t, fused=True, gates=gates, resid_dtype=resid_dtype, salt=9)
    G = [None if g is None else H.expand_gate(g, s.shape) for g, s in zip(gates, w.tensors)]
    so, sr, _ = walk.expected_and_compare(t, outs, resid, rh, resid_dtype=resid_dtype, G=G)
    _ok(so, "gated outs")
    _ok(sr, ("gated resid", resid_dtype))
    print("gated", kernel, resid_dtype, sr)
    # gates of None everywhere: the gated entry equals cb_extrapolate bit for bit
    a, ra, _ = walk.extrapolate(t, fused=True, salt=4)
    b_, rb, _ = walk.extrapolate(t, fused=True, salt=4, gates=[None] * len(w.tensors))
    for x, y in zip(ra, rb):
        assert torch.equal(x.view(torch.int16), y.view(torch.int16))
    walk.close()


def test_gated_residual_odd_shapes(cb, H):
    """Hidden sizes that are not multiples of 8 (scalar path), fp32 gates."""
    from test_gpu_a_parity import _odd_workload
    w = _odd_workload(4)
    nodes = [950.0, 900.0, 850.0, 800.0]
    walk = H.Walk(w, node_t=nodes)
    cb.cb_plan_set_shapes(walk.plan, [t.shape for t in w.tensors])
    for k, t in enumerate(nodes):
        walk.push(t, k)
    gates = _gates(w, torch.float32, 12)
    outs, resid, rh = walk.extrapolate(760.0, fused=True, gates=gates, gate_dtype="fp32", salt=2)
    G = [H.expand_gate(g, s.shape) for g, s in zip(gates, w.tensors)]
    so, sr, _ = walk.expected_and_compare(760.0, outs, resid, rh, G=G)
    _ok(so, "odd gated outs")
    _ok(sr, "odd gated resid")
    walk.close()


# Gate-row cases of the bulk kernel's gate staging: batch rows that are not a
# whole number of 4096-element tiles (a tile takes two gate rows), rows shorter
# than a tile (gates stay in global memory), and hidden sizes whose two gate
# rows fill (bf16) or overflow (fp32) the 32 KB staging limit.
_GATE_CASES = {
    "cross": [(4, 40, 1152)] * 3 + [(3, 24, 1024)] * 2,
    "short": [(8, 2, 1152)] * 2 + [(5, 3, 512)] * 2,
    "wide": [(2, 3, 8192)] * 2,
}


@pytest.mark.parametrize("case", sorted(_GATE_CASES))
@pytest.mark.parametrize("gate_dtype", ["bf16", "fp32"])
def test_gated_gate_rows(cb, H, case, gate_dtype):
    shapes = _GATE_CASES[case]
    groups = {}
    tensors = []
    for i, sh in enumerate(shapes):
        g = groups.setdefault(sh, len(groups))
        tensors.append(workloads.TensorSpec(g, i, sh, g))
    w = workloads.Workload(name=f"gate-rows-{case}", tensors=tensors, K=4, cache_dtype="bf16", T=0, r=0,
                           t_min=0.0, t_max=999.0, timesteps=[], degree=6, noise=0.1, seed=91)
    nodes = [960.0, 900.0, 840.0, 780.0]
    for kernel in ("bulk", "direct"):
        walk = H.Walk(w, node_t=nodes, kernel=kernel)
        cb.cb_plan_set_shapes(walk.plan, [t.shape for t in w.tensors])
        for k, t in enumerate(nodes):
            walk.push(t, k)
        gates = _gates(w, H.TORCH[gate_dtype], 31, skip={1})
        outs, resid, rh = walk.extrapolate(735.0, fused=True, gates=gates, gate_dtype=gate_dtype, salt=5)
        G = [None if g is None else H.expand_gate(g, s.shape) for g, s in zip(gates, w.tensors)]
        so, sr, _ = walk.expected_and_compare(735.0, outs, resid, rh, G=G)
        _ok(so, (case, kernel, "outs"))
        _ok(sr, (case, kernel, "resid"))
        walk.close()


@pytest.mark.parametrize("K", [1, 2, 3, 6, 8])
def test_gated_every_history_size(cb, H, K):
    """The gated kernels at every history size class (one and two CTAs per SM,
    with and without spilled registers), both kernels, staged gate rows."""
    shapes = _GATE_CASES["cross"]
    groups = {}
    tensors = []
    for i, sh in enumerate(shapes):
        g = groups.setdefault(sh, len(groups))
        tensors.append(workloads.TensorSpec(g, i, sh, g))
    w = workloads.Workload(name=f"gated-k{K}", tensors=tensors, K=K, cache_dtype="bf16", T=0, r=0,
                           t_min=0.0, t_max=999.0, timesteps=[], degree=6, noise=0.1, seed=92 + K)
    nodes = [980.0 - 41.0 * k for k in range(K)]
    for kernel in ("bulk", "direct"):
        walk = H.Walk(w, node_t=nodes, kernel=kernel)
        cb.cb_plan_set_shapes(walk.plan, [t.shape for t in w.tensors])
        for k, t in enumerate(nodes):
            walk.push(t, k)
        gates = _gates(w, torch.bfloat16, 40 + K, skip={2})
        t = nodes[-1] - 25.0
        outs, resid, rh = walk.extrapolate(t, fused=True, gates=gates, salt=K)
        G = [None if g is None else H.expand_gate(g, s.shape) for g, s in zip(gates, w.tensors)]
        so, sr, _ = walk.expected_and_compare(t, outs, resid, rh, G=G)
        _ok(so, (K, kernel, "outs"))
        _ok(sr, (K, kernel, "resid"))
        walk.close()


@pytest.mark.parametrize("src", ["fp32", "bf16"])
@pytest.mark.parametrize("odd", [False, True])
@pytest.mark.parametrize("kernel", ["auto", "bulk", "direct"])
def test_push_residual(cb, H, src, odd, kernel):
    """Full step with the fused epilogue (auto: its own kernel; bulk, direct:
    the skipped-step kernels on a one-entry history): the slots hold exactly
    what the plain push writes, and x <- x + sum_b g_b f_b (un-rounded
    features) matches the oracle's single rounding."""
    from test_gpu_a_parity import _odd_workload
    w = _odd_workload(3) if odd else workloads.scaled(workloads.pixart(), 32)
    w.cache_dtype = "bf16"
    nodes = [900.0, 800.0, 700.0]
    a = H.Walk(w, K=3, node_t=nodes, kernel=kernel)
    b = H.Walk(w, K=3, node_t=nodes)
    cb.cb_plan_set_shapes(a.plan, [t.shape for t in w.tensors])
    tdt = torch.float32 if src == "fp32" else torch.bfloat16
    for k, t in enumerate(nodes):
        feats = [workloads.trajectory(w, i, t, k, "cuda", out_dtype=tdt) for i in range(len(w.tensors))]
        gates = _gates(w, torch.bfloat16, 20 + k, skip={0})
        resid = [workloads.hidden_state(w, g, "cuda", salt=k) for g in range(a.n_groups)]
        rh = [H.host(r) for r in resid]
        cb.cb_cache_push_residual(a.plan, feats, H.CB[src], t, resid, cb.CB_BF16, gates, cb.CB_BF16)
        cb.cb_cache_push(b.plan, feats, H.CB[src], t)
        torch.cuda.synchronize()
        # the slot just written holds identical bytes (padding and unwritten slots are not compared)
        offs, slot = H.slot_layout([s_.numel for s_ in w.tensors], 2)
        for i, s_ in enumerate(w.tensors):
            lo = k * slot + offs[i]
            assert torch.equal(a.cache[lo:lo + 2 * s_.numel], b.cache[lo:lo + 2 * s_.numel]), (k, i)
        for g in range(a.n_groups):
            members = [i for i, s in enumerate(w.tensors) if s.group == g]
            F = [[H.host(feats[i])] for i in members]
            G = [None if gates[i] is None else H.expand_gate(gates[i], w.tensors[i].shape) for i in members]
            _, r64 = orc.extrapolate(F, [1.0], H.ORC[src], None, X=rh[g], x_dtype=orc.BF16,
                                     resid_dtype=orc.FP64, G=G)
            ref = orc.convert(r64, orc.FP64, orc.BF16)
            Fd = np.array([f[0].astype(np.float64) if src == "fp32" else H.bf16_to_f64(f[0]) for f in F])
            gb = np.array([np.ones_like(Fd[0]) if x is None else np.abs(x) for x in G])
            bound = (gb * np.abs(Fd)).sum(0) + np.abs(H.bf16_to_f64(rh[g]))
            st = H.compare_bf16(H.host(resid[g]), ref, r64, bound)
            assert st["bad"] == 0, (g, st)
            assert st["exact"] >= 0.99 * st["n"], st  # compensated sum: rounded once, like the oracle
    a.close()
    b.close()


@pytest.mark.parametrize("src", ["fp32", "bf16"])
@pytest.mark.parametrize("gated", [False, True])
@pytest.mark.parametrize("layout", ["groups-of-3", "pairs"])
def test_push_residual_kernels_bit_identical(cb, H, src, gated, layout):
    """The kernels that can run a full step's epilogue write the same slot
    bytes and the same hidden-state bits (one shared arithmetic). Every tensor
    sits in a group of three branches (with bf16 features and no gates the
    default then picks the epilogue kernel), or every item has one or two
    (groups of two and lone tensors: the bulk kernel): whole tiles, ragged
    tiles (6006 elements) and a hidden state off the 16-byte grid (scalar
    path). In the
    ragged last tile of a tensor the bulk kernel computes every element by the
    compensated path while the others take the guarded fast path vector by
    vector, so there the bulk kernel is held to the oracle's gate only."""
    nbr = 3 if layout == "groups-of-3" else 2
    tensors = [workloads.TensorSpec(0, b, (2, 3, 1001), 0) for b in range(nbr)]
    tensors += [workloads.TensorSpec(1, b, (2, 128, 1152), 1) for b in range(nbr)]
    tensors += [workloads.TensorSpec(2, b, (1, 7, 64), 2) for b in range(nbr)]
    if layout == "pairs":  # lone tensors: items of one member without a hidden state
        tensors += [workloads.TensorSpec(3 + i, 0, (1, 1, n), -1) for i, n in enumerate([1, 4097, 40000])]
    w = workloads.Workload(name="groups-of-3", tensors=tensors, K=3, cache_dtype="bf16", T=0, r=0, t_min=0.0,
                           t_max=999.0, timesteps=[], degree=6, noise=0.1, seed=55)
    nodes = [900.0, 800.0, 700.0]
    walks = {k: H.Walk(w, K=3, node_t=nodes, kernel=k) for k in ("auto", "bulk", "direct")}
    for wk in walks.values():
        cb.cb_plan_set_shapes(wk.plan, [t.shape for t in w.tensors])
    tdt = torch.float32 if src == "fp32" else torch.bfloat16
    ng = walks["auto"].n_groups
    offs, slot = H.slot_layout([s_.numel for s_ in w.tensors], 2)
    for k, t in enumerate(nodes):
        feats = [workloads.trajectory(w, i, t, k, "cuda", out_dtype=tdt) for i in range(len(w.tensors))]
        gates = _gates(w, torch.bfloat16, 40 + k, skip={1}) if gated else None
        out = {}
        for name, wk in walks.items():
            resid = [workloads.hidden_state(w, g, "cuda", salt=k) for g in range(ng)]
            x2 = resid[2].reshape(-1)
            shifted = torch.empty(x2.numel() + 1, dtype=x2.dtype, device="cuda")[1:]  # 2 bytes off the grid
            shifted.copy_(x2)
            resid[2] = shifted
            cb.cb_cache_push_residual(wk.plan, feats, H.CB[src], t, resid, cb.CB_BF16, gates, cb.CB_BF16)
            torch.cuda.synchronize()
            assert cb.cb_plan_device_status(wk.plan) == 0
            out[name] = resid
        # the default runs the epilogue kernel for ungated bf16 features in groups of three, else the bulk kernel
        epi = src == "bf16" and not gated and layout == "groups-of-3"
        ran = {"auto": "epilogue" if epi else "bulk", "bulk": "bulk", "direct": "direct"}
        for name in ("bulk", "direct"):
            for i, s_ in enumerate(w.tensors):  # the slot just written (padding and other slots are not)
                lo = k * slot + offs[i]
                assert torch.equal(walks["auto"].cache[lo:lo + 2 * s_.numel], walks[name].cache[lo:lo + 2 * s_.numel]), \
                    (k, name, i)
            for g in range(ng):
                a_, b_ = out["auto"][g].reshape(-1).view(torch.int16), out[name][g].reshape(-1).view(torch.int16)
                if (ran["auto"] == "bulk") != (ran[name] == "bulk"):  # the bulk kernel's whole tiles only
                    te = 4096 if src == "bf16" else 2048
                    whole = a_.numel() // te * te
                    a_, b_ = a_[:whole], b_[:whole]
                assert torch.equal(a_, b_), (k, name, g)
            # the bulk kernel's hidden states, whole and ragged tiles, against the oracle
            for g in range(ng):
                members = [i for i, s_ in enumerate(w.tensors) if s_.group == g]
                F = [[H.host(feats[i])] for i in members]
                G = None if gates is None else [None if gates[i] is None else H.expand_gate(gates[i],
                                                                                            w.tensors[i].shape)
                                                for i in members]
                x0 = H.host(workloads.hidden_state(w, g, "cuda", salt=k))
                _, r64 = orc.extrapolate(F, [1.0], H.ORC[src], None, X=x0, x_dtype=orc.BF16, resid_dtype=orc.FP64,
                                         G=G)
                Fd = np.array([f[0].astype(np.float64) if src == "fp32" else H.bf16_to_f64(f[0]) for f in F])
                gb = np.array([np.ones_like(Fd[0]) if (G is None or x is None) else np.abs(x)
                               for x in (G or [None] * len(members))])
                bound = (gb * np.abs(Fd)).sum(0) + np.abs(H.bf16_to_f64(x0))
                st = H.compare_bf16(H.host(out[name][g]), orc.convert(r64, orc.FP64, orc.BF16), r64, bound)
                assert st["bad"] == 0, (k, name, g, st)
        # and against the oracle's single rounding
        for g in range(ng):
            members = [i for i, s_ in enumerate(w.tensors) if s_.group == g]
            F = [[H.host(feats[i])] for i in members]
            G = None if gates is None else [None if gates[i] is None else H.expand_gate(gates[i], w.tensors[i].shape)
                                            for i in members]
            x0 = H.host(workloads.hidden_state(w, g, "cuda", salt=k))
            _, r64 = orc.extrapolate(F, [1.0], H.ORC[src], None, X=x0, x_dtype=orc.BF16, resid_dtype=orc.FP64, G=G)
            Fd = np.array([f[0].astype(np.float64) if src == "fp32" else H.bf16_to_f64(f[0]) for f in F])
            gb = np.array([np.ones_like(Fd[0]) if (G is None or x is None) else np.abs(x)
                           for x in (G or [None] * len(members))])
            bound = (gb * np.abs(Fd)).sum(0) + np.abs(H.bf16_to_f64(x0))
            st = H.compare_bf16(H.host(out["auto"][g]), orc.convert(r64, orc.FP64, orc.BF16), r64, bound)
            assert st["bad"] == 0, (k, g, st)
    for wk in walks.values():
        wk.close()


@pytest.mark.parametrize("src", ["fp32", "bf16"])
@pytest.mark.parametrize("kernel", ["auto", "bulk", "direct"])
@pytest.mark.parametrize("layout", ["groups-of-3", "pairs"])
def test_push_residual_cancellation(cb, H, src, kernel, layout):
    """Full-step epilogue where the hidden-state update cancels. Group 0: the
    first member's features are -x plus a residue, so x + sum_b f_b is a
    residue of the terms. Group 1: a small hidden state (~1e-6) and members a,
    b, -(a + b) + residue, which cancel among themselves (the fp32 sum a + b
    is rounded, so the fast path is off by many bf16 ulps, and only the
    members' part of the guard can see it). With pairs (groups of two) the
    members are -x + residue and a residue, then a and -a + residue. Every
    element must still be within one ulp of the oracle."""
    nbr = 3 if layout == "groups-of-3" else 2
    tensors = [workloads.TensorSpec(g, b, (2, 64, 1152), g) for g in range(2) for b in range(nbr)]
    w = workloads.Workload(name="cancel", tensors=tensors, K=2, cache_dtype="bf16", T=0, r=0, t_min=0.0,
                           t_max=999.0, timesteps=[], degree=6, noise=0.1, seed=57)
    walk = H.Walk(w, K=2, node_t=[900.0, 800.0], kernel=kernel)
    ng = walk.n_groups
    gen = torch.Generator(device="cuda").manual_seed(5)
    tdt = torch.float32 if src == "fp32" else torch.bfloat16
    small = 1e-6 if src == "fp32" else 1e-3  # a bf16 residue cannot be smaller than ~ulp(x)
    shape = w.tensors[0].shape
    resid = [workloads.hidden_state(w, 0, "cuda"),
             (1e-6 * torch.randn(shape, generator=gen, device="cuda")).to(torch.bfloat16)]
    rh = [H.host(r) for r in resid]
    x0 = resid[0].float()
    a = torch.randn(shape, generator=gen, device="cuda").to(tdt).float()
    b = torch.randn(shape, generator=gen, device="cuda").to(tdt).float()
    def residue():
        return small * torch.randn(shape, generator=gen, device="cuda")
    if nbr == 3:
        feats = [-x0 + residue(), residue(), residue(), a, b, -(a.double() + b.double()).float() + residue()]
    else:
        feats = [-x0 + residue(), residue(), a, -a + residue()]
    feats = [f.to(tdt) for f in feats]
    cb.cb_cache_push_residual(walk.plan, feats, H.CB[src], 900.0, resid, cb.CB_BF16)
    torch.cuda.synchronize()
    assert cb.cb_plan_device_status(walk.plan) == 0
    for g in range(ng):
        members = [i for i, s_ in enumerate(w.tensors) if s_.group == g]
        F = [[H.host(feats[i])] for i in members]
        _, r64 = orc.extrapolate(F, [1.0], H.ORC[src], None, X=rh[g], x_dtype=orc.BF16, resid_dtype=orc.FP64)
        Fd = np.array([f[0].astype(np.float64) if src == "fp32" else H.bf16_to_f64(f[0]) for f in F])
        bound = np.abs(Fd).sum(0) + np.abs(H.bf16_to_f64(rh[g]))
        st = H.compare_bf16(H.host(resid[g]), orc.convert(r64, orc.FP64, orc.BF16), r64, bound)
        assert st["bad"] == 0, (g, st)
        if src == "fp32":  # the case is what it claims: the update cancels for most elements
            assert np.median(np.abs(r64) / bound) < 1e-4, g
    walk.close()


@pytest.mark.parametrize("layout", ["lone", "groups"])
def test_maximum_plan(cb, H, layout):
    """A plan at the ABI's limits: CB_MAX_TENSORS tensors and CB_MAX_K history
    entries, either 256 lone tensors (256 work items) or 64 residual groups of
    CB_MAX_BRANCHES members with gated hidden states; both kernels, every
    element against the oracle."""
    rng = np.random.default_rng(31)
    n = cb.CB_MAX_TENSORS
    tensors = []
    if layout == "lone":
        for i in range(n):
            tensors.append(workloads.TensorSpec(i, 0, (1, int(rng.integers(1, 40)), 64), -1))
    else:
        for g in range(n // 4):
            sh = (int(rng.integers(1, 3)), int(rng.integers(1, 30)), int(rng.choice([64, 40])))
            tensors += [workloads.TensorSpec(g, m, sh, g) for m in range(4)]
    K = 8
    w = workloads.Workload(name=f"max-{layout}", tensors=tensors, K=K, cache_dtype="bf16", T=0, r=0,
                           t_min=0.0, t_max=999.0, timesteps=[], degree=6, noise=0.1, seed=313)
    nodes = [990.0 - 30.0 * k for k in range(K)]
    for kernel in ("bulk", "direct"):
        walk = H.Walk(w, node_t=nodes, kernel=kernel)
        cb.cb_plan_set_shapes(walk.plan, [t.shape for t in w.tensors])
        for k, t in enumerate(nodes):
            walk.push(t, k)
        t = nodes[-1] - 20.0
        if layout == "lone":
            outs, _, _ = walk.extrapolate(t)
            so, _, _ = walk.expected_and_compare(t, outs, None, None)
            _ok(so, (layout, kernel))
        else:
            gates = _gates(w, torch.bfloat16, 77)
            outs, resid, rh = walk.extrapolate(t, fused=True, gates=gates, salt=3)
            G = [H.expand_gate(g, s.shape) for g, s in zip(gates, w.tensors)]
            so, sr, _ = walk.expected_and_compare(t, outs, resid, rh, G=G)
            _ok(so, (layout, kernel, "outs"))
            _ok(sr, (layout, kernel, "resid"))
        walk.close()
