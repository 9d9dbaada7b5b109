"""Randomised GPU parity: many small seeded workloads that mix every launch
shape of the skipped-step kernels (history size K = 1..8, bf16 and fp32
caches, aligned and ragged hidden sizes, lone tensors and residual groups of
1..4 members, bf16 and fp32 predictions and hidden states, gates staged or
read from global memory, partial history, both kernels), each compared with
the oracle element by element (Sec. 3.3, Eq. for f_t; Sec. 3.1 residual).

Same gates as test_gpu_a_parity.py: bf16 within one ulp of the oracle's fp64
result rounded to bf16 (exact cancellations below 2^-40 sum|w F| counted
apart), fp32 within 2e-6 max|F|.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2608_23429_gb300 import workloads

pytestmark = pytest.mark.gpu

N_CASES = 64


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


def _random_case(seed: int):
    """A small workload: a few residual groups plus lone tensors, random shapes."""
    rng = np.random.default_rng(1000 + seed)
    K = int(rng.integers(1, 9))
    cache = "bf16" if rng.random() < 0.7 else "fp32"
    tensors = []
    n_groups = int(rng.integers(1, 4))
    for g in range(n_groups):
        b = int(rng.integers(1, 4))
        t = int(rng.integers(1, 48))
        h = int(rng.choice([64, 128, 512, 1152, 96, 7, 33, 1000]))
        nb = int(rng.integers(1, 5))
        tensors += [workloads.TensorSpec(g, m, (b, t, h), g) for m in range(nb)]
    for j in range(int(rng.integers(0, 3))):
        tensors.append(workloads.TensorSpec(10 + j, 0, (1, int(rng.integers(1, 20)), int(rng.choice([8, 17, 256]))), -1))
    w = workloads.Workload(name=f"random-{seed}", tensors=tensors, K=K, cache_dtype=cache, T=0, r=0, t_min=0.0,
                           t_max=999.0, timesteps=[], degree=6, noise=0.1, seed=500 + seed)
    spacing = float(rng.uniform(15.0, 60.0))
    nodes = [990.0 - spacing * k for k in range(K)]
    opts = dict(
        kernel=str(rng.choice(["bulk", "direct"])),
        out_dtype=str(rng.choice(["bf16", "fp32"])),
        resid_dtype="bf16" if rng.random() < 0.75 else "fp32",
        gated=bool(rng.random() < 0.5),
        gate_dtype="bf16" if rng.random() < 0.7 else "fp32",
        partial=bool(K > 1 and rng.random() < 0.3),
        target=nodes[-1] - float(rng.uniform(0.2, 1.5)) * spacing,
    )
    return w, nodes, opts


@pytest.mark.parametrize("seed", range(N_CASES))
def test_random_workload(cb, H, seed):
    w, nodes, o = _random_case(seed)
    walk = H.Walk(w, node_t=nodes, kernel=o["kernel"])
    cb.cb_plan_set_shapes(walk.plan, [t.shape for t in w.tensors])
    # partial history: extrapolate before H is full, from what it holds
    n_push = len(nodes)
    if o["partial"]:
        cb.cb_plan_set_option(walk.plan, cb.CB_OPT_PARTIAL_HISTORY, 1)
        n_push = max(1, len(nodes) - 1)
    for k in range(n_push):
        walk.push(nodes[k], k)  # the oracle's FIFO holds the same n_push entries
    gates = None
    G = None
    if o["gated"]:
        gen = torch.Generator(device="cuda").manual_seed(77 + seed)
        gdt = H.TORCH[o["gate_dtype"]]
        gates = [None if i % 3 == 1 else (0.5 * torch.randn(t.shape[0], t.shape[-1], generator=gen, device="cuda")).to(gdt)
                 for i, t in enumerate(w.tensors)]
        G = [None if g is None else H.expand_gate(g, s.shape) for g, s in zip(gates, w.tensors)]
    t = o["target"]
    outs, resid, rh = walk.extrapolate(t, out_dtype=o["out_dtype"], fused=True, resid_dtype=o["resid_dtype"],
                                       salt=seed, gates=gates, gate_dtype=o["gate_dtype"])
    so, sr, _ = walk.expected_and_compare(t, outs, resid, rh, out_dtype=o["out_dtype"],
                                          resid_dtype=o["resid_dtype"], G=G)
    _ok(so, (seed, o, "outs"))
    _ok(sr, (seed, o, "resid"))
    # the same step without hidden states (prediction-only launch shape)
    outs, _, _ = walk.extrapolate(t, out_dtype=o["out_dtype"])
    so, _, _ = walk.expected_and_compare(t, outs, None, None, out_dtype=o["out_dtype"])
    _ok(so, (seed, o, "prediction only"))
    walk.close()


@pytest.mark.parametrize("seed", range(0, N_CASES, 2))
def test_random_full_step_epilogue(cb, H, seed):
    """cb_cache_push_residual on random shapes, feature and cache types and
    gates: the slot holds exactly what cb_cache_push writes, and the hidden
    states match the oracle's x + sum_b g_b f_b rounded once."""
    w, nodes, o = _random_case(seed)
    rng = np.random.default_rng(7000 + seed)
    src = "fp32" if rng.random() < 0.5 else "bf16"
    K = max(2, w.K)
    a = H.Walk(w, K=K, node_t=[990.0 - 30.0 * k for k in range(K)])
    b = H.Walk(w, K=K, node_t=[990.0 - 30.0 * k for k in range(K)])
    cb.cb_plan_set_shapes(a.plan, [t.shape for t in w.tensors])
    esize = 2 if w.cache_dtype == "bf16" else 4
    offs, slot = H.slot_layout([s_.numel for s_ in w.tensors], esize)
    tdt = H.TORCH[src]
    for k in range(2):
        t = 990.0 - 30.0 * k
        feats = [workloads.trajectory(w, i, t, k, "cuda", out_dtype=tdt) for i in range(len(w.tensors))]
        gates = None
        G = None
        if o["gated"]:
            gen = torch.Generator(device="cuda").manual_seed(900 + seed + k)
            gates = [None if i % 3 == 2 else (0.5 * torch.randn(s_.shape[0], s_.shape[-1], generator=gen,
                                                                 device="cuda")).to(H.TORCH[o["gate_dtype"]])
                     for i, s_ in enumerate(w.tensors)]
            G = [None if g is None else H.expand_gate(g, s_.shape) for g, s_ in zip(gates, w.tensors)]
        resid = [workloads.hidden_state(w, g, "cuda", salt=k) for g in range(a.n_groups)]
        rh = [H.host(r) for r in resid]
        cb.cb_cache_push_residual(a.plan, feats, H.CB[src], t, resid, cb.CB_BF16, gates,
                                  H.CB[o["gate_dtype"]])
        cb.cb_cache_push(b.plan, feats, H.CB[src], t)
        torch.cuda.synchronize()
        assert cb.cb_plan_device_status(a.plan) == 0
        for i, s_ in enumerate(w.tensors):
            lo = k * slot + offs[i]
            assert torch.equal(a.cache[lo:lo + esize * s_.numel], b.cache[lo:lo + esize * s_.numel]), (seed, k, i)
        for g in range(a.n_groups):
            members = [i for i, s_ in enumerate(w.tensors) if s_.group == g]
            F = [[H.host(feats[i])] for i in members]
            Gm = None if G is None else [G[i] for i in members]
            _, r64 = orc.extrapolate(F, [1.0], H.ORC[src], None, X=rh[g], x_dtype=orc.BF16,
                                     resid_dtype=orc.FP64, G=Gm)
            ref = orc.convert(r64, orc.FP64, orc.BF16)
            Fd = np.array([f[0].astype(np.float64) if src == "fp32" else H.bf16_to_f64(f[0]) for f in F])
            gb = np.array([np.ones_like(Fd[0]) if (Gm is None or x is None) else np.abs(x)
                           for x in (Gm or [None] * len(members))])
            bound = (gb * np.abs(Fd)).sum(0) + np.abs(H.bf16_to_f64(rh[g]))
            st = H.compare_bf16(H.host(resid[g]), ref, r64, bound)
            assert st["bad"] == 0, (seed, k, g, st)
    a.close()
    b.close()
