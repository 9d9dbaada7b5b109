"""Helpers for the GPU parity tests.

``Walk`` drives a plan through a workload's schedule (Alg. 1): full steps push
freshly generated features through ``cb_cache_push``; skipped steps call
``cb_extrapolate``. The oracle mirrors the history buffer on the host with its
own FIFO, fed from the generator's bytes (never from the CUDA library), and
computes the expected values with its own weights. ``sample`` restricts the
host copies to a fixed set of element indices per tensor, so that full-size
workloads are checked on sampled outputs.
"""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle as orc
from paper_2608_23429_gb300 import chebboost as cb
from paper_2608_23429_gb300 import workloads

CB = {"bf16": cb.CB_BF16, "fp32": cb.CB_FP32}
ORC = {"bf16": orc.BF16, "fp32": orc.FP32}
TORCH = {"bf16": torch.bfloat16, "fp32": torch.float32}
KERNEL = {"auto": cb.CB_KERNEL_AUTO, "direct": cb.CB_KERNEL_DIRECT, "bulk": cb.CB_KERNEL_BULK}
FLOOR = 2.0 ** -40  # cancellation floor: |P| this small relative to sum|w F| is not resolvable


def host(t: torch.Tensor, idx: torch.Tensor | None = None) -> np.ndarray:
    t = t.detach().reshape(-1)
    if idx is not None:
        t = t[idx]
    t = t.contiguous().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16).copy()
    return t.numpy().copy()


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _step(bits: np.ndarray, k: int) -> np.ndarray:
    """Move each finite bf16 pattern k representable values up (k > 0) or down."""
    o = _ordered(bits) + k
    o = np.clip(o, -0x7F7F, 0x7F7F)
    return np.where(o < 0, (-o) | 0x8000, o).astype(np.uint16)


def _ordered(bits: np.ndarray) -> np.ndarray:
    b = bits.astype(np.int64)
    return np.where(b & 0x8000, -(b & 0x7FFF), b)


def compare_bf16(gpu: np.ndarray, ref: np.ndarray, ref64: np.ndarray, bound64: np.ndarray) -> dict:
    """Gate: within one bf16 ulp of the oracle rounded to bf16, except where the
    exact value cancels below 2^-40 * sum_j |w_j F_j| (counted separately)."""
    d = np.abs(_ordered(gpu) - _ordered(ref))
    floor = np.abs(bf16_to_f64(gpu) - ref64) <= FLOOR * bound64
    return dict(n=int(d.size), exact=int((d == 0).sum()), one_ulp=int((d == 1).sum()),
                floor=int(((d > 1) & floor).sum()), bad=int(((d > 1) & ~floor).sum()),
                max_ulp=int(d.max()) if d.size else 0)


def compare_fp32(gpu: np.ndarray, ref64: np.ndarray, max_f: float) -> dict:
    err = float(np.max(np.abs(gpu.astype(np.float64) - ref64))) if gpu.size else 0.0
    return dict(n=int(gpu.size), max_err=err, tol=2e-6 * max_f, bad=int(err > 2e-6 * max_f))


def merge(stats: list[dict]) -> dict:
    out: dict = {}
    for s in stats:
        for k, v in s.items():
            if k in ("max_ulp", "max_err", "tol"):
                out[k] = max(out.get(k, 0), v)
            else:
                out[k] = out.get(k, 0) + v
    return out


class Walk:
    def __init__(self, w: workloads.Workload, K: int | None = None, samples: int | None = None,
                 seed: int = 0, device: str = "cuda", node_t=None, kernel: str = "auto"):
        self.w = w
        self.K = K or w.K
        self.dev = torch.device(device)
        self.cdt = w.cache_dtype
        if node_t is None:
            self.full = library_schedule(w, self.K)
            node_t = [t for s, t in enumerate(w.timesteps) if self.full[s]]
        self.node_t = list(node_t)
        self.tensors = [(t.layer, t.branch, t.numel, t.group) for t in w.tensors]
        self.plan = cb.cb_plan_create(self.node_t, self.K, self.tensors, CB[self.cdt], w.t_min, w.t_max)
        self.cache = torch.empty(cb.cb_plan_cache_bytes(self.plan), dtype=torch.uint8, device=self.dev)
        cb.cb_plan_bind_cache(self.plan, self.cache, self.cache.numel())
        cb.cb_plan_set_option(self.plan, cb.CB_OPT_KERNEL, KERNEL[kernel])
        self.H = orc.History(self.K)
        self.n_groups = cb.cb_plan_num_groups(self.plan)
        # sampled element indices: one set per element space (group or lone tensor)
        self.idx = [None] * len(w.tensors)
        if samples is not None:
            g = torch.Generator().manual_seed(1234 + seed)
            spaces = {}
            for i, t in enumerate(w.tensors):
                key = ("g", t.group) if t.group >= 0 else ("t", i)
                if key not in spaces:
                    n = t.numel
                    k = min(samples, n)
                    pick = torch.randperm(n, generator=g)[:k]
                    edge = torch.tensor([0, 1, n - 2, n - 1][: min(4, n)], dtype=torch.int64)
                    spaces[key] = torch.unique(torch.cat([pick, edge])).to(self.dev)
                self.idx[i] = spaces[key]

    def close(self):
        cb.cb_plan_destroy(self.plan)

    # ---- full step
    def push(self, t: float, node_index: int, feats=None):
        if feats is None:
            feats = [workloads.trajectory(self.w, i, t, node_index, self.dev) for i in range(len(self.w.tensors))]
        fdt = "bf16" if feats[0].dtype == torch.bfloat16 else "fp32"
        cb.cb_cache_push(self.plan, feats, CB[fdt], t)
        host_vals = [orc.convert(host(f, self.idx[i]), ORC[fdt], ORC[self.cdt]) for i, f in enumerate(feats)]
        self.H.push(t, host_vals)
        return feats

    # ---- skipped step
    def extrapolate(self, t: float, out_dtype: str = "bf16", fused: bool = False, outs: bool = True,
                    resid_dtype: str = "bf16", ring=None, salt: int = 0, explicit=None, gates=None,
                    gate_dtype: str = "bf16"):
        w = self.w
        out_t = [torch.empty(s.shape, dtype=TORCH[out_dtype], device=self.dev) for s in w.tensors] if outs else None
        resid = None
        resid_host = None
        if fused:
            resid = [workloads.hidden_state(w, g, self.dev, TORCH[resid_dtype], salt=salt)
                     for g in range(self.n_groups)]
            resid_host = [host(resid[g], self._gidx(g)) for g in range(self.n_groups)]
        if gates is not None:
            cb.cb_extrapolate_gated(self.plan, t, out_t, CB[out_dtype], resid, CB[resid_dtype], gates,
                                    CB[gate_dtype])
        elif explicit is not None:
            cb.cb_extrapolate_weights(self.plan, explicit, out_t, CB[out_dtype], resid, CB[resid_dtype])
        elif ring is None:
            cb.cb_extrapolate(self.plan, t, out_t, CB[out_dtype], resid, CB[resid_dtype])
        else:
            slot_t, head = ring
            cb.cb_extrapolate_ring(self.plan, slot_t, head, t, out_t, CB[out_dtype], resid, CB[resid_dtype])
        torch.cuda.synchronize()
        assert cb.cb_plan_device_status(self.plan) == 0
        return out_t, resid, resid_host

    def _gidx(self, g):
        i = next(i for i, t in enumerate(self.w.tensors) if t.group == g)
        return self.idx[i]

    def expected_and_compare(self, t, out_t, resid, resid_host, out_dtype="bf16", resid_dtype="bf16",
                             times=None, nthreads=8, wts=None, G=None):
        """Oracle expectation for the live FIFO (or ``times`` relabelling it, or the
        explicit weights ``wts``) and the comparison."""
        w = self.w
        entries = self.H.entries()
        times = times if times is not None else [e[0] for e in entries]
        if wts is None:
            wts = orc.weights(times, t, w.t_min, w.t_max)
        cdt = ORC[self.cdt]
        stats_out, stats_res = [], []
        items = []
        if resid is not None:
            for g in range(self.n_groups):
                items.append(([i for i, s in enumerate(w.tensors) if s.group == g], g))
            lone = [i for i, s in enumerate(w.tensors) if s.group < 0]
            items += [([i], None) for i in lone]
        else:
            items = [([i], None) for i in range(len(w.tensors))]
        for members, g in items:
            F = [[e[1][i] for e in entries] for i in members]
            X = resid_host[g] if g is not None else None
            x_dt = ORC[resid_dtype]
            Gm = None if G is None else [G[i] for i in members]
            o64, r64 = orc.extrapolate(F, wts, cdt, orc.FP64, X=X, x_dtype=x_dt,
                                       resid_dtype=orc.FP64 if g is not None else None, nthreads=nthreads,
                                       G=Gm)
            Fd = np.array([[bf16_to_f64(f) if cdt == orc.BF16 else f.astype(np.float64) for f in row]
                           for row in F])  # [nb, K, n]
            bound = np.einsum("j,bjn->bn", np.abs(wts), np.abs(Fd))
            gbound = bound if Gm is None else np.array(
                [bound[b] * (1.0 if Gm[b] is None else np.abs(Gm[b])) for b in range(len(members))])
            for b, i in enumerate(members):
                if out_t is None:
                    continue
                gpu = host(out_t[i], self.idx[i])
                if out_dtype == "bf16":
                    ref = orc.convert(o64[b], orc.FP64, orc.BF16)
                    stats_out.append(compare_bf16(gpu, ref, o64[b], bound[b]))
                else:
                    stats_out.append(compare_fp32(gpu, o64[b], float(np.max(np.abs(Fd[b])))))
            if g is not None:
                gpu = host(resid[g], self.idx[members[0]])
                rb = gbound.sum(0) + np.abs(bf16_to_f64(X) if x_dt == orc.BF16 else X.astype(np.float64))
                if resid_dtype == "bf16":
                    ref = orc.convert(r64, orc.FP64, orc.BF16)
                    stats_res.append(compare_bf16(gpu, ref, r64, rb))
                else:
                    stats_res.append(compare_fp32(gpu, r64, float(np.max(np.abs(Fd)))))
        return merge(stats_out) if stats_out else None, merge(stats_res) if stats_res else None, wts


def library_schedule(w: workloads.Workload, K: int) -> np.ndarray:
    """The full-step mask the product drives its runs with (the library's
    cb_schedule_full), checked here against the oracle's own schedule."""
    mask, _ = cb.cb_schedule_full(w.T, w.r, w.s0, w.s1, K)
    assert np.array_equal(mask, orc.full_schedule(w.T, w.r, w.s0, w.s1, K)), (w.name, K)
    return mask


def schedule_steps(w: workloads.Workload, K: int):
    mask = library_schedule(w, K)
    return mask, [s for s in range(w.T) if not mask[s]]


def ceil_div(a, b):
    return -(-a // b)


def slot_layout(numels, esize):
    offs, o = [], 0
    for n in numels:
        offs.append(o)
        o = ceil_div(o + n * esize, 256) * 256
    return offs, o


def isfinite_all(*arrs):
    return all(np.all(np.isfinite(a)) for a in arrs)


def log2(x):
    return math.log2(x) if x > 0 else float("-inf")


def expand_gate(gate: torch.Tensor, shape, idx=None) -> np.ndarray:
    """A [batch, hidden] gate broadcast over tokens to the tensor's elements (fp64)."""
    b, t, h = shape
    g = gate.detach().float().cpu().numpy().astype(np.float64)
    full = np.broadcast_to(g[:, None, :], (b, t, h)).reshape(-1)
    return full if idx is None else full[idx.cpu().numpy()]
