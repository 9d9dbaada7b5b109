"""Seeded synthetic workloads shaped like the paper's cached branch outputs.

The paper caches, per DiT block, the outputs of the self-attention,
cross-attention and MLP branches (Sec. 3.1, B(x) = x + S + C + M) and feeds
them to the extrapolation of Sec. 3.3. Trained DiT-XL/2, PixArt-Sigma and
FLUX.1-dev activations are not available here; these generators stand in for
them with the same tensor shapes and smooth-trajectory structure:

* per element, coefficients c_d ~ N(0, 1) / (d + 1)^2 for d = 0..D and the
  trajectory F(tau) = sum_d c_d T_d(tau) (Chebyshev series, three-term
  recurrence), D = 3 for the tiny case and 6 otherwise;
* additive noise N(0, sigma^2) per (element, node), sigma = 0.1 (none on tiny);
* optionally a per-hidden-channel scale ~ LogNormal(0, 1) shared over batch,
  tokens and nodes (outlier channels);
* the hidden states for the fused residual: N(0, 1).

This module holds none of the method's arithmetic (no weights, no
extrapolation). Both the CUDA tests and the oracle consume the bytes it
produces, so the two sides see identical inputs. Seeds derive from 2025, the
seed the paper's experiments use.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch

BASE_SEED = 2025


@dataclass
class TensorSpec:
    layer: int
    branch: int
    shape: tuple
    group: int  # residual group (one hidden state per stream per block)

    @property
    def numel(self) -> int:
        n = 1
        for s in self.shape:
            n *= s
        return n


@dataclass
class Workload:
    name: str
    tensors: list
    K: int
    cache_dtype: str  # "bf16" | "fp32"
    T: int
    r: int
    t_min: float
    t_max: float
    timesteps: list  # t_s for s = 0..T-1 (sampling order)
    degree: int = 6
    noise: float = 0.1
    lognormal: bool = False
    seed: int = BASE_SEED
    fused: bool = False
    s0: int = 0
    s1: int = 0
    explicit_nodes: list = field(default_factory=list)    # tiny case only
    explicit_targets: list = field(default_factory=list)  # tiny case only

    @property
    def n_groups(self) -> int:
        return 1 + max(t.group for t in self.tensors)

    def group_numel(self, g: int) -> int:
        return next(t.numel for t in self.tensors if t.group == g)

    def group_shape(self, g: int) -> tuple:
        return next(t.shape for t in self.tensors if t.group == g)

    @property
    def slot_elems(self) -> int:
        return sum(t.numel for t in self.tensors)

    def esize(self) -> int:
        return 2 if self.cache_dtype == "bf16" else 4


def _ddpm_timesteps(T):
    return [999.0 * (1.0 - s / (T - 1)) for s in range(T)]


def _flow_timesteps(T):
    return [1.0 - s / (T - 1) for s in range(T)]


def _blocks(n_blocks, n_branches, shape, group_base=0):
    out = []
    for layer in range(n_blocks):
        for b in range(n_branches):
            out.append(TensorSpec(layer, b, shape, group_base + layer))
    return out


def tiny() -> Workload:
    return Workload(
        name="tiny", tensors=_blocks(2, 2, (1, 256, 1152)), K=4, cache_dtype="fp32",
        T=0, r=0, t_min=0.0, t_max=1000.0, timesteps=[], degree=3, noise=0.0,
        seed=BASE_SEED + 0, fused=False,
        explicit_nodes=[900.0, 800.0, 700.0, 600.0], explicit_targets=[575.0, 550.0, 500.0])


def dit256(K: int = 4) -> Workload:
    return Workload(
        name=f"dit-xl2-256-k{K}", tensors=_blocks(28, 2, (8, 256, 1152)), K=K, cache_dtype="bf16",
        T=50, r=4, t_min=0.0, t_max=999.0, timesteps=_ddpm_timesteps(50), seed=BASE_SEED + 1,
        fused=True)


def dit512() -> Workload:
    return Workload(
        name="dit-xl2-512", tensors=_blocks(28, 2, (4, 1024, 1152)), K=4, cache_dtype="bf16",
        T=50, r=5, t_min=0.0, t_max=999.0, timesteps=_ddpm_timesteps(50), seed=BASE_SEED + 2,
        lognormal=True)


def pixart() -> Workload:
    return Workload(
        name="pixart-sigma-1024", tensors=_blocks(28, 3, (2, 4096, 1152)), K=4, cache_dtype="bf16",
        T=20, r=3, t_min=0.0, t_max=999.0, timesteps=_ddpm_timesteps(20), seed=BASE_SEED + 3)


def flux() -> Workload:
    tensors = []
    g = 0
    for layer in range(19):  # double-stream blocks: image and text streams
        tensors.append(TensorSpec(layer, 0, (1, 4096, 3072), g))      # img attn
        tensors.append(TensorSpec(layer, 1, (1, 4096, 3072), g))      # img mlp
        tensors.append(TensorSpec(layer, 2, (1, 512, 3072), g + 1))   # txt attn
        tensors.append(TensorSpec(layer, 3, (1, 512, 3072), g + 1))   # txt mlp
        g += 2
    for layer in range(19, 57):  # single-stream blocks: merged attn || mlp output
        tensors.append(TensorSpec(layer, 0, (1, 4608, 3072), g))
        g += 1
    return Workload(
        name="flux1-dev-1024", tensors=tensors, K=5, cache_dtype="bf16", T=50, r=6,
        t_min=0.0, t_max=1.0, timesteps=_flow_timesteps(50), seed=BASE_SEED + 4)


PRESETS = {"tiny": tiny, "dit256": dit256, "dit256-k3": lambda: dit256(3), "dit512": dit512,
           "pixart": pixart, "flux": flux}


def scaled(w: Workload, factor: int) -> Workload:
    """The same workload with every tensor's token count divided by ``factor``
    (for parity runs the CPU oracle finishes in seconds)."""
    import copy
    w2 = copy.deepcopy(w)
    for t in w2.tensors:
        b, n, h = t.shape
        t.shape = (b, max(1, n // factor), h)
    w2.name = f"{w.name}/{factor}"
    return w2


def _seed(*parts: int) -> int:
    h = 1469598103934665603
    for p in parts:
        h = ((h ^ (int(p) & 0xFFFFFFFFFFFF)) * 1099511628211) % (1 << 63)
    return h


def _tau(w: Workload, t: float) -> float:
    # the trajectory is a function on [-1, 1]; the same affine map places it
    return 2.0 * (t - w.t_min) / (w.t_max - w.t_min) - 1.0


def trajectory(w: Workload, i: int, t: float, node_index: int, device, out_dtype=None,
               exact: bool = False, absolute: bool = False) -> torch.Tensor:
    """Branch output ``i`` at timestep ``t`` (the value a full step would cache).

    With ``exact`` the noise-free series is summed in fp64 from the same fp32
    coefficients (the analytic trajectory); with ``absolute`` as well, each
    term enters with its magnitude (a bound on the rounding of the fp32 sum).
    """
    spec = w.tensors[i]
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(_seed(w.seed, i, 1))
    tau = _tau(w, t)
    acc_dt = torch.float64 if exact else torch.float32
    F = torch.zeros(spec.shape, dtype=acc_dt, device=dev)
    t_prev, t_cur = 1.0, tau  # T_0, T_1
    for d in range(w.degree + 1):
        c = torch.randn(spec.shape, generator=g, device=dev, dtype=torch.float32)
        Td = 1.0 if d == 0 else (tau if d == 1 else None)
        if d >= 2:
            t_prev, t_cur = t_cur, 2.0 * tau * t_cur - t_prev
            Td = t_cur
        if absolute:
            F.add_(c.to(acc_dt).abs(), alpha=abs(Td) / float((d + 1) ** 2))
        else:
            F.add_(c.to(acc_dt), alpha=Td / float((d + 1) ** 2))
    if w.lognormal:
        gs = torch.Generator(device=dev)
        gs.manual_seed(_seed(w.seed, i, 3))
        scale = torch.exp(torch.randn(spec.shape[-1], generator=gs, device=dev, dtype=torch.float32))
    if exact:
        if w.lognormal:
            F.mul_(scale.to(acc_dt))
        return F if out_dtype is None else F.to(out_dtype)
    if w.noise > 0:
        gn = torch.Generator(device=dev)
        gn.manual_seed(_seed(w.seed, i, 2, node_index))
        F.add_(torch.randn(spec.shape, generator=gn, device=dev, dtype=torch.float32), alpha=w.noise)
    if w.lognormal:
        F.mul_(scale)
    dt = out_dtype or (torch.bfloat16 if w.cache_dtype == "bf16" else torch.float32)
    return F.to(dt)


def hidden_state(w: Workload, g_idx: int, device, dtype=torch.bfloat16, salt: int = 0) -> torch.Tensor:
    """The residual stream entering a block (one per residual group)."""
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(_seed(w.seed, 1000 + g_idx, 4, salt))
    return torch.randn(w.group_shape(g_idx), generator=g, device=dev, dtype=torch.float32).to(dtype)
