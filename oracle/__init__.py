"""Plain CPU oracle for ChebBooster's online extrapolation stage (test infrastructure).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py``
may import this package. The product path (the CUDA library and its binding) never
touches it, and the two share no code. The arithmetic lives in
``chebboost_oracle.c`` (fp64, written straight from the paper); this module builds
it with gcc and marshals numpy arrays into it. The one piece of logic kept here is
the history buffer H of Alg. 1: a FIFO of the n most recent (s_j, f_j) pairs whose
oldest entry is dropped when it is full (Sec. 3.3).
"""
from __future__ import annotations

import ctypes
import hashlib
import os
import platform
import subprocess
from collections import deque

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "chebboost_oracle.c")
_LIB = os.path.join(_HERE, "liborc.so")

BF16, FP32, FP64 = 0, 1, 2
_NP = {BF16: np.uint16, FP32: np.float32, FP64: np.float64}

_lib = None


_CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math", "-ffp-contract=off"]
_STAMP = os.path.join(_HERE, "liborc.stamp")


def _stamp() -> str:
    with open(_SRC, "rb") as fh:
        h = hashlib.sha256(fh.read())
    h.update(" ".join(_CFLAGS).encode())
    h.update(platform.machine().encode())
    return h.hexdigest()


def build(force: bool = False) -> str:
    """Compile the oracle with gcc into ``oracle/liborc.so``; an existing build is
    reused only when its stamp (source, flags, machine) matches."""
    stamp = _stamp()
    current = os.path.exists(_LIB) and os.path.exists(_STAMP) and open(_STAMP).read().strip() == stamp
    if force or not current:
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", *_CFLAGS, "-o", tmp, _SRC, "-lm", "-lpthread"])
        os.replace(tmp, _LIB)
        with open(_STAMP, "w") as fh:
            fh.write(stamp + "\n")
    return _LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB)
        D, I, P, I64 = ctypes.c_double, ctypes.c_int, ctypes.c_void_p, ctypes.c_int64
        L.orc_bf16_decode.argtypes, L.orc_bf16_decode.restype = [ctypes.c_uint16], D
        L.orc_bf16_encode.argtypes, L.orc_bf16_encode.restype = [D], ctypes.c_uint16
        L.orc_full_schedule.argtypes, L.orc_full_schedule.restype = [I, I, I, I, I, P], I
        L.orc_normalize.argtypes, L.orc_normalize.restype = [P, I, D, D, P], None
        L.orc_nodal.argtypes, L.orc_nodal.restype = [P, I, D], D
        L.orc_rho.argtypes, L.orc_rho.restype = [P, I, P], I
        L.orc_bary_coeff.argtypes, L.orc_bary_coeff.restype = [P, P, I, D, P], I
        L.orc_lagrange_basis.argtypes, L.orc_lagrange_basis.restype = [P, I, D, P], I
        L.orc_taylor_weights.argtypes, L.orc_taylor_weights.restype = [P, I, D, P], I
        L.orc_convert.argtypes, L.orc_convert.restype = [P, I, I64, P, I], None
        L.orc_extrapolate.argtypes = [I, I, P, I, P, P, I, I64, P, I, P, I, I]
        L.orc_extrapolate.restype = I
        L.orc_extrapolate_gated.argtypes = [I, I, P, I, P, P, I, I64, P, I, P, I, P, I]
        L.orc_extrapolate_gated.restype = I
        _lib = L
    return _lib


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


# ----------------------------------------------------------------- bf16 codec
def bf16_encode(x) -> np.ndarray:
    """fp64 -> bf16 bit patterns, round-to-nearest-even (one rounding)."""
    x = _f64(x).ravel()
    L = lib()
    return np.fromiter((L.orc_bf16_encode(float(v)) for v in x), dtype=np.uint16, count=x.size)


def bf16_decode(h) -> np.ndarray:
    h = np.ascontiguousarray(h, dtype=np.uint16).ravel()
    L = lib()
    return np.fromiter((L.orc_bf16_decode(int(v)) for v in h), dtype=np.float64, count=h.size)


def convert(src: np.ndarray, src_dtype: int, dst_dtype: int) -> np.ndarray:
    """The cache write: bit copy for bf16 -> bf16, else one RNE conversion."""
    src = np.ascontiguousarray(src, dtype=_NP[src_dtype]).ravel()
    dst = np.empty(src.size, dtype=_NP[dst_dtype])
    lib().orc_convert(_ptr(src), src_dtype, src.size, _ptr(dst), dst_dtype)
    return dst


# ------------------------------------------------------------------ schedule
def full_schedule(T: int, r: int, s0: int = 0, s1: int = 0, K: int = 0) -> np.ndarray:
    """Boolean mask of full-computation steps (Sec. 3.3 set F, then warm-up)."""
    out = np.zeros(T, dtype=np.uint8)
    n = lib().orc_full_schedule(T, r, s0, s1, K, _ptr(out))
    if n < 0:
        raise ValueError("invalid schedule parameters")
    return out.astype(bool)


def normalize(t, t_min: float, t_max: float) -> np.ndarray:
    t = _f64(t).ravel()
    tau = np.empty_like(t)
    lib().orc_normalize(_ptr(t), t.size, float(t_min), float(t_max), _ptr(tau))
    return tau


# ------------------------------------------------------------------- weights
def nodal(x, xq: float) -> float:
    x = _f64(x)
    return lib().orc_nodal(_ptr(x), x.size, float(xq))


def rho(x) -> np.ndarray:
    x = _f64(x)
    out = np.empty_like(x)
    if lib().orc_rho(_ptr(x), x.size, _ptr(out)) != 0:
        raise ValueError("duplicate nodes")
    return out


def bary_coeff(x, xq: float, rho_=None) -> np.ndarray:
    x = _f64(x)
    r = rho(x) if rho_ is None else _f64(rho_)
    w = np.empty_like(x)
    lib().orc_bary_coeff(_ptr(x), _ptr(r), x.size, float(xq), _ptr(w))
    return w


def lagrange_basis(x, xq: float) -> np.ndarray:
    x = _f64(x)
    out = np.empty_like(x)
    if lib().orc_lagrange_basis(_ptr(x), x.size, float(xq), _ptr(out)) != 0:
        raise ValueError("duplicate nodes")
    return out


def taylor_weights(x, xq: float) -> np.ndarray:
    """Truncated-Taylor weights with backward-difference derivatives (equispaced x)."""
    x = _f64(x)
    out = np.empty_like(x)
    if lib().orc_taylor_weights(_ptr(x), x.size, float(xq), _ptr(out)) != 0:
        raise ValueError("degenerate nodes")
    return out


def weights(node_t, t_target: float, t_min: float, t_max: float) -> np.ndarray:
    """The oracle's weights for one target: l_j(tau) on the normalised nodes."""
    return lagrange_basis(normalize(node_t, t_min, t_max), normalize([t_target], t_min, t_max)[0])


# ------------------------------------------------------------- extrapolation
def extrapolate(F, w, f_dtype: int, out_dtype: int | None = None, X=None, x_dtype: int = FP32,
                resid_dtype: int | None = None, nthreads: int = 1, G=None):
    """Per element: P_b = sum_j w_j F[b][j] (fp64) rounded once to ``out_dtype``;
    with ``resid_dtype`` set, also X + sum_b G_b P_b rounded once (G_b: optional
    per-element gates, 1 where absent).

    ``F`` is a list over branches b of lists over history entries j (oldest first),
    each a flat array of the same length in ``f_dtype`` (bf16 as uint16 bits).
    Returns ``(outs, resid)``; either is None when not requested.
    """
    K = len(w)
    nb = len(F)
    arrs = [np.ascontiguousarray(F[b][j], dtype=_NP[f_dtype]).ravel() for b in range(nb) for j in range(K)]
    n = arrs[0].size
    assert all(a.size == n for a in arrs)
    fptrs = (ctypes.c_void_p * len(arrs))(*[a.ctypes.data for a in arrs])
    w = _f64(w)
    outs = None
    optrs = None
    if out_dtype is not None:
        outs = [np.empty(n, dtype=_NP[out_dtype]) for _ in range(nb)]
        optrs = (ctypes.c_void_p * nb)(*[o.ctypes.data for o in outs])
    xa = None if X is None else np.ascontiguousarray(X, dtype=_NP[x_dtype]).ravel()
    resid = None if resid_dtype is None else np.empty(n, dtype=_NP[resid_dtype])
    garr = None
    gptrs = None
    if G is not None:  # per-member gates expanded to the element space (fp64), None = 1
        garr = [None if g is None else _f64(g).ravel() for g in G]
        assert all(g is None or g.size == n for g in garr)
        gptrs = (ctypes.c_void_p * nb)(*[None if g is None else g.ctypes.data for g in garr])
    rc = lib().orc_extrapolate_gated(
        K, nb, fptrs, f_dtype, _ptr(w), None if xa is None else _ptr(xa), x_dtype, n,
        optrs, out_dtype if out_dtype is not None else FP64,
        None if resid is None else _ptr(resid), resid_dtype if resid_dtype is not None else FP64,
        gptrs, int(nthreads))
    if rc != 0:
        raise RuntimeError(f"orc_extrapolate failed ({rc})")
    return outs, resid


class History:
    """The history buffer H of Alg. 1: the n most recent (s_j, f_j) pairs.

    ``push`` appends; when more than n entries are held the oldest is discarded
    (Sec. 3.3). ``entries()`` lists them oldest first.
    """

    def __init__(self, n: int):
        self.n = n
        self._h: deque = deque()

    def push(self, t: float, f) -> None:
        self._h.append((float(t), f))
        if len(self._h) > self.n:
            self._h.popleft()

    def full(self) -> bool:
        return len(self._h) == self.n

    def times(self) -> list[float]:
        return [t for t, _ in self._h]

    def entries(self) -> list:
        return list(self._h)
