"""ctypes binding of libchebboost (``include/chebboost.h``), same names, marshalling only.

Every call forwards to the C ABI: pointers may be given as ints, ``None`` or any
object with ``data_ptr()`` (a torch tensor); streams as ``None`` (legacy default
stream), an int handle, or an object with ``cuda_stream`` (``torch.cuda.Stream``).
A negative status raises :class:`CbError`. There is no fallback: importing this
module fails if the compiled library is missing.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libchebboost.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(
        f"{LIB_PATH} is not built; run `python -m paper_2608_23429_gb300.build` "
        "(the CUDA library is required, there is no CPU path)")

_lib = ctypes.CDLL(LIB_PATH)

CB_BF16, CB_FP32 = 0, 1
CB_MAX_K, CB_MAX_TENSORS, CB_MAX_BRANCHES, CB_CACHE_ALIGN, CB_STATUS_BYTES = 8, 256, 4, 256, 256
CB_MAX_NUMEL = 1 << 48
CB_OPT_KERNEL, CB_OPT_WAIT_NS, CB_OPT_TEST_WITHHOLD, CB_OPT_PARTIAL_HISTORY = 1, 2, 3, 4
CB_KERNEL_AUTO, CB_KERNEL_DIRECT, CB_KERNEL_BULK = 0, 1, 2
CB_DEV_CONSUMER_TIMEOUT, CB_DEV_PRODUCER_TIMEOUT, CB_DEV_DRAIN_TIMEOUT = 1, 2, 4
CB_OK, CB_ERR_ARG, CB_ERR_ALIGN, CB_ERR_NODES_DEGENERATE = 0, -1, -2, -3
CB_ERR_HISTORY_NOT_FULL, CB_ERR_ORDER, CB_ERR_UNBOUND, CB_ERR_CUDA, CB_ERR_LIMIT = -4, -5, -6, -7, -8


class cb_tensor_desc(ctypes.Structure):
    _fields_ = [("layer", ctypes.c_int32), ("branch", ctypes.c_int32), ("numel", ctypes.c_int64),
                ("group", ctypes.c_int32), ("reserved", ctypes.c_int32)]


_P, _I, _D, _SZ = ctypes.c_void_p, ctypes.c_int, ctypes.c_double, ctypes.c_size_t
_PP = ctypes.POINTER(ctypes.c_void_p)
_sig = {
    "cb_schedule_full": ([_I, _I, _I, _I, _I, _P, _P], _I),
    "cb_plan_create": ([_P, _I, _I, _P, _I, _I, _D, _D, ctypes.POINTER(_P)], _I),
    "cb_plan_cache_bytes": ([_P], _SZ),
    "cb_plan_bind_cache": ([_P, _P, _SZ], _I),
    "cb_cache_push": ([_P, _PP, _I, _D, _P], _I),
    "cb_extrapolate": ([_P, _D, _PP, _I, _PP, _I, _P], _I),
    "cb_extrapolate_ring": ([_P, _P, _I, _D, _PP, _I, _PP, _I, _P], _I),
    "cb_extrapolate_noalloc": ([_P, _P, _SZ, _P, _I, _D, _PP, _I, _PP, _I, _P, _P], _I),
    "cb_extrapolate_weights": ([_P, _P, _PP, _I, _PP, _I, _P], _I),
    "cb_plan_set_shapes": ([_P, _P], _I),
    "cb_extrapolate_gated": ([_P, _D, _PP, _I, _PP, _I, _PP, _I, _P], _I),
    "cb_cache_push_residual": ([_P, _PP, _I, _D, _PP, _I, _PP, _I, _P], _I),
    "cb_weights": ([_P, _D, _P], _I),
    "cb_taylor_weights": ([_P, _I, _D, _P], _I),
    "cb_plan_export_weights": ([_P, _P, _I, _P], _I),
    "cb_plan_history": ([_P, _P, _P, _P], _I),
    "cb_plan_reset": ([_P], _I),
    "cb_plan_set_option": ([_P, _I, ctypes.c_int64], _I),
    "cb_plan_device_status": ([_P, _P, _P], _I),
    "cb_plan_num_groups": ([_P], _I),
    "cb_plan_destroy": ([_P], None),
    "cb_status_string": ([_I], ctypes.c_char_p),
    "cb_last_error_message": ([], ctypes.c_char_p),
}
for _name, (_args, _res) in _sig.items():
    _f = getattr(_lib, _name)
    _f.argtypes, _f.restype = _args, _res

EXPORTED = tuple(_sig)


class CbError(RuntimeError):
    def __init__(self, status: int, call: str):
        msg = _lib.cb_status_string(status).decode()
        if status == CB_ERR_CUDA:
            msg += ": " + _lib.cb_last_error_message().decode()
        super().__init__(f"{call}: {msg} ({status})")
        self.status = status


def _check(rc: int, call: str) -> int:
    if rc < 0:
        raise CbError(rc, call)
    return rc


def _addr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


def ptr_array(xs):
    """The pointer array of a list of buffers (tensors, ints or None), in the
    form every call below also accepts: a loop over persistent buffers builds
    it once instead of on every call."""
    return (ctypes.c_void_p * len(xs))(*[_addr(x) for x in xs])


def _ptr_array(xs):
    if xs is None or isinstance(xs, ctypes.Array):
        return xs
    return ptr_array(xs)


# Tensor count, residual-group count, K and the partial-history option of every
# plan this module created: the library reads one pointer per tensor (or group)
# from each array and one weight per live history entry, so the lengths are
# checked here before a call.
_PLANS: dict = {}
_TENSORS, _GROUPS, _K, _PARTIAL = 0, 1, 2, 3


def _plan_key(plan) -> int | None:
    return plan.value if isinstance(plan, ctypes.c_void_p) else plan


def _dims(plan):
    return _PLANS.get(_plan_key(plan))


def _ptrs(plan, xs, per: int, call: str, what: str):
    """Pointer array of ``xs`` with one entry per tensor or per residual group."""
    if xs is None:
        return None
    d = _dims(plan)
    if d is not None and len(xs) != d[per]:
        unit = "tensors" if per == _TENSORS else "residual groups"
        raise CbError(CB_ERR_ARG, f"{call} ({what}: {len(xs)} pointers for {d[per]} {unit})")
    return _ptr_array(xs)


def _live(plan) -> int | None:
    """History entries a skipped step of this plan uses now: K once H is full,
    what H holds under the partial-history option, else 0 (the library then
    reports the history as not full). None for a plan made elsewhere."""
    d = _dims(plan)
    if d is None:
        return None
    count = ctypes.c_int(0)
    _check(_lib.cb_plan_history(plan, None, None, ctypes.byref(count)), "cb_plan_history")
    if count.value >= d[_K]:
        return d[_K]
    return count.value if d[_PARTIAL] else 0


def _weights_in(plan, w, call: str):
    """A caller's weight vector in a CB_MAX_K buffer padded with NaN: the library
    reads one entry per live history entry and rejects non-finite ones, so a
    vector of any other length is refused here."""
    w = np.ascontiguousarray(w, dtype=np.float64).ravel()
    d = _dims(plan)
    live = _live(plan)
    if w.size > (d[_K] if d is not None else CB_MAX_K) or (live and w.size != live):
        raise CbError(CB_ERR_ARG, f"{call} ({w.size} weights for {live} live history entries, "
                                  f"K = {d[_K] if d is not None else '?'})")
    buf = np.full(CB_MAX_K, np.nan)
    buf[:w.size] = w
    return buf


def _stream(s):
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return int(s.cuda_stream)


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def cb_schedule_full(T: int, r: int, s0: int = 0, s1: int = 0, K: int = 0):
    mask = np.zeros(T, dtype=np.uint8)
    n = ctypes.c_int(0)
    _check(_lib.cb_schedule_full(T, r, s0, s1, K, mask.ctypes.data, ctypes.byref(n)), "cb_schedule_full")
    return mask.astype(bool), n.value


def cb_plan_create(node_t, K: int, tensors, cache_dtype: int, t_min: float, t_max: float):
    """``tensors``: sequence of (layer, branch, numel, group)."""
    node_t = _f64(node_t)
    descs = (cb_tensor_desc * len(tensors))(*[cb_tensor_desc(int(l), int(b), int(n), int(g), 0)
                                             for (l, b, n, g) in tensors])
    plan = ctypes.c_void_p()
    _check(_lib.cb_plan_create(node_t.ctypes.data, node_t.size, K, ctypes.cast(descs, ctypes.c_void_p),
                               len(tensors), cache_dtype, float(t_min), float(t_max), ctypes.byref(plan)),
           "cb_plan_create")
    _PLANS[plan.value] = [len(tensors), int(_lib.cb_plan_num_groups(plan)), int(K), False]
    return plan


def cb_plan_cache_bytes(plan) -> int:
    return int(_lib.cb_plan_cache_bytes(plan))


def cb_plan_bind_cache(plan, dev_ptr, nbytes: int) -> None:
    _check(_lib.cb_plan_bind_cache(plan, _addr(dev_ptr), nbytes), "cb_plan_bind_cache")


def cb_cache_push(plan, feats, feat_dtype: int, t: float, stream=None) -> None:
    _check(_lib.cb_cache_push(plan, _ptrs(plan, feats, _TENSORS, "cb_cache_push", "feats"), feat_dtype, float(t),
                              _stream(stream)), "cb_cache_push")


def cb_extrapolate(plan, t_target: float, outs, out_dtype: int, resid=None, resid_dtype: int = CB_BF16,
                   stream=None) -> None:
    c = "cb_extrapolate"
    _check(_lib.cb_extrapolate(plan, float(t_target), _ptrs(plan, outs, _TENSORS, c, "outs"), out_dtype,
                               _ptrs(plan, resid, _GROUPS, c, "resid"), resid_dtype, _stream(stream)), c)


def cb_extrapolate_ring(plan, slot_t, head: int, t_target: float, outs, out_dtype: int, resid=None,
                        resid_dtype: int = CB_BF16, stream=None) -> None:
    c = "cb_extrapolate_ring"
    slot_t = _f64(slot_t).ravel()
    d = _dims(plan)
    if d is not None and slot_t.size != d[_K]:  # the library reads K slot times
        raise CbError(CB_ERR_ARG, f"{c} ({slot_t.size} slot times for K = {d[_K]})")
    _check(_lib.cb_extrapolate_ring(plan, slot_t.ctypes.data, head, float(t_target),
                                    _ptrs(plan, outs, _TENSORS, c, "outs"), out_dtype,
                                    _ptrs(plan, resid, _GROUPS, c, "resid"), resid_dtype, _stream(stream)), c)


def cb_extrapolate_noalloc(plan, hist, hist_bytes: int, slot_t, head: int, t_target: float, outs, out_dtype: int,
                           resid=None, resid_dtype: int = CB_BF16, status=None, stream=None) -> None:
    """The skipped step of cb_extrapolate_ring on a caller's history buffer
    ``hist`` (the K slots, no status block; the plan need not be bound), for
    callers that may not allocate device memory. ``status``: None, or a host
    buffer (pinned keeps the call asynchronous) that receives the launch's
    device status word once the stream gets there."""
    c = "cb_extrapolate_noalloc"
    slot_t = _f64(slot_t).ravel()
    d = _dims(plan)
    if d is not None and slot_t.size != d[_K]:  # the library reads K slot times
        raise CbError(CB_ERR_ARG, f"{c} ({slot_t.size} slot times for K = {d[_K]})")
    _check(_lib.cb_extrapolate_noalloc(plan, _addr(hist), int(hist_bytes), slot_t.ctypes.data, head,
                                       float(t_target), _ptrs(plan, outs, _TENSORS, c, "outs"), out_dtype,
                                       _ptrs(plan, resid, _GROUPS, c, "resid"), resid_dtype, _addr(status),
                                       _stream(stream)), c)


def cb_extrapolate_weights(plan, w_logical, outs, out_dtype: int, resid=None, resid_dtype: int = CB_BF16,
                           stream=None) -> None:
    c = "cb_extrapolate_weights"
    w = _weights_in(plan, w_logical, c)
    _check(_lib.cb_extrapolate_weights(plan, w.ctypes.data, _ptrs(plan, outs, _TENSORS, c, "outs"), out_dtype,
                                       _ptrs(plan, resid, _GROUPS, c, "resid"), resid_dtype, _stream(stream)), c)


def cb_plan_set_shapes(plan, shapes) -> None:
    """``shapes``: sequence of (batch, tokens, hidden), one per tensor."""
    bth = np.ascontiguousarray(np.asarray(shapes, dtype=np.int64).reshape(-1, 3))
    d = _dims(plan)
    if d is not None and bth.shape[0] != d[_TENSORS]:
        raise CbError(CB_ERR_ARG, f"cb_plan_set_shapes ({bth.shape[0]} shapes for {d[_TENSORS]} tensors)")
    _check(_lib.cb_plan_set_shapes(plan, bth.ctypes.data), "cb_plan_set_shapes")


def cb_extrapolate_gated(plan, t_target: float, outs, out_dtype: int, resid, resid_dtype: int, gates,
                         gate_dtype: int = CB_BF16, stream=None) -> None:
    c = "cb_extrapolate_gated"
    _check(_lib.cb_extrapolate_gated(plan, float(t_target), _ptrs(plan, outs, _TENSORS, c, "outs"), out_dtype,
                                     _ptrs(plan, resid, _GROUPS, c, "resid"), resid_dtype,
                                     _ptrs(plan, gates, _TENSORS, c, "gates"), gate_dtype, _stream(stream)), c)


def cb_cache_push_residual(plan, feats, feat_dtype: int, t: float, resid, resid_dtype: int = CB_BF16,
                           gates=None, gate_dtype: int = CB_BF16, stream=None) -> None:
    c = "cb_cache_push_residual"
    _check(_lib.cb_cache_push_residual(plan, _ptrs(plan, feats, _TENSORS, c, "feats"), feat_dtype, float(t),
                                       _ptrs(plan, resid, _GROUPS, c, "resid"), resid_dtype,
                                       _ptrs(plan, gates, _TENSORS, c, "gates"), gate_dtype, _stream(stream)), c)


def cb_weights(plan, t_target: float, n: int | None = None) -> np.ndarray:
    """Weights over the live history entries (K, or fewer under partial history),
    oldest first. ``n``, if given, must equal that count. The library writes one
    weight per live entry into a CB_MAX_K buffer."""
    live = _live(plan)
    if n is not None and (not 1 <= n <= CB_MAX_K or (live and n != live)):
        raise CbError(CB_ERR_ARG, f"cb_weights (n = {n} for {live} live history entries)")
    w = np.full(CB_MAX_K, np.nan)
    _check(_lib.cb_weights(plan, float(t_target), w.ctypes.data), "cb_weights")
    if live is None:
        live = n if n is not None else int(np.isfinite(w).sum())
    return w[:live].copy()


def cb_taylor_weights(node_t, t_target: float) -> np.ndarray:
    node_t = _f64(node_t)
    w = np.empty(node_t.size, dtype=np.float64)
    _check(_lib.cb_taylor_weights(node_t.ctypes.data, node_t.size, float(t_target), w.ctypes.data),
           "cb_taylor_weights")
    return w


def cb_plan_export_weights(plan, targets, K: int) -> np.ndarray:
    """One row of the plan's K weights per target (the library writes rows of K)."""
    targets = _f64(targets)
    d = _dims(plan)
    if (d is not None and K != d[_K]) or not 1 <= K <= CB_MAX_K:
        raise CbError(CB_ERR_ARG, f"cb_plan_export_weights (K = {K})")
    table = np.empty((targets.size, K), dtype=np.float64)
    _check(_lib.cb_plan_export_weights(plan, targets.ctypes.data, targets.size, table.ctypes.data),
           "cb_plan_export_weights")
    return table


def cb_plan_history(plan, K: int):
    """Slot times (the library writes the plan's K of them), oldest slot, count."""
    d = _dims(plan)
    if (d is not None and K != d[_K]) or not 1 <= K <= CB_MAX_K:
        raise CbError(CB_ERR_ARG, f"cb_plan_history (K = {K})")
    slot_t = np.empty(K, dtype=np.float64)
    head, count = ctypes.c_int(0), ctypes.c_int(0)
    _check(_lib.cb_plan_history(plan, slot_t.ctypes.data, ctypes.byref(head), ctypes.byref(count)),
           "cb_plan_history")
    return slot_t, head.value, count.value


def cb_plan_reset(plan) -> None:
    _check(_lib.cb_plan_reset(plan), "cb_plan_reset")


def cb_plan_set_option(plan, option: int, value: int) -> None:
    _check(_lib.cb_plan_set_option(plan, option, int(value)), "cb_plan_set_option")
    d = _dims(plan)
    if d is not None and option == CB_OPT_PARTIAL_HISTORY:
        d[_PARTIAL] = bool(value)


def cb_plan_device_status(plan, stream=None) -> int:
    st = ctypes.c_int(0)
    _check(_lib.cb_plan_device_status(plan, ctypes.byref(st), _stream(stream)), "cb_plan_device_status")
    return st.value


def cb_plan_num_groups(plan) -> int:
    return int(_lib.cb_plan_num_groups(plan))


def cb_plan_destroy(plan) -> None:
    _PLANS.pop(_plan_key(plan), None)
    _lib.cb_plan_destroy(plan)


def cb_status_string(status: int) -> str:
    return _lib.cb_status_string(status).decode()


def cb_last_error_message() -> str:
    return _lib.cb_last_error_message().decode()


def raw_status(name: str, *args) -> int:
    """Call an entry point and return its status instead of raising (tests)."""
    return getattr(_lib, name)(*args)
