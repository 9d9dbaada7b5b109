"""C ABI and host logic of libchebboost, on the CPU.

No test here launches a kernel: they cover the exported symbols, the
host-side schedule and weight precomputation (against the oracle), the slot
layout and every validation error that is returned before a launch.
"""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def cb():
    from paper_2608_23429_gb300 import build
    build.build()
    from paper_2608_23429_gb300 import chebboost
    return chebboost


def _declared():
    src = open(os.path.join(ROOT, "include", "chebboost.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(cb_\w+)\s*\(", src)))


def test_every_declared_symbol_is_exported(cb):
    names = _declared()
    assert len(names) >= 15
    lib = ctypes.CDLL(cb.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) <= set(cb.EXPORTED)


def test_constants_match_header(cb):
    """Every #define and enum value of the header has the same value in the binding."""
    src = re.sub(r"/\*.*?\*/", "", open(os.path.join(ROOT, "include", "chebboost.h")).read(), flags=re.S)
    consts = {m[0]: m[1] for m in re.findall(r"#define\s+(CB_\w+)\s+(.+)", src)}
    consts.update({m[0]: m[1] for m in re.findall(r"\b(CB_\w+)\s*=\s*(-?\d+)", src)})
    assert len(consts) >= 25
    for name, text in consts.items():
        value = eval(text.strip().replace("1LL", "1"), {})
        assert getattr(cb, name) == value, name


def test_status_strings(cb):
    for s in range(0, -9, -1):
        assert cb.cb_status_string(s) and cb.cb_status_string(s) != "unknown status"


def test_schedule_matches_oracle(cb, orc):
    rng = np.random.default_rng(3)
    for _ in range(300):
        T = int(rng.integers(1, 60))
        r = int(rng.integers(1, 9))
        s0, s1, K = int(rng.integers(0, 6)), int(rng.integers(0, 6)), int(rng.integers(0, 9))
        mask, n = cb.cb_schedule_full(T, r, s0, s1, K)
        ref = orc.full_schedule(T, r, s0, s1, K)
        assert np.array_equal(mask, ref), (T, r, s0, s1, K)
        assert n == int(ref.sum())


def _tensors(numels, groups=None):
    groups = groups or [-1] * len(numels)
    return [(i, 0, n, g) for i, (n, g) in enumerate(zip(numels, groups))]


def test_plan_create_errors(cb):
    E = cb.CbError
    nodes = [999.0, 900.0, 800.0, 700.0]
    ok = _tensors([100, 100])

    def status(**kw):
        args = dict(node_t=nodes, K=3, tensors=ok, cache_dtype=cb.CB_BF16, t_min=0.0, t_max=999.0)
        args.update(kw)
        try:
            p = cb.cb_plan_create(**args)
        except E as e:
            return e.status
        cb.cb_plan_destroy(p)
        return 0

    assert status() == 0
    assert status(K=0) == cb.CB_ERR_ARG
    assert status(K=9) == cb.CB_ERR_LIMIT
    assert status(node_t=nodes[:2]) == cb.CB_ERR_ARG
    assert status(node_t=[999.0, 900.0, 900.0, 700.0]) == cb.CB_ERR_NODES_DEGENERATE
    assert status(node_t=[999.0, 900.0, 950.0, 700.0]) == cb.CB_ERR_ARG
    assert status(t_min=5.0, t_max=5.0) == cb.CB_ERR_ARG
    assert status(t_min=float("nan")) == cb.CB_ERR_ARG
    assert status(cache_dtype=7) == cb.CB_ERR_ARG
    assert status(tensors=_tensors([100, 0])) == cb.CB_ERR_ARG
    assert status(tensors=_tensors([100, 101], [0, 0])) == cb.CB_ERR_ARG  # group numel mismatch
    assert status(tensors=_tensors([8] * 5, [0] * 5)) == cb.CB_ERR_LIMIT  # > CB_MAX_BRANCHES
    assert status(tensors=_tensors([8] * 257)) == cb.CB_ERR_LIMIT
    assert status(tensors=[(0, 0, 8, -2)]) == cb.CB_ERR_ARG
    assert status(tensors=[(0, 0, 8, cb.CB_MAX_TENSORS)]) == cb.CB_ERR_LIMIT  # group index
    assert status(tensors=_tensors([cb.CB_MAX_NUMEL])) == 0
    assert status(tensors=_tensors([8, cb.CB_MAX_NUMEL + 1])) == cb.CB_ERR_LIMIT


def test_cache_layout_and_bind(cb):
    numels = [1, 7, 128, 129, 1000]
    for dt, es in ((cb.CB_BF16, 2), (cb.CB_FP32, 4)):
        p = cb.cb_plan_create([3.0, 2.0, 1.0], 3, _tensors(numels), dt, 0.0, 3.0)
        slot = sum((n * es + 255) // 256 * 256 for n in numels)
        assert cb.cb_plan_cache_bytes(p) == 3 * slot + cb.CB_STATUS_BYTES
        with pytest.raises(cb.CbError) as e:
            cb.cb_plan_bind_cache(p, 0x1000 + 128, 3 * slot + cb.CB_STATUS_BYTES)
        assert e.value.status == cb.CB_ERR_ALIGN
        with pytest.raises(cb.CbError) as e:
            cb.cb_plan_bind_cache(p, 0x1000, 3 * slot + cb.CB_STATUS_BYTES - 1)
        assert e.value.status == cb.CB_ERR_ARG
        cb.cb_plan_destroy(p)


def test_validation_before_launch(cb):
    """Every error below is returned before any CUDA call (safe with or without a GPU)."""
    p = cb.cb_plan_create([999.0, 900.0, 800.0], 3, _tensors([64, 64], [0, 0]), cb.CB_BF16, 0.0, 999.0)
    st = cb.raw_status
    arr = lambda *xs: (ctypes.c_void_p * len(xs))(*xs)
    # unbound
    assert st("cb_cache_push", p, arr(0x1000, 0x2000), 0, 999.0, None) == cb.CB_ERR_UNBOUND
    assert st("cb_extrapolate", p, 850.0, arr(0x1000, 0x2000), 0, None, 0, None) == cb.CB_ERR_UNBOUND
    cb.cb_plan_bind_cache(p, 0x100000, cb.cb_plan_cache_bytes(p))  # never dereferenced below
    assert st("cb_cache_push", p, None, 0, 999.0, None) == cb.CB_ERR_ARG
    assert st("cb_cache_push", p, arr(0x1000, 0), 0, 999.0, None) == cb.CB_ERR_ARG
    assert st("cb_cache_push", p, arr(0x1001, 0x2000), 0, 999.0, None) == cb.CB_ERR_ALIGN
    assert st("cb_cache_push", p, arr(0x1002, 0x2000), 1, 999.0, None) == cb.CB_ERR_ALIGN
    assert st("cb_cache_push", p, arr(0x1000, 0x2000), 5, 999.0, None) == cb.CB_ERR_ARG
    assert st("cb_cache_push", p, arr(0x1000, 0x2000), 0, float("inf"), None) == cb.CB_ERR_ARG
    # history not full
    assert st("cb_extrapolate", p, 850.0, arr(0x1000, 0x2000), 0, None, 0, None) == cb.CB_ERR_HISTORY_NOT_FULL
    assert st("cb_extrapolate_ring", p, (ctypes.c_double * 3)(1, 2, 3), 0, 850.0, None, 0, None, 0,
              None) == cb.CB_ERR_HISTORY_NOT_FULL
    assert st("cb_extrapolate_ring", p, (ctypes.c_double * 3)(1, 2, 3), 3, 850.0, None, 0, None, 0,
              None) == cb.CB_ERR_ARG
    w = (ctypes.c_double * 3)()
    assert st("cb_weights", p, 850.0, w) == cb.CB_ERR_HISTORY_NOT_FULL
    slot_t, head, count = cb.cb_plan_history(p, 3)
    assert (head, count) == (0, 0)
    # options
    assert st("cb_plan_set_option", p, cb.CB_OPT_KERNEL, 7) == cb.CB_ERR_ARG
    assert st("cb_plan_set_option", p, cb.CB_OPT_WAIT_NS, -1) == cb.CB_ERR_ARG
    assert st("cb_plan_set_option", p, 99, 0) == cb.CB_ERR_ARG
    assert st("cb_plan_set_option", p, cb.CB_OPT_PARTIAL_HISTORY, 2) == cb.CB_ERR_ARG
    w3 = (ctypes.c_double * 3)(0.2, 0.3, 0.5)
    assert st("cb_extrapolate_weights", p, w3, arr(0x1000, 0x2000), 0, None, 0, None) == cb.CB_ERR_HISTORY_NOT_FULL
    assert st("cb_extrapolate_weights", p, None, arr(0x1000, 0x2000), 0, None, 0, None) == cb.CB_ERR_ARG
    for k in (cb.CB_KERNEL_DIRECT, cb.CB_KERNEL_BULK, cb.CB_KERNEL_AUTO):
        cb.cb_plan_set_option(p, cb.CB_OPT_KERNEL, k)
    # nothing has run since binding: the status read touches no device memory
    assert cb.cb_plan_device_status(p) == 0
    assert cb.cb_plan_num_groups(p) == 1
    cb.cb_plan_destroy(p)


def test_noalloc_validation_before_any_cuda_call(cb):
    """cb_extrapolate_noalloc checks its arguments before it touches CUDA (its
    per-device set-up included), so every malformed call below returns its
    code on a machine without a GPU. The plan is never bound: the call needs
    no arena."""
    p = cb.cb_plan_create([999.0, 900.0, 800.0], 3, _tensors([64, 64], [0, 0]), cb.CB_BF16, 0.0, 999.0)
    st = cb.raw_status
    arr = lambda *xs: (ctypes.c_void_p * len(xs))(*xs)
    need = cb.cb_plan_cache_bytes(p) - cb.CB_STATUS_BYTES  # the K slots, no status block
    times = (ctypes.c_double * 3)(999.0, 900.0, 800.0)
    outs = arr(0x1000, 0x2000)
    hist = 0x100000  # never dereferenced below
    call = lambda h, nbytes, t, head, tgt, o=outs: st("cb_extrapolate_noalloc", p, h, nbytes, t, head, tgt, o, 0,
                                                      None, 0, None, None)
    assert call(None, need, times, 0, 850.0) == cb.CB_ERR_ARG            # no history buffer
    assert call(hist + 16, need, times, 0, 850.0) == cb.CB_ERR_ALIGN     # not CB_CACHE_ALIGN-aligned
    assert call(hist, need - 1, times, 0, 850.0) == cb.CB_ERR_ARG        # shorter than the K slots
    assert call(hist, need, None, 0, 850.0) == cb.CB_ERR_ARG             # no slot times
    assert call(hist, need, times, 3, 850.0) == cb.CB_ERR_ARG            # head outside [0, K)
    assert call(hist, need, times, -1, 850.0) == cb.CB_ERR_ARG
    assert call(hist, need, times, 0, float("nan")) == cb.CB_ERR_ARG     # target not finite
    dup = (ctypes.c_double * 3)(999.0, 900.0, 999.0)
    assert call(hist, need, dup, 0, 850.0) == cb.CB_ERR_NODES_DEGENERATE
    bad = (ctypes.c_double * 3)(999.0, float("inf"), 800.0)
    assert call(hist, need, bad, 0, 850.0) == cb.CB_ERR_ARG
    assert st("cb_extrapolate_noalloc", None, hist, need, times, 0, 850.0, outs, 0, None, 0, None,
              None) == cb.CB_ERR_ARG                                    # no plan
    # the plan's own history is untouched, and it was never bound
    assert cb.cb_plan_history(p, 3)[1:] == (0, 0)
    cb.cb_plan_destroy(p)


def test_failed_launch_leaves_history_unchanged(cb):
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("needs a machine without a GPU (the push must fail at the CUDA call)")
    p = cb.cb_plan_create([999.0, 900.0], 2, _tensors([64]), cb.CB_BF16, 0.0, 999.0)
    cb.cb_plan_bind_cache(p, 0x100000, cb.cb_plan_cache_bytes(p))
    rc = cb.raw_status("cb_cache_push", p, (ctypes.c_void_p * 1)(0x1000), 0, 999.0, None)
    assert rc == cb.CB_ERR_CUDA
    assert cb.cb_last_error_message() != ""
    assert cb.cb_plan_history(p, 2)[2] == 0
    cb.cb_plan_destroy(p)


def _workload_nodes(w, orc):
    from paper_2608_23429_gb300 import chebboost as cb
    mask, _ = cb.cb_schedule_full(w.T, w.r, w.s0, w.s1, w.K)  # the product's schedule
    assert np.array_equal(mask, orc.full_schedule(w.T, w.r, w.s0, w.s1, w.K))
    ts = np.array(w.timesteps)
    return ts[mask], ts[~mask]


@pytest.mark.parametrize("name", ["dit256", "dit256-k3", "dit512", "pixart", "flux"])
def test_exported_weight_table_matches_oracle(cb, orc, name):
    """The precomputed weight table (Alg. 1 offline stage) for every skipped step of the
    schedule, against the oracle's Lagrange basis on the same K preceding nodes."""
    from paper_2608_23429_gb300 import workloads
    w = workloads.PRESETS[name]()
    nodes, targets = _workload_nodes(w, orc)
    p = cb.cb_plan_create(nodes, w.K, [(0, 0, 8, -1)], cb.CB_BF16, w.t_min, w.t_max)
    table = cb.cb_plan_export_weights(p, targets, w.K)
    for t, row in zip(targets, table):
        prev = nodes[nodes > t][-w.K:]  # timesteps decrease along the sampling order
        ref = orc.weights(prev, t, w.t_min, w.t_max)
        assert np.max(np.abs(row - ref)) <= 1e-12 * np.abs(ref).sum(), (name, t)
    cb.cb_plan_destroy(p)


def test_export_weights_edge_cases(cb, orc):
    p = cb.cb_plan_create([900.0, 800.0, 700.0, 600.0], 4, [(0, 0, 8, -1)], cb.CB_FP32, 0.0, 1000.0)
    tab = cb.cb_plan_export_weights(p, [575.0, 550.0, 500.0], 4)
    assert np.allclose(tab[2], [-1, 4, -6, 4], rtol=0, atol=1e-13)  # one spacing past the newest node
    with pytest.raises(cb.CbError) as e:
        cb.cb_plan_export_weights(p, [650.0], 4)  # only 3 nodes precede it
    assert e.value.status == cb.CB_ERR_HISTORY_NOT_FULL
    cb.cb_plan_destroy(p)


def test_taylor_weights_match_oracle(cb, orc):
    rng = np.random.default_rng(23)
    for _ in range(200):
        n = int(rng.integers(1, 9))
        h = float(rng.uniform(0.1, 50) * rng.choice([-1, 1]))
        x = float(rng.uniform(-500, 500)) + h * np.arange(n)
        xq = x[-1] + h * float(rng.uniform(0.05, 3))
        ref = orc.taylor_weights(x, xq)
        assert np.max(np.abs(cb.cb_taylor_weights(x, xq) - ref)) <= 1e-12 * np.abs(ref).sum()
    with pytest.raises(cb.CbError):
        cb.cb_taylor_weights([0.0, 1.0, 3.0], 4.0)  # not equispaced
    with pytest.raises(cb.CbError):
        cb.cb_taylor_weights([], 1.0)


def test_shapes_and_gate_validation(cb):
    st = cb.raw_status
    arr = lambda *xs: (ctypes.c_void_p * len(xs))(*xs)
    p = cb.cb_plan_create([999.0, 900.0], 2, [(0, 0, 2 * 4 * 8, 0), (0, 1, 2 * 4 * 8, 0), (1, 0, 64, -1)],
                          cb.CB_BF16, 0.0, 999.0)
    with pytest.raises(cb.CbError) as e:
        cb.cb_plan_set_shapes(p, [(2, 4, 8), (2, 4, 8), (1, 1, 63)])  # product != numel
    assert e.value.status == cb.CB_ERR_ARG
    with pytest.raises(cb.CbError) as e:
        cb.cb_plan_set_shapes(p, [(2, 4, 8), (4, 2, 8), (1, 1, 64)])  # one group, two shapes
    assert e.value.status == cb.CB_ERR_ARG
    # batch (2^61 + 8) x 8 x 1 wraps to 64 in 64-bit arithmetic: still rejected
    with pytest.raises(cb.CbError) as e:
        cb.cb_plan_set_shapes(p, [(2, 4, 8), (2, 4, 8), ((1 << 61) + 8, 8, 1)])
    assert e.value.status == cb.CB_ERR_ARG
    for bad in [(0, 8, 8), (1, 1 << 40, 1 << 40), (1, 1, 65), (3, 1, 21)]:
        with pytest.raises(cb.CbError) as e:
            cb.cb_plan_set_shapes(p, [(2, 4, 8), (2, 4, 8), bad])
        assert e.value.status == cb.CB_ERR_ARG, bad
    with pytest.raises(cb.CbError) as e:  # tokens * hidden >= 2^32
        big = cb.cb_plan_create([999.0, 900.0], 2, [(0, 0, 1 << 33, -1)], cb.CB_BF16, 0.0, 999.0)
        try:
            cb.cb_plan_set_shapes(big, [(1, 1 << 17, 1 << 16)])
        finally:
            cb.cb_plan_destroy(big)
    assert e.value.status == cb.CB_ERR_LIMIT
    cb.cb_plan_bind_cache(p, 0x100000, cb.cb_plan_cache_bytes(p))  # never dereferenced below
    gates = arr(0x3000, 0, 0)
    # history not full is reported before the gates are looked at
    assert st("cb_extrapolate_gated", p, 800.0, None, 0, arr(0x5000), 0, gates, 0, None) == \
        cb.CB_ERR_HISTORY_NOT_FULL
    # pushes with gates validate shapes and alignment before launching
    feats = arr(0x1000, 0x2000, 0x4000)
    assert st("cb_cache_push_residual", p, feats, 0, 999.0, arr(0x5000), 0, gates, 0, None) == cb.CB_ERR_ARG
    cb.cb_plan_set_shapes(p, [(2, 4, 8), (2, 4, 8), (1, 1, 64)])
    assert st("cb_cache_push_residual", p, feats, 0, 999.0, arr(0x5000), 0, arr(0x3001, 0, 0), 0, None) == \
        cb.CB_ERR_ALIGN
    assert st("cb_cache_push_residual", p, feats, 0, 999.0, arr(0x5001), 0, gates, 0, None) == cb.CB_ERR_ALIGN
    assert st("cb_cache_push_residual", p, feats, 0, 999.0, arr(0x5000), 0, gates, 9, None) == cb.CB_ERR_ARG
    cb.cb_plan_destroy(p)


def test_binding_checks_array_lengths(cb):
    """The binding refuses pointer lists, shapes, slot times and weight vectors
    whose length does not match the plan before the library reads them."""
    p = cb.cb_plan_create([999.0, 900.0, 800.0], 3, [(0, 0, 64, 0), (0, 1, 64, 0), (1, 0, 32, -1)],
                          cb.CB_BF16, 0.0, 999.0)
    two, three = [0x1000, 0x2000], [0x1000, 0x2000, 0x3000]
    calls = [
        lambda: cb.cb_cache_push(p, two, cb.CB_BF16, 999.0),
        lambda: cb.cb_extrapolate(p, 700.0, two, cb.CB_BF16),
        lambda: cb.cb_extrapolate(p, 700.0, three, cb.CB_BF16, resid=two),  # one residual group
        lambda: cb.cb_extrapolate_ring(p, [999.0, 900.0], 0, 700.0, three, cb.CB_BF16),
        lambda: cb.cb_extrapolate_weights(p, [0.1, 0.2, 0.3, 0.4], three, cb.CB_BF16),
        lambda: cb.cb_extrapolate_gated(p, 700.0, three, cb.CB_BF16, [0x5000], cb.CB_BF16, two),
        lambda: cb.cb_cache_push_residual(p, two, cb.CB_BF16, 999.0, [0x5000]),
        lambda: cb.cb_cache_push_residual(p, three, cb.CB_BF16, 999.0, two),
        lambda: cb.cb_plan_set_shapes(p, [(1, 8, 8), (1, 8, 8)]),
        lambda: cb.cb_weights(p, 700.0, 9),
        lambda: cb.cb_plan_export_weights(p, [700.0], 2),
        lambda: cb.cb_plan_history(p, 2),
    ]
    for i, call in enumerate(calls):
        with pytest.raises(cb.CbError) as e:
            call()
        assert e.value.status == cb.CB_ERR_ARG, i
    # lengths that match reach the library (which reports its own status)
    with pytest.raises(cb.CbError) as e:
        cb.cb_extrapolate(p, 700.0, three, cb.CB_BF16, resid=[0x5000])
    assert e.value.status == cb.CB_ERR_UNBOUND
    assert len(cb.cb_plan_history(p, 3)[0]) == 3
    cb.cb_plan_destroy(p)


def test_short_weight_vector_is_rejected_not_overread(cb):
    """cb_extrapolate_weights reads one weight per live entry: a shorter vector
    reaches the library padded with NaN and is refused as non-finite."""
    p = cb.cb_plan_create([999.0, 900.0], 2, [(0, 0, 64, -1)], cb.CB_BF16, 0.0, 999.0)
    cb.cb_plan_set_option(p, cb.CB_OPT_PARTIAL_HISTORY, 1)
    buf = cb._weights_in(p, [0.5], "test")
    assert buf.size == cb.CB_MAX_K and buf[0] == 0.5 and np.isnan(buf[1:]).all()
    cb.cb_plan_destroy(p)
    assert cb._dims(p) is None
