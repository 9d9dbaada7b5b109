"""The parity gates of the GPU tests, checked on the CPU.

The comparators in gpu_harness decide every GPU parity verdict, so they are
pinned here against values whose distances are known by construction: bf16
patterns a fixed number of representable values apart (also across zero),
cancellation cases inside and outside the 2^-40 floor, and fp32 errors just
inside and just outside 2e-6 max|F|.
"""
import numpy as np
import pytest


@pytest.fixture(scope="module")
def H():
    from paper_2608_23429_gb300 import build
    build.build()
    import oracle
    oracle.build()
    import gpu_harness
    return gpu_harness


def _ref(H, x):
    bits = H.orc.bf16_encode(np.asarray(x, np.float64))
    return bits, H.bf16_to_f64(bits)


def test_bf16_gate_counts_representable_steps(H):
    rng = np.random.default_rng(5)
    ref, ref64 = _ref(H, rng.standard_normal(4000) * 10.0 ** rng.integers(-30, 30, 4000))
    bound = np.abs(ref64)  # floor far below one ulp: it never applies here
    s = H.compare_bf16(ref, ref, ref64, bound)
    assert s["exact"] == s["n"] == 4000 and s["bad"] == 0 and s["max_ulp"] == 0
    for k in (1, -1):
        s = H.compare_bf16(H._step(ref, k), ref, ref64, bound)
        assert s["one_ulp"] == 4000 and s["bad"] == 0 and s["max_ulp"] == 1, k
    for k in (2, -2, 7):
        s = H.compare_bf16(H._step(ref, k), ref, ref64, bound)
        assert s["bad"] == 4000 and s["max_ulp"] == abs(k), k
    # one element off by two in a tensor that is otherwise exact fails the gate
    g = ref.copy()
    g[123] = H._step(ref[123:124], 2)[0]
    assert H.compare_bf16(g, ref, ref64, bound)["bad"] == 1


def test_bf16_gate_across_zero(H):
    z = np.zeros(1)
    # +0 and -0 are the same value
    s = H.compare_bf16(np.array([0x8000], np.uint16), np.array([0x0000], np.uint16), z, z)
    assert s["exact"] == 1
    # the smallest subnormals of either sign are two representable values apart
    pos, neg = np.array([0x0001], np.uint16), np.array([0x8001], np.uint16)
    s = H.compare_bf16(neg, pos, H.bf16_to_f64(pos), np.zeros(1))
    assert s["max_ulp"] == 2 and s["bad"] == 1
    s = H.compare_bf16(np.array([0x0000], np.uint16), pos, H.bf16_to_f64(pos), np.zeros(1))
    assert s["one_ulp"] == 1 and s["bad"] == 0


def test_bf16_cancellation_floor(H):
    # exact result 1e-30 after cancellation of terms of size ~1: the GPU's value
    # three times larger is many ulps away but within 2^-40 sum|w F|
    exact = np.array([1e-30])
    ref, _ = _ref(H, exact)
    gpu, _ = _ref(H, 3 * exact)
    s = H.compare_bf16(gpu, ref, exact, np.array([1.0]))
    assert s["max_ulp"] > 1 and s["floor"] == 1 and s["bad"] == 0
    # the same distance with terms of size 1e-20 is outside the floor
    s = H.compare_bf16(gpu, ref, exact, np.array([1e-20]))
    assert s["floor"] == 0 and s["bad"] == 1


def test_fp32_gate(H):
    rng = np.random.default_rng(6)
    ref = rng.uniform(-1, 1, 1000)
    ref[0] = 1.0  # max|F| = 1: tolerance 2e-6
    for err, bad in ((1.9e-6, 0), (2.1e-6, 1)):
        g = (ref + 0.0).astype(np.float32)
        g64 = g.astype(np.float64)
        # place one element exactly err away (in fp64 terms of the stored fp32 value)
        g[500] = np.float32(ref[500] + err)
        s = H.compare_fp32(g, np.where(np.arange(1000) == 500, ref, g64), 1.0)
        assert s["bad"] == bad and abs(s["max_err"] - abs(float(g[500]) - ref[500])) < 1e-12, err


def test_merge_adds_counts_and_keeps_maxima(H):
    a = dict(n=10, exact=8, one_ulp=2, floor=0, bad=0, max_ulp=1)
    b = dict(n=5, exact=3, one_ulp=1, floor=1, bad=0, max_ulp=9)
    m = H.merge([a, b])
    assert m == dict(n=15, exact=11, one_ulp=3, floor=1, bad=0, max_ulp=9)


def test_bench_parity_record_agrees_with_the_harness(H):
    """bench.py's parity record (the timed FLUX step against the oracle)
    counts exactly as the GPU tests' gate: the same ulp distances, the same
    cancellation floor, on patterns 0..3 values apart and on cancellations
    inside and outside the floor."""
    import bench
    rng = np.random.default_rng(11)
    ref, ref64 = _ref(H, rng.standard_normal(3000) * 10.0 ** rng.integers(-20, 20, 3000))
    bound = np.abs(ref64)
    gpu = ref.copy()
    gpu[:600] = H._step(ref[:600], 1)
    gpu[600:900] = H._step(ref[600:900], -2)
    gpu[900:1000] = H._step(ref[900:1000], 3)
    # exact value ~0 beside large terms: a gpu value within the floor passes, one outside fails
    ref64[1000:1100] = 0.0
    ref[1000:1100] = 0
    bound[1000:1100] = 2.0 ** 50
    gpu[1000:1050] = H.orc.bf16_encode(np.full(50, 2.0 ** 9))    # 2^9 <= 2^-40 * 2^50: inside the floor
    gpu[1050:1100] = H.orc.bf16_encode(np.full(50, 2.0 ** 11))   # outside it
    mine = bench.parity_stats(gpu, ref, ref64, bound)
    theirs = H.compare_bf16(gpu, ref, ref64, bound)
    assert mine == theirs
    assert mine["one_ulp"] == 600 and mine["floor"] == 50 and mine["bad"] == 300 + 100 + 50
