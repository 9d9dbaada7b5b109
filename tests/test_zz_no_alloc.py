"""cb_extrapolate_noalloc, the skipped step for callers that may not allocate
device memory, checked against cb_extrapolate_ring on the GPU.

Who calls it: an operator inside a framework or inference engine that lays out
every device buffer in advance and hands each operator only its inputs and
outputs. Such an operator may not call cudaMalloc. It can keep the history in
a buffer of exactly K slots, but it cannot add the status block that binding a
cache arena asks for. The call reads that buffer directly and records
device-side events in a status block the library holds itself.

This file is named to be collected last: a run that stops at its first failure
has then run every other test already. It also passes on its own in a fresh
process (the library's per-device set-up happens on the first call here).
"""
import pytest
import torch

from paper_2608_23429_gb300 import workloads

pytestmark = pytest.mark.gpu

K = 4
NODES = [999.0, 960.0, 921.0, 882.0, 843.0]  # five full steps into four slots: the ring has wrapped


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
    import oracle
    oracle.build()
    return gpu_harness


def _workload():
    """Lone tensors with ragged sizes (one element to many tiles) and two
    residual groups, bf16 cache."""
    tensors = [workloads.TensorSpec(i, 0, (1, 1, n), -1) for i, n in enumerate([1, 7, 4095, 4097, 12345, 300001])]
    tensors += [workloads.TensorSpec(20, b, (2, 3, 1001), 0) for b in range(3)]
    tensors += [workloads.TensorSpec(21, b, (1, 16, 512), 1) for b in range(2)]
    return workloads.Workload(name="noalloc", tensors=tensors, K=K, cache_dtype="bf16", T=0, r=0, t_min=0.0,
                              t_max=999.0, timesteps=[], degree=6, noise=0.1, seed=91)


def _bits(x):
    return x.view(torch.int16) if x.dtype == torch.bfloat16 else x.view(torch.int32)


def test_noalloc_matches_ring_on_two_calls(cb, H):
    w = _workload()
    walk = H.Walk(w, node_t=NODES, kernel="bulk")
    for k, t in enumerate(NODES):
        walk.push(t, k)
    slot_t, head, count = cb.cb_plan_history(walk.plan, K)
    assert count == K and head != 0
    slot_bytes = (cb.cb_plan_cache_bytes(walk.plan) - cb.CB_STATUS_BYTES) // K
    # the caller's history buffer: exactly the K slots, with no status block after them
    hist = torch.empty(K * slot_bytes, dtype=torch.uint8, device="cuda")
    hist.copy_(walk.cache[: K * slot_bytes])
    # a plan for the same tensors that is never bound to a cache arena
    plan = cb.cb_plan_create(NODES, K, walk.tensors, H.CB["bf16"], w.t_min, w.t_max)
    cb.cb_plan_set_option(plan, cb.CB_OPT_KERNEL, cb.CB_KERNEL_BULK)
    status = torch.full((1,), -1, dtype=torch.int32).pin_memory()
    torch.cuda.synchronize()

    # two calls in a row: predictions with the hidden states fused, then fp32 predictions alone
    for call, (t, out_dt, fused) in enumerate([(820.0, "bf16", True), (801.5, "fp32", False)]):
        ref_o, ref_r, rh = walk.extrapolate(t, out_dtype=out_dt, fused=fused, salt=call, ring=(slot_t, head))
        outs = [torch.full(s.shape, float("nan"), dtype=H.TORCH[out_dt], device="cuda") for s in w.tensors]
        resid = ([workloads.hidden_state(w, g, "cuda", torch.bfloat16, salt=call) for g in range(walk.n_groups)]
                 if fused else None)
        status.fill_(-1)
        cb.cb_extrapolate_noalloc(plan, hist, hist.numel(), slot_t, head, t, outs, H.CB[out_dt], resid,
                                  cb.CB_BF16, status=status)
        torch.cuda.synchronize()
        assert int(status[0]) == 0, call  # the shared word was cleared and nothing was recorded
        # the same kernel on the same bytes: identical to the bound plan's call
        for i, (a, b) in enumerate(zip(ref_o, outs)):
            assert torch.equal(_bits(a), _bits(b)), (call, i)
        if fused:
            for g, (a, b) in enumerate(zip(ref_r, resid)):
                assert torch.equal(_bits(a), _bits(b)), (call, g)
        # and within the parity gates of the oracle
        so, sr, _ = walk.expected_and_compare(t, outs, resid, rh, out_dtype=out_dt)
        assert so["bad"] == 0, (call, so)
        assert not fused or sr["bad"] == 0, (call, sr)

    # the unbound plan's own history is untouched
    assert cb.cb_plan_history(plan, K)[2] == 0
    # arguments are checked before anything is enqueued
    for args, code in [((hist, hist.numel() - 1, slot_t, head), cb.CB_ERR_ARG),
                       ((hist.data_ptr() + 16, hist.numel() - 16, slot_t, head), cb.CB_ERR_ALIGN),
                       ((hist, hist.numel(), slot_t, K), cb.CB_ERR_ARG)]:
        with pytest.raises(cb.CbError) as e:
            cb.cb_extrapolate_noalloc(plan, *args, 820.0, outs, cb.CB_FP32)
        assert e.value.status == code
    cb.cb_plan_destroy(plan)
    walk.close()
