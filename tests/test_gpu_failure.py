"""Failure detection on the GPU without a GPU fault.

Every shared-memory barrier wait in the kernels is bounded by %globaltimer; when it runs out the
kernel records DMS_ERR_TIMEOUT and exits normally.  The self-test entry point runs exactly that
wait on a barrier that nothing completes (a flag nobody sets), with a short limit, and the test
checks the status, the elapsed time, and that the context still works afterwards.
"""
import ctypes
import time

import pytest
import torch

import paper_2506_05345_gb300 as dms
import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dms.library()


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def test_bounded_wait_completes_when_arrived():
    assert dms.dms_selftest_bounded_wait(1, 50_000_000, _stream()) == dms.DMS_OK


def test_bounded_wait_times_out_and_context_survives():
    t0 = time.perf_counter()
    code = dms.dms_selftest_bounded_wait(0, 30_000_000, _stream())  # 30 ms, nobody arrives
    dt = time.perf_counter() - t0
    assert code == dms.DMS_ERR_TIMEOUT
    assert dt >= 0.025
    # the context is intact: a decode step still runs and matches the oracle
    from _harness import Run
    wl = workloads.Workload(name="after-timeout", batch=1, layers=1, q_heads=4, kv_heads=1,
                            window=8, prefill=((100, False),), decode_steps=2, p_evict=0.5)
    r = Run(wl, fused=True)
    try:
        r.prefill()
        for s in range(2):
            q, out = r.step(s)
            r.check_outputs(q, out)
        r.check_retained()
    finally:
        r.close()


def test_selftest_rejects_bad_limits():
    assert dms.dms_selftest_bounded_wait(0, 10, _stream()) == dms.DMS_ERR_INVALID_ARGUMENT


def test_cluster_flag_wait_times_out_and_falls_back():
    """A cluster launch whose head flags never arrive (the self-test makes it wait for a value
    no launch publishes, 2 ms limit): every head's wait gives up, DMS_ERR_TIMEOUT is recorded,
    the launch falls back to the dependency wait and still computes the oracle's result; the
    next launches run normally, and a reset clears the sticky error."""
    import _harness
    import workloads
    wl = workloads.Workload(name="stale-flag", batch=1, layers=1, q_heads=20, kv_heads=4,
                            window=32, prefill=((600, False),), decode_steps=8, p_evict=0.6)
    r = _harness.Run(wl, fused=True, decode_kernel=dms.DMS_DECODE_CLUSTER)
    try:
        assert r.cache.decode_plan(wl.gqa_group)["kernel"] == dms.DMS_DECODE_CLUSTER
        r.prefill()
        for s in range(2):  # the layer's state is now last written by flag-publishing launches
            q, out = r.step(s)
            r.check_outputs(q, out)
        assert r.cache.stats()["device_error"] == 0
        code = dms.library().dms_selftest_stale_flag(ctypes.c_void_p(r.cache.handle), 0, 2_000_000)
        assert code == dms.DMS_OK
        q, out = r.step(2)
        r.check_outputs(q, out)  # the fallback read the completed state
        assert r.cache.stats()["device_error"] == dms.DMS_ERR_TIMEOUT
        for s in range(3, 6):
            q, out = r.step(s)
            r.check_outputs(q, out)
        r.cache.reset()
        assert r.cache.stats()["device_error"] == 0
    finally:
        r.close()
