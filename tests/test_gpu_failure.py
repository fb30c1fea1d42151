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
