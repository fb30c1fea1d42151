"""GPU parity at the full per-layer sizes of the benchmark workloads.

One layer of each workload at its full size, driven exactly as bench.py drives it (default cache
options, the fused single-token append + decode step):
  * retained sets of every (sequence, KV head) bit-exact against the oracle at the start and end
    of decoding and at >= 8 steps in between;
  * attention outputs of a seeded sample of (step, sequence, KV head) groups -- all G query heads
    of each, >= 256 (step, sequence, query head) tuples per workload -- within max-abs 2e-2 and
    mean-abs 2e-3, the sample always including the longest and the shortest head.
"""
import numpy as np
import pytest
import torch

import paper_2506_05345_gb300 as dms
import workloads
from _harness import Run

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dms.library()


def _sweep(name):
    for w in workloads.sweep_workloads():
        if w.name == name:
            return w
    raise KeyError(name)


def _full_size(wl, steps=None, n_checks=10, pairs_per_check=None, seed=0):
    steps = wl.decode_steps if steps is None else steps
    B, H, G = wl.batch, wl.kv_heads, wl.gqa_group
    if pairs_per_check is None:  # >= 256 (b, hq) tuples over the output checks
        pairs_per_check = max(2, int(np.ceil(256 / (G * n_checks))))
    rng = np.random.default_rng(seed)
    check_steps = sorted(set(np.linspace(0, steps - 1, n_checks).astype(int).tolist()))
    r = Run(wl, fused=True)
    try:
        r.prefill()
        r.check_retained()
        n_tuples = 0
        for s in range(steps):
            q, out = r.step(s)
            if s in check_steps:
                st = r.check_retained()  # every head, bit-exact
                counts = st["counts"][0]
                flat = rng.choice(B * H, size=min(pairs_per_check, B * H), replace=False)
                pairs = {(int(x) // H, int(x) % H) for x in flat}
                bl, hl = np.unravel_index(np.argmax(counts), counts.shape)
                bs, hs = np.unravel_index(np.argmin(counts), counts.shape)
                pairs |= {(int(bl), int(hl)), (int(bs), int(hs))}
                r.check_outputs(q, out, pairs=sorted(pairs))
                n_tuples += len(pairs) * G
        assert n_tuples >= 256
        return r.summary()
    finally:
        r.close()


def test_qwen7b_b64_ctx8192_p075():
    """B 64, 28 q / 4 kv heads, prefill 7936 + 256 fused decode steps, P(evict) 0.75."""
    _full_size(workloads.QWEN7B_B64_8K)


def test_qwen32b_b8_ctx32768_koutliers():
    """B 8, 40 q / 8 kv heads, prefill 32512 + 256 steps, P(evict) 0.875, x8 K outlier channels."""
    _full_size(workloads.QWEN32B_B8_32K)


def test_qwen32b_32threads_shared_prefix_beta82():
    """32 threads of a shared 2048-token prefix + 16128 own tokens + 256 steps, ragged heads."""
    wl = workloads.QWEN32B_THREADS32
    mx, mean = _full_size(wl)
    r = 1.0 - workloads.head_evict_prob(wl, 0)  # retained fraction per KV head
    assert r.max() / r.min() > 2.0  # strongly ragged heads in this layer


@pytest.mark.parametrize("name", [
    "sweep-cr1-b16-ctx16384",   # dense (no evictions)
    "sweep-cr2-b64-ctx4096",
    "sweep-cr4-b1-ctx65536",
    "sweep-cr8-b256-ctx4096",
    "sweep-cr8-b16-ctx65536",
])
def test_sweep_points(name):
    """Points of the compression x batch x context sweep at full per-layer size (32 steps)."""
    _full_size(_sweep(name), steps=32, n_checks=8)
