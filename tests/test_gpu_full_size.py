"""GPU parity at the full per-layer sizes of the benchmark workloads.

The named workloads run two layers of one cache at full per-layer size, driven exactly as
bench.py drives them (default cache options, every step the fused single-token append + decode
of each layer in order); the sweep points run one layer.  Checked:
  * retained sets of every (layer, sequence, KV head) bit-exact against the oracle at the start
    and end of decoding and at >= 8 steps in between;
  * attention outputs of a seeded sample of (layer, step, sequence, KV head) groups -- all G
    query heads of each, >= 256 (step, sequence, query head) tuples per layer -- within max-abs
    2e-2 and mean-abs 2e-3, the sample always including the layer's longest and shortest head.
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


def _full_size(wl, steps=None, n_checks=10, pairs_per_check=None, seed=0, layers=1):
    steps = wl.decode_steps if steps is None else steps
    B, H, G = wl.batch, wl.kv_heads, wl.gqa_group
    if pairs_per_check is None:  # >= 256 (b, hq) tuples per layer over the output checks
        pairs_per_check = max(2, int(np.ceil(256 / (G * n_checks))))
    rng = np.random.default_rng(seed)
    check_steps = sorted(set(np.linspace(0, steps - 1, n_checks).astype(int).tolist()))
    assert len(check_steps) >= min(steps, 8) and check_steps[0] == 0 and check_steps[-1] == steps - 1
    r = Run(wl, fused=True, layers=layers)
    try:
        r.prefill()
        for layer in range(layers):
            r.check_retained(layer=layer)
        n_tuples = [0] * layers
        for s in range(steps):
            outs = r.step_all(s)
            if s in check_steps:
                for layer, (q, out) in enumerate(outs):
                    st = r.check_retained(layer=layer)  # every head, bit-exact
                    counts = st["counts"][layer]
                    flat = rng.choice(B * H, size=min(pairs_per_check, B * H), replace=False)
                    pairs = {(int(x) // H, int(x) % H) for x in flat}
                    bl, hl = np.unravel_index(np.argmax(counts), counts.shape)
                    bs, hs = np.unravel_index(np.argmin(counts), counts.shape)
                    pairs |= {(int(bl), int(hl)), (int(bs), int(hs))}
                    r.check_outputs(q, out, pairs=sorted(pairs), layer=layer)
                    n_tuples[layer] += len(pairs) * G
        assert min(n_tuples) >= min(256, B * H * G * len(check_steps))
        return r.summary()
    finally:
        r.close()


def test_qwen7b_b64_ctx8192_p075():
    """B 64, 28 q / 4 kv heads, prefill 7936 + 256 fused decode steps, P(evict) 0.75; two layers."""
    _full_size(workloads.QWEN7B_B64_8K, layers=2)


def test_qwen32b_b8_ctx32768_koutliers():
    """B 8, 40 q / 8 kv heads, prefill 32512 + 256 steps, P(evict) 0.875, x8 K outlier channels;
    two layers."""
    _full_size(workloads.QWEN32B_B8_32K, layers=2)


def test_qwen32b_32threads_shared_prefix_beta82():
    """32 threads of a shared 2048-token prefix + 16128 own tokens + 256 steps, ragged heads;
    two layers (each with its own Beta(8,2) eviction probabilities)."""
    wl = workloads.QWEN32B_THREADS32
    _full_size(wl, layers=2)
    for layer in range(2):
        r = 1.0 - workloads.head_evict_prob(wl, layer)  # retained fraction per KV head
        assert r.max() / r.min() > 2.0  # strongly ragged heads in this layer


def test_one_layer_alternating_with_another_of_odd_page_table_stride():
    """Two layers whose page tables start off 16-byte boundaries (batch 1, 3 KV heads, 21 pages
    per head): layer 1's table begins 63 int32 entries in, and the decode prefetches each
    layer's table.  Steps alternate layers, so every decode may read its layer's state early."""
    wl = workloads.Workload(name="odd-stride", batch=1, layers=2, q_heads=12, kv_heads=3,
                            window=256, prefill=((1280, False),), decode_steps=40, p_evict=0.5)
    assert (wl.batch * wl.kv_heads * -(-wl.context // 64)) % 4 != 0
    _full_size(wl, n_checks=8, layers=2)


# Every point at 8x compression, the largest point (dense, batch 256, 64K context: 68.7 GB of
# KV in one layer) and one point of each other compression.
SWEEP_POINTS = ([f"sweep-cr8-b{b}-ctx{c}" for b in (1, 16, 64, 256) for c in (4096, 16384, 65536)] +
                ["sweep-cr1-b256-ctx65536", "sweep-cr1-b16-ctx16384", "sweep-cr2-b64-ctx4096",
                 "sweep-cr4-b1-ctx65536"])


@pytest.mark.parametrize("name", SWEEP_POINTS)
def test_sweep_points(name):
    """Points of the compression x batch x context sweep at full per-layer size (32 steps; the
    16 largest-footprint steps for points of 64K context and batch 64 or more)."""
    wl = _sweep(name)
    big = wl.batch >= 64 and wl.context >= 65536
    _full_size(wl, steps=16 if big else 32, n_checks=8)
