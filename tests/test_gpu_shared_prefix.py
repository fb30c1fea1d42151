"""Shared-prompt pages: a prompt identical in every sequence is appended once, its frozen pages
mapped into every sequence (read-only).  The cache must behave exactly like the one filled with
the replicated prompt (outputs and retained positions bit for bit), with fewer pool pages, and
match the fp64 oracle.
"""
import statistics

import numpy as np
import pytest
import torch

import oracle
import paper_2506_05345_gb300 as dms
import workloads
from _harness import MAX_ABS, MEAN_ABS

pytestmark = pytest.mark.gpu
D = 128


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dms.library()


def _kvl(B, n, H, p, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    k = torch.randn((B, n, H, D), generator=g, device="cuda").to(torch.bfloat16)
    v = torch.randn((B, n, H, D), generator=g, device="cuda").to(torch.bfloat16)
    lg = (torch.randn((B, n, H), generator=g, device="cuda")
          + statistics.NormalDist().inv_cdf(p)).to(torch.bfloat16)
    return k, v, lg


def _fill(shared, B, H, G, w, n_pre, n_own, steps, p, policy, seed=0, hist=None):
    cache = dms.DmsCache(layers=1, kv_heads=H, window=w, capacity=n_pre + n_own + steps, batch=B,
                         eviction_policy=policy)
    kp, vp, lp = _kvl(1, n_pre, H, p, seed)
    if shared:
        cache.append_shared_prefix(0, kp, vp, lp)
    else:
        cache.append_and_evict(0, kp.expand(B, -1, -1, -1).contiguous(),
                               vp.expand(B, -1, -1, -1).contiguous(), lp.expand(B, -1, -1).contiguous())
    parts = [(kp.expand(B, -1, -1, -1), vp.expand(B, -1, -1, -1), lp.expand(B, -1, -1))]
    if n_own:
        k, v, lg = _kvl(B, n_own, H, p, seed + 1)
        cache.append_and_evict(0, k, v, lg)
        parts.append((k, v, lg))
    outs = []
    for s in range(steps):
        k, v, lg = _kvl(B, 1, H, p, seed + 100 + s)
        g = torch.Generator(device="cuda").manual_seed(seed + 200 + s)
        q = torch.randn((B, H * G, D), generator=g, device="cuda").to(torch.bfloat16)
        outs.append(cache.append_and_decode(0, k, v, lg, q, gqa_group=G).clone())
        parts.append((k, v, lg))
        if hist is not None:
            hist.append(q)
    return cache, outs, parts


@pytest.mark.parametrize("policy", [dms.DMS_EVICT_DELAYED, dms.DMS_EVICT_IMMEDIATE])
@pytest.mark.parametrize("n_pre,w", [(700, 32), (2048, 256), (20, 64)])
def test_shared_prefix_equals_replicated(policy, n_pre, w):
    B, H, G, n_own, steps = 4, 2, 4, 300, 16
    a, out_a, _ = _fill(True, B, H, G, w, n_pre, n_own, steps, 0.8, policy)
    b, out_b, _ = _fill(False, B, H, G, w, n_pre, n_own, steps, 0.8, policy)
    try:
        for s, (x, y) in enumerate(zip(out_a, out_b)):
            assert torch.equal(x, y), s
        assert np.array_equal(a.export_positions(0), b.export_positions(0))
        sa, sb = a.stats(), b.stats()
        assert sa["device_error"] == 0 and sb["device_error"] == 0
        assert sa["total_retained"] == sb["total_retained"]
        if n_pre > w + 64 * 2:  # some whole pages are frozen: they are stored once
            assert sa["pages_in_use"] < sb["pages_in_use"], (sa, sb)
        else:
            assert sa["pages_in_use"] <= sb["pages_in_use"]
    finally:
        a.close()
        b.close()


def test_shared_prefix_matches_oracle():
    B, H, G, w, n_pre, n_own, steps = 3, 2, 4, 24, 400, 50, 10
    qs = []
    cache, outs, parts = _fill(True, B, H, G, w, n_pre, n_own, steps, 0.75, 0, seed=5, hist=qs)
    try:
        K = workloads.bf16_bits(torch.cat([p[0] for p in parts], 1))
        V = workloads.bf16_bits(torch.cat([p[1] for p in parts], 1))
        L = workloads.bf16_bits(torch.cat([p[2] for p in parts], 1))
        j = K.shape[1] - 1
        pos = cache.export_positions(0)
        cnt = cache.stats(with_counts=True)["counts"][0]
        Q = workloads.bf16_bits(qs[-1])
        got = outs[-1].float().cpu().numpy()
        errs = []
        for b in range(B):
            for h in range(H):
                assert np.array_equal(np.sort(pos[b, h, :int(cnt[b, h])]),
                                      oracle.retained(L[b, :, h], j, w))
                ref = oracle.decode(Q[b, h * G:(h + 1) * G], K[b, :, h], V[b, :, h], L[b, :, h], j, w)
                errs.append(np.abs(got[b, h * G:(h + 1) * G] - ref).ravel())
        e = np.concatenate(errs)
        assert e.max() <= MAX_ABS and e.mean() <= MEAN_ABS
    finally:
        cache.close()


def test_shared_prefix_requires_empty_layer():
    with dms.DmsCache(layers=1, kv_heads=2, window=8, capacity=256, batch=2) as cache:
        k, v, lg = _kvl(1, 10, 2, 0.5, 1)
        cache.append_shared_prefix(0, k, v, lg)
        code = dms.dms_append_shared_prefix(cache.handle, 0, k.data_ptr(), v.data_ptr(),
                                            lg.data_ptr(), 10, None)
        assert code == dms.DMS_ERR_STATE
