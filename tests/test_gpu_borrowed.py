"""GPU parity of decisions taken from a borrowed query neuron (App. B), through the C ABI.

The decision logit of (sequence b, KV head h) at each token is element 0 of query head
h * G; the attention takes that element as 0.  Retained sets bit-exact and outputs within
max-abs 2e-2 / mean-abs 2e-3 against the fp64 oracle fed with ``oracle.borrowed``; the
borrowed entry points equal the plain ones fed with the extracted logits and the zeroed
queries bit for bit.
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


def _inputs(B, H, G, n, p, seed):
    """k, v [B, n, H, D] and q [B, n, H * G, D] bf16; element 0 of each group's first query
    head carries a decision logit with P(> 0) = p."""
    g = torch.Generator(device="cuda").manual_seed(seed)
    k = torch.randn((B, n, H, D), generator=g, device="cuda").to(torch.bfloat16)
    v = torch.randn((B, n, H, D), generator=g, device="cuda").to(torch.bfloat16)
    q = torch.randn((B, n, H * G, D), generator=g, device="cuda")
    mu = statistics.NormalDist().inv_cdf(p)
    q[:, :, ::G, 0] = torch.randn((B, n, H), generator=g, device="cuda") + mu
    return k, v, q.to(torch.bfloat16)


def _explicit(q, G):
    """The logits and the zeroed queries the plain entry points need for the same step."""
    lg = q[..., ::G, 0].contiguous()
    qz = q.clone()
    qz[..., ::G, 0] = 0
    return lg, qz


class History:
    def __init__(self):
        self.k, self.v, self.q = [], [], []

    def add(self, k, v, q):
        self.k.append(k)
        self.v.append(v)
        self.q.append(q)

    def bits(self, G):
        K = workloads.bf16_bits(torch.cat(self.k, 1))
        V = workloads.bf16_bits(torch.cat(self.v, 1))
        L, _ = oracle.borrowed(workloads.bf16_bits(torch.cat(self.q, 1)), G)  # [B, T, H]
        return K, V, L


def _check(cache, hist, q_step, out, G, w, errs, retained=True):
    K, V, L = hist.bits(G)
    B, T, H = L.shape
    j = T - 1
    if retained:
        pos = cache.export_positions(0)
        counts = cache.stats(with_counts=True)["counts"][0]
        for b in range(B):
            for h in range(H):
                n = int(counts[b, h])
                assert np.array_equal(np.sort(pos[b, h, :n]), oracle.retained(L[b, :, h], j, w)), (b, h)
    _, q_att = oracle.borrowed(workloads.bf16_bits(q_step), G)  # [B, H * G, D]
    got = out.float().cpu().numpy()
    for b in range(B):
        for h in range(H):
            ref = oracle.decode(q_att[b, h * G:(h + 1) * G], K[b, :, h], V[b, :, h], L[b, :, h], j, w)
            e = np.abs(got[b, h * G:(h + 1) * G] - ref).ravel()
            assert e.max() <= MAX_ABS, (b, h, e.max())
            errs.append(e)


@pytest.mark.parametrize("B,H,G,w,P,steps,p,kernel", [
    (2, 3, 4, 40, 257, 40, 0.7, dms.DMS_DECODE_TILED),
    (1, 2, 16, 16, 130, 24, 0.8, dms.DMS_DECODE_TILED),   # two n-tiles (G > 8)
    (3, 4, 1, 8, 70, 24, 0.6, dms.DMS_DECODE_TILED),      # MHA: every head lends its element 0
    (2, 3, 4, 40, 257, 16, 0.7, dms.DMS_DECODE_SIMPLE),   # cross-check kernel (two launches)
])
def test_borrowed_matches_oracle(B, H, G, w, P, steps, p, kernel):
    k, v, q = _inputs(B, H, G, P, p, 1)
    with dms.DmsCache(layers=1, kv_heads=H, window=w, capacity=P + steps, batch=B,
                      decode_kernel=kernel) as cache:
        cache.append_and_evict_borrowed(0, k, v, q, G)
        hist = History()
        hist.add(k, v, q)
        errs = []
        for s in range(steps):
            k1, v1, q1 = _inputs(B, H, G, 1, p, 100 + s)
            out = cache.append_and_decode_borrowed(0, k1, v1, q1[:, 0], gqa_group=G)
            hist.add(k1, v1, q1)
            _check(cache, hist, q1[:, 0], out, G, w, errs, retained=(s % 4 == 0 or s == steps - 1))
        assert cache.stats()["device_error"] == 0
        assert np.concatenate(errs).mean() <= MEAN_ABS


def _run(B, H, G, w, P, steps, mode):
    """Outputs of every step and the final retained positions for one calling mode."""
    k, v, q = _inputs(B, H, G, P, 0.75, 7)
    outs = []
    with dms.DmsCache(layers=1, kv_heads=H, window=w, capacity=P + steps, batch=B) as cache:
        if mode == "explicit":
            lg, _ = _explicit(q, G)
            cache.append_and_evict(0, k, v, lg)
        else:
            cache.append_and_evict_borrowed(0, k, v, q, G)
        for s in range(steps):
            k1, v1, q1 = _inputs(B, H, G, 1, 0.75, 200 + s)
            qs = q1[:, 0].contiguous()
            if mode == "explicit":
                lg1, qz = _explicit(q1, G)
                out = cache.append_and_decode(0, k1, v1, lg1, qz[:, 0].contiguous(), gqa_group=G)
            elif mode == "fused":
                out = cache.append_and_decode_borrowed(0, k1, v1, qs, gqa_group=G)
            else:  # separate calls
                cache.append_and_evict_borrowed(0, k1, v1, q1, G)
                out = cache.decode_attention_borrowed(0, qs, gqa_group=G)
            assert torch.equal(qs, q1[:, 0]), "the caller's q must not be modified"
            outs.append(out.clone())
        pos = cache.export_positions(0)
        assert cache.stats()["device_error"] == 0
    return outs, pos


@pytest.mark.parametrize("G", [4, 7, 16])
def test_borrowed_equals_explicit_and_separate(G):
    B, H, w, P, steps = 4, 2, 24, 333, 20
    ref_out, ref_pos = _run(B, H, G, w, P, steps, "explicit")
    for mode in ("fused", "separate"):
        outs, pos = _run(B, H, G, w, P, steps, mode)
        assert np.array_equal(pos, ref_pos), mode
        for s, (a, b) in enumerate(zip(outs, ref_out)):
            assert torch.equal(a, b), (mode, s)


def test_borrowed_rejects_bad_arguments():
    with dms.DmsCache(layers=1, kv_heads=2, window=8, capacity=64, batch=1) as cache:
        k, v, q = _inputs(1, 2, 4, 1, 0.5, 3)
        assert dms.dms_append_and_evict_borrowed(cache.handle, 0, k.data_ptr(), v.data_ptr(),
                                                 q.data_ptr(), 1, 17,
                                                 None) == dms.DMS_ERR_INVALID_ARGUMENT
        assert dms.dms_append_and_decode_borrowed(cache.handle, 0, k.data_ptr(), v.data_ptr(),
                                                  q.data_ptr() + 2, q.data_ptr(), 4, 0.0,
                                                  None) == dms.DMS_ERR_INVALID_ARGUMENT
