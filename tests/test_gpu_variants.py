"""GPU parity of the variants: window sizes 16 and 512 (Sec. 5 ablations use a 16-token
window; 512 is a larger one), and the immediate-eviction ablation (Sec. 5: token i is evicted
by the decision of token i + w instead of its own), through the C ABI against the fp64 oracle.
Retained sets bit-exact; outputs within max-abs 2e-2 / mean-abs 2e-3.
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
IMM = dms.DMS_EVICT_IMMEDIATE


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dms.library()


def _kvl(B, n, H, p, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    k = torch.randn((B, n, H, D), generator=g, device="cuda").to(torch.bfloat16)
    v = torch.randn((B, n, H, D), generator=g, device="cuda").to(torch.bfloat16)
    mu = statistics.NormalDist().inv_cdf(p)
    lg = (torch.randn((B, n, H), generator=g, device="cuda") + mu).to(torch.bfloat16)
    return k, v, lg


def _q(B, H, G, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    return torch.randn((B, H * G, D), generator=g, device="cuda").to(torch.bfloat16)


def _run(B, H, G, w, chunks, steps, p, policy=0, mode="fused", check=True, seed=0, **kw):
    """Bulk appends of the given chunk sizes, then decode steps; checks retained sets and
    outputs against the oracle under the policy.  Returns (outputs, final positions)."""
    imm = policy == IMM
    T = sum(chunks) + steps
    Ks, Vs, Ls, outs, errs = [], [], [], [], []
    with dms.DmsCache(layers=1, kv_heads=H, window=w, capacity=T, batch=B,
                      eviction_policy=policy, **kw) as cache:
        for i, n in enumerate(chunks):
            k, v, lg = _kvl(B, n, H, p, seed * 1000 + i)
            cache.append_and_evict(0, k, v, lg)
            Ks.append(k), Vs.append(v), Ls.append(lg)
        for s in range(steps):
            k, v, lg = _kvl(B, 1, H, p, seed * 1000 + 500 + s)
            q = _q(B, H, G, seed * 1000 + 900 + s)
            Ks.append(k), Vs.append(v), Ls.append(lg)
            if mode == "fused":
                out = cache.append_and_decode(0, k, v, lg, q, gqa_group=G)
            else:
                cache.append_and_evict(0, k, v, lg)
                out = cache.decode_attention(0, q, gqa_group=G)
            outs.append(out.clone())
            if not check:
                continue
            K = workloads.bf16_bits(torch.cat(Ks, 1))
            V = workloads.bf16_bits(torch.cat(Vs, 1))
            L = workloads.bf16_bits(torch.cat(Ls, 1))
            j = K.shape[1] - 1
            Q = workloads.bf16_bits(q)
            got = out.float().cpu().numpy()
            if s % 4 == 0 or s == steps - 1:
                pos = cache.export_positions(0)
                cnt = cache.stats(with_counts=True)["counts"][0]
                for b in range(B):
                    for h in range(H):
                        n = int(cnt[b, h])
                        want = oracle.retained(L[b, :, h], j, w, immediate=imm)
                        assert np.array_equal(np.sort(pos[b, h, :n]), want), (s, b, h)
            for b in range(B):
                for h in range(H):
                    ref = oracle.decode(Q[b, h * G:(h + 1) * G], K[b, :, h], V[b, :, h], L[b, :, h],
                                        j, w, immediate=imm)
                    e = np.abs(got[b, h * G:(h + 1) * G] - ref).ravel()
                    assert e.max() <= MAX_ABS, (s, b, h, e.max())
                    errs.append(e)
        assert cache.stats()["device_error"] == 0
        pos = cache.export_positions(0)
    if errs:
        assert np.concatenate(errs).mean() <= MEAN_ABS
    return outs, pos


@pytest.mark.parametrize("w", [16, 512])
@pytest.mark.parametrize("mode", ["fused", "separate"])
def test_window_sizes_delayed(w, mode):
    _run(B=2, H=2, G=4, w=w, chunks=(700, 1, 130), steps=24, p=0.8, mode=mode)


@pytest.mark.parametrize("w", [0, 1, 16, 64])
@pytest.mark.parametrize("mode", ["fused", "separate"])
def test_immediate_eviction(w, mode):
    _run(B=2, H=3, G=4, w=w, chunks=(300, 1, 77, 200), steps=20, p=0.7, policy=IMM, mode=mode)


def test_immediate_eviction_simple_kernel():
    _run(B=1, H=2, G=5, w=16, chunks=(250,), steps=12, p=0.7, policy=IMM,
         decode_kernel=dms.DMS_DECODE_SIMPLE)


def test_immediate_w0_equals_delayed():
    a, pa = _run(B=2, H=2, G=4, w=0, chunks=(200, 33), steps=10, p=0.6, policy=IMM, check=False)
    b, pb = _run(B=2, H=2, G=4, w=0, chunks=(200, 33), steps=10, p=0.6, policy=0, check=False)
    assert np.array_equal(pa, pb)
    assert all(torch.equal(x, y) for x, y in zip(a, b))


@pytest.mark.parametrize("policy", [0, IMM])
def test_bulk_equals_token_by_token(policy):
    """One bulk append leaves the same retained sets as the same tokens appended one by one."""
    B, H, w, n = 2, 2, 16, 180
    k, v, lg = _kvl(B, n, H, 0.7, 42)
    sets = []
    for bulk in (True, False):
        with dms.DmsCache(layers=1, kv_heads=H, window=w, capacity=n, batch=B,
                          eviction_policy=policy) as cache:
            if bulk:
                cache.append_and_evict(0, k, v, lg)
            else:
                for t in range(n):
                    cache.append_and_evict(0, k[:, t:t + 1].contiguous(), v[:, t:t + 1].contiguous(),
                                           lg[:, t:t + 1].contiguous())
            pos = cache.export_positions(0)
            sets.append([[sorted(x for x in pos[b, h] if x >= 0) for h in range(H)] for b in range(B)])
    assert sets[0] == sets[1]


@pytest.mark.parametrize("kernel", [dms.DMS_PREFILL_TCGEN05, dms.DMS_PREFILL_MMA_SYNC])
@pytest.mark.parametrize("w,policy", [(16, 0), (512, 0), (16, IMM), (64, IMM)])
def test_prefill_variants(w, policy, kernel):
    B, P, H, G = 2, 700, 2, 4
    g = torch.Generator(device="cuda").manual_seed(w + policy)
    q = torch.randn((B, P, H * G, D), generator=g, device="cuda").to(torch.bfloat16)
    k, v, lg = _kvl(B, P, H, 0.7, 7 + w)
    out = dms.prefill_attention(q, k, v, lg, window=w, eviction_policy=policy, kernel=kernel)
    Q, K, V, L = (workloads.bf16_bits(t) for t in (q, k, v, lg))
    got = out.float().cpu().numpy()
    errs = []
    for b in range(B):
        for j in range(0, P, 3):
            for h in range(H):
                ref = oracle.decode(Q[b, j, h * G:(h + 1) * G], K[b, :, h], V[b, :, h], L[b, :, h],
                                    j, w, immediate=policy == IMM)
                errs.append(np.abs(got[b, j, h * G:(h + 1) * G] - ref).ravel())
    e = np.concatenate(errs)
    assert e.max() <= MAX_ABS and e.mean() <= MEAN_ABS, (e.max(), e.mean())
