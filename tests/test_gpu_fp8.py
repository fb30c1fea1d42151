"""fp8 E4M3 page format (DMS_KV_FP8_E4M3): the CUDA path through the C ABI against the fp64
oracle.  Stored codes and scales bit-exact against the oracle's quantisation of the input rows
(the E4M3 rounding decides integer codes, so both sides take it in fp32); retained sets
bit-exact and equal to a bf16 cache's; attention outputs within max-abs 2e-2 / mean-abs 2e-3 of
the oracle's attention over the dequantised rows.
"""
import statistics

import numpy as np
import pytest
import torch

import oracle
import paper_2506_05345_gb300 as dms
import workloads
from _harness import MAX_ABS, MEAN_ABS, Run

pytestmark = pytest.mark.gpu
FP8 = dms.DMS_KV_FP8_E4M3
D = 128


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dms.library()


def small(**kw):
    base = dict(name="f8", batch=2, layers=1, q_heads=8, kv_heads=2, window=32,
                prefill=((300, False),), decode_steps=6, p_evict=0.75)
    base.update(kw)
    return workloads.Workload(**base)


def _run(wl, fused=False, codes_every=3, **kw):
    r = Run(wl, kv_format=FP8, fused=fused, **kw)
    try:
        r.prefill()
        r.check_retained()
        r.check_codes()
        for s in range(wl.decode_steps):
            q, out = r.step(s)
            r.check_outputs(q, out)
            if s % codes_every == 0 or s == wl.decode_steps - 1:
                r.check_retained()
                r.check_codes()
        return r.summary()
    finally:
        r.close()


# fp8 pages are read both by the flat split (the default for these few-head shapes) and by
# the per-head clusters (DMS_DECODE_CLUSTER; G <= 8)
KERNELS = pytest.mark.parametrize("kernel", [dms.DMS_DECODE_TILED, dms.DMS_DECODE_CLUSTER],
                                  ids=["split", "cluster"])


@KERNELS
@pytest.mark.parametrize("w", [0, 1, 16, 63, 64, 256])
def test_fp8_windows(w, kernel):
    _run(small(window=w, prefill=((333, False),)), decode_kernel=kernel)


@KERNELS
@pytest.mark.parametrize("G", [1, 4, 7, 8, 9, 16])
def test_fp8_gqa_groups(G, kernel):
    _run(small(q_heads=2 * G, decode_steps=4), decode_kernel=kernel)


@KERNELS
@pytest.mark.parametrize("prefill", [1, 15, 16, 17, 63, 64, 65, 129, 1000])
def test_fp8_page_boundaries(prefill, kernel):
    _run(small(prefill=((prefill, False),), window=20, p_evict=0.5, decode_steps=5),
         decode_kernel=kernel)


@pytest.mark.parametrize("p", [0.0, 1.0])
def test_fp8_no_and_total_eviction(p):
    _run(small(p_evict=p, prefill=((200, False),), window=8))


@KERNELS
def test_fp8_fused_entry_point(kernel):
    """dms_append_and_decode on an fp8 cache: the single-token append (quantising the new
    rows) fused into the decode launch."""
    _run(small(), fused=True, decode_kernel=kernel)


@pytest.mark.parametrize("batch,kv_heads,fused", [(1, 1, True), (1, 2, False), (8, 8, True)])
def test_fp8_cluster_stored_codes(batch, kv_heads, fused):
    """fp8 pages on per-head clusters (down to 2 CTAs per head for 64 heads) with more pages
    per CTA than stages and a 2000-token window at P(evict) 0.9, so that new tokens take slots
    in pages staged early: stored codes and scales bit-exact after the steps, outputs and
    retained sets against the oracle."""
    wl = small(batch=batch, kv_heads=kv_heads, q_heads=kv_heads * 5, window=2000,
               prefill=((4000 if batch > 1 else 8000, False),), decode_steps=30, p_evict=0.9)
    r = Run(wl, kv_format=FP8, fused=fused, decode_kernel=dms.DMS_DECODE_CLUSTER)
    try:
        assert r.cache.decode_plan(wl.gqa_group)["kernel"] == dms.DMS_DECODE_CLUSTER
        r.prefill()
        for s in range(wl.decode_steps):
            q, out = r.step(s)
            if s % 10 == 9:
                r.check_outputs(q, out)
                r.check_retained()
        r.check_codes()
        r.summary()
    finally:
        r.close()


def test_fp8_llama_shape_long():
    """Batch 1, 32 q / 8 kv heads, prefill 4096 + 32 steps, w = 256, P(evict) 0.875."""
    wl = workloads.Workload(**{**workloads.LLAMA_B1_4K.__dict__, "decode_steps": 32})
    mx, mean = _run(wl, codes_every=16)
    assert mx <= MAX_ABS and mean <= MEAN_ABS


def test_fp8_positions_equal_bf16_cache():
    """The page format changes nothing about which tokens are kept or where."""
    wl = small(prefill=((500, False),), decode_steps=5)
    runs = [Run(wl, kv_format=f) for f in (dms.DMS_KV_BF16, FP8)]
    try:
        for r in runs:
            r.prefill()
            for s in range(wl.decode_steps):
                r.step(s)
        assert np.array_equal(runs[0].cache.export_positions(0), runs[1].cache.export_positions(0))
        st = [r.cache.stats() for r in runs]
        assert st[0]["total_retained"] == st[1]["total_retained"]
    finally:
        for r in runs:
            r.close()


def _kvl(B, n, H, p, seed, zero_every=0):
    g = torch.Generator(device="cuda").manual_seed(seed)
    k = (torch.randn((B, n, H, D), generator=g, device="cuda") *
         torch.exp(torch.randn((B, n, H, 1), generator=g, device="cuda"))).to(torch.bfloat16)
    v = torch.randn((B, n, H, D), generator=g, device="cuda").to(torch.bfloat16)
    if zero_every:
        k[:, ::zero_every] = 0
        v[:, 1::zero_every] = 0
    lg = (torch.randn((B, n, H), generator=g, device="cuda")
          + statistics.NormalDist().inv_cdf(p)).to(torch.bfloat16)
    return k, v, lg


def _oracle_check(cache, K, V, L, q, out, G, w, immediate=False, q_att=None):
    B, T, H, _ = K.shape
    j = T - 1
    Kb, Vb, Lb = workloads.bf16_bits(K), workloads.bf16_bits(V), workloads.bf16_bits(L)
    Q = q_att if q_att is not None else workloads.bf16_bits(q)
    got = out.float().cpu().numpy()
    errs = []
    for b in range(B):
        for h in range(H):
            kc, ks = oracle.quantize_rows_e4m3(Kb[b, :, h])
            vc, vs = oracle.quantize_rows_e4m3(Vb[b, :, h])
            ref = oracle.decode_fp8(Q[b, h * G:(h + 1) * G], kc, ks, vc, vs, Lb[b, :, h], j, w,
                                    immediate=immediate)
            errs.append(np.abs(got[b, h * G:(h + 1) * G] - ref).ravel())
    e = np.concatenate(errs)
    assert np.all(np.isfinite(got))
    assert e.max() <= MAX_ABS and e.mean() <= MEAN_ABS, (e.max(), e.mean())


def test_fp8_zero_rows_and_wide_row_scales():
    """Rows of zeros (scale 0, codes 0) and key rows whose scales span e^+-3."""
    B, H, G, w, n = 2, 2, 4, 16, 400
    with dms.DmsCache(layers=1, kv_heads=H, window=w, capacity=n + 3, batch=B,
                      kv_format=FP8) as cache:
        k, v, lg = _kvl(B, n, H, 0.6, 3, zero_every=5)
        cache.append_and_evict(0, k, v, lg)
        hist = [(k, v, lg)]
        for s in range(3):
            ks, vs, ls = _kvl(B, 1, H, 0.6, 10 + s)
            q = torch.randn((B, H * G, D), device="cuda").to(torch.bfloat16)
            out = cache.append_and_decode(0, ks, vs, ls, q, gqa_group=G)
            hist.append((ks, vs, ls))
            K, V, L = (torch.cat([x[i] for x in hist], 1) for i in range(3))
            _oracle_check(cache, K, V, L, q, out, G, w)
        k8, v8, sc = cache.export_kv(0)
        pos = cache.export_positions(0)
        Kb = workloads.bf16_bits(K)
        for b in range(B):
            for h in range(H):
                for s_, p_ in enumerate(pos[b, h]):
                    if p_ < 0 or p_ >= n or p_ % 5:
                        continue
                    assert sc[b, h, s_, 0] == 0 and not k8[b, h, s_].any()
                    assert not Kb[b, p_, h].any()


def test_fp8_immediate_eviction():
    B, H, G, w, n, steps = 2, 2, 4, 24, 300, 4
    with dms.DmsCache(layers=1, kv_heads=H, window=w, capacity=n + steps, batch=B,
                      kv_format=FP8, eviction_policy=dms.DMS_EVICT_IMMEDIATE) as cache:
        k, v, lg = _kvl(B, n, H, 0.7, 4)
        cache.append_and_evict(0, k, v, lg)
        hist = [(k, v, lg)]
        for s in range(steps):
            ks, vs, ls = _kvl(B, 1, H, 0.7, 20 + s)
            cache.append_and_evict(0, ks, vs, ls)
            hist.append((ks, vs, ls))
            q = torch.randn((B, H * G, D), device="cuda").to(torch.bfloat16)
            out = cache.decode_attention(0, q, gqa_group=G)
            K, V, L = (torch.cat([x[i] for x in hist], 1) for i in range(3))
            _oracle_check(cache, K, V, L, q, out, G, w, immediate=True)


def test_fp8_borrowed_decisions():
    """App. B decisions from each group's first query head, on an fp8 cache."""
    B, H, G, w, n, steps = 2, 2, 4, 16, 200, 3
    with dms.DmsCache(layers=1, kv_heads=H, window=w, capacity=n + steps, batch=B,
                      kv_format=FP8) as cache:
        qs, ks_, vs_ = [], [], []
        g = torch.Generator(device="cuda").manual_seed(6)
        qp = torch.randn((B, n, H * G, D), generator=g, device="cuda").to(torch.bfloat16)
        kp = torch.randn((B, n, H, D), generator=g, device="cuda").to(torch.bfloat16)
        vp = torch.randn((B, n, H, D), generator=g, device="cuda").to(torch.bfloat16)
        cache.append_and_evict_borrowed(0, kp, vp, qp, gqa_group=G)
        qs.append(qp), ks_.append(kp), vs_.append(vp)
        for s in range(steps):
            q = torch.randn((B, 1, H * G, D), generator=g, device="cuda").to(torch.bfloat16)
            k = torch.randn((B, 1, H, D), generator=g, device="cuda").to(torch.bfloat16)
            v = torch.randn((B, 1, H, D), generator=g, device="cuda").to(torch.bfloat16)
            out = cache.append_and_decode_borrowed(0, k, v, q[:, 0], gqa_group=G)
            qs.append(q), ks_.append(k), vs_.append(v)
            Q = workloads.bf16_bits(torch.cat(qs, 1))
            L, _ = oracle.borrowed(Q, G)
            _, q_att = oracle.borrowed(workloads.bf16_bits(q[:, 0]), G)
            Lt = torch.from_numpy(L.view(np.int16)).view(torch.bfloat16)
            _oracle_check(cache, torch.cat(ks_, 1), torch.cat(vs_, 1), Lt, None, out, G, w,
                          q_att=q_att)


def test_fp8_shared_prefix():
    """A shared prompt on an fp8 cache: frozen pages (and their scales) mapped into every
    sequence; outputs equal to the replicated prompt bit for bit, and to the oracle."""
    B, H, G, w, n, steps = 3, 2, 4, 16, 300, 3
    outs = []
    for shared in (True, False):
        with dms.DmsCache(layers=1, kv_heads=H, window=w, capacity=n + steps, batch=B,
                          kv_format=FP8) as cache:
            kp, vp, lp = _kvl(1, n, H, 0.7, 8)
            if shared:
                cache.append_shared_prefix(0, kp, vp, lp)
            else:
                cache.append_and_evict(0, kp.expand(B, -1, -1, -1).contiguous(),
                                       vp.expand(B, -1, -1, -1).contiguous(),
                                       lp.expand(B, -1, -1).contiguous())
            hist = [(kp.expand(B, -1, -1, -1), vp.expand(B, -1, -1, -1), lp.expand(B, -1, -1))]
            run = []
            for s in range(steps):
                k, v, lg = _kvl(B, 1, H, 0.7, 30 + s)
                g = torch.Generator(device="cuda").manual_seed(40 + s)
                q = torch.randn((B, H * G, D), generator=g, device="cuda").to(torch.bfloat16)
                out = cache.append_and_decode(0, k, v, lg, q, gqa_group=G)
                hist.append((k, v, lg))
                run.append(out.clone())
                if shared:
                    K, V, L = (torch.cat([x[i] for x in hist], 1) for i in range(3))
                    _oracle_check(cache, K, V, L, q, out, G, w)
            outs.append(run)
    for a, b in zip(*outs):
        assert torch.equal(a, b)
