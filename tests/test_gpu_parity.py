"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle.

Retained sets bit-exact; outputs within max-abs 2e-2 / mean-abs 2e-3.
"""
import dataclasses

import numpy as np
import pytest
import torch

import paper_2506_05345_gb300 as dms
import workloads
from _harness import MAX_ABS, MEAN_ABS, Run

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dms.library()


def small(**kw):
    base = dict(name="t", batch=2, layers=1, q_heads=8, kv_heads=2, window=32,
                prefill=((300, False),), decode_steps=8, p_evict=0.75)
    base.update(kw)
    return workloads.Workload(**base)


def _run_all_steps(wl, check_every=1, retained_every=4, **cache_kw):
    r = Run(wl, **cache_kw)
    try:
        r.prefill()
        r.check_retained()
        for s in range(wl.decode_steps):
            q, out = r.step(s)
            if s % check_every == 0 or s == wl.decode_steps - 1:
                r.check_outputs(q, out)
            if s % retained_every == 0 or s == wl.decode_steps - 1:
                r.check_retained()
        return r.summary()
    finally:
        r.close()


# ---------------------------------------------------------------- the small config, in full


@pytest.mark.parametrize("kernel,fused", [(dms.DMS_DECODE_TILED, False), (dms.DMS_DECODE_TILED, True),
                                          (dms.DMS_DECODE_SPLIT, False), (dms.DMS_DECODE_SPLIT, True),
                                          (dms.DMS_DECODE_SIMPLE, False)])
def test_llama_b1_ctx4352_every_step(kernel, fused):
    """Batch 1, 32 q / 8 kv heads, prefill 4096 + 256 decode steps, w = 256, P(evict) 0.875:
    every step, every query head; retained sets every 16 steps.  The default kernel runs the
    8 heads as per-head clusters; DMS_DECODE_SPLIT as the flat split over all SMs."""
    wl = workloads.LLAMA_B1_4K
    mx, mean = _run_all_steps(wl, check_every=1, retained_every=16, decode_kernel=kernel,
                              fused=fused)
    assert mx <= MAX_ABS and mean <= MEAN_ABS


# ---------------------------------------------------------------- edge cases


# The small shapes below run both as per-head clusters (DMS_DECODE_CLUSTER; the default
# kernel takes these only for enough heads) and as the flat split over all SMs.
TILED_KERNELS = pytest.mark.parametrize("kernel", [dms.DMS_DECODE_CLUSTER, dms.DMS_DECODE_SPLIT],
                                        ids=["cluster", "split"])


@TILED_KERNELS
@pytest.mark.parametrize("fused", [False, True])
@pytest.mark.parametrize("w", [0, 1, 15, 63, 64, 255, 256])
def test_windows(w, fused, kernel):
    _run_all_steps(small(window=w, prefill=((333, False),), decode_steps=6), fused=fused,
                   decode_kernel=kernel)


@TILED_KERNELS
@pytest.mark.parametrize("fused", [False, True])
@pytest.mark.parametrize("G", [1, 3, 4, 5, 7, 8, 9, 16])
def test_gqa_groups(G, fused, kernel):
    _run_all_steps(small(q_heads=2 * G, kv_heads=2, decode_steps=4), fused=fused,
                   decode_kernel=kernel)


@TILED_KERNELS
@pytest.mark.parametrize("fused", [False, True])
@pytest.mark.parametrize("prefill", [1, 2, 63, 64, 65, 127, 128, 129, 1000])
def test_page_boundaries(prefill, fused, kernel):
    _run_all_steps(small(prefill=((prefill, False),), decode_steps=5, window=20, p_evict=0.5),
                   fused=fused, decode_kernel=kernel)


@TILED_KERNELS
@pytest.mark.parametrize("w", [0, 3, 40])
def test_fused_decode_from_empty_cache(w, kernel):
    """The fused step appends and attends from the very first token (pages opened in-kernel)."""
    wl = small(window=w, prefill=(), decode_steps=150, p_evict=0.6)
    _run_all_steps(wl, check_every=7, retained_every=10, fused=True, decode_kernel=kernel)


@pytest.mark.parametrize("fused", [False, True])
@pytest.mark.parametrize("batch,kv_heads,G,prefill", [
    (1, 1, 5, 5000), (1, 8, 5, 20000), (2, 8, 5, 3000), (1, 16, 5, 700), (3, 6, 5, 1500),
    (5, 8, 5, 1200), (8, 8, 8, 900), (8, 8, 3, 9000), (16, 8, 5, 700), (12, 8, 8, 2500)])
def test_cluster_shapes(batch, kv_heads, G, prefill, fused):
    """Head counts over the cluster sizes' range (1 to 128 heads: clusters of 16 CTAs down to 1),
    with heads of many pages (5000 and 20000 tokens at P(evict) 0.2: up to 250 pages over a
    cluster) and of few (a head of 700 tokens leaves most of its cluster's CTAs without
    pages), and clusters smaller than the group (40 heads of G = 5 and 64 heads of G = 8,
    whose query-head rows are shared out over the cluster's CTAs)."""
    wl = small(batch=batch, kv_heads=kv_heads, q_heads=kv_heads * G, window=100,
               prefill=((prefill, False),), decode_steps=3, p_evict=0.2)
    r = Run(wl, decode_kernel=dms.DMS_DECODE_CLUSTER)
    plan = r.cache.decode_plan(G)
    r.close()
    assert plan["kernel"] == dms.DMS_DECODE_CLUSTER, plan
    _run_all_steps(wl, fused=fused, decode_kernel=dms.DMS_DECODE_CLUSTER)


def test_fused_matches_separate_bitwise():
    """dms_append_and_decode gives the same retained sets and the same bits as the two calls."""
    wl = small(batch=3, kv_heads=4, q_heads=28, window=30, prefill=((700, False),), decode_steps=40,
               p_evict=0.7)
    a, b = Run(wl, fused=False), Run(wl, fused=True)
    try:
        a.prefill()
        b.prefill()
        for s_ in range(wl.decode_steps):
            _, oa = a.step(s_)
            _, ob = b.step(s_)
            assert torch.equal(oa, ob), s_
        pa, pb = a.cache.export_positions(0), b.cache.export_positions(0)
        for bb in range(wl.batch):
            for h in range(wl.kv_heads):
                assert np.array_equal(np.sort(pa[bb, h][pa[bb, h] >= 0]), np.sort(pb[bb, h][pb[bb, h] >= 0]))
        a.check_retained()
        b.check_retained()
    finally:
        a.close()
        b.close()


@pytest.mark.parametrize("p", [0.0, 1.0])
def test_no_and_total_eviction(p):
    """p = 0: dense (CR 1).  p = 1: every token is flagged, only the window survives."""
    wl = small(p_evict=p, prefill=((400, False),), window=40, decode_steps=5)
    r = Run(wl)
    try:
        r.prefill()
        st = r.check_retained()
        expect = 400 if p == 0.0 else 41
        assert np.all(st["counts"] == expect)
        for s in range(wl.decode_steps):
            q, out = r.step(s)
            r.check_outputs(q, out)
        r.check_retained()
        r.summary()
    finally:
        r.close()


def test_w0_all_evict_single_token():
    """w = 0 and every decision 1: one token remains and the output is v_j (bf16)."""
    wl = small(window=0, p_evict=1.0, prefill=((70, False),), decode_steps=3)
    r = Run(wl)
    try:
        r.prefill()
        for s in range(3):
            q, out = r.step(s)
            st = r.check_retained()
            assert np.all(st["counts"] == 1)
            G = wl.gqa_group
            want = r.V[:, r.t - 1].repeat_interleave(G, dim=1)
            assert torch.equal(out, want)
    finally:
        r.close()


@pytest.mark.parametrize("fused", [False, True])
def test_ragged_heads_mixed_probabilities(fused):
    """Heads with P(evict) from 0 to 1 in one layer: very different n_h per head."""
    wl = small(batch=3, kv_heads=4, q_heads=20, window=24, prefill=((900, False),), decode_steps=6)
    r = Run(wl, fused=fused)
    try:
        B, H = wl.batch, wl.kv_heads
        p = [0.0, 0.5, 0.95, 1.0]
        k, v, lg = workloads.gen_kv(wl, 0, "prefill0", 900, r.dev, p_override=p)
        r.append(k, v, lg)
        r.check_retained()
        for s in range(wl.decode_steps):
            q, out = r.step(s, p_override=p)
            r.check_outputs(q, out)
        st = r.check_retained()
        assert st["counts"].max() > 5 * st["counts"].min()
        r.summary()
    finally:
        r.close()


def test_special_logits():
    """NaN, +-0, -inf keep; +inf and tiny positives evict (Sec. 3.2 sign rule)."""
    wl = small(window=4, prefill=((64, False),), decode_steps=0)
    r = Run(wl)
    try:
        vals = torch.tensor([float("nan"), 0.0, -0.0, float("-inf"), float("inf"), 1e-38,
                             -1e-38, 3.0], dtype=torch.float32)
        B, H = wl.batch, wl.kv_heads
        lg = vals.repeat(8)[None, :, None].expand(B, 64, H).contiguous().to(torch.bfloat16).to(r.dev)
        k, v, _ = workloads.gen_kv(wl, 0, "p", 64, r.dev)
        r.append(k, v, lg)
        st = r.check_retained()
        # kept outside the window: NaN, +0, -0, -inf, -1e-38 (5 of every 8)
        assert int(st["counts"][0, 0, 0]) == len(np.arange(0, 59)[np.isin(np.arange(59) % 8,
                                                                           [0, 1, 2, 3, 6])]) + 5
    finally:
        r.close()


def test_bulk_then_decode_equals_sequential():
    """Bulk prefill of P tokens gives the same retained sets as P single-token appends."""
    wl = small(batch=2, kv_heads=2, window=16, prefill=((150, False),), decode_steps=0)
    a, b = Run(wl), Run(wl)
    try:
        k, v, lg = workloads.gen_kv(wl, 0, "prefill0", 150, a.dev)
        a.append(k, v, lg)
        for t in range(150):
            b.append(k[:, t:t + 1].contiguous(), v[:, t:t + 1].contiguous(), lg[:, t:t + 1].contiguous())
        a.check_retained()
        b.check_retained()
        pa, pb = a.cache.export_positions(0), b.cache.export_positions(0)
        for bb in range(2):
            for h in range(2):
                assert np.array_equal(np.sort(pa[bb, h][pa[bb, h] >= 0]), np.sort(pb[bb, h][pb[bb, h] >= 0]))
        # mixed: bulk chunks of uneven size then singles, still the oracle's sets
        c = Run(wl)
        try:
            for lo, hi in ((0, 7), (7, 100), (100, 101), (101, 150)):
                c.append(k[:, lo:hi].contiguous(), v[:, lo:hi].contiguous(), lg[:, lo:hi].contiguous())
            c.check_retained()
        finally:
            c.close()
    finally:
        a.close()
        b.close()


@pytest.mark.parametrize("fused", [False, True])
@pytest.mark.parametrize("min_pages,ctas", [(1, 4), (1, 1), (1000000, 1), (3, 2)])
def test_split_shapes(min_pages, ctas, fused):
    """Heads split over many CTAs (multi-piece combine) and one CTA walking all heads."""
    wl = small(batch=2, kv_heads=3, q_heads=15, window=40, prefill=((2500, False),), decode_steps=3,
               p_evict=0.3)
    _run_all_steps(wl, min_pages_per_cta=min_pages, ctas_per_sm=ctas, fused=fused)


def test_empty_cache_gives_zeros():
    wl = small()
    r = Run(wl)
    try:
        q = workloads.gen_q(wl, 0, "q", r.dev)
        out = r.cache.decode_attention(0, q, gqa_group=wl.gqa_group)
        torch.cuda.synchronize()
        assert torch.count_nonzero(out) == 0
    finally:
        r.close()


@pytest.mark.parametrize("kw", [{"decode_kernel": dms.DMS_DECODE_CLUSTER}, {"min_pages_per_cta": 1}],
                         ids=["cluster", "split1"])
def test_deterministic_outputs(kw):
    wl = small(prefill=((3000, False),), decode_steps=1, window=64)
    r = Run(wl, **kw)
    try:
        r.prefill()
        q, out = r.step(0)
        again = [r.cache.decode_attention(0, q, gqa_group=wl.gqa_group) for _ in range(3)]
        for o in again:
            assert torch.equal(o, out)
    finally:
        r.close()


def test_stats_and_capacity_errors():
    wl = small(prefill=((200, False),), decode_steps=2, window=16)
    r = Run(wl, capacity=203)
    try:
        r.prefill()
        r.step(0)
        r.step(1)
        st = r.cache.stats(with_counts=True)
        assert st["total_appended"] == 202 * wl.batch * wl.kv_heads
        assert st["total_retained"] == int(st["counts"].sum())
        assert st["total_evicted"] == st["total_appended"] - st["total_retained"]
        pages = int(np.sum((st["counts"] + 63) // 64))
        assert st["pages_in_use"] == pages
        assert st["max_retained"] == st["counts"].max()
        k, v, lg = workloads.gen_kv(wl, 0, "over", 2, r.dev)
        with pytest.raises(dms.DmsError) as ei:
            r.cache.append_and_evict(0, k, v, lg)  # 202 + 2 > capacity 203
        assert ei.value.code == dms.DMS_ERR_CAPACITY
    finally:
        r.close()


def test_pool_exhaustion_is_sticky():
    """A page pool too small for the batch sets the sticky capacity error."""
    wl = small(batch=2, kv_heads=2, prefill=((200, False),), decode_steps=0, p_evict=0.0)
    r = Run(wl, pool_tokens=64 * 6)  # 4 heads need 4 pages each
    try:
        r.prefill()
        st = r.cache.stats()
        assert st["device_error"] == dms.DMS_ERR_CAPACITY
        r.cache.reset()
        assert r.cache.stats()["device_error"] == 0
    finally:
        r.close()


def test_reset_and_reuse():
    wl = small(prefill=((500, False),), decode_steps=2)
    r = Run(wl)
    try:
        r.prefill()
        r.cache.reset()
        r.t = 0
        r.K.zero_()
        r.prefill()
        for s in range(2):
            q, out = r.step(s)
            r.check_outputs(q, out)
        r.check_retained()
        assert r.cache.stats()["peak_pages"] > 0
    finally:
        r.close()


@pytest.mark.parametrize("kernel", [dms.DMS_DECODE_CLUSTER, dms.DMS_DECODE_SPLIT],
                         ids=["cluster", "split"])
@pytest.mark.parametrize("fused", [True, False])
@pytest.mark.parametrize("B,Hkv,P", [(2, 2, 500), (1, 3, 560)], ids=["aligned", "odd-table"])
def test_multilayer_interleaved_steps(fused, kernel, B, Hkv, P):
    """Three layers advanced together, as a model decodes: each step visits layer 0, 1, 2.
    Consecutive launches serve different layers, so the fused kernel reads the layer's state
    and stages its first pages before waiting for the previous launch.  In the second shape a
    layer's page table holds 3 heads x 9 pages = 27 entries, so the tables of layers 1 and 2
    start off a 16-byte boundary (the L2 prefetch of the table must stay aligned)."""
    import oracle
    from _harness import MAX_ABS, MEAN_ABS
    L, G, w, steps = 3, 4, 24, 12
    wl = small(batch=B, kv_heads=Hkv, q_heads=Hkv * G, window=w)
    dev = torch.device("cuda")
    cache = dms.DmsCache(layers=L, kv_heads=Hkv, window=w, capacity=P + steps, batch=B,
                         decode_kernel=kernel)
    hist = []
    try:
        for l in range(L):
            k, v, lg = workloads.gen_kv(wl, l, "prefill", P, dev, p_override=[0.6 + 0.1 * l] * Hkv)
            cache.append_and_evict(l, k, v, lg)
            hist.append([k, v, lg])
        errs = []
        for s_ in range(steps):
            outs = []
            for l in range(L):
                k, v, lg = workloads.gen_kv(wl, l, f"d{s_}", 1, dev)
                q = workloads.gen_q(wl, l, f"d{s_}", dev)  # written right before the call
                if fused:
                    out = cache.append_and_decode(l, k, v, lg, q, gqa_group=G)
                else:
                    cache.append_and_evict(l, k, v, lg)
                    out = cache.decode_attention(l, q, gqa_group=G)
                for i, t in enumerate((k, v, lg)):
                    hist[l][i] = torch.cat([hist[l][i], t], 1)
                outs.append((q, out))
            if s_ % 3 == 2 or s_ == steps - 1:
                j = P + s_
                for l, (q, out) in enumerate(outs):
                    K, V, LG = (workloads.bf16_bits(t) for t in hist[l])
                    Q = workloads.bf16_bits(q)
                    got = out.float().cpu().numpy()
                    for b in range(B):
                        for h in range(Hkv):
                            ref = oracle.decode(Q[b, h * G:(h + 1) * G], K[b, :, h], V[b, :, h],
                                                LG[b, :, h], j, w)
                            errs.append(np.abs(got[b, h * G:(h + 1) * G] - ref).ravel())
                    pos = cache.export_positions(l)
                    for b in range(B):
                        for h in range(Hkv):
                            have = np.sort(pos[b, h][pos[b, h] >= 0])
                            assert np.array_equal(have, oracle.retained(LG[b, :, h], j, w)), (l, b, h)
        e = np.concatenate(errs)
        assert e.max() <= MAX_ABS and e.mean() <= MEAN_ABS, (e.max(), e.mean())
        assert cache.stats()["device_error"] == 0
    finally:
        cache.close()


def test_cluster_early_start_across_mixed_calls():
    """The per-head completion flags of the cluster kernel: fused steps (which publish),
    plain decodes in between (which read the state early and publish nothing), single and
    bulk appends and a reset (after which the next launch waits for its dependency
    first), on one layer of 1 x 4 heads; outputs and retained sets against the oracle
    after every call, and no device error."""
    wl = small(batch=1, kv_heads=4, q_heads=20, window=30, prefill=((700, False),),
               decode_steps=20, p_evict=0.6)  # capacity 720: 12 tokens appended per round
    r = Run(wl, decode_kernel=dms.DMS_DECODE_CLUSTER)
    assert r.cache.decode_plan(wl.gqa_group)["kernel"] == dms.DMS_DECODE_CLUSTER
    try:
        r.prefill()
        plan = ["fused", "fused", "decode", "fused", "append1", "decode", "fused", "bulk",
                "fused", "fused", "decode", "decode", "fused"]
        for round_ in range(2):
            for i, what in enumerate(plan):
                tag = f"r{round_}s{i}"
                if what in ("fused", "append1", "bulk"):
                    n = 5 if what == "bulk" else 1
                    k, v, lg = workloads.gen_kv(wl, 0, tag, n, r.dev)
                    q = workloads.gen_q(wl, 0, tag, r.dev)
                    if what == "fused":
                        out = r.cache.append_and_decode(0, k, v, lg, q, gqa_group=wl.gqa_group)
                        r.record(k, v, lg)
                        r.check_outputs(q, out)
                    else:
                        r.append(k, v, lg)
                else:
                    q = workloads.gen_q(wl, 0, tag, r.dev)
                    out = r.cache.decode_attention(0, q, gqa_group=wl.gqa_group)
                    r.check_outputs(q, out)
                r.check_retained()
            if round_ == 0:  # start again from an empty layer
                r.cache.reset()
                r.t = 0
                r.prefill()
        r.summary()
    finally:
        r.close()


def test_decode_plan():
    """Which kernel runs: the default takes per-head clusters for a batch-1 8-head cache (6
    CTAs each while the layer is short, <= 8192 tokens, up to 10 beyond), for 64 heads
    (clusters of 2 on GB300) and for 128 (one CTA per head); the flat split for more heads
    than SMs, or for few heads whose clusters would cover under half of the SMs.
    DMS_DECODE_CLUSTER takes clusters whenever every head's cluster fits (bf16 or fp8
    pages); G > 8 and the simple kernel never do."""
    nsm = torch.cuda.get_device_properties(0).multi_processor_count

    def plan(B, H, G=5, tokens=0, **kw):
        with dms.DmsCache(layers=1, kv_heads=H, window=16, capacity=tokens + 256, batch=B,
                          **kw) as c:
            if tokens:
                g = torch.Generator(device="cuda").manual_seed(0)
                k = torch.randn((B, tokens, H, 128), generator=g, device="cuda").to(torch.bfloat16)
                lg = torch.zeros((B, tokens, H), device="cuda").to(torch.bfloat16)
                c.append_and_evict(0, k, k, lg)
            return c.decode_plan(G)

    assert plan(1, 8) == {"kernel": dms.DMS_DECODE_CLUSTER, "ctas": 48, "cluster_size": 6}
    assert plan(1, 8, tokens=8191)["cluster_size"] == 6   # the next step reads 8192 tokens
    p = plan(1, 8, tokens=8192)
    assert p["kernel"] == dms.DMS_DECODE_CLUSTER and 6 <= p["cluster_size"] <= 10
    assert p["ctas"] == 8 * p["cluster_size"]
    if nsm == 152:
        assert p["cluster_size"] == 10
    p = plan(8, 8)  # 64 heads: the largest size that fits is small
    assert p["kernel"] == dms.DMS_DECODE_CLUSTER and p["cluster_size"] >= 2
    if nsm == 152:
        assert p == {"kernel": dms.DMS_DECODE_CLUSTER, "ctas": 128, "cluster_size": 2}
    p = plan(16, 8)  # 128 heads: one CTA per head
    assert p["kernel"] == dms.DMS_DECODE_CLUSTER and p["ctas"] == 128 * p["cluster_size"]
    if nsm == 152:
        assert p["cluster_size"] == 1
    assert plan(32, 8)["kernel"] == dms.DMS_DECODE_SPLIT  # 256 heads: more than SMs
    assert plan(1, 2)["kernel"] == dms.DMS_DECODE_SPLIT
    assert plan(1, 2, decode_kernel=dms.DMS_DECODE_CLUSTER) == {
        "kernel": dms.DMS_DECODE_CLUSTER, "ctas": 12, "cluster_size": 6}
    assert plan(1, 8, G=9)["kernel"] == dms.DMS_DECODE_SPLIT
    assert plan(1, 8, kv_format=dms.DMS_KV_FP8_E4M3)["kernel"] == dms.DMS_DECODE_CLUSTER
    assert plan(1, 8, decode_kernel=dms.DMS_DECODE_SPLIT)["kernel"] == dms.DMS_DECODE_SPLIT
    assert plan(1, 8, decode_kernel=dms.DMS_DECODE_SIMPLE) == {
        "kernel": dms.DMS_DECODE_SIMPLE, "ctas": 8, "cluster_size": 0}
    assert plan(1, 8, min_pages_per_cta=1)["kernel"] == dms.DMS_DECODE_SPLIT


@pytest.mark.parametrize("batch,kv_heads", [(1, 1), (1, 2)])
def test_cluster_stored_rows_after_fused_steps(batch, kv_heads):
    """Fused steps on per-head clusters whose CTAs stream more pages than they have stages,
    with a window of 4000 tokens at P(evict) 0.9: the slots the window's tokens hold are
    spread over the whole head, so the new token usually takes a slot in a page its CTA
    staged early and has reused since.  Every stored K/V row stays bit-exact (the row at
    each retained slot is its position's input), and outputs and retained sets match the
    oracle."""
    wl = small(batch=batch, kv_heads=kv_heads, q_heads=kv_heads * 5, window=4000,
               prefill=((8000, False),), decode_steps=40, p_evict=0.9)
    r = Run(wl, fused=True, decode_kernel=dms.DMS_DECODE_CLUSTER)
    try:
        plan = r.cache.decode_plan(wl.gqa_group)
        assert plan["kernel"] == dms.DMS_DECODE_CLUSTER
        r.prefill()
        pages = int(r.cache.stats(with_counts=True)["counts"].max() + 63) // 64
        assert pages > 6 * plan["cluster_size"]  # more pages per CTA than stages
        for s in range(wl.decode_steps):
            q, out = r.step(s)
            if s % 10 == 9:
                r.check_outputs(q, out)
                r.check_retained()
        r.check_codes()
        r.summary()
    finally:
        r.close()
