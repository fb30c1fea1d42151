"""GPU parity of the sparse DMS prefill attention (Sec. 3.1 mask / Fig. 1b, Sec. 3.2), through
the C ABI.  Every output row j equals the fp64 oracle's decode at position j (the retained
set R_j of reading 1) within max-abs 2e-2 / mean-abs 2e-3.
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


def _inputs(B, P, H, G, p, seed, borrowed=False):
    g = torch.Generator(device="cuda").manual_seed(seed)
    q = torch.randn((B, P, H * G, D), generator=g, device="cuda")
    k = torch.randn((B, P, H, D), generator=g, device="cuda").to(torch.bfloat16)
    v = torch.randn((B, P, H, D), generator=g, device="cuda").to(torch.bfloat16)
    if p >= 1:
        lg = torch.full((B, P, H), 1.0, device="cuda")
    elif p <= 0:
        lg = torch.full((B, P, H), -1.0, device="cuda")
    else:
        lg = torch.randn((B, P, H), generator=g, device="cuda") + statistics.NormalDist().inv_cdf(p)
    if borrowed:
        q[:, :, ::G, 0] = lg
    return q.to(torch.bfloat16), k, v, lg.to(torch.bfloat16)


def _ws_error(ws):
    code, err = dms.dms_prefill_device_error(ws.data_ptr(), None)
    assert code == dms.DMS_OK
    return err


def _check_rows(q, k, v, lg, out, w, G, rows=None, q_att=None):
    """Compare output rows [(b, j, h)] (all G query heads of KV head h) with the oracle."""
    B, P, H, _ = k.shape
    Q = workloads.bf16_bits(q if q_att is None else q_att)
    K, V, L = workloads.bf16_bits(k), workloads.bf16_bits(v), workloads.bf16_bits(lg)
    got = out.float().cpu().numpy()
    if rows is None:
        rows = [(b, j, h) for b in range(B) for j in range(P) for h in range(H)]
    errs = []
    for b, j, h in rows:
        ref = oracle.decode(Q[b, j, h * G:(h + 1) * G], K[b, :, h], V[b, :, h], L[b, :, h], j, w)
        errs.append(np.abs(got[b, j, h * G:(h + 1) * G] - ref).ravel())
    e = np.concatenate(errs)
    assert np.all(np.isfinite(got)), "non-finite output"
    assert e.max() <= MAX_ABS, e.max()
    assert e.mean() <= MEAN_ABS, e.mean()
    return e


KERNELS = [dms.DMS_PREFILL_TCGEN05, dms.DMS_PREFILL_MMA_SYNC]


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("B,P,H,G,w,p", [
    (2, 300, 2, 4, 32, 0.75),     # partial last tile, retained + window keys
    (1, 1000, 1, 4, 64, 0.9),     # many retained tiles
    (1, 77, 2, 1, 8, 0.5),        # MHA, a single partial tile
    (1, 200, 1, 16, 0, 1.0),      # w = 0, everything evicted: each query sees itself only
    (1, 130, 1, 4, 500, 0.6),     # window covers the prompt: dense causal
    (2, 257, 1, 4, 128, 0.0),     # nothing evicted: dense causal
    (1, 1, 1, 1, 0, 1.0),         # one token
    (1, 129, 2, 7, 3, 0.7),       # G = 7, tile boundary + 1
    (2, 1200, 2, 8, 64, 0.75),    # 320 (head, tile) units: > 2 per CTA of the persistent kernel
    (2, 1100, 3, 7, 16, 0.5),     # 378 units, G = 7; each CTA ends on one-tile units
])
def test_prefill_matches_oracle(B, P, H, G, w, p, kernel):
    q, k, v, lg = _inputs(B, P, H, G, p, seed=P + G)
    ws_bytes = dms.dms_prefill_workspace_bytes(B, P, H)[1]
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    out = torch.full_like(q, float("nan"))  # every row must be written
    dms.prefill_attention(q, k, v, lg, window=w, workspace=ws, out=out, kernel=kernel)
    torch.cuda.synchronize()
    assert _ws_error(ws) == dms.DMS_OK
    _check_rows(q, k, v, lg, out, w, G)
    # bitwise deterministic
    out2 = dms.prefill_attention(q, k, v, lg, window=w, workspace=ws, kernel=kernel)
    assert torch.equal(out, out2)


def test_prefill_special_logits():
    """NaN and -0 keep, +inf and the smallest positive subnormal evict (Sec. 3.2 sign rule)."""
    B, P, H, G, w = 1, 400, 2, 4, 16
    q, k, v, lg = _inputs(B, P, H, G, 0.5, seed=9)
    bits = lg.view(torch.int16)
    specials = torch.tensor([0x7FC0, 0x8000, 0x7F80, 0x0001, 0xFF80, 0x0000], dtype=torch.int32)
    idx = torch.arange(0, P, 7, device="cuda")
    bits[0, idx, :] = specials[torch.arange(len(idx)) % len(specials)].to(torch.int16).to("cuda")[:, None]
    out = dms.prefill_attention(q, k, v, lg, window=w)
    _check_rows(q, k, v, lg, out, w, G)


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("G", [1, 4, 16])
def test_prefill_borrowed_equals_explicit(G, kernel):
    B, P, H, w = 2, 350, 2, 40
    q, k, v, lg = _inputs(B, P, H, G, 0.8, seed=G, borrowed=True)
    q_keep = q.clone()
    out_b = dms.prefill_attention(q, k, v, None, window=w, kernel=kernel)
    assert torch.equal(q, q_keep), "the caller's q must not be modified"
    lg_x = q[:, :, ::G, 0].contiguous()
    qz = q.clone()
    qz[:, :, ::G, 0] = 0
    out_x = dms.prefill_attention(qz, k, v, lg_x, window=w, kernel=kernel)
    assert torch.equal(out_b, out_x)
    rows = [(b, j, h) for b in range(B) for j in range(0, P, 5) for h in range(H)]
    _check_rows(q, k, v, lg_x, out_b, w, G, rows=rows, q_att=qz)


def test_prefill_last_row_matches_decode_step():
    """Row P - 1 of the prefill equals a decode after appending the same P tokens."""
    B, P, H, G, w = 3, 700, 2, 4, 64
    q, k, v, lg = _inputs(B, P, H, G, 0.75, seed=21)
    out = dms.prefill_attention(q, k, v, lg, window=w)
    with dms.DmsCache(layers=1, kv_heads=H, window=w, capacity=P, batch=B) as cache:
        cache.append_and_evict(0, k[:, :P - 1].contiguous(), v[:, :P - 1].contiguous(),
                               lg[:, :P - 1].contiguous())
        dec = cache.append_and_decode(0, k[:, P - 1:].contiguous(), v[:, P - 1:].contiguous(),
                                      lg[:, P - 1:].contiguous(), q[:, P - 1].contiguous(),
                                      gqa_group=G)
    diff = (out[:, P - 1].float() - dec.float()).abs()
    assert diff.max().item() <= 2 * MAX_ABS


@pytest.mark.parametrize("kernel", KERNELS)
def test_prefill_full_prompt_sampled(kernel):
    """Qwen-R1-7B attention shape (28 / 4 heads), 7936-token prompt, P(evict) 0.75: >= 256
    sampled (sequence, query, KV head) rows, always including the first and last query."""
    B, P, H, G, w = 4, 7936, 4, 7, 256
    q, k, v, lg = _inputs(B, P, H, G, 0.75, seed=77)
    ws = torch.empty(dms.dms_prefill_workspace_bytes(B, P, H)[1], dtype=torch.uint8,
                     device="cuda")
    out = dms.prefill_attention(q, k, v, lg, window=w, workspace=ws, kernel=kernel)
    torch.cuda.synchronize()
    assert _ws_error(ws) == dms.DMS_OK
    rng = np.random.default_rng(5)
    rows = {(int(rng.integers(B)), int(rng.integers(P)), int(rng.integers(H))) for _ in range(300)}
    rows |= {(b, j, h) for b in range(B) for j in (0, 127, 128, w, P - 1) for h in range(H)}
    _check_rows(q, k, v, lg, out, w, G, rows=sorted(rows))


def test_prefill_rejects_bad_arguments():
    B, P, H, G = 1, 64, 1, 4
    q, k, v, lg = _inputs(B, P, H, G, 0.5, seed=1)
    out = torch.empty_like(q)
    need = dms.dms_prefill_workspace_bytes(B, P, H)[1]
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    args = lambda **kw: dict(dict(q=q.data_ptr(), k=k.data_ptr(), v=v.data_ptr(),  # noqa: E731
                                  lg=lg.data_ptr(), ws=ws.data_ptr(), wb=need, out=out.data_ptr(),
                                  G=G, w=8), **kw)

    def call(a):
        return dms.dms_prefill_attention(a["q"], a["k"], a["v"], a["lg"], B, P, H, a["G"], a["w"],
                                         0.0, a["ws"], a["wb"], a["out"], None)
    assert call(args()) == dms.DMS_OK
    assert call(args(wb=need - 1)) == dms.DMS_ERR_CAPACITY
    assert call(args(q=q.data_ptr() + 2)) == dms.DMS_ERR_INVALID_ARGUMENT
    assert call(args(ws=ws.data_ptr() + 8)) == dms.DMS_ERR_INVALID_ARGUMENT
    assert call(args(G=17)) == dms.DMS_ERR_INVALID_ARGUMENT
    assert call(args(w=-1)) == dms.DMS_ERR_INVALID_ARGUMENT
    torch.cuda.synchronize()


def test_prefill_kernels_agree():
    """The tcgen05 and the mma.sync kernels compute the same tiles: equal within rounding."""
    B, P, H, G, w = 2, 1500, 2, 7, 256
    q, k, v, lg = _inputs(B, P, H, G, 0.8, seed=31)
    a = dms.prefill_attention(q, k, v, lg, window=w, kernel=dms.DMS_PREFILL_TCGEN05)
    b = dms.prefill_attention(q, k, v, lg, window=w, kernel=dms.DMS_PREFILL_MMA_SYNC)
    assert (a.float() - b.float()).abs().max().item() <= 2e-2
