"""dms_decode_attention_paged_noalloc: decode over caller-owned pages with no allocation.

This entry point serves callers that cannot call cudaMalloc (their device memory
is owned by another allocator); the library uses a static device array for the
split-K scratch instead.  The test fills a regular cache through the C ABI,
rebuilds the same retained rows in caller-owned torch buffers in the documented
page layout -- at shuffled pool pages, with unused pages full of NaN between
them, so that a kernel ignoring the page table would fail -- and checks the
allocation-free call against dms_decode_attention on two calls in a row, within
the parity tolerance of the other GPU tests, for a group that fits one n-tile
(G = 5) and one that needs two (G = 16).  After each call the device-side status
the static array holds is read back and must be DMS_OK.  A second test makes a
bounded wait give up on that status word (a barrier nothing completes, a short
limit) and checks that the timeout is reported, and that the next decode clears it.

The file name sorts last so that a run stopping at the first failure has already
run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2506_05345_gb300 as dms
import workloads
from _harness import MAX_ABS, MEAN_ABS, Run

pytestmark = pytest.mark.gpu

NAN_BF16 = 0x7FC0


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _caller_owned_pages(r: Run, seed: int):
    """Pages, page table and counts holding the cache's retained rows, slot for slot,
    at shuffled pool pages; unused pool pages and rows past each count hold NaN."""
    wl = r.wl
    B, H, D = wl.batch, wl.kv_heads, wl.head_dim
    pos = r.cache.export_positions(0)                       # [B, H, capacity], slot order
    counts = r.cache.stats(with_counts=True)["counts"][0]   # [B, H]
    max_pages = int((counts.max() + 63) // 64) + 1          # one spare entry per head
    heads = B * H
    n_pool = heads * max_pages + 2 * heads                  # unused pages between the heads
    rng = np.random.default_rng(seed)
    perm = rng.permutation(n_pool)
    page_table = np.full((heads, max_pages), -1, dtype=np.int32)
    pool = torch.full((n_pool, 2, 64, 16, 8), 0, dtype=torch.int16, device=r.dev)
    pool.fill_(NAN_BF16)
    pool = pool.view(torch.bfloat16)
    rows = torch.arange(64, device=r.dev)[:, None]
    chunk_idx = (torch.arange(16, device=r.dev)[None, :] ^ (rows & 7))  # physical <- logical
    nxt = 0
    for b in range(B):
        for h in range(H):
            n = int(counts[b, h])
            p = torch.as_tensor(pos[b, h, :n].astype(np.int64), device=r.dev)
            npg = (n + 63) // 64
            ids = perm[nxt:nxt + npg]
            nxt += npg
            page_table[b * H + h, :npg] = ids
            idx = torch.as_tensor(ids.astype(np.int64), device=r.dev)
            for half, src in ((0, r.K), (1, r.V)):
                x = torch.full((npg * 64, D), float("nan"), dtype=torch.bfloat16, device=r.dev)
                x[:n] = src[b, p, h]
                x = x.view(npg, 64, 16, 8)
                # logical chunk c of row r sits at physical chunk c ^ (r & 7)
                y = torch.gather(x, 2, chunk_idx[None, :, :, None].expand(npg, 64, 16, 8))
                pool[idx, half] = y
    pt = torch.as_tensor(page_table.reshape(-1), device=r.dev)
    cnt = torch.as_tensor(counts.reshape(-1).astype(np.int32), device=r.dev)
    return pool, pt, cnt, max_pages


def _noalloc(pool, page_table, cnt, B, H, max_pages, q, G):
    out = torch.empty_like(q)
    code = dms.dms_decode_attention_paged_noalloc(
        ctypes.c_void_p(pool.data_ptr()), ctypes.c_void_p(page_table.data_ptr()),
        ctypes.c_void_p(cnt.data_ptr()), B, H, max_pages, ctypes.c_void_p(q.data_ptr()),
        ctypes.c_void_p(out.data_ptr()), G, 0.0, _stream())
    return code, out


def _device_status():
    code, status = dms.dms_decode_noalloc_device_error(_stream())
    assert code == dms.DMS_OK, dms._native.status_string(code)
    return status


@pytest.mark.parametrize("q_heads", [20, 64])  # G = 5 (one n-tile), G = 16 (two n-tiles)
def test_noalloc_matches_cache_decode_twice(q_heads):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    wl = workloads.Workload(name=f"noalloc{q_heads}", batch=3, layers=1, q_heads=q_heads,
                            kv_heads=4, window=48, prefill=((1500, False),), decode_steps=2,
                            p_evict=0.8)
    r = Run(wl)
    try:
        r.prefill()
        B, H, G = wl.batch, wl.kv_heads, wl.gqa_group
        for call in range(2):  # two calls in a row share (and must re-clear) the scratch
            q, ref = r.step(call)
            pool, pt, cnt, max_pages = _caller_owned_pages(r, seed=call)
            code, out = _noalloc(pool, pt, cnt, B, H, max_pages, q, G)
            assert code == dms.DMS_OK, dms._native.status_string(code)
            torch.cuda.synchronize()
            assert _device_status() == dms.DMS_OK
            e = (out.float() - ref.float()).abs()
            assert torch.isfinite(out.float()).all()
            assert e.max().item() <= MAX_ABS and e.mean().item() <= MEAN_ABS, (call, e.max().item())
            r.check_outputs(q, out)  # and against the fp64 oracle
    finally:
        r.close()


def test_noalloc_timeout_is_reported_then_cleared():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    # a bounded wait that nothing completes gives up after 2 ms on the static error word
    assert dms.dms_selftest_noalloc_timeout(2_000_000, _stream()) == dms.DMS_OK
    assert _device_status() == dms.DMS_ERR_TIMEOUT
    assert _device_status() == dms.DMS_ERR_TIMEOUT  # reading does not clear it
    # the context stays usable, and the next decode clears the word and succeeds
    wl = workloads.Workload(name="noalloc-after-timeout", batch=2, layers=1, q_heads=8,
                            kv_heads=2, window=16, prefill=((300, False),), decode_steps=1,
                            p_evict=0.5)
    r = Run(wl)
    try:
        r.prefill()
        q, ref = r.step(0)
        pool, pt, cnt, max_pages = _caller_owned_pages(r, seed=7)
        code, out = _noalloc(pool, pt, cnt, wl.batch, wl.kv_heads, max_pages, q, wl.gqa_group)
        assert code == dms.DMS_OK
        torch.cuda.synchronize()
        assert _device_status() == dms.DMS_OK
        r.check_outputs(q, out)
    finally:
        r.close()


def test_noalloc_rejects_batches_beyond_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dev = torch.device("cuda")
    q = torch.zeros((1000, 1, 128), dtype=torch.bfloat16, device=dev)
    pool = torch.zeros((1, 2, 64, 128), dtype=torch.bfloat16, device=dev)
    pt = torch.zeros((1000,), dtype=torch.int32, device=dev)
    cnt = torch.zeros((1000,), dtype=torch.int32, device=dev)
    code, _ = _noalloc(pool, pt, cnt, 1000, 1, 1, q, 1)  # 1000 heads + SMs > 1024 records
    assert code == dms.DMS_ERR_CAPACITY
    code, _ = _noalloc(pool, pt, cnt, 1, 1, 1, q[:1], 17)  # group above 16
    assert code == dms.DMS_ERR_INVALID_ARGUMENT
    code = dms.dms_decode_attention_paged_noalloc(  # page table not 4-byte aligned
        ctypes.c_void_p(pool.data_ptr()), ctypes.c_void_p(pt.data_ptr() + 2),
        ctypes.c_void_p(cnt.data_ptr()), 1, 1, 1, ctypes.c_void_p(q.data_ptr()),
        ctypes.c_void_p(q.data_ptr()), 1, 0.0, _stream())
    assert code == dms.DMS_ERR_INVALID_ARGUMENT
