"""dms_decode_attention_paged_noalloc: decode over caller-owned pages with no allocation.

This entry point serves callers that cannot call cudaMalloc (their device memory
is owned by another allocator); the library uses a static device array for the
split-K scratch instead.  The test fills a regular cache through the C ABI,
rebuilds the same retained rows in caller-owned torch buffers in the documented
page layout, and checks the allocation-free call against dms_decode_attention on
two calls in a row, within the parity tolerance of the other GPU tests.

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


def _caller_owned_pages(r: Run):
    """Pages, page table and counts holding the cache's retained rows, slot for slot."""
    wl = r.wl
    B, H, D = wl.batch, wl.kv_heads, wl.head_dim
    pos = r.cache.export_positions(0)                       # [B, H, capacity], slot order
    counts = r.cache.stats(with_counts=True)["counts"][0]   # [B, H]
    max_pages = int((counts.max() + 63) // 64)
    heads = B * H
    pool = torch.zeros((heads * max_pages, 2, 64, 16, 8), dtype=torch.bfloat16, device=r.dev)
    rows = torch.arange(64, device=r.dev)[:, None]
    chunk_idx = (torch.arange(16, device=r.dev)[None, :] ^ (rows & 7))  # physical <- logical
    for b in range(B):
        for h in range(H):
            n = int(counts[b, h])
            p = torch.as_tensor(pos[b, h, :n].astype(np.int64), device=r.dev)
            npg = (n + 63) // 64
            for half, src in ((0, r.K), (1, r.V)):
                x = torch.zeros((npg * 64, D), dtype=torch.bfloat16, device=r.dev)
                x[:n] = src[b, p, h]
                x = x.view(npg, 64, 16, 8)
                # logical chunk c of row r sits at physical chunk c ^ (r & 7)
                y = torch.gather(x, 2, chunk_idx[None, :, :, None].expand(npg, 64, 16, 8))
                base = (b * H + h) * max_pages
                pool[base:base + npg, half] = y
    page_table = torch.arange(heads * max_pages, dtype=torch.int32, device=r.dev)
    cnt = torch.as_tensor(counts.reshape(-1).astype(np.int32), device=r.dev)
    return pool, page_table, cnt, max_pages


def _noalloc(pool, page_table, cnt, B, H, max_pages, q, G):
    out = torch.empty_like(q)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    code = dms.dms_decode_attention_paged_noalloc(
        ctypes.c_void_p(pool.data_ptr()), ctypes.c_void_p(page_table.data_ptr()),
        ctypes.c_void_p(cnt.data_ptr()), B, H, max_pages, ctypes.c_void_p(q.data_ptr()),
        ctypes.c_void_p(out.data_ptr()), G, 0.0, stream)
    return code, out


def test_noalloc_matches_cache_decode_twice():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    wl = workloads.Workload(name="noalloc", batch=3, layers=1, q_heads=20, kv_heads=4, window=48,
                            prefill=((1500, False),), decode_steps=2, p_evict=0.8)
    r = Run(wl)
    try:
        r.prefill()
        B, H, G = wl.batch, wl.kv_heads, wl.gqa_group
        for call in range(2):  # two calls in a row share (and must re-clear) the scratch
            q, ref = r.step(call)
            pool, pt, cnt, max_pages = _caller_owned_pages(r)
            code, out = _noalloc(pool, pt, cnt, B, H, max_pages, q, G)
            assert code == dms.DMS_OK, dms._native.status_string(code)
            torch.cuda.synchronize()
            e = (out.float() - ref.float()).abs()
            assert torch.isfinite(out.float()).all()
            assert e.max().item() <= MAX_ABS and e.mean().item() <= MEAN_ABS, (call, e.max().item())
            r.check_outputs(q, out)  # and against the fp64 oracle
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
