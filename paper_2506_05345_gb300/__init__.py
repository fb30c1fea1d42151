"""DMS decode on one GB300: Python face of libdms (include/dms.h).

Dynamic Memory Sparsification (arXiv 2506.05345) keeps, per (layer, sequence,
KV head), only the tokens whose eviction decision is 0 plus the last `window`
ones (delayed eviction, Sec. 3.1); decode attention reads only those.

Two layers of API, both thin:
  * the C names (``dms_cache_create``, ``dms_append_and_evict``,
    ``dms_decode_attention``, ``dms_cache_stats``, ...) re-exported from the
    ctypes binding, taking raw pointers exactly like the C ABI;
  * ``DmsCache``, which takes torch CUDA tensors, checks their shapes, and
    passes ``data_ptr()`` and the current stream.
PyTorch provides device memory and streams only; all computation is in the
library's CUDA kernels.  Nothing here falls back to a CPU implementation.
"""
from __future__ import annotations

import ctypes

import numpy as np

from . import _native
from ._native import (DMS_EVICT_DELAYED, DMS_EVICT_IMMEDIATE,  # noqa: F401
                      DMS_PREFILL_MMA_SYNC, DMS_PREFILL_TCGEN05,  # noqa: F401
                      DMS_DECODE_CLUSTER, DMS_DECODE_SIMPLE, DMS_DECODE_SPLIT,  # noqa: F401
                      DMS_DECODE_TILED,  # noqa: F401
                      DMS_ERR_CAPACITY,  # noqa: F401
                      DMS_KV_BF16, DMS_KV_FP8_E4M3,  # noqa: F401
                      DMS_ERR_INVALID_ARGUMENT, DMS_ERR_STATE, DMS_ERR_TIMEOUT, DMS_OK,
                      DmsLibraryError,
                      dms_options, dms_stats)

HEAD_DIM = 128


class DmsError(RuntimeError):
    def __init__(self, code: int, what: str):
        self.code = int(code)
        try:
            msg = _native.status_string(code)
        except DmsLibraryError:
            msg = f"status {code}"
        super().__init__(f"{what}: {msg} (status {code})")


def _check(code: int, what: str):
    if code != DMS_OK:
        raise DmsError(code, what)


def library():
    """The loaded libdms (raises DmsLibraryError if it is not built)."""
    return _native.load()


# ---- C names, same arguments as the header (raw pointers / ints) -------------

def dms_cache_create(layers, kv_heads, head_dim, window, capacity, opt: dms_options):
    out = ctypes.c_void_p()
    code = library().dms_cache_create(layers, kv_heads, head_dim, window, capacity,
                                      ctypes.byref(opt), ctypes.byref(out))
    return code, out.value


def dms_cache_destroy(cache):
    return library().dms_cache_destroy(cache)


def dms_cache_reset(cache, stream):
    return library().dms_cache_reset(cache, stream)


def dms_append_and_evict(cache, layer, k_ptr, v_ptr, logit_ptr, n_tokens, stream):
    return library().dms_append_and_evict(cache, layer, k_ptr, v_ptr, logit_ptr, n_tokens, stream)


def dms_decode_attention(cache, layer, q_ptr, out_ptr, gqa_group, sm_scale, stream):
    return library().dms_decode_attention(cache, layer, q_ptr, out_ptr, gqa_group,
                                          float(sm_scale), stream)


def dms_append_and_decode(cache, layer, k_ptr, v_ptr, logit_ptr, q_ptr, out_ptr, gqa_group,
                          sm_scale, stream):
    return library().dms_append_and_decode(cache, layer, k_ptr, v_ptr, logit_ptr, q_ptr, out_ptr,
                                           gqa_group, float(sm_scale), stream)


def dms_append_shared_prefix(cache, layer, k_ptr, v_ptr, logit_ptr, n_tokens, stream):
    return library().dms_append_shared_prefix(cache, layer, k_ptr, v_ptr, logit_ptr, n_tokens,
                                              stream)


def dms_append_and_evict_borrowed(cache, layer, k_ptr, v_ptr, q_ptr, n_tokens, gqa_group, stream):
    return library().dms_append_and_evict_borrowed(cache, layer, k_ptr, v_ptr, q_ptr, n_tokens,
                                                   gqa_group, stream)


def dms_decode_attention_borrowed(cache, layer, q_ptr, out_ptr, gqa_group, sm_scale, stream):
    return library().dms_decode_attention_borrowed(cache, layer, q_ptr, out_ptr, gqa_group,
                                                   float(sm_scale), stream)


def dms_append_and_decode_borrowed(cache, layer, k_ptr, v_ptr, q_ptr, out_ptr, gqa_group,
                                   sm_scale, stream):
    return library().dms_append_and_decode_borrowed(cache, layer, k_ptr, v_ptr, q_ptr, out_ptr,
                                                    gqa_group, float(sm_scale), stream)


def dms_prefill_workspace_bytes(batch, n_tokens, kv_heads):
    out = ctypes.c_size_t(0)
    code = library().dms_prefill_workspace_bytes(batch, n_tokens, kv_heads, ctypes.byref(out))
    return code, out.value


def dms_prefill_attention(q_ptr, k_ptr, v_ptr, logit_ptr, batch, n_tokens, kv_heads, gqa_group,
                          window, sm_scale, ws_ptr, ws_bytes, out_ptr, stream):
    return library().dms_prefill_attention(q_ptr, k_ptr, v_ptr, logit_ptr, batch, n_tokens,
                                           kv_heads, gqa_group, window, float(sm_scale), ws_ptr,
                                           ws_bytes, out_ptr, stream)


def dms_prefill_attention_borrowed(q_ptr, k_ptr, v_ptr, batch, n_tokens, kv_heads, gqa_group,
                                   window, sm_scale, ws_ptr, ws_bytes, out_ptr, stream):
    return library().dms_prefill_attention_borrowed(q_ptr, k_ptr, v_ptr, batch, n_tokens,
                                                    kv_heads, gqa_group, window, float(sm_scale),
                                                    ws_ptr, ws_bytes, out_ptr, stream)


def dms_prefill_device_error(ws_ptr, stream):
    out = ctypes.c_int(0)
    code = library().dms_prefill_device_error(ws_ptr, stream, ctypes.byref(out))
    return code, out.value


def dms_prefill_attention_ex(q_ptr, k_ptr, v_ptr, logit_ptr, batch, n_tokens, kv_heads,
                             gqa_group, window, eviction_policy, kernel, sm_scale, ws_ptr,
                             ws_bytes, out_ptr, stream):
    return library().dms_prefill_attention_ex(q_ptr, k_ptr, v_ptr, logit_ptr, batch, n_tokens,
                                              kv_heads, gqa_group, window, eviction_policy, kernel,
                                              float(sm_scale), ws_ptr, ws_bytes, out_ptr, stream)


def prefill_attention(q, k, v, decision_logit=None, window: int = 256, gqa_group=None,
                      sm_scale: float = 0.0, workspace=None, out=None, stream=None,
                      eviction_policy: int = 0, kernel: int = -1):
    """Sparse DMS prefill attention of a whole prompt (no cache involved).

    q: [B, P, Hkv * G, 128], k, v: [B, P, Hkv, 128], decision_logit: [B, P, Hkv] bf16 CUDA
    tensors; decision_logit=None takes the decisions from element 0 of each group's first
    query head (App. B).  Returns out [B, P, Hkv * G, 128] bf16.  The workspace (uint8
    CUDA tensor) is allocated when not given.
    """
    import torch
    B, P, Hkv, D = k.shape
    if gqa_group is None:
        gqa_group = q.shape[2] // Hkv
    code, nbytes = dms_prefill_workspace_bytes(B, P, Hkv)
    _check(code, "dms_prefill_workspace_bytes")
    if workspace is None:
        workspace = torch.empty(nbytes, dtype=torch.uint8, device=q.device)
    if out is None:
        out = torch.empty_like(q)
    qp = _bf16_cuda(q, (B, P, Hkv * gqa_group, D), "q")
    kp = _bf16_cuda(k, (B, P, Hkv, D), "k")
    vp = _bf16_cuda(v, (B, P, Hkv, D), "v")
    op = _bf16_cuda(out, (B, P, Hkv * gqa_group, D), "out")
    if workspace.dtype != torch.uint8 or not workspace.is_cuda:
        raise TypeError("workspace must be a uint8 CUDA tensor")
    wp = ctypes.c_void_p(workspace.data_ptr())
    wb = workspace.numel()
    if eviction_policy != 0 or kernel >= 0:
        lp = None if decision_logit is None else _bf16_cuda(decision_logit, (B, P, Hkv),
                                                            "decision_logit")
        code = dms_prefill_attention_ex(qp, kp, vp, lp, B, P, Hkv, gqa_group, window,
                                        eviction_policy,
                                        DMS_PREFILL_TCGEN05 if kernel < 0 else kernel,
                                        sm_scale, wp, wb, op, _stream_ptr(stream))
        _check(code, "dms_prefill_attention_ex")
    elif decision_logit is None:
        code = dms_prefill_attention_borrowed(qp, kp, vp, B, P, Hkv, gqa_group, window, sm_scale,
                                              wp, wb, op, _stream_ptr(stream))
        _check(code, "dms_prefill_attention_borrowed")
    else:
        lp = _bf16_cuda(decision_logit, (B, P, Hkv), "decision_logit")
        code = dms_prefill_attention(qp, kp, vp, lp, B, P, Hkv, gqa_group, window, sm_scale, wp,
                                     wb, op, _stream_ptr(stream))
        _check(code, "dms_prefill_attention")
    return out


def dms_cache_stats(cache, stats: dms_stats, counts_ptr, stream):
    return library().dms_cache_stats(cache, ctypes.byref(stats), counts_ptr, stream)


def dms_cache_export_positions(cache, layer, host_pos_ptr, stream):
    return library().dms_cache_export_positions(cache, layer, host_pos_ptr, stream)


def dms_cache_export_kv(cache, layer, host_k_ptr, host_v_ptr, host_scales_ptr, stream):
    return library().dms_cache_export_kv(cache, layer, host_k_ptr, host_v_ptr, host_scales_ptr,
                                         stream)


def dms_cache_layer_length(cache, layer):
    out = ctypes.c_int64()
    code = library().dms_cache_layer_length(cache, layer, ctypes.byref(out))
    return code, out.value


def dms_decode_plan(cache, layer, gqa_group):
    """(code, kernel, ctas, cluster_size) of the next fused decode step of `layer`."""
    k, n, c = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
    code = library().dms_decode_plan(cache, layer, gqa_group, ctypes.byref(k), ctypes.byref(n),
                                     ctypes.byref(c))
    return code, k.value, n.value, c.value


def dms_decode_attention_paged_noalloc(pool_ptr, page_table_ptr, counts_ptr, batch, kv_heads,
                                       max_pages, q_ptr, out_ptr, gqa_group, sm_scale, stream):
    """Decode over caller-owned pages with the library's static scratch (no allocation)."""
    return library().dms_decode_attention_paged_noalloc(
        pool_ptr, page_table_ptr, counts_ptr, batch, kv_heads, max_pages, q_ptr, out_ptr,
        gqa_group, float(sm_scale), stream)


def dms_decode_noalloc_device_error(stream):
    """(status of the call, device-side status of the last allocation-free decode)."""
    out = ctypes.c_int(0)
    code = library().dms_decode_noalloc_device_error(stream, ctypes.byref(out))
    return code, out.value


def dms_selftest_noalloc_timeout(limit_ns, stream):
    return library().dms_selftest_noalloc_timeout(int(limit_ns), stream)


def dms_selftest_bounded_wait(arrive, limit_ns, stream):
    return library().dms_selftest_bounded_wait(int(arrive), int(limit_ns), stream)


# ---- torch-facing wrapper ---------------------------------------------------

def _stream_ptr(stream=None):
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _bf16_cuda(t, shape, name):
    import torch
    if not isinstance(t, torch.Tensor) or not t.is_cuda or t.dtype != torch.bfloat16:
        raise TypeError(f"{name} must be a CUDA bfloat16 tensor")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


class DmsCache:
    """Per-head sparsified KV cache for `layers` layers of `batch` x `kv_heads` heads."""

    def __init__(self, layers: int, kv_heads: int, window: int, capacity: int, batch: int,
                 head_dim: int = HEAD_DIM, pool_tokens: int = 0,
                 decode_kernel: int = DMS_DECODE_TILED, ctas_per_sm: int = 0,
                 min_pages_per_cta: int = 0, eviction_policy: int = 0,
                 kv_format: int = DMS_KV_BF16):
        self._h = None
        opt = dms_options()
        opt.kv_format = kv_format
        opt.batch = batch
        opt.pool_tokens = pool_tokens
        opt.decode_kernel = decode_kernel
        opt.ctas_per_sm = ctas_per_sm
        opt.min_pages_per_cta = min_pages_per_cta
        opt.eviction_policy = eviction_policy
        code, h = dms_cache_create(layers, kv_heads, head_dim, window, capacity, opt)
        _check(code, "dms_cache_create")
        self._h = h
        self.layers, self.kv_heads, self.window = layers, kv_heads, window
        self.capacity, self.batch, self.head_dim = capacity, batch, head_dim
        self.kv_format = kv_format

    def close(self):
        if self._h is not None:
            dms_cache_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    @property
    def handle(self):
        return self._h

    def reset(self, stream=None):
        _check(dms_cache_reset(self._h, _stream_ptr(stream)), "dms_cache_reset")

    def append_and_evict(self, layer: int, k, v, decision_logit, stream=None):
        """k, v: [batch, n, kv_heads, 128] bf16; decision_logit: [batch, n, kv_heads] bf16."""
        n = k.shape[1]
        B, H, D = self.batch, self.kv_heads, self.head_dim
        kp = _bf16_cuda(k, (B, n, H, D), "k")
        vp = _bf16_cuda(v, (B, n, H, D), "v")
        lp = _bf16_cuda(decision_logit, (B, n, H), "decision_logit")
        _check(dms_append_and_evict(self._h, layer, kp, vp, lp, n, _stream_ptr(stream)),
               "dms_append_and_evict")

    def decode_attention(self, layer: int, q, out=None, gqa_group: int | None = None,
                         sm_scale: float = 0.0, stream=None):
        """q, out: [batch, kv_heads * gqa_group, 128] bf16.  Returns out."""
        import torch
        B, H, D = self.batch, self.kv_heads, self.head_dim
        if gqa_group is None:
            gqa_group = q.shape[1] // H
        if out is None:
            out = torch.empty_like(q)
        qp = _bf16_cuda(q, (B, H * gqa_group, D), "q")
        op = _bf16_cuda(out, (B, H * gqa_group, D), "out")
        _check(dms_decode_attention(self._h, layer, qp, op, gqa_group, sm_scale,
                                    _stream_ptr(stream)), "dms_decode_attention")
        return out

    def append_and_decode(self, layer: int, k, v, decision_logit, q, out=None,
                          gqa_group: int | None = None, sm_scale: float = 0.0, stream=None):
        """One decode step of one layer (single-token append + decode in one launch)."""
        import torch
        B, H, D = self.batch, self.kv_heads, self.head_dim
        if gqa_group is None:
            gqa_group = q.shape[1] // H
        if out is None:
            out = torch.empty_like(q)
        kp = _bf16_cuda(k, (B, 1, H, D), "k")
        vp = _bf16_cuda(v, (B, 1, H, D), "v")
        lp = _bf16_cuda(decision_logit, (B, 1, H), "decision_logit")
        qp = _bf16_cuda(q, (B, H * gqa_group, D), "q")
        op = _bf16_cuda(out, (B, H * gqa_group, D), "out")
        _check(dms_append_and_decode(self._h, layer, kp, vp, lp, qp, op, gqa_group, sm_scale,
                                     _stream_ptr(stream)), "dms_append_and_decode")
        return out

    def append_shared_prefix(self, layer: int, k, v, decision_logit, stream=None):
        """A prompt identical in every sequence, given once: k, v [1, n, kv_heads, 128],
        decision_logit [1, n, kv_heads] bf16; the layer must be empty.  Its frozen pages
        are stored once and shared by all sequences."""
        n = k.shape[1]
        H, D = self.kv_heads, self.head_dim
        kp = _bf16_cuda(k, (1, n, H, D), "k")
        vp = _bf16_cuda(v, (1, n, H, D), "v")
        lp = _bf16_cuda(decision_logit, (1, n, H), "decision_logit")
        _check(dms_append_shared_prefix(self._h, layer, kp, vp, lp, n, _stream_ptr(stream)),
               "dms_append_shared_prefix")

    # ---- decisions from the borrowed query neuron (App. B): element 0 of each group's
    # first query head is the decision logit and is taken as 0 by the attention.

    def append_and_evict_borrowed(self, layer: int, k, v, q, gqa_group: int, stream=None):
        """k, v: [batch, n, kv_heads, 128]; q: [batch, n, kv_heads * gqa_group, 128] bf16."""
        n = k.shape[1]
        B, H, D = self.batch, self.kv_heads, self.head_dim
        kp = _bf16_cuda(k, (B, n, H, D), "k")
        vp = _bf16_cuda(v, (B, n, H, D), "v")
        qp = _bf16_cuda(q, (B, n, H * gqa_group, D), "q")
        _check(dms_append_and_evict_borrowed(self._h, layer, kp, vp, qp, n, gqa_group,
                                             _stream_ptr(stream)), "dms_append_and_evict_borrowed")

    def decode_attention_borrowed(self, layer: int, q, out=None, gqa_group: int | None = None,
                                  sm_scale: float = 0.0, stream=None):
        """As decode_attention, with element 0 of each group's first query head taken as 0."""
        import torch
        B, H, D = self.batch, self.kv_heads, self.head_dim
        if gqa_group is None:
            gqa_group = q.shape[1] // H
        if out is None:
            out = torch.empty_like(q)
        qp = _bf16_cuda(q, (B, H * gqa_group, D), "q")
        op = _bf16_cuda(out, (B, H * gqa_group, D), "out")
        _check(dms_decode_attention_borrowed(self._h, layer, qp, op, gqa_group, sm_scale,
                                             _stream_ptr(stream)), "dms_decode_attention_borrowed")
        return out

    def append_and_decode_borrowed(self, layer: int, k, v, q, out=None,
                                   gqa_group: int | None = None, sm_scale: float = 0.0,
                                   stream=None):
        """One decode step with the decisions read from q (one launch when fusable)."""
        import torch
        B, H, D = self.batch, self.kv_heads, self.head_dim
        if gqa_group is None:
            gqa_group = q.shape[1] // H
        if out is None:
            out = torch.empty_like(q)
        kp = _bf16_cuda(k, (B, 1, H, D), "k")
        vp = _bf16_cuda(v, (B, 1, H, D), "v")
        qp = _bf16_cuda(q, (B, H * gqa_group, D), "q")
        op = _bf16_cuda(out, (B, H * gqa_group, D), "out")
        _check(dms_append_and_decode_borrowed(self._h, layer, kp, vp, qp, op, gqa_group, sm_scale,
                                              _stream_ptr(stream)),
               "dms_append_and_decode_borrowed")
        return out

    def stats(self, stream=None, with_counts: bool = False):
        st = dms_stats()
        counts = None
        cptr = None
        if with_counts:
            counts = np.zeros((self.layers, self.batch, self.kv_heads), dtype=np.int32)
            cptr = ctypes.c_void_p(counts.ctypes.data)
        code = dms_cache_stats(self._h, st, cptr, _stream_ptr(stream))
        d = {f: getattr(st, f) for f, _ in dms_stats._fields_ if f != "reserved"}
        if code not in (DMS_OK, st.device_error):
            _check(code, "dms_cache_stats")
        if with_counts:
            d["counts"] = counts
        return d

    def export_positions(self, layer: int, stream=None) -> np.ndarray:
        """[batch, kv_heads, capacity] int32 positions in slot order, -1 past n_h."""
        out = np.empty((self.batch, self.kv_heads, self.capacity), dtype=np.int32)
        _check(dms_cache_export_positions(self._h, layer, ctypes.c_void_p(out.ctypes.data),
                                          _stream_ptr(stream)), "dms_cache_export_positions")
        return out

    def export_kv(self, layer: int, stream=None):
        """Stored rows of `layer` in head_dim order: (k, v, scales) with k, v of shape
        [batch, kv_heads, capacity, 128] (uint16 bf16 bits, or uint8 E4M3 codes for an
        fp8 cache) and scales [batch, kv_heads, capacity, 2] float32 (key, value) for fp8
        caches, None otherwise; zero past each head's n_h."""
        shape = (self.batch, self.kv_heads, self.capacity, self.head_dim)
        fp8 = self.kv_format == DMS_KV_FP8_E4M3
        dt = np.uint8 if fp8 else np.uint16
        k, v = np.empty(shape, dtype=dt), np.empty(shape, dtype=dt)
        sc = np.empty(shape[:3] + (2,), dtype=np.float32) if fp8 else None
        _check(dms_cache_export_kv(self._h, layer, ctypes.c_void_p(k.ctypes.data),
                                   ctypes.c_void_p(v.ctypes.data),
                                   ctypes.c_void_p(sc.ctypes.data) if fp8 else None,
                                   _stream_ptr(stream)), "dms_cache_export_kv")
        return k, v, sc

    def layer_length(self, layer: int) -> int:
        code, n = dms_cache_layer_length(self._h, layer)
        _check(code, "dms_cache_layer_length")
        return n

    def decode_plan(self, gqa_group: int, layer: int = 0) -> dict:
        """The kernel the next fused decode step of `layer` runs, its CTAs, cluster size."""
        code, kernel, ctas, cluster = dms_decode_plan(self._h, layer, gqa_group)
        _check(code, "dms_decode_plan")
        return {"kernel": kernel, "ctas": ctas, "cluster_size": cluster}
