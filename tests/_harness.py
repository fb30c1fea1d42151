"""Drives the CUDA path through the C ABI and checks it against the fp64 oracle.

The full appended history (K, V, logits) of every layer under test is kept on the
device so that any (layer, sequence, KV head) can be handed to the oracle at any step.
Tolerances: retained sets bit-exact; attention outputs max-abs <= 2e-2 and
mean-abs <= 2e-3 against the fp64 oracle on the same bf16 inputs.  An fp8 cache
(kv_format=DMS_KV_FP8_E4M3) is checked against the oracle's attention over its own
quantisation of the history; its stored codes and scales bit-exact.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
import paper_2506_05345_gb300 as dms
import workloads

MAX_ABS = 2e-2
MEAN_ABS = 2e-3


class Run:
    """A cache of `layers` layers driven through the C ABI, with every layer's appended history
    (K, V, decision logits) kept on the device; layer l draws the inputs of workload layer
    `layer + l`.  Steps append the new token and decode every layer in order, as the bench does."""

    # Largest K or V tensor generated at once (elements); bigger prompts are appended in chunks.
    CHUNK_ELEMS = 1 << 28

    def __init__(self, wl: workloads.Workload, device="cuda", layer: int = 0,
                 capacity: int | None = None, fused: bool = False, layers: int = 1, **cache_kw):
        self.wl, self.layer, self.dev = wl, layer, torch.device(device)
        self.fused = fused  # decode steps through dms_append_and_decode
        self.fp8 = cache_kw.get("kv_format", dms.DMS_KV_BF16) == dms.DMS_KV_FP8_E4M3
        self.T = capacity or wl.context
        self.n_layers = layers
        B, H, D = wl.batch, wl.kv_heads, wl.head_dim
        self.cache = dms.DmsCache(layers=layers, kv_heads=H, window=wl.window, capacity=self.T,
                                  batch=B, **cache_kw)
        self.Ks = [torch.zeros((B, self.T, H, D), dtype=torch.bfloat16, device=self.dev)
                   for _ in range(layers)]
        self.Vs = [torch.zeros_like(k) for k in self.Ks]
        self.Ls = [torch.zeros((B, self.T, H), dtype=torch.bfloat16, device=self.dev)
                   for _ in range(layers)]
        self.ts = [0] * layers
        self.errs = []

    # layer 0's history (the single-layer view most tests use)
    K = property(lambda self: self.Ks[0])
    V = property(lambda self: self.Vs[0])
    L = property(lambda self: self.Ls[0])

    @property
    def t(self):
        return self.ts[0]

    @t.setter
    def t(self, value):
        self.ts[0] = value

    def close(self):
        self.cache.close()

    def record(self, k, v, lg, layer=0):
        n, t = k.shape[1], self.ts[layer]
        self.Ks[layer][:, t:t + n] = k
        self.Vs[layer][:, t:t + n] = v
        self.Ls[layer][:, t:t + n] = lg
        self.ts[layer] = t + n

    def append(self, k, v, lg, layer=0):
        self.cache.append_and_evict(layer, k, v, lg)
        self.record(k, v, lg, layer)

    def prefill(self):
        wl = self.wl
        per_token = wl.batch * wl.kv_heads * wl.head_dim
        chunk = max(64, self.CHUNK_ELEMS // per_token)
        for layer in range(self.n_layers):
            for i, (n, shared) in enumerate(wl.prefill):
                for c0 in range(0, n, chunk):
                    nc = min(chunk, n - c0)
                    tag = f"prefill{i}" + (f"c{c0}" if n > chunk else "")
                    if shared:
                        k, v, lg = workloads.gen_kv(wl, self.layer + layer, tag, nc, self.dev,
                                                    batch=1)
                        B = wl.batch
                        k = k.expand(B, -1, -1, -1).contiguous()
                        v = v.expand(B, -1, -1, -1).contiguous()
                        lg = lg.expand(B, -1, -1).contiguous()
                    else:
                        k, v, lg = workloads.gen_kv(wl, self.layer + layer, tag, nc, self.dev)
                    self.append(k, v, lg, layer)
                    del k, v, lg

    def step_layer(self, s: int, layer: int = 0, p_override=None):
        k, v, lg = workloads.gen_kv(self.wl, self.layer + layer, f"decode{s}", 1, self.dev,
                                    p_override=p_override)
        q = workloads.gen_q(self.wl, self.layer + layer, f"decode{s}", self.dev)
        if self.fused:
            out = self.cache.append_and_decode(layer, k, v, lg, q, gqa_group=self.wl.gqa_group)
            self.record(k, v, lg, layer)
        else:
            self.append(k, v, lg, layer)
            out = self.cache.decode_attention(layer, q, gqa_group=self.wl.gqa_group)
        return q, out

    def step(self, s: int, p_override=None):
        """Decode step s of layer 0 (single-layer runs)."""
        return self.step_layer(s, 0, p_override)

    def step_all(self, s: int):
        """Decode step s of every layer, in layer order; [(q, out)] per layer."""
        return [self.step_layer(s, layer) for layer in range(self.n_layers)]

    # ---- checks

    def logits_host(self, layer=0) -> np.ndarray:
        return workloads.bf16_bits(self.Ls[layer][:, :self.ts[layer]])

    def check_retained(self, heads=None, layer=0):
        """Retained positions of every (b, h) of `layer` equal the oracle's R_j, bit for bit."""
        j = self.ts[layer] - 1
        pos = self.cache.export_positions(layer)
        L = self.logits_host(layer)
        B, H = self.wl.batch, self.wl.kv_heads
        heads = heads if heads is not None else [(b, h) for b in range(B) for h in range(H)]
        st = self.cache.stats(with_counts=True)
        assert st["device_error"] == 0, st
        for b, h in heads:
            row = pos[b, h]
            n = int(st["counts"][layer, b, h])
            assert np.all(row[:n] >= 0) and np.all(row[n:] == -1), (b, h)
            have = np.sort(row[:n])
            want = oracle.retained(L[b, :, h], j, self.wl.window)
            assert np.array_equal(have, want), (layer, b, h, len(have), len(want))
        return st

    def check_outputs(self, q, out, pairs=None, record=True, layer=0):
        """Outputs of the given (b, h) KV heads (all G query heads each) of `layer` vs the
        oracle."""
        j = self.ts[layer] - 1
        G, B, H = self.wl.gqa_group, self.wl.batch, self.wl.kv_heads
        pairs = pairs if pairs is not None else [(b, h) for b in range(B) for h in range(H)]
        Q = workloads.bf16_bits(q)
        got = out.float().cpu().numpy()
        errs = []
        for b, h in pairs:
            k = workloads.bf16_bits(self.Ks[layer][b, :j + 1, h])
            v = workloads.bf16_bits(self.Vs[layer][b, :j + 1, h])
            lg = workloads.bf16_bits(self.Ls[layer][b, :j + 1, h])
            if self.fp8:
                kc, ks = oracle.quantize_rows_e4m3(k)
                vc, vs = oracle.quantize_rows_e4m3(v)
                ref = oracle.decode_fp8(Q[b, h * G:(h + 1) * G], kc, ks, vc, vs, lg, j,
                                        self.wl.window)
            else:
                ref = oracle.decode(Q[b, h * G:(h + 1) * G], k, v, lg, j, self.wl.window)
            errs.append(np.abs(got[b, h * G:(h + 1) * G].astype(np.float64) - ref).ravel())
        e = np.concatenate(errs)
        assert np.all(np.isfinite(got)), "non-finite output"
        if record:
            self.errs.append(e)
        assert e.max() <= MAX_ABS, e.max()
        return e

    def check_codes(self, heads=None):
        """Stored rows of every retained slot equal the input row at the slot's position:
        bf16 bits, or (fp8) the oracle's E4M3 codes and fp32 scales, bit for bit."""
        k_st, v_st, sc = self.cache.export_kv(0)
        pos = self.cache.export_positions(0)
        counts = self.cache.stats(with_counts=True)["counts"][0]
        B, H = self.wl.batch, self.wl.kv_heads
        heads = heads if heads is not None else [(b, h) for b in range(B) for h in range(H)]
        for b, h in heads:
            n = int(counts[b, h])
            p = pos[b, h, :n]
            k = workloads.bf16_bits(self.K[b, :, h])[p]
            v = workloads.bf16_bits(self.V[b, :, h])[p]
            if self.fp8:
                kc, ks = oracle.quantize_rows_e4m3(k)
                vc, vs = oracle.quantize_rows_e4m3(v)
                assert np.array_equal(k_st[b, h, :n], kc), (b, h)
                assert np.array_equal(v_st[b, h, :n], vc), (b, h)
                assert np.array_equal(sc[b, h, :n, 0], ks) and np.array_equal(sc[b, h, :n, 1], vs)
            else:
                assert np.array_equal(k_st[b, h, :n], k) and np.array_equal(v_st[b, h, :n], v)
            assert not k_st[b, h, n:].any() and not v_st[b, h, n:].any()

    def summary(self):
        e = np.concatenate(self.errs) if self.errs else np.zeros(1)
        assert e.mean() <= MEAN_ABS, e.mean()
        return float(e.max()), float(e.mean())
