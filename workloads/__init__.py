"""Seeded synthetic inputs for DMS decode, shaped like the paper's workloads.

This module draws random numbers and nothing else: it holds none of the
method's arithmetic (no decisions, no retained sets, no attention).  Both the
CUDA path and the CPU oracle are fed from it; neither side imports the other.

The paper evaluates on reasoning benchmarks (AIME 24, MATH 500, GPQA,
LiveCodeBench; Sec. 4) with retrofitted Qwen-R1 / Llama models.  Neither the
data nor the weights are used here: these tensors stand in for them with the
models' attention shapes (Sec. 4, GQA).

Recipe (per (workload, layer, phase, step) a fresh ``torch.Generator`` seeded
from a stable hash):
  * q, k, v ~ N(0, 1) rounded to bf16 (round-to-nearest-even).
  * Optional outlier channels in K: a seeded 1 % of the head_dim channels
    (rounded up to 2) are scaled x8 for every head and token.
  * Decision logits ~ N(mu_h, 1) rounded to bf16, with mu_h = Phi^-1(p_h) so
    that P(logit > 0) = p_h, the per-head eviction probability.  p_h = 0 is the
    no-eviction (CR 1) case: all logits are -1.
  * Ragged heads: p_h = 1 - 0.625 (1 - b_h), b_h ~ Beta(8, 2) per (layer, KV
    head), which makes the mean retained fraction 1/8 (8x aggregate
    compression) and retained lengths strongly uneven across heads.
"""
from __future__ import annotations

import dataclasses
import statistics
import zlib
from typing import Optional, Sequence

import numpy as np

HEAD_DIM = 128


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape of one synthetic decode workload (one replica, one GPU)."""
    name: str
    batch: int
    layers: int
    q_heads: int
    kv_heads: int
    window: int
    # Bulk appends before decoding: list of (token count, shared_across_batch).
    prefill: tuple
    decode_steps: int
    p_evict: float = 0.875          # per-head eviction probability (uniform heads)
    ragged_beta: bool = False       # draw p_h from the Beta(8,2) recipe instead
    k_outliers: bool = False
    head_dim: int = HEAD_DIM
    seed: int = 1234

    @property
    def gqa_group(self) -> int:
        return self.q_heads // self.kv_heads

    @property
    def context(self) -> int:
        return sum(n for n, _ in self.prefill) + self.decode_steps

    @property
    def prefill_tokens(self) -> int:
        return sum(n for n, _ in self.prefill)


def _wl(name, B, L, Hq, Hkv, prefill, steps, p, **kw) -> Workload:
    return Workload(name=name, batch=B, layers=L, q_heads=Hq, kv_heads=Hkv, window=256,
                    prefill=tuple(prefill), decode_steps=steps, p_evict=p, **kw)


# The five shapes (names say what they are, with their sizes).
LLAMA_B1_4K = _wl("llama-gqa32x8-b1-ctx4352-p0.875", 1, 1, 32, 8, [(4096, False)], 256, 0.875)
QWEN7B_B64_8K = _wl("qwen-r1-7b-b64-ctx8192-p0.75-28l", 64, 28, 28, 4, [(7936, False)], 256, 0.75)
QWEN32B_B8_32K = _wl("qwen-r1-32b-b8-ctx32768-p0.875-64l-koutlier", 8, 64, 40, 8,
                     [(32512, False)], 256, 0.875, k_outliers=True)
QWEN32B_THREADS32 = _wl("qwen-r1-32b-32threads-prefix2048+16384-beta82-64l", 32, 64, 40, 8,
                        [(2048, True), (16128, False)], 256, 0.875, ragged_beta=True)

WORKLOADS = {w.name: w for w in (LLAMA_B1_4K, QWEN7B_B64_8K, QWEN32B_B8_32K, QWEN32B_THREADS32)}


def sweep_workloads(max_bytes: float = 180e9) -> list:
    """Compression {1,2,4,8}x x batch {1,16,64,256} x context {4K,16K,64K}, Qwen-R1-32B dims.

    Layers per point = min(64, floor(max_bytes / dense per-layer KV bytes)); points whose
    single layer does not fit are dropped.
    """
    out = []
    for cr in (1, 2, 4, 8):
        p = 0.0 if cr == 1 else 1.0 - 1.0 / cr
        for B in (1, 16, 64, 256):
            for ctx in (4096, 16384, 65536):
                per_layer = B * 8 * ctx * HEAD_DIM * 2 * 2
                L = int(min(64, max_bytes // per_layer))
                if L < 1:
                    continue
                out.append(_wl(f"sweep-cr{cr}-b{B}-ctx{ctx}", B, L, 40, 8,
                               [(ctx - 256, False)], 256, p))
    return out


def stable_seed(*parts) -> int:
    """Stable 63-bit seed from any printable parts (same on every machine)."""
    h = zlib.crc32("|".join(str(p) for p in parts).encode())
    h2 = zlib.adler32("#".join(str(p) for p in parts).encode())
    return ((h << 31) ^ h2) & ((1 << 63) - 1)


def head_evict_prob(wl: Workload, layer: int) -> np.ndarray:
    """Per-KV-head eviction probability p_h for one layer (float64, [kv_heads])."""
    if wl.ragged_beta:
        rng = np.random.default_rng(stable_seed(wl.seed, wl.name, layer, "beta"))
        b = rng.beta(8.0, 2.0, size=wl.kv_heads)
        return 1.0 - 0.625 * (1.0 - b)
    return np.full(wl.kv_heads, float(wl.p_evict))


def logit_means(p: Sequence[float]) -> Optional[np.ndarray]:
    """mu_h = Phi^-1(p_h); None when p_h = 0 for all heads (the all -1 CR-1 case)."""
    p = np.asarray(p, dtype=np.float64)
    if np.all(p <= 0.0):
        return None
    nd = statistics.NormalDist()
    return np.array([nd.inv_cdf(min(max(x, 1e-9), 1 - 1e-9)) if x > 0 else -8.0 for x in p])


def outlier_channels(wl: Workload) -> np.ndarray:
    """Seeded K outlier channels: ceil(1 % of head_dim), at least 2."""
    rng = np.random.default_rng(stable_seed(wl.seed, wl.name, "outliers"))
    n = max(2, int(np.ceil(0.01 * wl.head_dim)))
    return np.sort(rng.choice(wl.head_dim, size=n, replace=False))


def _gen(device, seed):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def gen_kv(wl: Workload, layer: int, phase: str, n_tokens: int, device="cpu",
           batch: Optional[int] = None, p_override=None):
    """k, v [B, n, Hkv, D] bf16 and decision logits [B, n, Hkv] bf16 for one append.

    ``phase`` names the append (e.g. "prefill0", "decode17"); ``batch`` overrides
    the workload batch (used for a shared prefix drawn once with batch 1).
    """
    import torch
    B = wl.batch if batch is None else batch
    Hkv, D = wl.kv_heads, wl.head_dim
    g = _gen(device, stable_seed(wl.seed, wl.name, layer, phase))
    k = torch.randn((B, n_tokens, Hkv, D), generator=g, device=device, dtype=torch.float32)
    if wl.k_outliers:
        ch = torch.as_tensor(outlier_channels(wl), device=device)
        k[..., ch] *= 8.0
    k = k.to(torch.bfloat16)
    v = torch.randn((B, n_tokens, Hkv, D), generator=g, device=device,
                    dtype=torch.float32).to(torch.bfloat16)
    p = head_evict_prob(wl, layer) if p_override is None else np.asarray(p_override, dtype=float)
    mu = logit_means(p)
    if mu is None:
        logit = torch.full((B, n_tokens, Hkv), -1.0, device=device, dtype=torch.bfloat16)
    else:
        z = torch.randn((B, n_tokens, Hkv), generator=g, device=device, dtype=torch.float32)
        logit = (z + torch.as_tensor(mu, device=device, dtype=torch.float32)).to(torch.bfloat16)
    return k, v, logit


def gen_q(wl: Workload, layer: int, phase: str, device="cpu", batch: Optional[int] = None):
    """q [B, Hq, D] bf16 for one decode step."""
    import torch
    B = wl.batch if batch is None else batch
    g = _gen(device, stable_seed(wl.seed, wl.name, layer, phase, "q"))
    return torch.randn((B, wl.q_heads, wl.head_dim), generator=g, device=device,
                       dtype=torch.float32).to(torch.bfloat16)


def bf16_bits(t) -> np.ndarray:
    """Host uint16 view of a bf16 torch tensor (copies to host if needed)."""
    import torch
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def kv_bytes_per_token_head(head_dim: int = HEAD_DIM, elem_bytes: int = 2) -> int:
    """Algorithmic bytes read per retained token, per KV head, per layer: K + V rows.

    This is the unit of the paper's KV-read model (App. H: 4 * d_kv bytes per token
    and layer at 2 bytes per element, d_kv = kv_heads * head_dim), i.e. 512 B at
    head_dim 128.
    """
    return 2 * head_dim * elem_bytes
