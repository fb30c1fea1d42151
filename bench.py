"""DMS decode benchmark on GB300: retained KV tokens read per second.

One step = one decode step of the whole model: for every layer, the fused
append + delayed eviction of the new token (all sequences, all KV heads) and the
split-K decode attention over the retained sets (GQA).  The default workload is
the 8x-compressed Qwen-R1-32B shape: 64 layers, 40 query / 8 KV heads, head_dim
128, batch 8, context 32768 (prefill 32512, then decode), window 256,
P(evict) = 0.875, 1 % of the key channels scaled x8.  The Qwen-R1-7B shape (4x)
and the others are selected with --workload.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Prints one JSON line.  `value` = retained KV tokens read per second over the
whole step (device-resident inputs, CUDA events, barrier + synchronize around K
steps, max over ranks).  `e2e` repeats it through the C ABI with the step inputs
copied from pinned host memory and the outputs copied back inside the timed
region.  `roofline` reports the decode kernel against the measured HBM copy
bandwidth.  `cpu_baseline` times the fp64 CPU oracle on a bounded sample.
Multi-GPU (torchrun): every rank runs an independent replica (weak scaling, no
collective on the data path).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads  # noqa: E402

METRIC = "retained KV tokens read/s and decode-attn µs/layer-step; % of GB300 HBM peak"
UNIT = "tokens/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
DECODE_SRCS = [os.path.join(ROOT, "paper_2506_05345_gb300", "csrc", f)
               for f in ("dms_decode.cu", "dms_ptx.cuh", "dms_internal.cuh")]
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "decode_traffic.json")
TRAFFIC_FILE_FP8 = os.path.join(ROOT, "profiles", "decode_traffic_fp8.json")
# dms_options.decode_kernel values (include/dms.h)
DECODE_KERNELS = {"tiled": 0, "simple": 1, "split": 2, "cluster": 3}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default=workloads.QWEN32B_B8_32K.name)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--dense", action="store_true", help="no evictions (CR 1) with the same shape")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--kv-fp8", action="store_true",
                    help="fp8 E4M3 page format (per-row fp32 scales)")
    ap.add_argument("--decode-kernel", default="tiled", choices=list(DECODE_KERNELS),
                    help="tiled (default: per-head clusters or the flat split), split, cluster, "
                         "simple")
    ap.add_argument("--ctas-per-sm", type=int, default=0)
    ap.add_argument("--min-pages", type=int, default=0)
    ap.add_argument("--separate", action="store_true",
                    help="append and decode as two launches instead of the fused step")
    ap.add_argument("--borrowed", action="store_true",
                    help="decision logits carried by element 0 of each group's first query head "
                         "(App. B) instead of a separate tensor")
    ap.add_argument("--prefill", action="store_true",
                    help="time the sparse prefill attention of the workload's prompt instead of "
                         "the decode step")
    ap.add_argument("--shared-prefix", action="store_true",
                    help="append the workload's shared prompt once and share its frozen pages "
                         "between the sequences")
    ap.add_argument("--prefill-kernel", default="tcgen05", choices=["tcgen05", "mma_sync"],
                    help="prefill attention kernel (with --prefill)")
    ap.add_argument("--batch", type=int, default=0,
                    help="override the batch (small cases for profiling)")
    ap.add_argument("--layers", type=int, default=0,
                    help="override the layer count (small cases for profiling)")
    return ap.parse_args()


def get_workload(args):
    wl = workloads.WORKLOADS.get(args.workload)
    if wl is None:
        for s in workloads.sweep_workloads():
            if s.name == args.workload:
                wl = s
    if wl is None:
        raise SystemExit(f"unknown workload {args.workload}")
    import dataclasses
    if args.layers > 0:
        wl = dataclasses.replace(wl, layers=args.layers)
    if args.batch > 0:
        wl = dataclasses.replace(wl, batch=args.batch)
    if args.dense:
        wl = dataclasses.replace(wl, p_evict=0.0, ragged_beta=False, name=wl.name + "-dense")
    return wl


def measured_bf16_peak():
    """Measured dense bf16 peak (TFLOP/s): the burst figure, for a kernel timed alone."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def decode_source_sha():
    """Hash of every source the decode kernel is compiled from."""
    h = hashlib.sha256()
    for path in DECODE_SRCS:
        with open(path, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def traffic_per_launch(units_per_launch, fp8=False):
    """DRAM bytes per decode launch from the committed ncu summary, scaled to this
    launch's units; None if there is none or the kernel changed since."""
    try:
        with open(TRAFFIC_FILE_FP8 if fp8 else TRAFFIC_FILE) as f:
            t = json.load(f)
    except Exception:
        return None
    if t.get("kernel_source_sha") != decode_source_sha():
        return None
    per_unit = t["dram_bytes_per_launch"] / t["units_per_launch"]
    return per_unit * units_per_launch


class Clocks:
    """nvidia-smi sampling during the timed region."""
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
            return
        t0 = time.time()
        while time.time() - t0 < 5.0 and os.path.getsize(self.path) == 0:
            time.sleep(0.01)

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 7:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[0]) for r in rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[3 + i].lower() == "active"})
        return {"sm_mhz": float(np.median(sm)) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


def check_world(gpus, world):
    """--gpus N must equal the number of ranks the launcher started (torchrun's WORLD_SIZE,
    1 without a launcher): the bench never spreads itself over GPUs it was not given."""
    if gpus != world:
        raise SystemExit(
            f"bench.py: --gpus {gpus} but {world} rank(s) were launched (WORLD_SIZE); for N > 1 "
            f"run: python -m torch.distributed.run --nnodes=1 --nproc-per-node {gpus} "
            f"--master-addr 127.0.0.1 --master-port <port> bench.py --gpus {gpus} ...")


def dist_setup(args):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    check_world(getattr(args, "gpus", world), world)
    pg = None
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() and args.impl == "ours" else "gloo"
        dist.init_process_group(backend=backend)
        pg = dist
    return world, rank, local, pg


def barrier(pg, dev=None):
    if pg is not None:
        pg.barrier()


def max_over_ranks(pg, x, dev):
    if pg is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(pg, x, dev):
    if pg is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    pg.all_reduce(t, op=pg.ReduceOp.SUM)
    return float(t.item())


def aggregate_throughput(pg, units, elapsed_ms, dev):
    """Whole-job throughput: units processed by all ranks / the slowest rank's time.

    Returns (units per second, max elapsed ms).  Each rank runs an independent replica
    (weak scaling); this reduction is the only cross-rank traffic.
    """
    t_max = max_over_ranks(pg, elapsed_ms, dev)
    total = sum_over_ranks(pg, units, dev)
    return total / (t_max * 1e-3), t_max


def replica_tag(rank):
    """Seed tag of a rank's replica: every rank draws its own batch of sequences."""
    return f"rank{rank}"


# ============================================================================ ours


def expected_retained_per_layer(wl):
    """Retained tokens of one layer at the start of decoding, in expectation:
    B * sum_h (T - p_h (T - w - 1)) (Sec. 3.1 delayed eviction; layer 0's p_h)."""
    T = wl.prefill_tokens
    p = workloads.head_evict_prob(wl, 0)
    evictable = max(0, T - wl.window - 1)
    return float(wl.batch * np.sum(T - p * evictable))


def decode_config(args, wl, world, warmup, steps):
    """The `config` object of a decode line; the GPU arm and the reference arm print the same."""
    D = wl.head_dim
    bytes_per_unit = 2 * D + 8 if args.kv_fp8 else workloads.kv_bytes_per_token_head(D)
    per_layer_mb = expected_retained_per_layer(wl) * bytes_per_unit / 1e6
    if per_layer_mb * wl.layers > 2 * 129.0:
        l2 = (f"no flush: ~{per_layer_mb:.0f} MB of retained KV per layer x {wl.layers} layers "
              "rotate, larger than the 129 MB L2")
    else:
        l2 = (f"not flushed: ~{per_layer_mb:.1f} MB of retained KV per layer x {wl.layers} "
              "layer(s) stays in the 129 MB L2 (a latency-bound shape)")
    return {"workload": wl.name, "batch_per_gpu": wl.batch, "layers": wl.layers,
            "q_heads": wl.q_heads,
            "kv_format": "fp8_e4m3 (per-row fp32 scales)" if args.kv_fp8 else "bf16",
            "kv_heads": wl.kv_heads, "head_dim": D, "window": wl.window,
            "prefill": wl.prefill_tokens,
            "timed_positions": [wl.prefill_tokens + warmup, wl.prefill_tokens + warmup + steps - 1],
            "p_evict": (None if wl.ragged_beta else wl.p_evict),
            "ragged_beta": wl.ragged_beta,
            "shared_prefix_pages": bool(getattr(args, "shared_prefix", False) and
                                        any(sh for _, sh in wl.prefill)),
            "l2": l2, "parallelism": f"replicas x{world}"}


def run_ours(args, wl, world, rank, local, pg):
    import torch

    import paper_2506_05345_gb300 as dms

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    B, L, H, G, D = wl.batch, wl.layers, wl.kv_heads, wl.gqa_group, wl.head_dim
    Hq = H * G
    K_, W_ = args.steps, args.warmup
    K2 = max(1, min(K_, 20))  # extra steps with per-kernel events (roofline durations)
    E_K, E_W = (0, 0) if args.no_e2e else (min(K_, 50), 2)
    decode_needed = max(wl.decode_steps, W_ + K_ + K2 + E_W + E_K)
    capacity = wl.prefill_tokens + decode_needed
    seed_tag = replica_tag(rank)
    cache = dms.DmsCache(layers=L, kv_heads=H, window=wl.window, capacity=capacity, batch=B,
                         ctas_per_sm=args.ctas_per_sm, min_pages_per_cta=args.min_pages,
                         kv_format=dms.DMS_KV_FP8_E4M3 if args.kv_fp8 else dms.DMS_KV_BF16,
                         decode_kernel=DECODE_KERNELS[args.decode_kernel])
    stream = torch.cuda.current_stream()

    # ---- sampled heads for the parity check and the CPU baseline (layer 0)
    rng = np.random.default_rng(workloads.stable_seed(wl.name, "sample", rank))
    n_sample = min(8, B * H)
    flat = rng.choice(B * H, size=n_sample, replace=False)
    sample = [(int(x) // H, int(x) % H) for x in flat]
    hist = {s: {"k": [], "v": [], "l": []} for s in sample}

    # ---- prefill (untimed)
    t_setup = time.time()
    # Prefill in bulk appends of at most ~2^28 elements per K / V tensor.
    chunk = max(64, (1 << 28) // (B * H * D))
    for layer in range(L):
        for i, (n, shared) in enumerate(wl.prefill):
            for c0 in range(0, n, chunk):
                nc = min(chunk, n - c0)
                tag = f"{seed_tag}prefill{i}" + (f"c{c0}" if n > chunk else "")
                if shared and args.shared_prefix and cache.layer_length(layer) == 0:
                    k, v, lg = workloads.gen_kv(wl, layer, tag, nc, dev, batch=1)
                    cache.append_shared_prefix(layer, k, v, lg)  # stored once, pages shared
                    k, v, lg = k.expand(B, -1, -1, -1), v.expand(B, -1, -1, -1), lg.expand(B, -1, -1)
                elif shared:
                    k, v, lg = workloads.gen_kv(wl, layer, tag, nc, dev, batch=1)
                    k = k.expand(B, -1, -1, -1).contiguous()
                    v = v.expand(B, -1, -1, -1).contiguous()
                    lg = lg.expand(B, -1, -1).contiguous()
                    cache.append_and_evict(layer, k, v, lg)
                else:
                    k, v, lg = workloads.gen_kv(wl, layer, tag, nc, dev)
                    cache.append_and_evict(layer, k, v, lg)
                if layer == 0 and rank == 0:
                    for (b, h) in sample:
                        hist[(b, h)]["k"].append(workloads.bf16_bits(k[b, :, h]))
                        hist[(b, h)]["v"].append(workloads.bf16_bits(v[b, :, h]))
                        hist[(b, h)]["l"].append(workloads.bf16_bits(lg[b, :, h]))
                del k, v, lg
    torch.cuda.synchronize()
    st0 = cache.stats()
    if st0["device_error"]:
        raise RuntimeError(f"device error after prefill: {st0}")
    # the kernel the fused steps launch (per-head clusters or the flat split)
    plan = cache.decode_plan(G, 0)
    plan["kernel"] = {v: k for k, v in DECODE_KERNELS.items()}[plan["kernel"]]
    kernel_name = {"cluster": "decode_cluster_kernel", "simple": "decode_simple_kernel"}.get(
        plan["kernel"], "decode_tiled_kernel")

    # ---- step inputs, resident in HBM before the timed region
    n_dev_steps = W_ + K_ + K2
    ins = []
    for s in range(n_dev_steps):
        per = []
        for layer in range(L):
            k, v, lg = workloads.gen_kv(wl, layer, f"{seed_tag}decode{s}", 1, dev)
            q = workloads.gen_q(wl, layer, f"{seed_tag}decode{s}", dev)
            if args.borrowed:  # the same decisions, carried by the borrowed neuron
                q[:, ::G, 0] = lg[:, 0]
            per.append((k, v, lg, q))
        ins.append(per)
    outs = [torch.empty((B, Hq, D), dtype=torch.bfloat16, device=dev) for _ in range(L)]

    ev_dec = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(L)] for _ in range(K2)]
    ev_app = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(L)] for _ in range(K2)]

    # The C-ABI calls of every step, marshalled before any timing (shapes were checked
    # when the tensors were made): the timed loops only call the library.
    import ctypes
    lib = dms.library()
    vp = ctypes.c_void_p
    hnd, sptr = vp(cache.handle), vp(stream.cuda_stream)

    def step_calls(layer, kp, vp_, lp, qp, op):
        """One layer's decode step as a tuple of (C function, arguments)."""
        if args.borrowed and args.separate:
            return ((lib.dms_append_and_evict_borrowed, (hnd, layer, kp, vp_, qp, 1, G, sptr)),
                    (lib.dms_decode_attention_borrowed, (hnd, layer, qp, op, G, 0.0, sptr)))
        if args.borrowed:
            return ((lib.dms_append_and_decode_borrowed,
                     (hnd, layer, kp, vp_, qp, op, G, 0.0, sptr)),)
        if args.separate:
            return ((lib.dms_append_and_evict, (hnd, layer, kp, vp_, lp, 1, sptr)),
                    (lib.dms_decode_attention, (hnd, layer, qp, op, G, 0.0, sptr)))
        return ((lib.dms_append_and_decode, (hnd, layer, kp, vp_, lp, qp, op, G, 0.0, sptr)),)
    calls = []
    for s in range(n_dev_steps):
        per = []
        for layer in range(L):
            k, v, lg, q = ins[s][layer]
            kp, vp_, lp, qp, op = (vp(t.data_ptr()) for t in (k, v, lg, q, outs[layer]))
            per.append(step_calls(layer, kp, vp_, lp, qp, op))
        calls.append(per)
    codes = []

    def do_step(s, timed_idx=None):
        for layer in range(L):
            seq = calls[s][layer]
            if len(seq) == 1:  # one launch: single-token append fused into the decode
                if timed_idx is not None:
                    ev_dec[timed_idx][layer][0].record(stream)
                fn, a = seq[0]
                codes.append(fn(*a))
                if timed_idx is not None:
                    ev_dec[timed_idx][layer][1].record(stream)
                continue
            (fa, aa), (fd, ad) = seq
            if timed_idx is not None:
                ev_app[timed_idx][layer][0].record(stream)
            codes.append(fa(*aa))
            if timed_idx is not None:
                ev_app[timed_idx][layer][1].record(stream)
                ev_dec[timed_idx][layer][0].record(stream)
            codes.append(fd(*ad))
            if timed_idx is not None:
                ev_dec[timed_idx][layer][1].record(stream)

    for s in range(W_):
        do_step(s)
    torch.cuda.synchronize()
    st_before = cache.stats()
    clocks = Clocks(local)
    if rank == 0:
        clocks.start()
    barrier(pg)
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    # Timed region: K whole steps back to back, no events between kernels (an event
    # between two kernels would serialise their programmatic overlap).
    t_start.record(stream)
    for i in range(K_):
        do_step(W_ + i)
    t_end.record(stream)
    torch.cuda.synchronize()
    barrier(pg)
    clk = clocks.stop() if rank == 0 else None
    elapsed_ms = t_start.elapsed_time(t_end)
    st_after = cache.stats()
    if st_after["device_error"]:
        raise RuntimeError(f"device error during timed steps: {st_after}")
    if any(c != 0 for c in codes):
        raise RuntimeError(f"library call failed during timed steps: {sorted(set(codes))}")
    # Second timed region: K2 further steps with CUDA events around every append
    # and decode launch, for the per-kernel durations of the roofline.
    torch.cuda.synchronize()
    for i in range(K2):
        do_step(W_ + K_ + i, timed_idx=i)
    torch.cuda.synchronize()
    st_k2 = cache.stats()
    # tokens read per step: every head reads n_h after its append; n_h grows by 0 or 1
    # per step, so the per-step total is interpolated between the two snapshots
    # (the error is below the growth over the run, < 0.2 % here).
    tok_first = st_before["total_retained"]
    tok_last = st_after["total_retained"]
    tokens_read = K_ * 0.5 * (tok_first + tok_last)
    dec_ms = [ev_dec[i][layer][0].elapsed_time(ev_dec[i][layer][1])
              for i in range(K2) for layer in range(L)]
    app_ms = ([ev_app[i][layer][0].elapsed_time(ev_app[i][layer][1])
               for i in range(K2) for layer in range(L)] if args.separate else [0.0])
    # bf16: K and V rows, 2 * 2 * D bytes; fp8: 2 * D codes and two fp32 scales
    bytes_per_unit = 2 * D + 8 if args.kv_fp8 else workloads.kv_bytes_per_token_head(D)
    if args.separate:
        # two kernels per layer-step: the decode launches' own event-bracketed durations
        units_per_launch = 0.5 * (tok_last + st_k2["total_retained"]) / L
        dec_avg_s = float(np.mean(dec_ms)) * 1e-3
        duration_source = "mean CUDA-event duration of the decode launches (second timed region)"
    else:
        # the fused kernel is the only kernel of the timed region: its average launch
        # duration is the timed region's elapsed time over its K * L launches
        units_per_launch = 0.5 * (tok_first + tok_last) / L
        dec_avg_s = elapsed_ms * 1e-3 / (K_ * L)
        duration_source = "timed region elapsed / (steps * layers); the only kernel in the region"

    value, elapsed_max_ms = aggregate_throughput(pg, tokens_read, elapsed_ms, dev)

    # ---- parity sample (layer 0, last timed step) and CPU baseline
    parity = None
    cpu_baseline = None
    if rank == 0:
        import oracle
        Gs = G
        last = n_dev_steps - 1
        for s in range(n_dev_steps):
            k, v, lg, q = ins[s][0]
            for (b, h) in sample:
                hist[(b, h)]["k"].append(workloads.bf16_bits(k[b, :, h]))
                hist[(b, h)]["v"].append(workloads.bf16_bits(v[b, :, h]))
                hist[(b, h)]["l"].append(workloads.bf16_bits(lg[b, :, h]))
        q_last = workloads.bf16_bits(ins[last][0][3])
        got = outs[0].float().cpu().numpy()
        j = wl.prefill_tokens + n_dev_steps - 1
        errs = []
        cases = []
        for (b, h) in sample:
            kk = np.concatenate(hist[(b, h)]["k"])
            vv = np.concatenate(hist[(b, h)]["v"])
            ll = np.concatenate(hist[(b, h)]["l"])
            qq = q_last[b, h * Gs:(h + 1) * Gs]
            if args.borrowed:  # the attention takes the borrowed element as 0 (App. B)
                qq = oracle.borrowed(qq, Gs)[1]
            if args.kv_fp8:  # the oracle quantises the history itself
                kk = oracle.quantize_rows_e4m3(kk)
                vv = oracle.quantize_rows_e4m3(vv)
                ref = oracle.decode_fp8(qq, *kk, *vv, ll, j, wl.window)
            else:
                ref = oracle.decode(qq, kk, vv, ll, j, wl.window)
            errs.append(np.abs(got[b, h * Gs:(h + 1) * Gs] - ref).ravel())
            cases.append((qq, kk, vv, ll, len(oracle.retained(ll, j, wl.window))))
        e = np.concatenate(errs)
        parity = {"sampled_kv_heads": len(sample), "max_abs": float(e.max()),
                  "mean_abs": float(e.mean()), "ok": bool(e.max() <= 2e-2 and e.mean() <= 2e-3)}
        # CPU oracle: repeat the sampled heads' decode until the budget is spent
        tok = 0
        calls = 0
        t0 = time.perf_counter()
        while True:
            for (qq, kk, vv, ll, n) in cases:
                if args.kv_fp8:
                    oracle.decode_fp8(qq, *kk, *vv, ll, j, wl.window)
                else:
                    oracle.decode(qq, kk, vv, ll, j, wl.window)
                tok += n
                calls += 1
            if time.perf_counter() - t0 >= args.cpu_seconds:
                break
        cpu_s = time.perf_counter() - t0
        cpu_baseline = {"value": tok / cpu_s, "unit": UNIT, "cores": 1, "kind": "oracle",
                        "sample": f"{calls} fp64 oracle decodes of sampled (layer 0, seq, KV head) "
                                  f"groups ({G} query heads each) at position {j}, "
                                  f"{cpu_s:.1f} s single-threaded"}

    # ---- end to end through the C ABI with host buffers
    # Each step's inputs (k, v, decision logits, q of every layer) sit in one pinned host slab
    # and reach the device in one copy; the step's outputs go back in one copy.  Copies run on
    # their own streams into double-buffered device slabs, so the upload of step s + 1 and the
    # download of step s overlap the kernels of the neighbouring step; every copy is inside
    # the timed region.
    e2e = None
    if E_K > 0:
        n_e = E_W + E_K
        kb, lb, qb = B * H * D * 2, B * H * 2, B * Hq * D * 2
        al = lambda x: (x + 255) // 256 * 256  # noqa: E731
        o_k, o_v, o_l, o_q = 0, al(kb), 2 * al(kb), 2 * al(kb) + al(lb)
        slab = al(o_q + qb)
        host_in = torch.empty((n_e, L, slab), dtype=torch.uint8, pin_memory=True)
        for s in range(n_e):
            for layer in range(L):
                k, v, lg = workloads.gen_kv(wl, layer, f"{seed_tag}e2e{s}", 1, dev)
                q = workloads.gen_q(wl, layer, f"{seed_tag}e2e{s}", dev)
                if args.borrowed:
                    q[:, ::G, 0] = lg[:, 0]
                row = host_in[s, layer]
                for off, t in ((o_k, k), (o_v, v), (o_l, lg), (o_q, q)):
                    b = t.reshape(-1).view(torch.uint8)
                    row[off:off + b.numel()].copy_(b.cpu())
        dev_in = [torch.empty((L, slab), dtype=torch.uint8, device=dev) for _ in range(2)]
        dev_out = [torch.empty((L, B, Hq, D), dtype=torch.bfloat16, device=dev)
                   for _ in range(2)]
        host_out = [torch.empty((L, B, Hq, D), dtype=torch.bfloat16, pin_memory=True)
                    for _ in range(2)]
        h2d = L * slab
        d2h = host_out[0].numel() * host_out[0].element_size()
        e_calls = []
        for i in range(2):
            base = dev_in[i].data_ptr()
            per = []
            for layer in range(L):
                lb0 = base + layer * slab
                kp, vp_, lp, qp = (vp(lb0 + o) for o in (o_k, o_v, o_l, o_q))
                op = vp(dev_out[i][layer].data_ptr())
                per.append(step_calls(layer, kp, vp_, lp, qp, op))
            e_calls.append(per)
        up, down = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        ev = lambda: torch.cuda.Event()  # noqa: E731
        in_ready, in_free = [ev(), ev()], [ev(), ev()]
        out_ready, out_free = [ev(), ev()], [ev(), ev()]

        def e2e_step(s, first):
            i = s & 1
            if not first[i]:
                up.wait_event(in_free[i])  # the kernels of step s - 2 have read slab i
            with torch.cuda.stream(up):
                dev_in[i].copy_(host_in[s], non_blocking=True)
            in_ready[i].record(up)
            stream.wait_event(in_ready[i])
            if not first[i]:
                stream.wait_event(out_free[i])  # step s - 2's outputs have left slab i
            for seq in e_calls[i]:
                for fn, a in seq:
                    codes.append(fn(*a))
            in_free[i].record(stream)
            out_ready[i].record(stream)
            down.wait_event(out_ready[i])
            with torch.cuda.stream(down):
                host_out[i].copy_(dev_out[i], non_blocking=True)
            out_free[i].record(down)
            first[i] = False

        first = [True, True]
        for s in range(E_W):
            e2e_step(s, first)
        torch.cuda.synchronize()
        sb = cache.stats()
        barrier(pg)
        a = torch.cuda.Event(enable_timing=True)
        z = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        up.wait_event(a)
        down.wait_event(a)
        for s in range(E_K):
            e2e_step(E_W + s, first)
        stream.wait_event(out_free[0])
        stream.wait_event(out_free[1])
        z.record(stream)
        torch.cuda.synchronize()
        barrier(pg)
        sa = cache.stats()
        if any(codes):
            raise RuntimeError(f"C ABI returned {sorted(set(codes))}")
        e_val, e_ms = aggregate_throughput(
            pg, E_K * 0.5 * (sb["total_retained"] + sa["total_retained"]), a.elapsed_time(z), dev)
        e2e = {"value": e_val, "unit": UNIT, "h2d_bytes_per_step": int(h2d),
               "d2h_bytes_per_step": int(d2h), "ms_per_step": e_ms / E_K, "steps": E_K,
               "copies": "one packed pinned H2D and one D2H per step on their own streams, "
                         "double-buffered device slabs"}

    if rank != 0:
        cache.close()
        return None

    peak, peak_kind = measured_peak()
    achieved_gbs = units_per_launch * bytes_per_unit / dec_avg_s / 1e9
    traffic = traffic_per_launch(units_per_launch, fp8=args.kv_fp8)
    res = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K_,
        "warmup": W_, "ms_per_step": elapsed_max_ms / K_, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None,
        "dtype": "fp8 E4M3 K/V codes, f16 MMA, fp32 accumulate" if args.kv_fp8 else "bf16",
        "data": "synthetic",
        "impl": "ours",
        "config": decode_config(args, wl, world, W_, K_),
        "step_mode": ("separate append + decode launches" if args.separate else
                      "fused single-token append + decode, one launch per layer") +
                     ("; decisions from element 0 of each group's first query head (App. B)"
                      if args.borrowed else ""),
        "decode_us_per_layer_step": dec_avg_s * 1e6,
        "isolated_launch_us": float(np.mean(dec_ms)) * 1e3,
        "append_us_per_layer_step": (float(np.mean(app_ms)) * 1e3 if args.separate else None),
        "retained_tokens_per_layer_step": units_per_launch,
        "compression": (wl.prefill_tokens + n_dev_steps) * B * H / units_per_launch,
        "hbm_frac_of_nominal_8tbs": achieved_gbs / NOMINAL_HBM_GBS,
        "roofline": {"kernel": kernel_name + (" (fp8 pages)" if args.kv_fp8 else "") +
                               ("" if args.separate else " (append fused)"),
                     "launch": plan,
                     "bound": "hbm", "achieved": achieved_gbs,
                     "peak": peak, "unit": "GB/s", "frac": achieved_gbs / peak,
                     "peak_kind": f"{peak_kind} copy bandwidth (read + write; the kernel only "
                                  "reads, so a fraction a little above 1 is possible)",
                     "frac_of_nominal_8tbs": achieved_gbs / NOMINAL_HBM_GBS,
                     "traffic": traffic,
                     "algorithmic_bytes_per_launch": units_per_launch * bytes_per_unit,
                     "duration": duration_source},
        "cpu_baseline": cpu_baseline,
        "e2e": e2e,
        "gpu_launches": (2 if args.separate else 1) * L * K_,
        "clocks": clk,
        "parity_sample": parity,
        "setup_s": time.time() - t_setup,
    }
    cache.close()
    return res


# ============================================================================ reference (oracle)


def run_reference(args, wl, world, rank):
    """The fp64 CPU oracle on the host cores, same workload and metric, bounded sample."""
    import oracle
    import torch
    if rank != 0:
        return None
    B, H, G, D = wl.batch, wl.kv_heads, wl.gqa_group, wl.head_dim
    rng = np.random.default_rng(workloads.stable_seed(wl.name, "refsample"))
    n_sample = 4
    flat = rng.choice(B * H, size=n_sample, replace=False)
    sample = [(int(x) // H, int(x) % H) for x in flat]
    # history of the sampled heads (layer 0), generated on the CPU with the same recipe
    sub = workloads.Workload(**{**wl.__dict__, "batch": 1, "name": wl.name})
    hist = {}
    for (b, h) in sample:
        ks, vs, ls = [], [], []
        for i, (n, _shared) in enumerate(wl.prefill):
            k, v, lg = workloads.gen_kv(sub, 0, f"ref{b}prefill{i}", n, "cpu")
            ks.append(workloads.bf16_bits(k[0, :, h]))
            vs.append(workloads.bf16_bits(v[0, :, h]))
            ls.append(workloads.bf16_bits(lg[0, :, h]))
        hist[(b, h)] = [ks, vs, ls]
    steps = args.warmup + args.steps
    per_step_s = []
    per_step_tok = []
    for s in range(steps):
        tok = 0
        t0 = time.perf_counter()
        for (b, h) in sample:
            k, v, lg = workloads.gen_kv(sub, 0, f"ref{b}decode{s}", 1, "cpu")
            q = workloads.gen_q(sub, 0, f"ref{b}decode{s}", "cpu")
            ks, vs, ls = hist[(b, h)]
            ks.append(workloads.bf16_bits(k[0, :, h]))
            vs.append(workloads.bf16_bits(v[0, :, h]))
            ls.append(workloads.bf16_bits(lg[0, :, h]))
            kk, vv, ll = np.concatenate(ks), np.concatenate(vs), np.concatenate(ls)
            j = len(ll) - 1
            qq = workloads.bf16_bits(q[0, h * G:(h + 1) * G])
            t1 = time.perf_counter()
            if getattr(args, "kv_fp8", False):  # the oracle quantises the history itself
                oracle.decode_fp8(qq, *oracle.quantize_rows_e4m3(kk),
                                  *oracle.quantize_rows_e4m3(vv), ll, j, wl.window)
            else:
                oracle.decode(qq, kk, vv, ll, j, wl.window)
            per_step_s.append(time.perf_counter() - t1)
            tok += len(oracle.retained(ll, j, wl.window))
        per_step_tok.append(tok)
    timed_s = sum(per_step_s[args.warmup * n_sample:])
    timed_tok = sum(per_step_tok[args.warmup:])
    value = timed_tok / timed_s
    return {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * timed_s / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": decode_config(args, wl, world, args.warmup, args.steps),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": f"{n_sample} sampled (layer 0, seq, KV head) groups per step, "
                                       f"{G} query heads each, fp64 single-threaded"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


PREFILL_METRIC = "sparse DMS prefill attention TFLOP/s (4*128 flop per visible (query head, key) pair)"


def prefill_pairs(lg, window):
    """Visible (query, key) pairs per KV head, summed: sum_j |R_j| with
    |R_j| = j + 1 - #{i <= j - w - 1 : alpha_i = 1} (alpha_i = [logit_i > 0])."""
    import torch
    B, P, H = lg.shape
    alpha = (lg.float() > 0).to(torch.int64)           # NaN keeps, +inf evicts
    cum = torch.cumsum(alpha, dim=1)                   # [B, P, H]
    out_sum = cum[:, :max(0, P - window - 1)].sum().item()
    return B * H * P * (P + 1) // 2 - out_sum


def run_prefill(args, wl, world, rank, local, pg):
    """One step = the sparse prefill attention (pack pre-pass + attention kernel) of the
    workload's whole prompt, for every layer in the rotation."""
    import ctypes

    import torch

    import paper_2506_05345_gb300 as dms

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    B, H, G, D = wl.batch, wl.kv_heads, wl.gqa_group, wl.head_dim
    P, w, Hq = wl.prefill_tokens, wl.window, wl.kv_heads * wl.gqa_group
    L = max(1, min(args.layers or 2, wl.layers))
    K_, W_ = args.steps, args.warmup
    seed_tag = replica_tag(rank)
    ins = []
    for layer in range(L):
        k, v, lg = workloads.gen_kv(wl, layer, f"{seed_tag}prompt", P, dev)
        g = torch.Generator(device=dev).manual_seed(workloads.stable_seed(wl.name, layer, seed_tag, "pq"))
        q = torch.randn((B, P, Hq, D), generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
        if args.borrowed:
            q[:, :, ::G, 0] = lg
        ins.append((q, k, v, lg))
    code, ws_bytes = dms.dms_prefill_workspace_bytes(B, P, H)
    if code != dms.DMS_OK:
        raise RuntimeError(f"dms_prefill_workspace_bytes: {code}")
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    outs = [torch.empty((B, P, Hq, D), dtype=torch.bfloat16, device=dev) for _ in range(L)]
    pairs = [prefill_pairs(lg, w) for (_, _, _, lg) in ins]
    flops_per_step = sum(pairs) * G * 4 * D
    lib = dms.library()
    vp = ctypes.c_void_p
    sptr = vp(torch.cuda.current_stream().cuda_stream)
    kernel = dms.DMS_PREFILL_TCGEN05 if args.prefill_kernel == "tcgen05" else dms.DMS_PREFILL_MMA_SYNC
    calls = []
    for layer in range(L):
        q, k, v, lg = ins[layer]
        calls.append((lib.dms_prefill_attention_ex,
                      (vp(q.data_ptr()), vp(k.data_ptr()), vp(v.data_ptr()),
                       None if args.borrowed else vp(lg.data_ptr()), B, P, H, G, w, 0, kernel,
                       0.0, vp(ws.data_ptr()), ws_bytes, vp(outs[layer].data_ptr()), sptr)))
    codes = []

    def step():
        for fn, a in calls:
            codes.append(fn(*a))

    for _ in range(W_):
        step()
    torch.cuda.synchronize()
    clocks = Clocks(local)
    barrier(pg, dev)
    clocks.start()
    a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record()
    for _ in range(K_):
        step()
    z.record()
    torch.cuda.synchronize()
    clk = clocks.stop()
    barrier(pg, dev)
    if any(codes):
        raise RuntimeError(f"C ABI returned {sorted(set(codes))}")
    code, err = dms.dms_prefill_device_error(ws.data_ptr(), None)
    if code != dms.DMS_OK or err != dms.DMS_OK:
        raise RuntimeError(f"prefill device error {err}")
    ms = a.elapsed_time(z)
    ms_max = max_over_ranks(pg, ms, dev)
    t_layer = ms_max / 1e3 / (K_ * L)
    value = sum_over_ranks(pg, flops_per_step * K_, dev) / (ms_max / 1e3) / 1e12
    if rank != 0:
        return None
    # ---- parity sample (layer 0) and CPU baseline: the fp64 oracle on sampled rows
    import oracle
    q, k, v, lg = ins[0]
    rng = np.random.default_rng(workloads.stable_seed(wl.name, "prefill-sample"))
    rows = {(int(rng.integers(B)), int(rng.integers(P)), int(rng.integers(H))) for _ in range(24)}
    rows |= {(0, P - 1, 0), (B - 1, 0, H - 1)}
    rows = sorted(rows)
    got = outs[0]
    errs, cases = [], []
    for b, j, h in rows:
        qq = workloads.bf16_bits(q[b, j, h * G:(h + 1) * G])
        if args.borrowed:
            qq = oracle.borrowed(qq, G)[1]
        kk, vv = workloads.bf16_bits(k[b, :, h]), workloads.bf16_bits(v[b, :, h])
        ll = workloads.bf16_bits(lg[b, :, h])
        ref = oracle.decode(qq, kk, vv, ll, j, w)
        errs.append(np.abs(got[b, j, h * G:(h + 1) * G].float().cpu().numpy() - ref).ravel())
        cases.append((qq, kk, vv, ll, j, len(oracle.retained(ll, j, w))))
    e = np.concatenate(errs)
    parity = {"sampled_rows": len(rows), "max_abs": float(e.max()), "mean_abs": float(e.mean()),
              "ok": bool(e.max() <= 2e-2 and e.mean() <= 2e-3)}
    flops_cpu, t0, n = 0, time.time(), 0
    while time.time() - t0 < args.cpu_seconds or n == 0:
        qq, kk, vv, ll, j, nr = cases[n % len(cases)]
        oracle.decode(qq, kk, vv, ll, j, w)
        flops_cpu += nr * G * 4 * D
        n += 1
    cpu_s = time.time() - t0
    peak, peak_kind = measured_bf16_peak()
    achieved = flops_per_step / L / t_layer / 1e12
    dense_pairs = B * H * P * (P + 1) // 2
    return {
        "metric": PREFILL_METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
        "steps": K_, "warmup": W_, "ms_per_step": ms_max / K_, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "impl": "ours",
        "config": {"workload": wl.name + "-prompt", "batch_per_gpu": B, "prompt_tokens": P,
                   "q_heads": Hq, "kv_heads": H, "head_dim": D, "window": w,
                   "p_evict": 0.0 if args.dense else wl.p_evict, "layers": L,
                   "decisions": "borrowed query neuron (App. B)" if args.borrowed else "logit tensor",
                   "l2": "no flush: each layer's prompt (q, k, v, out, workspace) is several GB",
                   "parallelism": f"replicas x{world}"},
        "us_per_layer": t_layer * 1e6,
        "prompt_tokens_per_s_per_layer": B * P / t_layer,
        "visible_pairs_per_layer": pairs[0], "dense_causal_pairs_per_layer": dense_pairs,
        "sparsity": 1.0 - pairs[0] / dense_pairs,
        "roofline": {"kernel": ("prefill_tc_kernel (tcgen05)" if kernel == dms.DMS_PREFILL_TCGEN05
                               else "prefill_attn_kernel (mma.sync)") + " + pack pre-pass",
                     "bound": "tensor",
                     "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "peak_kind": f"{peak_kind} dense bf16 (burst)",
                     "traffic": None,
                     "algorithmic_flops_per_layer": flops_per_step / L,
                     "duration": "timed region elapsed / (steps * layers)"},
        "cpu_baseline": {"value": flops_cpu / cpu_s / 1e12, "unit": "TFLOP/s", "cores": 1,
                         "kind": "oracle",
                         "sample": f"{n} fp64 oracle decodes of {len(cases)} sampled (sequence, "
                                   f"query, KV head) rows of layer 0, {cpu_s:.1f} s single-threaded"},
        "e2e": None, "gpu_launches": 3 * L * K_, "clocks": clk, "parity_sample": parity,
    }


def main():
    args = parse()
    wl = get_workload(args)
    world, rank, local, pg = dist_setup(args)
    if args.impl == "reference":
        res = run_reference(args, wl, world, rank)
    elif args.prefill:
        res = run_prefill(args, wl, world, rank, local, pg)
    else:
        res = run_ours(args, wl, world, rank, local, pg)
    if rank == 0 and res is not None:
        print(json.dumps(res), flush=True)
    if pg is not None:
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
