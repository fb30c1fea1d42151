"""The multi-rank host logic of bench.py on CPU: two gloo ranks on 127.0.0.1.

Each rank runs an independent replica (weak scaling, no collective on the data path); the only
cross-rank traffic is the timing reduction.  Checks: process-group set-up from the launcher's
environment, max-over-ranks time, whole-job throughput = units of all ranks / slowest time,
distinct replica seeds, and that only rank 0 runs (and prints) the reference arm.
"""
import os
import socket
import types

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    w, r, local, pg = bench.dist_setup(types.SimpleNamespace(impl="reference"))
    try:
        elapsed_ms = [4.0, 10.0][rank]
        units = [1000.0, 3000.0][rank]
        value, t_max = bench.aggregate_throughput(pg, units, elapsed_ms, "cpu")
        bench.barrier(pg)
        ref = bench.run_reference(types.SimpleNamespace(warmup=1, steps=1), None, w, r) \
            if r != 0 else "skipped-on-rank0"
        q.put((r, w, value, t_max, bench.replica_tag(r), ref))
    finally:
        pg.destroy_process_group()


def test_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, w0, v0, t0, tag0, _), (r1, w1, v1, t1, tag1, ref1) = out
    assert (r0, r1) == (0, 1) and w0 == w1 == 2
    assert t0 == t1 == 10.0                     # max over ranks
    assert v0 == v1 == pytest.approx(4000.0 / 10e-3)  # all units / slowest time
    assert tag0 != tag1                         # independent replicas
    assert ref1 is None                         # the reference arm runs on rank 0 only


def test_gpus_flag_must_match_the_launched_ranks():
    """--gpus N without N launched ranks is an error, not a silent one-GPU run."""
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    import bench
    bench.check_world(1, 1)
    bench.check_world(2, 2)
    with pytest.raises(SystemExit):
        bench.check_world(8, 1)
    env = {k: v for k, v in os.environ.items() if k not in ("WORLD_SIZE", "RANK", "LOCAL_RANK")}
    run = subprocess.run([sys.executable, "bench.py", "--gpus", "2", "--impl", "reference",
                          "--steps", "1", "--warmup", "1"], cwd=root, env=env,
                         capture_output=True, text=True, timeout=300)
    assert run.returncode != 0
    assert "--gpus 2 but 1 rank(s)" in run.stderr
    assert not [ln for ln in run.stdout.splitlines() if ln.startswith("{")]
