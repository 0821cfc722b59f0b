"""The N > 1 bench path on CPU: gloo ranks agree on the maximum step time.

bench.py runs one independent replica per GPU (the path has no exchange
step) and reports the slowest rank's step time; this checks that reduction
with world size 2 over gloo, without a GPU.
"""

import os
import socket

import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    w, r, local = bench.dist_env()
    assert (w, r, local) == (world, rank, rank)
    bench.barrier(world)
    out[rank] = bench.reduce_max(1.5 + 2.0 * rank, world)
    dist.destroy_process_group()


def test_reduce_max_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    assert dict(out) == {0: 3.5, 1: 3.5}


def test_single_rank_is_identity():
    import bench
    assert bench.reduce_max(4.25, 1) == 4.25


def _reference_run(rank: int, world: int):
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = {**os.environ, "RANK": str(rank), "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)}
    p = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config", "tiny", "--steps", "2",
                        "--warmup", "0", "--reference-step-seconds", "0.3"],
                       cwd=root, env=env, capture_output=True, text=True, timeout=600)
    lines = [json.loads(x) for x in p.stdout.splitlines() if x.startswith("{")]
    return p.returncode, lines


def test_reference_arm_runs_on_rank_zero_only():
    """Under two ranks the oracle arm runs once: rank 0 prints the line, the
    other rank exits 0 without work; the oracle's throughput is its own
    (tokens per step over seconds per step), not multiplied by the rank count."""
    rc1, lines1 = _reference_run(1, 2)
    assert rc1 == 0 and lines1 == []
    rc0, lines0 = _reference_run(0, 2)
    assert rc0 == 0 and len(lines0) == 1
    line = lines0[0]
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["value"] == line["cpu_baseline"]["value"] == line["e2e"]["value"]
    # value: the step's tokens over the step time extrapolated from the
    # measured samples (ms_per_step is the measured sample time per step)
    per_step = line["config"]["tokens_per_step"] / (line["extrapolated_full_step_ms"] / 1e3)
    assert abs(line["value"] - per_step) <= 0.01 * per_step
    assert line["extrapolated"] is True and line["ms_per_step"] > 0
