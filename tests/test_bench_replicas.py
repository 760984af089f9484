"""bench.py's multi-process path on CPU: world size 2 over gloo (127.0.0.1).
Each rank runs an independent replica of the workload; the step time is
reduced with a max over ranks and the value counts the work of every rank.
Only the host-side plumbing is exercised here (no GPU)."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    w, r, l = bench.dist_setup()
    assert (w, r, l) == (world, rank, rank)
    bench.barrier(w)
    t = bench.reduce_max(1.5 + rank, w)       # per-rank step times 1.5 and 2.5 ms
    # a replica run measures the step only: no projection (nor the other
    # configurations or the CPU baseline), whatever the flags say
    extras = bench.plan_extras(bench.parse_args([]), w, r, "stress14b")
    assert extras == {"projection": False, "per_config": False, "cpu_baseline": False}, extras
    try:
        bench.time_projection(None, None, None, None, None, 0.0, w)
        reached = True
    except RuntimeError:
        reached = False
    assert not reached
    out[rank] = t
    import torch.distributed as dist
    dist.destroy_process_group()


def test_two_replicas_take_the_max_step_time():
    port = _free_port()
    out = mp.Manager().dict()
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    assert out[0] == pytest.approx(2.5) and out[1] == pytest.approx(2.5)


def test_single_gpu_runs_the_extras():
    import bench
    args = bench.parse_args([])
    assert bench.plan_extras(args, 1, 0, "stress14b") == {
        "projection": True, "per_config": True, "cpu_baseline": True}
    args = bench.parse_args(["--no-projection", "--no-per-config", "--no-cpu-baseline"])
    assert not any(bench.plan_extras(args, 1, 0, "stress14b").values())
    assert bench.DEFAULT_WORKLOAD == "stress14b"


def test_config_describes_replicas():
    import bench
    from paper_2609_22283_gb300 import inputs as I
    c = bench.config_of(I.WORKLOADS["prog4"], 4)
    assert c["parallelism"] == "4 independent replicas"
    assert c["workload"] == "prog4" and c["kv_tokens_per_node"] == [32760] * 4
    assert bench.attn_flops(I.WORKLOADS["clean1"]) == pytest.approx(4 * 4680 * 18720 * 128 * 12)
