"""Multi-GPU runs of bench.py are replicas: each rank runs the whole layer
stack on its own GPU with no data-path collective, and the job's throughput
is all ranks' tokens over the slowest rank's time.  These tests run that
host logic (and the reference arm's rank handling) as two gloo ranks on the
CPU."""
import io
import json
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, results):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", init_method="tcp://127.0.0.1:%d" % port, rank=rank, world_size=world)
    import bench
    r, w, _ = bench.dist_env()
    # rank r took 1 + r seconds for its 100 tokens
    value, slowest = bench.replica_throughput(100, 1.0 + r, w, "cpu")

    class Args:
        workload, batch, seed, p, steps, warmup, gpus = "tiny_relu_f32", 2, 0, 0.7, 2, 1, world
        pool, no_flush = 64, False

    out = io.StringIO()
    with redirect_stdout(out):
        bench.run_reference(Args())
    results[rank] = (r, w, value, slowest, out.getvalue())
    dist.destroy_process_group()


def bench_workload(name):
    sys.path.insert(0, ROOT)
    from paper_2605_28283_gb300 import workloads as wl
    return wl.WORKLOADS[name]


def test_two_replicas_report_all_tokens_over_the_slowest_rank():
    import torch.multiprocessing as mp
    pytest.importorskip("torch.distributed")
    with mp.get_context("spawn").Manager() as m:  # no fork of this (multi-threaded) process
        results = m.dict()
        mp.spawn(_rank_main, args=(2, _free_port(), results), nprocs=2, join=True)
        res = dict(results)
    for rank in (0, 1):
        r, w, value, slowest, out = res[rank]
        assert (r, w) == (rank, 2)
        assert slowest == 2.0 and value == pytest.approx(100.0)  # 2 ranks x 100 tokens / 2 s
    # the reference arm runs and prints on rank 0 only
    lines = [l for l in res[0][4].splitlines() if l.startswith("{")]
    assert len(lines) == 1
    rec = json.loads(lines[0])
    assert rec["impl"] == "reference" and rec["cpu_baseline"]["kind"] == "oracle" and rec["value"] > 0
    # the reference arm states its host cores and prints the GPU arm's config dict
    assert {"cpu_count", "affinity_cores", "omp_threads"} <= set(rec["cpu_baseline"])
    import bench
    assert rec["config"] == bench.config_dict(bench_workload("tiny_relu_f32"), 2, 0.7, 64, 2, False)
    assert res[1][4].strip() == ""
