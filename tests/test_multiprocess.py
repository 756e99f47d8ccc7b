"""The N > 1 path of bench.py on CPU with gloo ranks (world size 2): each rank
decodes its own batch (weak scaling, nothing exchanged on the data path), the
step time is the max over ranks, the rate counts every rank's pixels, and the
reference arm prints one line from rank 0 only."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    from paper_2609_09020_gb300 import workloads as wk
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    wl = bench.shard_workload(wk.WORKLOADS["c5"], rank)
    ms = bench.max_over_ranks(0.8 + 0.3 * rank, world)       # rank 1 is the slower one
    el = bench.max_over_ranks(2.0 - rank, world)
    gathered = [None] * world
    dist.all_gather_object(gathered, wl.seeds)
    if rank == 0:
        q.put((ms, el, gathered, bench.whole_job_rate(64 * 512 * 768, world, ms)))
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_and_reduce():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    ms, el, seeds, rate = q.get(timeout=5)
    assert ms == pytest.approx(1.1) and el == pytest.approx(2.0)
    assert len(seeds[0]) == len(seeds[1]) == 64 and not set(seeds[0]) & set(seeds[1])
    assert tuple(seeds[0]) == tuple(range(100, 164))
    assert rate == pytest.approx(2 * 64 * 512 * 768 / 1.1e-3 / 1e6)


def test_reference_arm_under_torchrun_two_ranks():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--workload", "c1", "--steps", "1",
           "--warmup", "3", "--ref-step-s", "0.2"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    sys.path.insert(0, ROOT)
    import bench
    # the same metric, unit and direction as our arm, on the named workload
    assert (d["metric"], d["unit"], d["higher_is_better"]) == (bench.METRIC, bench.UNIT, True)
    assert d["config"]["workload"].startswith("c1: 1 x 256x256")
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["cpu_baseline"]["cores"] >= 1 and "c1" in d["cpu_baseline"]["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
    assert d["ms_per_step"] >= 0.9 * 200  # one step is a bounded sample of 0.2 s
