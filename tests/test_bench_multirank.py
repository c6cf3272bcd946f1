"""The multi-rank host logic of bench.py on CPU (gloo, world size 2): the max over ranks that
the timed region reports, and the reference arm under torchrun (rank 0 alone prints one line,
the other rank exits 0 without work).  The GPU arm itself needs a GPU per rank."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, values, out):
    import torch
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    import bench

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        got = bench.max_over_ranks(values[rank], world, torch.device("cpu"))
        out[rank] = got
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    world, port = 2, _free_port()
    values = [3.25, 7.5]
    with mp.get_context("spawn").Manager() as mgr:  # no fork of a threaded process
        out = mgr.dict()
        mp.spawn(_rank_main, args=(world, port, values, out), nprocs=world, join=True)
        assert out[0] == out[1] == max(values)


def test_max_over_ranks_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.max_over_ranks(2.5, 1, None) == 2.5


@pytest.mark.timeout(300)
def test_reference_arm_under_torchrun_world2():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2", "--master-addr",
           "127.0.0.1", "--master-port", str(port), "bench.py", "--impl", "reference", "--gpus", "2",
           "--workload", "fp32_256x512_r16", "--steps", "2", "--warmup", "3"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=280, env=env)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [ln for ln in res.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, res.stdout
    rec = json.loads(lines[0])
    assert rec["impl"] == "reference" and rec["higher_is_better"] is False
    assert rec["value"] > 0 and rec["cpu_baseline"]["kind"] == "oracle"
    assert rec["e2e"]["h2d_bytes_per_step"] == 0


def test_stored_traffic_entries_name_their_sources():
    """Every stored per-launch DRAM figure names the sources of its kernel, and bench.py reports
    it only while their hash matches (a changed kernel gets traffic null until re-captured)."""
    sys.path.insert(0, ROOT)
    import bench

    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        tj = json.load(f)
    assert tj
    for key, ent in tj.items():
        assert ent["sources"] and ent["bytes_per_launch"] > 0, key
        for name in ent["sources"]:
            assert os.path.exists(os.path.join(ROOT, "paper_2512_13728_gb300", "csrc", name)), (key, name)
        assert len(ent["src_hash"]) == 12
        assert bench.sources_hash(ent["sources"]) != bench.sources_hash(ent["sources"][:-1])
