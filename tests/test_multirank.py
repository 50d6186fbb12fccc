"""The N > 1 path of bench.py on CPU ranks (gloo, world size 2, 127.0.0.1): the job time is
the slowest rank's, the rate counts every rank's fits, and under torchrun the reference arm
runs on rank 0 only (the other ranks exit 0 without work or output)."""
import importlib.util
import os
import socket
import subprocess
import sys

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        b = _bench()
        # rank r took 10 + 5 r ms: every rank must see the slowest, 15 ms
        got = b.max_over_ranks(10.0 + 5.0 * rank, dist, "cpu")
        dist.barrier()
        with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
            f.write(repr(got))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_two_gloo_ranks(tmp_path):
    world = 2
    mp.spawn(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    for r in range(world):
        assert float((tmp_path / f"rank{r}.txt").read_text()) == 15.0


def test_single_rank_and_rate():
    b = _bench()
    assert b.max_over_ranks(3.5, None, "cpu") == 3.5
    # two ranks, 5 fits of 8 iterations each, slowest rank 1 s: 80 iterations/s
    assert b.whole_job_rate(2, 5, 8, 1000.0) == 80.0
    assert b.whole_job_rate(1, 10, 8, 500.0) == 160.0


def test_reference_arm_non_zero_rank_exits_quietly():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--steps", "1", "--warmup", "0"],
                         env=env, capture_output=True, text=True, timeout=300)
    assert out.returncode == 0, out.stderr
    assert out.stdout.strip() == ""
