"""The bench's multi-rank logic on CPU (two gloo ranks, no GPU): every rank
replays its own streams (distinct seeds, distinct data), the job time is the
slowest rank's, the whole-job rate counts every rank's units; under torchrun
the reference arm runs on rank 0 only."""
import os
import socket
import subprocess
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def rank_main(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    import crc_synth as S
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        ms = bench.max_over_ranks(3.0 + 2.0 * rank, world, "cpu")   # ranks took 3 and 5 ms
        rate = bench.job_rate(1000, world, ms)
        w = S.TINY.with_(B=1, T=4)
        h = S.hidden(w, seed=bench.rank_seed(rank))
        digest = torch.tensor([float(np.asarray(h, dtype=np.float64).sum())], dtype=torch.float64)
        seen = [torch.zeros(1, dtype=torch.float64) for _ in range(world)]
        dist.all_gather(seen, digest)
        dist.barrier()
        np.save(os.path.join(out_dir, f"rank{rank}.npy"),
                np.array([ms, rate] + [float(x.item()) for x in seen]))
    finally:
        dist.destroy_process_group()


def test_two_ranks_slowest_rank_and_own_streams(tmp_path):
    import torch.multiprocessing as mp
    port = free_port()
    mp.start_processes(rank_main, args=(2, port, str(tmp_path)), nprocs=2, start_method="spawn")
    r0, r1 = (np.load(tmp_path / f"rank{r}.npy") for r in range(2))
    assert r0[0] == r1[0] == 5.0                        # the slowest rank's time everywhere
    assert r0[1] == r1[1] == pytest.approx(2 * 1000 / 0.005)
    assert r0[2] != r0[3]                               # different streams per rank
    assert list(r0[2:]) == list(r1[2:])


def test_reference_arm_runs_on_rank_zero_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--gpus", "2", "--steps", "1", "--warmup", "1"],
                       capture_output=True, text=True, env=env, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == ""
