"""The multi-rank glue of bench.py (weak scaling: every rank compresses its
own trajectory, the job time is the slowest rank's) on two gloo ranks on the
CPU.  No GPU and no data-path collective are involved."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world), RANK=str(rank),
                      LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, r, lr = bench.dist_env()
        assert (w, r, lr) == (world, rank, rank)
        # every rank reports the slowest rank's time
        ms = bench.max_over_ranks(1.0 + rank * 0.5, torch.device("cpu"), w)
        # whole-job throughput counts every rank's units
        v = bench.job_throughput(w, 28, ms)
        # each rank's inputs are its own trajectory (seeded by rank)
        from paper_2603_00188_gb300 import synth
        wl = synth.trajectory(n_steps=2, gh=4, gw=5, n_text=3, hq=4, hkv=2, w=2, seed=(0, r))
        digest = float(np.asarray(wl.k, dtype=np.float64).sum())
        t = torch.tensor([digest], dtype=torch.float64)
        gathered = [torch.zeros(1, dtype=torch.float64) for _ in range(w)]
        dist.all_gather(gathered, t)
        out[rank] = (ms, v, [float(g.item()) for g in gathered])
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.start_processes(_rank_main, args=(world, port, out), nprocs=world, start_method="spawn", join=True)
        res = dict(out)
    assert set(res) == {0, 1}
    for r in range(world):
        ms, v, digests = res[r]
        assert ms == pytest.approx(1.5)
        import bench
        assert v == pytest.approx(world * bench.N_TOK * 28 / 1.5e-3)
        assert digests[0] != digests[1]      # the ranks' inputs differ
    assert res[0][2] == res[1][2]
