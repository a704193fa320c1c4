"""The N > 1 bench path on CPU: two gloo ranks, each with its own replica
workload, and the max-over-ranks timing reduction (no collective is on the
data path; the archive shards by (sequence, layer) stream)."""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        import synth
        cfg = bench.rank_workload(rank)
        # this rank's first head vector: a replica of its own
        x = synth.kv_elements(cfg, 0, 0, 0, 0, np.arange(4)).astype(np.float64)
        # timings: rank r takes (r + 1) ms, its e2e 10 - r ms
        got = bench.max_over_ranks([rank + 1.0, 10.0 - rank], "cpu")
        dist.barrier()
        q.put((rank, cfg.cfg_id, x.tolist(), got))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_replicas_and_max_timing():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = {}
    for _ in range(world):
        rank, cid, x, got = q.get(timeout=120)
        out[rank] = (cid, x, got)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    import synth
    assert out[0][0] == synth.CFG3.cfg_id and out[1][0] == synth.CFG3.cfg_id + 1000
    assert out[0][1] != out[1][1]                          # each rank archives its own data
    for r in range(world):
        assert out[r][2] == [2.0, 10.0]                    # the job's time is the slowest rank's
