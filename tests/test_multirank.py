"""The multi-GPU path of bench.py on CPU: two gloo ranks (world size 2).

Pairs are independent, so each rank decodes its own batch and the only
collectives are the barrier and the maximum over ranks of the timed region.
These tests check the host logic of that path: distinct inputs per rank, the
maximum reduction, the whole-job throughput, and that the reference arm runs
on rank 0 only.
"""
import hashlib
import io
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import bench
    import synth
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        cfg = synth.config("tiny")
        lat, mask, labels = bench.decode_inputs(cfg, bench.rank_seed_offset(rank))
        digest = hashlib.sha256(lat.tobytes() + mask.tobytes() + labels.tobytes()).hexdigest()
        digests = [None] * world
        dist.all_gather_object(digests, digest)
        mx = bench.max_over_ranks([1.0 + rank, 10.0 - rank, 5.0], "cpu")
        dist.barrier()
        # the reference arm prints only on rank 0; the others return at once
        args = type("A", (), {"warmup": 0, "steps": 1, "gpus": world, "select": "least_similar"})()
        out = io.StringIO()
        if rank != 0:
            with redirect_stdout(out):
                bench.run_reference(args, cfg, plan=None)
        q.put((rank, digests, mx, out.getvalue()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_inputs_and_reduce_timings():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    results = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    by_rank = dict((r[0], r) for r in results)
    digests = by_rank[0][1]
    assert digests == by_rank[1][1] and digests[0] != digests[1]     # each rank its own batch
    for r in range(world):
        assert by_rank[r][2] == [2.0, 10.0, 5.0]                      # maximum over ranks
    assert by_rank[1][3] == ""                                        # reference arm silent off rank 0


def test_job_throughput_counts_all_ranks():
    import bench
    assert bench.job_images_per_s(1, 32, 5, 1000.0) == pytest.approx(160.0)
    assert bench.job_images_per_s(4, 32, 5, 1000.0) == pytest.approx(640.0)
    assert bench.rank_seed_offset(0) != bench.rank_seed_offset(1)
