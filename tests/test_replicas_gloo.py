"""The bench's multi-GPU path on CPU: the step shards by module with no
exchange, so with N > 1 each rank owns every N-th module and steps only
those; the job's time is the maximum over ranks (barrier and all-reduce MAX,
here over gloo, world size 2) and the job's value is ms per full-model step
(the slowest shard's step plus its refresh amortised over 200 steps); the
reference arm runs on rank 0 only and the other ranks exit without output."""

import io
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    # rank r measured 10 + 5 r ms: the job takes the slowest replica
    t = bench.job_time_ms(10.0 + 5.0 * rank, world)
    dist.barrier()
    # the reference arm: rank 0 alone works and prints
    buf = io.StringIO()
    with redirect_stdout(buf):
        if rank != 0:
            bench.run_reference(type("A", (), dict(workload="llama7b_layer", steps=1, warmup=0, gpus=world,
                                                  cpu_seconds=1.0, proj_rule="left", state_dtype="f32"))())
    out.put((rank, t, bench.job_value(t, 200.0), buf.getvalue(), bench.shard_modules(224, rank, world)))
    dist.destroy_process_group()


def test_shards_take_the_slowest_rank_and_cover_every_module_once():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=60) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    owned = []
    for rank, t, value, printed, shard in res:
        assert t == 15.0                      # max over ranks
        assert value == pytest.approx(15.0 + 1.0)   # slowest shard's step + refresh / 200
        if rank != 0:
            assert printed == ""              # non-zero ranks of the reference arm stay silent
        owned += shard
        # each shard holds every module type of the 7-per-layer model equally often
        types = [i % 7 for i in shard]
        assert all(types.count(k) == 16 for k in range(7))
    assert sorted(owned) == list(range(224))
