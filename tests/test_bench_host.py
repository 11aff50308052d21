"""Host-side logic of the multi-GPU benchmark, on CPU with gloo.

Every rank processes its own B sequences (the path has no exchange step, so
there is no collective on the data path); the job's time is the slowest
rank's.  Two gloo ranks check that the shards are disjoint and cover
[0, world*B), that the regenerated shard inputs differ between ranks, and
that the timing reduction returns the max over ranks.
"""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, B, out):
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    import gen
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        seqs = list(bench.shard(rank, B))
        gathered = [None] * world
        dist.all_gather_object(gathered, seqs)
        w = gen.make_workload(B, 2, 64, "f32", seed=9)
        inp = gen.generate_sequences(w, seqs)
        first_u = [None] * world
        dist.all_gather_object(first_u, float(inp["u"][0, 0]))
        t = bench.max_over_ranks(1.5 + rank, dist)
        out[rank] = (gathered, first_u, t)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_sequences_and_take_the_max_time():
    world, B = 2, 3
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_worker, args=(world, port, B, out), nprocs=world, join=True)
        res = dict(out)
    gathered, first_u, t = res[0]
    allseq = sorted(s for part in gathered for s in part)
    assert allseq == list(range(world * B))
    assert set(gathered[0]).isdisjoint(gathered[1])
    assert first_u[0] != first_u[1]
    assert res[0][2] == res[1][2] == 2.5


def test_traffic_figures_follow_the_kernel_code_not_its_comments():
    # The bench reports a kernel's captured DRAM traffic only while the
    # kernel's code is the code it was captured from: comments and spacing
    # do not count, a changed statement does.
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    src = "int f(int x) {\n  // the square\n  return x * x; /* (exact) */\n}\n"
    assert bench._code_only(src) == bench._code_only("int f(int x) {  return x * x;\n\n}")
    assert bench._code_only(src) != bench._code_only(src.replace("x * x", "x + x"))
    for k in bench.KERNEL_SOURCES:
        assert len(bench.kernel_source_hash(k)) == 16
