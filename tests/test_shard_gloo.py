"""Multi-rank path on the CPU (gloo, world size 2).

Fork decode shards by independent traces: each rank takes the traces
t % world == rank and computes their forks with no data-path collective.
The test computes each shard with the oracle on its own rank, gathers the
results through gloo only to check them, and compares with the unsharded
oracle result; it also checks that the shards partition the forks exactly.
"""

import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _spec():
    from paper_2606_17518_gb300 import workloads as wl
    return wl.WorkloadSpec(name="shard", num_traces=5, prefix_len=(20, 90), forks=(1, 4),
                           suffix_len=(0, 40), hq=8, hkv=2, dqk=16, dv=16, page_size=8, seed=21)


def _rank_main(rank, world, port, results):
    import sys
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist

    import oracle
    from paper_2606_17518_gb300 import workloads as wl
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w = wl.make_workload(_spec())
    part = wl.shard_traces(w, rank, world)
    o, lse = (oracle.fork_attn_decode(part) if part["total_forks"]
              else (np.zeros((0, w["hq"], w["dv"])), np.zeros((0, w["hq"]))))
    gathered = [None] * world
    dist.all_gather_object(gathered, (part["global_forks"].tolist(), o, lse))
    if rank == 0:
        results.put(gathered)
    dist.barrier()
    dist.destroy_process_group()


def test_trace_shards_reproduce_full_result():
    from paper_2606_17518_gb300 import workloads as wl
    import oracle
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    gathered = q.get(timeout=300)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    w = wl.make_workload(_spec())
    o_full, l_full = oracle.fork_attn_decode(w)
    seen = []
    for forks, o, lse in gathered:
        seen += forks
        for i, f in enumerate(forks):
            np.testing.assert_allclose(o[i], o_full[f], rtol=0, atol=1e-12)
            np.testing.assert_allclose(lse[i], l_full[f], rtol=0, atol=1e-12)
    assert sorted(seen) == list(range(w["total_forks"]))


def test_shard_with_more_ranks_than_traces():
    from paper_2606_17518_gb300 import workloads as wl
    w = wl.make_workload(_spec())
    parts = [wl.shard_traces(w, r, 8) for r in range(8)]
    assert sum(p["num_traces"] for p in parts) == w["num_traces"]
    assert sum(p["total_forks"] for p in parts) == w["total_forks"]
    assert parts[7]["num_traces"] == 0 and parts[7]["total_forks"] == 0
