"""The sharded (multi-GPU) path's host logic on the CPU with two gloo ranks:
each rank owns an independent replica of the workload (its own seeds, its own
paged cache), runs the crop + append bookkeeping of a bench step, and the only
collective is the max over ranks of the step time (outside the data path)."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        import bench
        import oracle
        import paper_2609_04875_gb300 as pe
        w = bench.make_workload("agent_batch", replica=rank)
        # each rank's host bookkeeping for one step, checked against the oracle
        c = pe.PagedKVCache(1, w.num_kv_heads, w.head_dim, w.page_size, w.num_pages, len(w.agents),
                            w.max_pages_per_seq, init_free_order=w.init_free_order(), host_only=True)
        o = oracle.OracleKVCache(1, w.num_kv_heads, w.head_dim, w.page_size, w.num_pages, len(w.agents),
                                 w.max_pages_per_seq, init_free_order=w.init_free_order(), store_values=False)
        seqs = [c.seq_create() for _ in w.agents]
        for s, a in zip(seqs, w.agents):
            o.seq_create()
            c.append_kv(s, n_tokens=a.T)
            o.append(s, n_tokens=a.T)
        c.crop_batch(seqs, [a.tau for a in w.agents])
        cu = [0]
        for a in w.agents:
            cu.append(cu[-1] + a.S)
        c.append_kv_batch(seqs, cu_tokens=cu)
        for s, a in zip(seqs, w.agents):
            o.crop(s, a.tau)
        for s, a in zip(seqs, w.agents):
            o.append(s, n_tokens=a.S)
        ok = c.free_list() == o.free_list() and all(c.page_table(s) == o.page_table(s) for s in seqs)
        ok = ok and all(c.seq_info(s) == (a.T, a.S) for s, a in zip(seqs, w.agents))
        # timing aggregation: the job's time is the slowest rank's
        local_ms = 10.0 + rank
        agg = bench.reduce_max(local_ms, True)
        seeds = [None] * world
        dist.all_gather_object(seeds, (w.seed, [a.T for a in w.agents][:4]))
        q.put((rank, ok, agg, seeds, w.total_suffix))
    finally:
        dist.destroy_process_group()


def test_two_rank_replicas_gloo():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    results = [q.get(timeout=300) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    results.sort()
    for rank, ok, agg, seeds, tokens in results:
        assert ok, f"rank {rank}: bookkeeping differs from the oracle"
        assert agg == 11.0, "max over ranks"
        assert seeds[0] != seeds[1], "replicas must draw from different seeds"
    # whole-job throughput = all ranks' tokens / the slowest rank's time
    total = sum(r[4] for r in results)
    assert total > results[0][4]
