"""The multi-GPU path is page sharding with no data-path collective: each rank decodes its own
pages (pages never see each other), and the benchmark reduces only its timing. These checks run
the host side of that path as two gloo ranks on the CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2608_06146_gb300.engine import shard_pages


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, num_pages, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = shard_pages(num_pages, rank, world)
        gathered = [None] * world
        dist.all_gather_object(gathered, mine)
        import bench
        t = bench.max_over_ranks(torch, world, float(rank + 1) * 1.5)
        dist.barrier()
        q.put((rank, gathered, t))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("num_pages", [32, 7, 1])
def test_two_gloo_ranks_partition_pages_and_reduce_timing(num_pages):
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, num_pages, q)) for r in range(world)]
    for p in procs:
        p.start()
    results = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, gathered, t in results:
        flat = sorted(x for shard in gathered for x in shard)
        assert flat == list(range(num_pages)), "shards must partition the pages"
        assert max(len(s) for s in gathered) - min(len(s) for s in gathered) <= 1
        assert t == 3.0, "max over ranks of (rank+1)*1.5"


def test_shard_pages_rejects_bad_rank():
    with pytest.raises(ValueError):
        shard_pages(4, 2, 2)


def _loop_rank_main(rank, world, port, q):
    """One rank of a sharded Algorithm 1 run: its own scheduler over its shard of the pages, the host
    side of the loop (the device append and decode need a GPU per rank)."""
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import numpy as np

        from paper_2608_06146_gb300 import inputs
        from paper_2608_06146_gb300 import padoc_attn as pa
        pa.load_library()
        wl = inputs.serving_batch(seed=3, num_pages=9)
        mine = shard_pages(len(wl.pages), rank, world)
        pages = [wl.pages[p] for p in mine]
        src = inputs.LoopTokenSource(pages)
        nb = sum(-(-(pg.prefix_len + pg.layout_len) // 16) + sum(-(-n // 16) for n in pg.branch_len) for pg in pages)
        m = pa.Mpd(nb)
        for p in range(len(pages)):
            P, nf, leos, _ = src.admission(p)
            _, _, new = m.add_page(P, nf, leos)
            src.admitted(p, new)
        decoded = []
        while m.status()[1] > 0:
            ids, _ = m.begin_step()
            src.rows(ids)
            for r in src.token_rows(ids):   # local packed row -> (global page, page-local position)
                lp = int(np.searchsorted(src.base, r, side="right") - 1)
                decoded.append((mine[lp], int(r - src.base[lp])))
            nf, eos = src.events(ids)
            src.forked(ids, nf, m.end_step(nf, eos))
        gathered = [None] * world
        dist.all_gather_object(gathered, (decoded, m.status()[2] == nb))
        q.put((rank, gathered))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_run_the_loop_on_their_page_shards():
    """Sharded Algorithm 1: together the ranks decode every layout and branch token of every page
    exactly once, and each rank's pool is whole again at the end."""
    from paper_2608_06146_gb300 import build as pbuild
    from paper_2608_06146_gb300 import inputs
    pbuild.build()
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_loop_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    results = [q.get(timeout=300) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    wl = inputs.serving_batch(seed=3, num_pages=9)
    want = sorted((p, j) for p, pg in enumerate(wl.pages) for j in range(pg.prefix_len, pg.packed_len))
    for _, gathered in results:
        got = sorted(t for dec, _ in gathered for t in dec)
        assert got == want
        assert all(whole for _, whole in gathered)
