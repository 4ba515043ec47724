"""The N > 1 path's host logic with world_size-2 gloo process groups on CPU.

Each rank routes its shard with the CPU oracle (standing in for its GPU) and
the gathered outputs must equal one process routing the whole batch; the
max-over-ranks timing reduction is checked the same way.
"""

import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2607_08565_gb300.shard import rank_batches, request_range, shard_batch


def test_request_ranges_partition():
    for n in (0, 1, 7, 8192, 8193):
        for world in (1, 2, 3, 8):
            ranges = [request_range(n, r, world) for r in range(world)]
            assert ranges[0][0] == 0 and ranges[-1][1] == n
            assert all(a[1] == b[0] for a, b in zip(ranges, ranges[1:]))
            sizes = [hi - lo for lo, hi in ranges]
            assert max(sizes) - min(sizes) <= 1
    ids = [rank_batches(r, 4, 3) for r in range(4)]
    flat = sorted(sum(ids, []))
    assert flat == list(range(12))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, result_q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import oracle
    from synth import burst_trace

    tr = burst_trace(num_instances=8, block_size=16, n_sessions=200, batch_size=301,
                     len_lo=64, len_hi=900)
    p = tr.params
    ox = oracle.OracleIndex(p.num_instances)
    for s in range(tr.n_sessions):
        h = oracle.block_hashes(tr.session_prefix(s), p.block_size)
        for t in tr.session_tiers(s):
            ox.insert(h, t)
    bt = tr.batch(0)
    tok, off, lo, hi = shard_batch(bt.tokens, bt.offsets, rank, world)
    out = ox.route_batch(p.block_size, 2, 0, tok, off, bt.load, 1, 4, 2)
    # gather every rank's slice (gloo all_gather of equal-size padded rows)
    n_max = request_range(bt.n_requests, 0, world)[1]
    pad = np.full((4, n_max), -1, dtype=np.int64)
    for j, f in enumerate(("instance", "local_hit", "global_hit", "session_key")):
        pad[j, :hi - lo] = out[f].astype(np.int64) if f != "session_key" else \
            out[f].view(np.int64)
    parts = [torch.empty(4, n_max, dtype=torch.int64) for _ in range(world)]
    dist.all_gather(parts, torch.from_numpy(pad))
    elapsed = torch.tensor([float(rank + 1)])
    dist.all_reduce(elapsed, op=dist.ReduceOp.MAX)
    if rank == 0:
        full = ox.route_batch(p.block_size, 2, 0, bt.tokens, bt.offsets, bt.load, 1, 4, 2)
        ok = elapsed.item() == float(world)
        for r in range(world):
            a, b = request_range(bt.n_requests, r, world)
            got = parts[r].numpy()[:, :b - a]
            for j, f in enumerate(("instance", "local_hit", "global_hit", "session_key")):
                want = full[f][a:b].astype(np.int64) if f != "session_key" else \
                    full[f][a:b].view(np.int64)
                ok = ok and np.array_equal(got[j], want)
        result_q.put(bool(ok))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_sharded_routing_matches_single_process():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for pr in procs:
        pr.start()
    ok = q.get(timeout=180)
    for pr in procs:
        pr.join(timeout=60)
    assert ok
    assert all(pr.exitcode == 0 for pr in procs)
