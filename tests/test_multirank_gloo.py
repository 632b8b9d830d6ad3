"""The multi-GPU host path on CPU: two gloo ranks exercise the timing exchange (max over ranks, token
gather, job throughput) and the trajectory sharding the pass uses across GPUs.  No GPU is touched."""
import os
import socket

import pytest

from paper_2609_22158_gb300 import multirank as MR


def _free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update({"WORLD_SIZE": str(world), "RANK": str(rank), "LOCAL_RANK": str(rank),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    try:
        w, r, l = MR.rank_env()
        dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=r, world_size=w)
        # each rank times a different step; the job's time is the slowest rank's
        ms = MR.max_over_ranks([3.25, 4.5][r], dist)
        tokens = MR.gather_tokens([32768, 20000][r], dist)
        value = MR.job_throughput(tokens, ms * 1e-3)
        # every rank derives its own trajectories from the same list without talking to the others
        mine = list(MR.shard(16, w, r))
        seeds = MR.rank_seed(1234, r)
        dist.barrier()
        q.put((r, w, l, ms, tokens, value, mine, seeds))
        dist.destroy_process_group()
    except Exception as e:  # reported to the parent, which fails the test
        q.put(("error", rank, repr(e)))


def test_two_gloo_ranks_exchange_timing_and_shard_work():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in range(2)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert not any(x[0] == "error" for x in res), res
    res.sort()
    (r0, w0, l0, ms0, tok0, v0, mine0, s0), (r1, w1, l1, ms1, tok1, v1, mine1, s1) = res
    assert (r0, r1, w0, w1, l0, l1) == (0, 1, 2, 2, 0, 1)
    assert ms0 == ms1 == 4.5                      # max over ranks, seen by every rank
    assert tok0 == tok1 == [32768, 20000]         # rank order
    assert v0 == v1 == pytest.approx((32768 + 20000) / 4.5e-3)
    assert mine0 + mine1 == list(range(16)) and len(mine0) == len(mine1) == 8
    assert s0 != s1


@pytest.mark.parametrize("n,world", [(16, 1), (16, 3), (5, 8), (0, 2), (7, 7)])
def test_shard_covers_every_item_once(n, world):
    parts = [list(MR.shard(n, world, r)) for r in range(world)]
    assert sum(parts, []) == list(range(n))
    sizes = [len(p) for p in parts]
    assert max(sizes) - min(sizes) <= 1


def test_single_process_defaults(monkeypatch):
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    assert MR.rank_env() == (1, 0, 0)
    assert MR.max_over_ranks(2.5) == 2.5
    assert MR.gather_tokens(123) == [123]
    with pytest.raises(ValueError):
        MR.job_throughput([1], 0.0)


def _failing_worker(rank, world, port, q):
    import datetime
    import torch.distributed as dist
    os.environ.update({"WORLD_SIZE": str(world), "RANK": str(rank), "LOCAL_RANK": str(rank),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world,
                            timeout=datetime.timedelta(seconds=10))
    if rank == 1:
        # this rank fails between steps, before the timing exchange: it never joins the collective
        q.put((rank, "raised"))
        raise SystemExit(3)
    try:
        MR.max_over_ranks(1.0, dist)
        q.put((rank, "no error"))
    except Exception as e:  # the surviving rank learns of it from its next collective
        q.put((rank, "detected: " + type(e).__name__))


def test_a_failed_rank_is_detected_by_the_next_collective():
    """A rank that leaves between steps (an exception on the host, no GPU involved) makes the other
    rank's next timing exchange fail with an error instead of hanging."""
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_failing_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
    assert res[1] == "raised" and procs[1].exitcode == 3
    assert res[0].startswith("detected"), res[0]
