"""The multi-process path of bench.py (one replica per GPU, N > 1) exercised on the CPU: two ranks
over gloo, launched like torchrun launches them (RANK, WORLD_SIZE, LOCAL_RANK, MASTER_ADDR
127.0.0.1). Each rank builds its own token shard (seed = rank) and routes it independently (the
oracle stands in for the GPU path here); the only collectives are the barrier, the max of the rank
times, and, for metrics only, an E-int sum of the expert counts. A rank that dies between steps
makes the survivor's next collective fail with an error (gloo, a 20 s process-group timeout), so the
job ends instead of hanging."""
import multiprocessing as mp
import os
import socket

import numpy as np


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch

    import bench
    import synth
    from oracle import clearmoe as O

    w, r, local, dist = bench.init_replicas("gloo")
    try:
        shape = synth.DEIT_TINY_FP32.with_(T=2 * 197, n_cal=1000, seed=r)
        L = synth.make_layer(shape)
        counts = O.route(L["x"], L["Wg"], L["bg"])["counts"]
        c = torch.tensor(counts, dtype=torch.int64)
        dist.all_reduce(c)
        ms = bench.max_over_ranks(1.5 + r, dist, device="cpu")
        q.put(dict(rank=r, world=w, local=local, x0=L["x"][0].copy(), counts=counts,
                   global_counts=c.numpy(), ms=ms, rate=bench.whole_job_rate(shape.T, w, 10, ms)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_replicas_over_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted((q.get(timeout=300) for _ in procs), key=lambda d: d["rank"])
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [d["world"] for d in res] == [2, 2] and [d["local"] for d in res] == [0, 1]
    assert not np.array_equal(res[0]["x0"], res[1]["x0"]), "ranks must hold different shards"
    total = res[0]["counts"] + res[1]["counts"]
    for d in res:
        assert np.array_equal(d["global_counts"], total)
        assert d["ms"] == 2.5  # the slowest rank's time
        assert abs(d["rate"] - 2 * 394 * 10 / 2.5e-3) < 1e-6 * d["rate"]


def test_single_process_needs_no_collective(monkeypatch):
    import bench
    monkeypatch.delenv("WORLD_SIZE", raising=False)
    w, r, local, dist = bench.init_replicas("gloo")
    assert (w, r, dist) == (1, 0, None)
    assert bench.max_over_ranks(3.0, None) == 3.0


def _dying_rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank), CLEARMOE_PG_TIMEOUT_S="20")
    import time

    import bench

    try:
        w, r, local, dist = bench.init_replicas("gloo")
        dist.barrier()  # one step completed by both ranks
        if r == 1:
            os._exit(3)  # dies between steps: no collective of its own in flight
        t0 = time.time()
        try:
            bench.max_over_ranks(1.0, dist, device="cpu")
            q.put(("completed", time.time() - t0))
        except Exception as exc:  # the failure reaches the survivor as an error, not a hang
            q.put((type(exc).__name__, time.time() - t0))
    except Exception as exc:
        q.put((f"setup failed: {exc!r}", -1.0))
    # os._exit skips the queue's feeder thread: flush the message to the pipe first, or the
    # parent may never receive it
    q.close()
    q.join_thread()
    os._exit(0)


def test_a_dead_rank_fails_the_next_collective():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_dying_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        outcome, waited = q.get(timeout=120)
    finally:
        for p in procs:
            p.join(timeout=30)
            if p.is_alive():  # only this test's own children
                p.kill()
                p.join()
    assert not outcome.startswith("setup failed"), outcome
    assert procs[1].exitcode == 3
    assert outcome != "completed", "the survivor's collective completed without its peer"
    assert waited < 60, f"the survivor learned of the failure only after {waited:.0f} s"
