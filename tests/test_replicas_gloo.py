"""The multi-GPU host path on the CPU, with two gloo ranks.

The compression path has no exchange between (layer, document, head) units,
so N GPUs run N independent replicas: each rank draws its own data (its own
seed), the only cross-rank operations are barriers and the maximum of the step
times, and the whole-job value counts every rank's tokens.  Each rank here also
runs the oracle on its own tiny layer, to show the replicas need nothing from
one another.
"""
import os
import socket
import time

import pytest


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, queue):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from oracle import taskpress_oracle as O
        from paper_2608_03276_gb300 import replicas, synth
        r, wsz, local = replicas.dist_env()
        w = synth.WORKLOADS[1].with_(doc_lens=(300,))
        x = synth.make_layer(w.with_(seed=replicas.rank_seed(w.seed, r)))
        out = O.compress_layer(x.q, x.k, x.v, x.doc_offsets, n_heads_q=w.n_heads_q,
                               n_heads_kv=w.n_heads_kv, keep_ratio=w.keep_ratio)
        replicas.barrier()
        ms = replicas.max_over_ranks(10.0 + 5.0 * r)
        value = replicas.whole_job_value(w.n_total, 2, wsz, ms)
        kept = [out["idx"][(0, h)].tolist() for h in range(w.n_heads_kv)]
        queue.put((r, wsz, local, x.digest(), ms, value, kept))
    finally:
        dist.destroy_process_group()


def test_two_gloo_replicas():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, queue)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        res = sorted(queue.get(timeout=180) for _ in range(2))
    finally:
        for p in procs:
            p.join(timeout=60)
    assert all(p.exitcode == 0 for p in procs)
    (r0, w0, l0, d0, ms0, v0, k0), (r1, w1, l1, d1, ms1, v1, k1) = res
    assert (r0, r1) == (0, 1) and w0 == w1 == 2 and (l0, l1) == (0, 1)
    assert d0 != d1, "every rank must draw its own data"
    assert ms0 == ms1 == 15.0, "every rank reports the slowest rank's time"
    assert v0 == v1 == pytest.approx(300 * 2 * 2 / 15e-3)
    assert k0 != k1


def test_single_process_defaults(monkeypatch):
    from paper_2608_03276_gb300 import replicas
    for var in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(var, raising=False)
    assert replicas.dist_env() == (0, 1, 0)
    assert replicas.max_over_ranks(12.5) == 12.5
    assert replicas.rank_seed(7, 0) == 7 and replicas.rank_seed(7, 1) != 7
    replicas.barrier()


def _dying_worker(rank, world, port, queue):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    from paper_2608_03276_gb300 import replicas
    replicas.init("gloo", timeout_s=10.0)
    replicas.barrier()  # step 1: both ranks present
    if rank == 1:
        os._exit(3)  # rank 1 dies between steps, with nothing in flight
    t0 = time.perf_counter()
    try:
        replicas.barrier()  # step 2: the survivor must get an error, not block
        queue.put(("no error", time.perf_counter() - t0))
    except Exception as e:  # noqa: BLE001 - any collective error is the detection
        queue.put((type(e).__name__, time.perf_counter() - t0))


def test_dead_rank_is_detected():
    """A rank that exits between steps makes the survivor's next barrier fail
    within the replica group's timeout instead of blocking it."""
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_dying_worker, args=(r, 2, port, queue)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        what, waited = queue.get(timeout=120)
    finally:
        for p in procs:
            p.join(timeout=60)
            if p.is_alive():
                p.kill()
    assert what != "no error"
    assert waited < 60.0
    assert procs[1].exitcode == 3
