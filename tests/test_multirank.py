"""The N > 1 host path of bench.py on CPU: two gloo ranks, each building its
own batch of the same shape (weak scaling: units are independent, no data-path
collective), then the timing and byte aggregation the GPU ranks do over NCCL
(max over ranks of the step time, sum over ranks of the bytes)."""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, queue):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    import torch.distributed as td
    td.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        import oracle
        wl = bench.make_workload("long", rank, oracle.alloc_from_scores)
        tot, score, evicted = bench.workload_bytes(wl)
        max_r, sum_r = bench.rank_reducers(True, "cpu")
        step_ms = 4.0 + rank  # a stand-in for the rank's measured step time
        queue.put(dict(rank=rank, tot=tot, lens=[int(x) for x in wl.lens], budget=[int(x) for x in wl.budget],
                       shape=(wl.L, wl.B, wl.H_kv, wl.S_cap), max_ms=max_r(step_ms), all_bytes=sum_r(tot),
                       all_evicted=sum_r(evicted)))
        td.barrier()
    finally:
        td.destroy_process_group()


def test_two_rank_weak_scaling_aggregation():
    import multiprocessing as mp
    import oracle
    import bench
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted([q.get(timeout=120) for _ in range(2)], key=lambda d: d["rank"])
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    a, b = res
    # each rank holds its own batch of the same shape
    assert a["shape"] == b["shape"]
    assert a["lens"] != b["lens"]
    # the aggregate every rank reports: max of the times, sum of the bytes
    assert a["max_ms"] == b["max_ms"] == 5.0
    assert a["all_bytes"] == b["all_bytes"] == a["tot"] + b["tot"]
    # and it equals the bytes of the two batches computed here independently
    expect = sum(bench.workload_bytes(bench.make_workload("long", r, oracle.alloc_from_scores))[0] for r in range(2))
    assert a["all_bytes"] == expect
    assert np.isclose(a["all_evicted"], b["all_evicted"])
