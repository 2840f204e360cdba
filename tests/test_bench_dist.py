"""Multi-rank logic of bench.py on CPU with gloo, world size 2: every rank
decodes its own batch (independent sequences, no data-path collective), the
step time is the max over ranks and the throughput counts every rank's batch;
the end-to-end figure is aggregated the same way."""
import os
import socket

import pytest
import torch
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    import workloads
    dist.init_process_group("gloo", rank=rank, world_size=world)
    r, w, l = bench.dist_env()
    wl = bench.shard_workload(workloads.WORKLOADS["llama3_8b"], r)
    step_s = 0.010 * (r + 1)                      # rank 1 is the slow one
    slowest = bench.max_over_ranks(step_s, w, torch.device("cpu"))
    value, _ = bench.aggregate([slowest] * w, wl.B)
    L = workloads.ctx_lengths(wl)
    e2e = bench.aggregate_e2e({"value": 0.0, "unit": "tokens/s", "ms_per_step": 0.3 + 0.1 * r,
                               "h2d_bytes_per_step": 100, "d2h_bytes_per_step": 7},
                              wl.B, w, torch.device("cpu"))
    dist.barrier()
    q.put((r, wl.seed, slowest, value, L.tolist(), e2e))
    dist.destroy_process_group()


def test_two_rank_weak_scaling_logic():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    res = sorted(q.get(timeout=120) for _ in ps)
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, s0, t0, v0, L0, e0), (r1, s1, t1, v1, L1, e1) = res
    assert s0 != s1 and L0 != L1                  # independent batches
    assert t0 == t1 == pytest.approx(0.020)       # max over ranks
    assert v0 == v1 == pytest.approx(2 * 64 / 0.020)
    # end to end: both ranks' sequences over the slower rank's 0.4 ms step
    assert e0 == e1
    assert e0["ms_per_step"] == pytest.approx(0.4) and e0["value"] == pytest.approx(2 * 64 / 0.4e-3, rel=1e-6)
    assert (e0["h2d_bytes_per_step"], e0["d2h_bytes_per_step"]) == (200, 14)
