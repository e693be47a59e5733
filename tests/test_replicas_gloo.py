"""Multi-GPU runs of the serving step are independent replicas (the path has no
exchange step): every rank serves its own seeded batch and the job's time is
the slowest rank's. The host side of that is checked here with two gloo ranks
on the CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        from paper_2608_08684_gb300 import synth
        wl = bench.replica_workload(synth.WORKLOADS["tiny"], rank)
        # this rank's own batch: keys of layer 0
        k = synth.layer_keys(wl, 0)
        local_ms = 10.0 + 5.0 * rank
        total = bench.max_over_ranks(local_ms, world, torch.device("cpu"))
        ms_step, value = bench.job_throughput(total, 4, wl.batch * wl.seq_len, world)
        out[rank] = (wl.seed, float(k.float().sum()), total, ms_step, value)
    finally:
        dist.destroy_process_group()


def test_two_replicas_max_time_and_distinct_batches():
    world = 2
    port = _free_port()
    # the manager's server process is spawned too: forking this
    # multi-threaded process could deadlock the child
    with mp.get_context("spawn").Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert sorted(res) == [0, 1]
    seeds = {res[r][0] for r in res}
    assert len(seeds) == 2, "each replica is seeded apart"
    assert res[0][1] != res[1][1], "each replica serves its own batch"
    for r in res:
        total, ms_step, value = res[r][2:]
        assert total == pytest.approx(15.0), "the slowest rank's time on every rank"
        assert ms_step == pytest.approx(15.0 / 4)
        from paper_2608_08684_gb300 import synth
        wl = synth.WORKLOADS["tiny"]
        assert value == pytest.approx(world * wl.batch * wl.seq_len / (ms_step / 1e3))


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(7.5, 1, torch.device("cpu")) == 7.5
    from paper_2608_08684_gb300 import synth
    wl = synth.WORKLOADS["tiny"]
    assert bench.replica_workload(wl, 0) is wl
