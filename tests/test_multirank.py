"""The benchmark's N > 1 host path (one process per GPU, independent samples,
max-over-ranks timing, whole-job throughput) on CPU with gloo ranks."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import bench
    from paper_2511_22533_gb300 import synth
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms_local = [120.0, 180.0][rank]
    ms = bench.max_over_ranks(ms_local, world)
    value = bench.whole_job_throughput(25, 4, world, ms)
    S = synth.latents(synth.SHAPES["tiny"], 1, bench.rank_seed(rank))
    out[rank] = (ms, value, float(S[0, 0, 0]))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_gloo_ranks_aggregate():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(90)
        assert p.exitcode == 0
    (ms0, v0, s0), (ms1, v1, s1) = out[0], out[1]
    assert ms0 == ms1 == 180.0                       # max over ranks
    assert v0 == v1 == pytest.approx(25 * 4 * 2 / 0.18)  # all ranks' steps / slowest time
    assert s0 != s1                                   # ranks sample different inputs


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(42.0, 1) == 42.0
    assert bench.whole_job_throughput(25, 10, 1, 500.0) == pytest.approx(500.0)
