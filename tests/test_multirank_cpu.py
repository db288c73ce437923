"""The multi-process host logic of bench.py on CPU: two gloo ranks.

bench.py --gpus N runs one process per GPU, each on its own token batch
(the path has no data exchange: tokens are independent), and only the
timing is reduced (max over ranks). These tests run that reduction, the
whole-job throughput and the per-rank inputs across two real processes
with the gloo backend; no GPU is involved.
"""

import multiprocessing as mp
import os
import socket
import sys

import pytest

from tests.conftest import ROOT


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    try:
        sys.path.insert(0, ROOT)
        os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                          MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
        import numpy as np
        import torch.distributed as dist
        dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
        import bench
        from paper_2606_04945_gb300 import inputs
        # per-rank step times: the job takes as long as its slowest rank
        ms, ms_e2e = bench.reduce_max([0.1 + 0.05 * rank, 0.4 - 0.1 * rank], "cpu")
        # each rank's own token batch (a small case of the same generator)
        case = inputs.random_linear(bench.rank_seed(rank), 16, 512, 64)
        first = float(case.X[0, :8].sum())
        firsts = [None] * world
        dist.all_gather_object(firsts, first)
        # the reference arm prints on rank 0 only
        ref = None if rank == 0 else bench.run_reference(_Args())
        dist.barrier()
        dist.destroy_process_group()
        q.put((rank, ms, ms_e2e, firsts, ref, np.isfinite(first)))
    except Exception as e:  # report instead of hanging the parent
        q.put((rank, "error", repr(e), None, None, None))


class _Args:
    steps = 1
    warmup = 0
    ref_sample_tokens = 4


def test_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    world = 2
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = {}
    try:
        for _ in range(world):
            r = q.get(timeout=180)
            res[r[0]] = r
    finally:
        for p in procs:
            p.join(timeout=30)
            if p.is_alive():
                p.kill()
    for r in range(world):
        assert res[r][1] != "error", res[r][2]
    for r in range(world):
        _, ms, ms_e2e, firsts, ref, finite = res[r]
        assert ms == pytest.approx(0.15) and ms_e2e == pytest.approx(0.4)   # max over ranks
        assert firsts[0] != firsts[1] and finite                           # distinct batches
    assert res[1][4] is None                                               # rank 1 prints nothing


def test_job_throughput_is_weak_scaling():
    sys.path.insert(0, ROOT)
    import bench
    ops = 2 * 1024 * (12288 + 4096) * 4096
    one = bench.job_tops(ops, 0.1, 1)
    assert bench.job_tops(ops, 0.1, 4) == pytest.approx(4 * one)
    assert bench.job_tops(ops, 0.2, 2) == pytest.approx(one)
    assert len({bench.rank_seed(r) for r in range(8)}) == 8


def test_reference_line_matches_our_arm():
    """The reference arm's line (rank 0, the oracle on a small sample) has
    our arm's metric, unit, direction and config for the same arguments,
    and the keys the contract asks of it."""
    sys.path.insert(0, ROOT)
    import bench

    class Args(_Args):
        no_graph = False
        step_form = "grouped"

    line = bench.run_reference(Args())
    assert line["impl"] == "reference"
    assert line["metric"] == bench.METRIC and line["unit"] == bench.UNIT and line["higher_is_better"] is True
    assert line["config"] == bench.arm_config(Args()) == bench.config_dict(True, True)
    assert line["value"] > 0 and line["cpu_baseline"]["value"] == line["value"]
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
