"""The multi-rank path of bench.py on CPU: two gloo ranks, each timing its own
token batch; the job's time is the slowest rank's and its throughput counts
every rank's work. The data path has no collective; only the timing is reduced."""

import multiprocessing as mp
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # Rank r's step took 1 + r ms on the device and 10 - r ms end to end.
        ms, e2e = bench.reduce_over_ranks([1.0 + rank, 10.0 - rank], dist, "cpu")
        q.put((rank, ms, e2e, bench.job_tops(2e9, world, ms), bench.rank_seed_base(rank)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_report_the_slowest_rank_and_all_work():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        results = sorted(q.get(timeout=120) for _ in range(2))
    finally:
        for p in procs:
            p.join(timeout=60)
    assert all(p.exitcode == 0 for p in procs)
    for rank, ms, e2e, tops, _ in results:
        assert ms == 2.0 and e2e == 10.0          # maxima over both ranks, on every rank
        assert tops == pytest.approx(2e9 * 2 / 2e-3 / 1e12)
    assert results[0][4] != results[1][4]       # each rank draws its own batch


def test_single_process_needs_no_collective():
    assert bench.reduce_over_ranks([3.0, 4.0]) == [3.0, 4.0]
    assert bench.job_tops(1e12, 1, 1000.0) == pytest.approx(1.0)


def test_reference_arm_runs_on_rank_zero_only():
    class Args:
        workload, steps, warmup, ref_budget = "toy", 1, 0, 0.1
    assert bench.run_reference(Args, rank=1, world=2) is None


def test_reference_arm_line_on_rank_zero():
    """The reference arm times the float64 oracle on a bounded token sample and prints the
    base contract's keys, with an end-to-end figure that copies nothing."""
    class Args:
        workload, steps, warmup, ref_budget = "toy", 2, 1, 0.5
    line = bench.run_reference(Args, rank=0, world=1)
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC and line["unit"] == bench.UNIT
    assert line["value"] > 0 and line["higher_is_better"] is True and line["steps"] == 2
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"] == {"value": line["value"], "unit": bench.UNIT, "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
    assert 4 <= line["config"]["tokens_per_step"] <= 16
