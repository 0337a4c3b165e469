"""The benchmark's multi-rank host logic on CPU ranks (gloo, world size 2):
the slowest rank's time is every rank's, the job value counts every rank's
bytes, and the reference arm runs on rank 0 only."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = bench.max_over_ranks(1.5 + rank, world, "cpu")   # rank 1 is slower
        gbs = bench.job_gbs(1_000_000_000, world, ms)
        ref = bench.run_reference(None, rank, world) if rank != 0 else "rank0"
        out.put((rank, ms, gbs, ref))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_job_value_gloo():
    world = 2
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(out.get(timeout=10) for _ in range(world))
    for rank, ms, gbs, ref in got:
        assert ms == 2.5                      # the slowest rank's time, on every rank
        assert gbs == pytest.approx(2 * 1e9 / 2.5e-3 / 1e9)
    assert got[1][3] is None                  # the reference arm: rank 0 only


def test_single_rank_is_identity():
    assert bench.max_over_ranks(3.25, 1, "cpu") == 3.25
    assert bench.job_gbs(537_000_000, 1, 1.0) == pytest.approx(537.0)


def test_oracle_sample_units_and_bytes():
    """The reference arm's bounded sample: rows of a single case (its inputs
    cut to the same elements), whole cases of a batch."""
    from paper_2608_02712_gb300 import workloads
    single = [workloads.c5(shape=(64, 256), first_k=16)]
    assert bench.sample_units(single) == 64
    t, nbytes = bench.oracle_step_time(single, 8)
    assert t > 0 and nbytes == 8 * 256 * 4 * 2
    batch = [workloads.fuzz(s) for s in range(3)]
    assert bench.sample_units(batch) == 3
    t, nbytes = bench.oracle_step_time(batch, 2)
    assert nbytes == sum(bench.case_bytes(c) for c in batch[:2])
    assert "cases of the batch" in bench.sample_text(batch, 2, nbytes)


def test_full_size_flags():
    class A:
        c2_batch, c5_rows, no_inputs = 8, 32768, False
    assert bench.full_size(A)
    A.c5_rows = 4096
    assert not bench.full_size(A)


def test_no_inputs_case_is_the_plain_pair():
    """--no-inputs: the same candidate/reference pair, its inputs dropped and
    its workload named without the input."""
    with_in = bench.make_cases("c5", "cpu", c5_rows=2)
    plain = bench.make_cases("c5", "cpu", c5_rows=2, no_inputs=True)
    assert with_in[0]["name"] == "c5_fp32_2x65536_input" and len(with_in[0]["inputs"]) == 1
    assert plain[0]["name"] == "c5_fp32_2x65536" and plain[0]["inputs"] == []
    # bitwise (the candidate holds NaN)
    assert torch.equal(plain[0]["cand"].view(torch.int32), with_in[0]["cand"].view(torch.int32))
    assert torch.equal(plain[0]["ref"], with_in[0]["ref"])
