"""The scan's wait limit, without a fault: the test hook NMV_FAULT_INJECT=stall
makes every warp announce the bytes of its first stage and issue no copy,
so its bounded wait on the stage's mbarrier runs out (after about 2 s).
The call must return NMV_ETIMEOUT (no hang, nothing left allocated), and the
CUDA context must stay usable: the next call, without the hook, is correct."""
import os

import pytest
import torch

import oracle
from _parity import assert_same
from paper_2608_02712_gb300 import NmvError, nmv, validate, workloads

pytestmark = pytest.mark.gpu


def test_wait_limit_reports_timeout_and_the_context_survives(monkeypatch):
    case = workloads.c1(device="cuda", shape=(256, 1024))
    args = dict(rtol=case["rtol"], atol=case["atol"], tile=case["tile"], first_k=case["first_k"])
    monkeypatch.setenv("NMV_FAULT_INJECT", "stall")
    with pytest.raises(NmvError) as e:
        validate(case["cand"], case["ref"], **args)
    assert e.value.status == nmv.NMV_ETIMEOUT
    assert "did not complete" in str(e.value)
    monkeypatch.delenv("NMV_FAULT_INJECT")
    torch.cuda.synchronize()
    got = validate(case["cand"], case["ref"], **args)
    assert_same(got, oracle.validate(case["cand"].cpu(), case["ref"].cpu(), **args), "after the timeout")
