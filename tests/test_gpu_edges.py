"""GPU parity at the edges of the scan's fp32 proofs and of its launch plan
(workloads.edge): tolerances where the pre-filter is switched off (rtol
above 1/2, atol above 2^100) or sits at 1/4 and 1/2; differences at and
either side of |r|/4 (where c - r stops being provably exact in fp32);
subnormal references; tiles above the shared-memory profile size; tile grids
wider than the shared-memory histogram window; cases of millions of
elements.  Each case is compared with the oracle field by field, alone, in
one mixed batch, and through buffers that are not 16-byte aligned."""
import pytest
import torch

import oracle
from _parity import assert_same
from paper_2608_02712_gb300 import validate, validate_batch, workloads

pytestmark = pytest.mark.gpu

N_EDGE = 120


def _oracle(case):
    cpu = lambda t: t.cpu()
    return oracle.validate(cpu(case["cand"]), cpu(case["ref"]),
                           inputs=[cpu(x) for x in case["inputs"]], rtol=case["rtol"],
                           atol=case["atol"], tile=case["tile"], first_k=case["first_k"])


@pytest.mark.parametrize("seed", range(N_EDGE))
def test_edge_parity(seed):
    case = workloads.edge(seed, device="cuda")
    got = validate(case["cand"], case["ref"], rtol=case["rtol"], atol=case["atol"],
                   tile=case["tile"], first_k=case["first_k"])
    assert_same(got, _oracle(case), case["name"])


def test_edge_batch():
    cases = [workloads.edge(s, device="cuda") for s in range(0, N_EDGE, 3)]
    got = validate_batch(cases)
    for c, g in zip(cases, got["results"]):
        assert_same(g, _oracle(c), c["name"] + " (batch)")


@pytest.mark.parametrize("seed", range(0, N_EDGE, 5))
def test_edge_parity_unaligned(seed):
    case = workloads.edge(seed, device="cuda")
    shift = lambda t: torch.cat([t.reshape(-1)[:1], t.reshape(-1)])[1:].view(t.shape)
    c, r = shift(case["cand"]), shift(case["ref"])
    got = validate(c, r, rtol=case["rtol"], atol=case["atol"], tile=case["tile"],
                   first_k=case["first_k"])
    assert_same(got, _oracle(case), case["name"] + " (unaligned)")
