"""GPU parity at the workloads' full sizes, in the launch configuration the
benchmark times: the whole 512-case sweep in one batch call, and a case of
more than 2^32 elements with random values, each compared with the oracle
field by field."""
import numpy as np
import pytest
import torch

import oracle
from _parity import assert_same
from paper_2608_02712_gb300 import validate, validate_batch, workloads

pytestmark = pytest.mark.gpu


def _oracle(case):
    cpu = lambda t: t.cpu()
    return oracle.validate(cpu(case["cand"]), cpu(case["ref"]),
                           inputs=[cpu(x) for x in case["inputs"]], rtol=case["rtol"],
                           atol=case["atol"], tile=case["tile"], first_k=case["first_k"])


def test_c3_full_size_batch():
    """The full-coverage sweep at its configured size: 512 pairs of up to
    4 Mi elements (rank 1-5, fp32/fp16/bf16, half of them faulted) in ONE
    nmv_validate_batch call; every case against the oracle, and the batch
    pass count (the sweep's "x% matched cases")."""
    cases = workloads.c3(device="cuda")
    assert len(cases) == workloads.C3_COUNT
    got = validate_batch(cases)
    n_pass = 0
    for c, g in zip(cases, got["results"]):
        w = _oracle(c)
        assert_same(g, w, c["name"])
        n_pass += int(w["pass"])
    assert got["n_pass"] == n_pass


def test_beyond_32_bits_random_values():
    """bf16 [4099, 1048583] (4.3e9 elements > 2^32, 8.6 GB per tensor):
    random values with accumulation-style noise, isolated faults on both
    sides of index 2^32, NaN/-Inf on both sides, and a band of wrong rows
    past 2^32; the whole result against one oracle pass."""
    free, _ = torch.cuda.mem_get_info()
    if free < (80 << 30):
        pytest.skip("needs 80 GiB of free device memory")
    shape = (4099, 1048583)
    numel = shape[0] * shape[1]
    assert numel > (1 << 32)
    g = torch.Generator(device="cuda").manual_seed(31)
    ref = torch.randn(shape, generator=g, device="cuda", dtype=torch.bfloat16)
    cand = torch.empty_like(ref)
    for r0 in range(0, shape[0], 512):   # row chunks keep the fp32 temporaries small
        rr = ref[r0:r0 + 512].float()
        cand[r0:r0 + 512] = (rr * (1.0 + torch.randn(rr.shape, generator=g, device="cuda")
                                   * 2.0 ** -9)).to(torch.bfloat16)
    del rr
    cf = cand.view(-1)
    two32 = 1 << 32
    for i in (3, 1 << 31, two32 - 2, two32 - 1, two32, two32 + 1, two32 + 4097, numel - 1):
        cf[i] = cf[i].float() + 3.0
    cf[two32 - 5] = float("nan")
    cf[two32 + 5] = float("-inf")
    cand[4097:4099, 1000:1300] += 1.0  # rows past 2^32 (4097 * 1048583 > 2^32)
    got = validate(cand, ref, rtol=1.6e-2, atol=1e-3, tile=(128, 4096), first_k=1024)
    assert got["numel"] == numel and not got["pass"]
    host = {"cand": cand.cpu(), "ref": ref.cpu(), "inputs": [], "rtol": 1.6e-2, "atol": 1e-3,
            "tile": (128, 4096), "first_k": 1024}
    del cand, ref, cf
    want = _oracle(host)
    assert_same(got, want, "bf16 beyond 2^32")
    assert (np.asarray(want["fk_index"]) >= two32).any()
