"""nmv_validate_noalloc: the entry point for callers that must not allocate.

Some callers cannot let a library call cudaMalloc: a process whose framework
allocator has reserved nearly all device memory up front, or latency-critical
code that cannot take the device-wide synchronisation of cudaMalloc/cudaFree.
nmv_validate_noalloc serves them from a fixed scratch array in the library and
from output arrays the caller owns.  These tests call it through the C ABI and
check it against nmv_validate, which allocates its workspace as it needs, with
the same tolerance as the oracle parity tests.  Every case runs two calls in a
row, because the scratch keeps the previous call's contents.

The file name sorts last so that a run stopping at the first failure has run
every other test first; the tests also pass alone in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

from _parity import assert_same
from paper_2608_02712_gb300 import NmvError, nmv, validate, validate_noalloc, workloads


def _dev(case):
    return {k: (v.cuda() if isinstance(v, torch.Tensor) else
                [x.cuda() for x in v] if k == "inputs" else v) for k, v in case.items()}


def _both(case):
    args = dict(inputs=case["inputs"], rtol=case["rtol"], atol=case["atol"], tile=case["tile"],
                first_k=case["first_k"])
    want = validate(case["cand"], case["ref"], **args)
    first = validate_noalloc(case["cand"], case["ref"], **args)
    second = validate_noalloc(case["cand"], case["ref"], **args)
    return want, first, second


def _cases():
    yield workloads.c1()
    yield workloads.c2(shape=(2, 512, 640))
    yield workloads.c4(numel=(1 << 20) + 37)
    yield workloads.c5(shape=(512, 1024), first_k=4096)
    for seed in (3, 11, 29, 57):
        yield workloads.fuzz(seed)


@pytest.mark.gpu
@pytest.mark.parametrize("case", list(_cases()), ids=lambda c: c["name"])
def test_noalloc_matches_validate_twice(case):
    case = _dev(case)
    want, first, second = _both(case)
    assert_same(first, want, case["name"] + " (first call)")
    assert_same(second, want, case["name"] + " (second call)")


@pytest.mark.gpu
def test_noalloc_after_a_different_case():
    # A larger case with many mismatches leaves maps and records in the
    # scratch; a clean case right after must not see any of them.
    dirty = _dev(workloads.c1())
    validate_noalloc(dirty["cand"], dirty["ref"], rtol=dirty["rtol"], atol=dirty["atol"],
                     tile=dirty["tile"], first_k=dirty["first_k"])
    ref = torch.randn(300, 257, device="cuda")
    got = validate_noalloc(ref.clone(), ref, rtol=1e-5, atol=1e-8, tile=(64, 64), first_k=16)
    want = validate(ref.clone(), ref, rtol=1e-5, atol=1e-8, tile=(64, 64), first_k=16)
    assert_same(got, want, "clean after dirty")
    assert got["mismatch"] == 0 and got["tile_hist"].sum() == 0 and got["k_out"] == 0


@pytest.mark.gpu
def test_noalloc_rejects_a_case_beyond_the_scratch():
    x = torch.zeros(2048, 2048, device="cuda")
    # 2048 x 2048 one-element tiles: 32 MiB of histogram alone
    with pytest.raises(NmvError) as e:
        validate_noalloc(x, x, rtol=0.0, atol=0.0, tile=(1, 1), first_k=0)
    assert e.value.status == nmv.NMV_EINVAL
    assert "scratch" in str(e.value)
    # nmv_validate has no such limit
    assert validate(x, x, rtol=0.0, atol=0.0, tile=(1, 1), first_k=0)["pass"]


def test_noalloc_requires_caller_arrays():
    lib = nmv.load()
    shape = (ctypes.c_int64 * 1)(16)
    buf = (ctypes.c_float * 16)()
    t = nmv.Tensor(ctypes.cast(buf, ctypes.c_void_p), 0, 1, ctypes.cast(shape, ctypes.POINTER(ctypes.c_int64)))
    c = nmv.Case()
    c.cand = t
    c.ref = nmv.Tensor(t.data, t.dtype, t.rank, t.shape)
    c.rtol, c.atol = 1e-5, 1e-8
    c.tile_rows, c.tile_cols, c.first_k = 1, 4, 2
    r = nmv.Result()  # no arrays set
    assert lib.nmv_validate_noalloc(ctypes.byref(c), None, ctypes.byref(r)) == nmv.NMV_EINVAL
    assert b"caller arrays" in lib.nmv_last_error()
    assert lib.nmv_validate_noalloc(None, None, ctypes.byref(r)) == nmv.NMV_EINVAL
    assert lib.nmv_validate_noalloc(ctypes.byref(c), None, None) == nmv.NMV_EINVAL
