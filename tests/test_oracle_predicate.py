"""Pins for P1, the pass predicate (the tolerance check tau of Section 3.2,
Eq. 1), against torch.isclose on fp64-upcast tensors (equal_nan=False), at
exact tolerance boundaries and on special-value tables."""
import itertools
import math

import numpy as np
import pytest
import torch

from paper_2608_02712_gb300 import workloads


def _oracle_fail_mask(oracle_lib, cand, ref, rtol, atol):
    n = cand.numel()
    res = oracle_lib.validate(cand, ref, rtol=rtol, atol=atol, tile=(1, 1) if n == 0 else (1, 1),
                              first_k=n)
    mask = np.zeros(n, bool)
    mask[res["fk_index"]] = True
    assert res["mismatch"] == int(mask.sum())
    return mask, res


def _isclose_fail_mask(cand, ref, rtol, atol):
    ok = torch.isclose(cand.double().reshape(-1), ref.double().reshape(-1),
                       rtol=rtol, atol=atol, equal_nan=False)
    return (~ok).numpy()


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16, torch.bfloat16, torch.int32])
@pytest.mark.parametrize("seed", range(6))
def test_matches_torch_isclose_random(oracle_lib, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    n = 5000
    if dtype == torch.int32:
        ref = torch.randint(-50, 50, (n,), generator=g, dtype=torch.int32)
        cand = ref + torch.randint(-3, 4, (n,), generator=g, dtype=torch.int32)
        tols = [(0.0, 0.0), (0.05, 1.0), (0.0, 2.0), (0.5, 0.0)]
    else:
        ref = (torch.randn(n, generator=g) * 10 ** (seed - 2)).to(dtype)
        rel = torch.randn(n, generator=g) * 2e-3
        cand = (ref.float() * (1 + rel)).to(dtype)
        sp = workloads.SPECIALS[dtype]
        idx = torch.randint(0, n, (200,), generator=g)
        cand[idx[:100]] = torch.tensor([sp[i % len(sp)] for i in range(100)], dtype=dtype)
        ref[idx[100:]] = torch.tensor([sp[(3 * i) % len(sp)] for i in range(100)], dtype=dtype)
        tols = [(1e-3, 1e-5), (0.0, 1e-3), (2e-3, 0.0), (0.0, 0.0), (1e-2, 1e-8)]
    for rtol, atol in tols:
        got, _ = _oracle_fail_mask(oracle_lib, cand, ref, rtol, atol)
        want = _isclose_fail_mask(cand, ref, rtol, atol)
        assert (got == want).all(), (rtol, atol, np.nonzero(got != want)[0][:10])


def test_special_value_table(oracle_lib):
    vals = [0.0, -0.0, 1.0, -1.0, float("inf"), float("-inf"), float("nan"), 1e-45, 3.4e38]
    pairs = list(itertools.product(vals, vals))
    c = torch.tensor([p[0] for p in pairs], dtype=torch.float32)
    r = torch.tensor([p[1] for p in pairs], dtype=torch.float32)
    for rtol, atol in [(0.0, 0.0), (1e-3, 1e-5), (1.0, 10.0)]:
        got, _ = _oracle_fail_mask(oracle_lib, c, r, rtol, atol)
        want = _isclose_fail_mask(c, r, rtol, atol)
        assert (got == want).all()
    # hand-checked consequences of P1
    _, res = _oracle_fail_mask(oracle_lib, c, r, 1.0, 10.0)
    fails = set(res["fk_index"].tolist())
    idx = {p: i for i, p in enumerate(pairs) if not any(map(math.isnan, p))}
    assert idx[(float("inf"), float("inf"))] not in fails          # same-sign Inf passes
    assert idx[(float("inf"), float("-inf"))] in fails             # opposite Inf fails
    assert idx[(1.0, float("inf"))] in fails                       # finite vs Inf fails
    assert idx[(0.0, -0.0)] not in fails                           # +0 == -0
    nan_rows = [i for i, p in enumerate(pairs) if any(map(math.isnan, p))]
    assert set(nan_rows) <= fails                                  # NaN never passes


def test_exact_atol_boundary(oracle_lib):
    g = torch.Generator().manual_seed(11)
    c = torch.randn(64, generator=g)
    r = torch.randn(64, generator=g)
    for i in range(64):
        ci, ri = c[i:i + 1], r[i:i + 1]
        d = abs(float(ci.double()) - float(ri.double()))
        ok, _ = _oracle_fail_mask(oracle_lib, ci, ri, 0.0, d)
        assert not ok[0], "boundary equality must pass"
        below = math.nextafter(d, 0.0)
        bad, _ = _oracle_fail_mask(oracle_lib, ci, ri, 0.0, below)
        assert bad[0], "one ulp under the boundary must fail"


def test_exact_rtol_boundary(oracle_lib):
    # |1.5 - 1.0| = 0.5 = 0.5 * |1.0| exactly
    c = torch.tensor([1.5], dtype=torch.float32)
    r = torch.tensor([1.0], dtype=torch.float32)
    ok, _ = _oracle_fail_mask(oracle_lib, c, r, 0.5, 0.0)
    assert not ok[0]
    bad, _ = _oracle_fail_mask(oracle_lib, c, r, math.nextafter(0.5, 0.0), 0.0)
    assert bad[0]
    # asymmetric: the scale is |r|, not |c|
    ok2, _ = _oracle_fail_mask(oracle_lib, r, c, 1.0 / 3.0, 0.0)   # 0.5 <= 0.5
    assert not ok2[0]
    bad2, _ = _oracle_fail_mask(oracle_lib, c, r, 1.0 / 3.0, 0.0)  # 0.5 > 1/3
    assert bad2[0]


def test_no_fused_multiply_add(oracle_lib):
    """fl(atol + fl(rtol*|r|)) differs from the singly rounded atol + rtol*|r|
    for these draws; a candidate exactly at the singly rounded threshold must
    be judged against the two-rounding value."""
    from fractions import Fraction
    rng = np.random.default_rng(5)
    found = 0
    for _ in range(200000):
        r = float(rng.uniform(0.5, 2.0))
        rtol = float(rng.uniform(1e-3, 1e-1))
        atol = float(rng.uniform(1e-3, 1e-1))
        two = atol + rtol * abs(r)
        fused = float(Fraction(atol) + Fraction(rtol) * Fraction(abs(r)))
        if fused == two:
            continue
        c = r + fused
        if c - r != fused or Fraction(c) - Fraction(r) != Fraction(fused):
            continue
        found += 1
        assert oracle_lib.pass_predicate(c, r, rtol, atol) == (fused <= two)
        if found >= 50:
            break
    assert found >= 10
