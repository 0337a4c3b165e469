"""Pins for the oracle's deep forensics (oracle.forensics): an independent
numpy restatement on random cases (bit views for the ulp distance,
np.frexp for the fp16 spacing, np.maximum.at / np.bincount for the growth
curve and the marginals, torch.isclose for the predicate), hand-built cases
with known answers, and the cumsum case of the paper's Table 1."""
import math

import numpy as np
import pytest
import torch

from paper_2608_02712_gb300 import workloads

_IV = {torch.float32: np.int32, torch.float16: np.int16, torch.bfloat16: np.int16, torch.int32: np.int32}


def ordv(t):
    if t.dtype == torch.int32:
        return t.reshape(-1).numpy().astype(np.int64)
    width = 32 if t.dtype == torch.float32 else 16
    iv = torch.int32 if width == 32 else torch.int16
    b = t.reshape(-1).view(iv).numpy().astype(np.int64) & ((1 << width) - 1)
    sign = b >> (width - 1)
    mag = b & ((1 << (width - 1)) - 1)
    return np.where(sign == 1, -mag, mag)


def brute(cand, ref, rtol, atol, axis, near_ulps, near_fraction, growth_factor):
    with np.errstate(invalid="ignore", over="ignore"):
        return _brute(cand, ref, rtol, atol, axis, near_ulps, near_fraction, growth_factor)


def _brute(cand, ref, rtol, atol, axis, near_ulps, near_fraction, growth_factor):
    shape = tuple(cand.shape)
    rank = len(shape)
    c = cand.double().reshape(-1).numpy()
    r = ref.double().reshape(-1).numpy()
    n = c.size
    ok = torch.isclose(torch.from_numpy(c), torch.from_numpy(r), rtol=rtol, atol=atol).numpy()
    fin = np.isfinite(c) & np.isfinite(r)
    u = np.abs(ordv(cand) - ordv(ref))
    bins = np.where(u == 0, 0, np.minimum(np.array([int(v).bit_length() for v in u], np.int64), 33))
    hist = np.bincount(bins[fin], minlength=34).astype(np.int64)
    mis = ~ok
    fm = mis & fin
    if fm.any():
        mu = int(u[fm].max())
        arg = int(np.flatnonzero(fm & (u == mu))[0])
    else:
        mu, arg = -1, -1
    d = np.abs(c - r)
    m, e = np.frexp(np.abs(r))
    sp = np.ldexp(1.0, np.maximum(e - 1, -14) - 10)
    sp = np.where(r == 0, 2.0 ** -24, sp)
    within = int((fm & (d <= sp)).sum())
    nonfin = int((mis & ~fin).sum())
    ax = axis % rank if rank else 0
    length = shape[ax] if rank else 1
    coords = np.unravel_index(np.arange(n), shape) if rank else [np.zeros(n, np.int64)]
    growth = np.zeros(length)
    if rank:
        np.maximum.at(growth, coords[ax][fin], d[fin])
    else:
        growth[:] = d[fin].max() if fin.any() else 0.0
    marg = [np.bincount(coords[a][mis], minlength=shape[a]).astype(np.int64) for a in range(rank)]
    q = max(1, length // 4)
    lo = hi = 0.0
    if length:
        for v in growth[:q]:
            lo += v
        for v in growth[length - q:]:
            hi += v
        lo, hi = lo / q, hi / q
    mismatch = int(mis.sum())
    flags = 0
    if mismatch and not nonfin and mu <= near_ulps and mismatch <= near_fraction * n:
        flags |= 1
    if mismatch and not nonfin and within == mismatch:
        flags |= 2
    if length >= 4 and hi > 0 and hi >= growth_factor * lo:
        flags |= 4
    return {"mismatch": mismatch, "n_finite_pairs": int(fin.sum()), "ulp_hist": hist,
            "max_ulp_mismatch": mu, "argmax_ulp_mismatch": arg, "mism_nonfinite": nonfin,
            "mism_within_f16": within, "flags": flags, "growth": growth,
            "growth_lo": lo, "growth_hi": hi, "marginals": marg}


def check(res, want):
    for k, w in want.items():
        g = res[k]
        if k == "marginals":
            assert len(g) == len(w) and all(np.array_equal(a, b) for a, b in zip(g, w)), k
        elif isinstance(w, np.ndarray):
            assert np.array_equal(np.asarray(g).view(np.int64) if np.asarray(g).dtype == np.float64 else g,
                                  w.view(np.int64) if w.dtype == np.float64 else w), (k, g, w)
        elif isinstance(w, float):
            assert np.float64(g).tobytes() == np.float64(w).tobytes(), (k, g, w)
        else:
            assert g == w, (k, g, w)


def _random_case(seed):
    case = workloads.fuzz(seed)
    g = torch.Generator().manual_seed(seed)
    rank = case["cand"].dim()
    axis = int(torch.randint(-max(rank, 1), max(rank, 1), (1,), generator=g)) if rank else 0
    near_ulps = int(torch.randint(0, 64, (1,), generator=g))
    near_fraction = float(torch.rand(1, generator=g)) * 0.1
    growth = 1.0 + float(torch.rand(1, generator=g)) * 4
    return case, axis, near_ulps, near_fraction, growth


@pytest.mark.parametrize("seed", range(150))
def test_forensics_fuzz_against_brute_force(oracle_lib, seed):
    case, axis, nu, nf, gf = _random_case(seed)
    args = dict(rtol=case["rtol"], atol=case["atol"], axis=axis, near_ulps=nu, near_fraction=nf,
                growth_factor=gf)
    res = oracle_lib.forensics(case["cand"], case["ref"], **args)
    check(res, brute(case["cand"], case["ref"], case["rtol"], case["atol"], axis, nu, nf, gf))


def test_forensics_ulp_distances_by_hand(oracle_lib):
    tiny = float(np.float32(np.frombuffer(np.uint32(1).tobytes(), np.float32)[0]))
    c = torch.tensor([0.0, -0.0, 1.0, tiny, 1.0, 3.0], dtype=torch.float32)
    r = torch.tensor([-0.0, 0.0, float(np.nextafter(np.float32(1), np.float32(2))), -tiny, 1.0, 1.0],
                     dtype=torch.float32)
    res = oracle_lib.forensics(c, r, rtol=0.0, atol=0.0)
    # u: 0, 0, 1, 2 (crossing zero), 0, 3 * 2^22 (1.0 -> 2.0 is 2^23 values,
    # 2.0 -> 3.0 another 2^22), which lies in [2^23, 2^24): bin 24
    h = res["ulp_hist"]
    assert h[0] == 3 and h[1] == 1 and h[2] == 1 and h[24] == 1 and h.sum() == 6
    assert res["mismatch"] == 3 and res["max_ulp_mismatch"] == 3 << 22 and res["argmax_ulp_mismatch"] == 5
    i = torch.tensor([5, -7, 100], dtype=torch.int32)
    res = oracle_lib.forensics(i, torch.tensor([5, 7, 90], dtype=torch.int32), rtol=0.0, atol=0.0)
    assert res["max_ulp_mismatch"] == 14 and res["argmax_ulp_mismatch"] == 1
    assert res["ulp_hist"][0] == 1 and res["ulp_hist"][4] == 2   # 14 and 10 lie in [8, 16)


def test_forensics_f16_spacing_boundary(oracle_lib):
    """|c - r| exactly one fp16 spacing of r counts as within, the next
    float above does not; r below 2^-14 uses the subnormal spacing 2^-24."""
    r = torch.tensor([1.0, 1.0, 3.0, 1e-6, 0.0], dtype=torch.float32)
    sp = [2.0 ** -10, 2.0 ** -10, 2.0 ** -9, 2.0 ** -24, 2.0 ** -24]
    c = torch.tensor([1.0 + sp[0], float(np.nextafter(np.float32(1.0 + sp[1]), np.float32(2))),
                      3.0 - sp[2], 1e-6 + sp[3], sp[4]], dtype=torch.float32)
    res = oracle_lib.forensics(c, r, rtol=0.0, atol=0.0)
    assert res["mismatch"] == 5 and res["mism_within_f16"] == 4
    assert not res["flags"] & 2
    res = oracle_lib.forensics(c[[0, 2, 3, 4]], r[[0, 2, 3, 4]], rtol=0.0, atol=0.0)
    assert res["flags"] & 2 and res["mism_within_f16"] == res["mismatch"] == 4


def test_forensics_growth_and_marginals_closed_form(oracle_lib):
    """d = (j + 1) * 1e-3 at column j of a [3, 8] pair: growth[j] = that,
    growth_lo = mean of columns 0-1, growth_hi = mean of columns 6-7; every
    element mismatches, so each row marginal is 8 and each column's 3."""
    r = torch.zeros(3, 8)
    d = (torch.arange(8, dtype=torch.float64) + 1) * 1e-3
    c = (r.double() + d).float()
    res = oracle_lib.forensics(c, r, rtol=0.0, atol=0.0, axis=1, growth_factor=4.0)
    want = c[0].double().numpy()
    assert np.array_equal(res["growth"], want)
    assert res["growth_lo"] == (want[0] + want[1]) / 2 and res["growth_hi"] == (want[6] + want[7]) / 2
    assert res["flags"] & 4            # 7.5e-3 >= 4 * 1.5e-3
    assert res["marginals"][0].tolist() == [8, 8, 8] and res["marginals"][1].tolist() == [3] * 8
    res = oracle_lib.forensics(c, r, rtol=0.0, atol=0.0, axis=0)
    assert res["axis_len"] == 3 and not res["flags"] & 4   # fewer than 4 entries


def test_forensics_near_pass(oracle_lib):
    r = torch.randn(1000, generator=torch.Generator().manual_seed(3))
    c = r.clone()
    c[10] = float(np.nextafter(np.float32(c[10]), np.float32(np.inf)))
    c[20] = float(np.nextafter(np.float32(c[20]), np.float32(-np.inf)))
    res = oracle_lib.forensics(c, r, rtol=0.0, atol=0.0, near_ulps=1, near_fraction=0.002)
    assert res["mismatch"] == 2 and res["max_ulp_mismatch"] == 1 and res["flags"] & 1
    assert not oracle_lib.forensics(c, r, rtol=0.0, atol=0.0, near_ulps=0, near_fraction=0.002)["flags"] & 1
    assert not oracle_lib.forensics(c, r, rtol=0.0, atol=0.0, near_ulps=1, near_fraction=0.001)["flags"] & 1
    c[30] = float("nan")
    assert not oracle_lib.forensics(c, r, rtol=0.0, atol=0.0, near_ulps=1, near_fraction=0.01)["flags"] & 1


def test_cumsum_divergence_compounds_along_the_axis(oracle_lib):
    """The cumsum case (Table 1): the pure-FP32 candidate fails against the
    per-step FP16 reference with errors that grow along the scan axis; the
    per-step-rounded candidate (the repair) matches exactly."""
    case = workloads.cumsum_fp16(rows=32, cols=1024)
    res = oracle_lib.forensics(case["cand"], case["ref"], rtol=case["rtol"], atol=case["atol"])
    assert res["mismatch"] > 0 and res["flags"] & 4
    assert res["growth_hi"] > 10 * res["growth_lo"]
    assert res["marginals"][1][-256:].sum() > res["marginals"][1][:256].sum()
    fixed = workloads.cumsum_fp16(rows=32, cols=1024, repaired=True)
    res = oracle_lib.forensics(fixed["cand"], fixed["ref"], rtol=fixed["rtol"], atol=fixed["atol"])
    assert res["mismatch"] == 0 and res["ulp_hist"][0] == 32 * 1024 and res["flags"] == 0
