"""Pins for P2-P6 of the oracle against vectorised numpy/torch brute force on
small random cases: torch.isclose decides the pass mask, np.argmax (first
occurrence) the argmax, math.fsum the exactly rounded sum of squares,
np.add.at / np.bincount the localisation maps, np.flatnonzero the first-K."""
import math

import numpy as np
import pytest
import torch

from paper_2608_02712_gb300 import workloads

_IV = {torch.float32: torch.int32, torch.float16: torch.int16,
       torch.bfloat16: torch.int16, torch.int32: torch.int32}


def brute(case):
    cand, ref = case["cand"], case["ref"]
    rtol, atol = case["rtol"], case["atol"]
    th, tw = case["tile"]
    k = case["first_k"]
    shape = tuple(cand.shape)
    c = cand.double().reshape(-1).numpy()
    r = ref.double().reshape(-1).numpy()
    n = c.size
    ok = torch.isclose(torch.from_numpy(c), torch.from_numpy(r), rtol=rtol, atol=atol,
                       equal_nan=False).numpy()
    bad = np.flatnonzero(~ok)
    m2, n2 = (1, 1) if len(shape) == 0 else (int(np.prod(shape[:-1], dtype=np.int64)), shape[-1])
    ncols = max(n2, 1)
    rows, cols = bad // ncols, bad % ncols
    gr = -(-m2 // th) if n else 0
    gc = -(-n2 // tw) if n else 0
    hist = np.zeros((gr, gc), np.int64)
    np.add.at(hist, (rows // th, cols // tw), 1)
    out = {
        "mismatch": bad.size,
        "cand_nan": int(np.isnan(c).sum()), "cand_posinf": int(np.isposinf(c).sum()),
        "cand_neginf": int(np.isneginf(c).sum()), "ref_nan": int(np.isnan(r).sum()),
        "ref_posinf": int(np.isposinf(r).sum()), "ref_neginf": int(np.isneginf(r).sum()),
        "tile_hist": hist,
        "row_prof": np.bincount(rows % th, minlength=th).astype(np.int64),
        "col_prof": np.bincount(cols % tw, minlength=tw).astype(np.int64),
        "fk_index": bad[:k],
    }
    fin = np.isfinite(c) & np.isfinite(r)
    out["n_finite_pairs"] = int(fin.sum())
    fidx = np.flatnonzero(fin)
    d = c[fin] - r[fin]
    a = np.abs(d)
    if fidx.size:
        j = int(np.argmax(a))
        out["max_abs"], out["argmax_abs"] = float(a[j]), int(fidx[j])
        out["sse"] = math.fsum((d * d).tolist())
    else:
        out["max_abs"], out["argmax_abs"], out["sse"] = 0.0, -1, 0.0
    nz = r[fin] != 0
    if nz.any():
        rel = a[nz] / np.abs(r[fin][nz])
        j = int(np.argmax(rel))
        out["max_rel"], out["argmax_rel"] = float(rel[j]), int(fidx[nz][j])
    else:
        out["max_rel"], out["argmax_rel"] = 0.0, -1
    # P6 from bit views
    cb = cand.reshape(-1).view(_IV[cand.dtype]).numpy().astype(np.int64)
    rb = ref.reshape(-1).view(_IV[ref.dtype]).numpy().astype(np.int64)
    flags = 0
    eq = []
    thr = max(1, -(-n // 100))
    pt = -1
    for j, x in enumerate(case["inputs"]):
        if x.dtype != cand.dtype or x.numel() != n:
            eq.append(-1)
            continue
        xb = x.reshape(-1).view(_IV[x.dtype]).numpy().astype(np.int64)
        e = int(((cb == xb) & (rb != xb)).sum())
        eq.append(e)
        if e >= thr:
            flags |= 1
            if pt < 0:
                pt = j
    if n >= 1 and (c == 0).all():
        flags |= 2
    if n >= 2 and (cb == cb[0]).all():
        flags |= 4
    if n >= 1 and (r == 0).all():
        flags |= 8
    if n >= 2 and (rb == rb[0]).all():
        flags |= 16
    out["flags"], out["input_eq"], out["passthrough_input"] = flags, np.array(eq, np.int64), pt
    out["fk_cand"], out["fk_ref"] = c[bad[:k]], r[bad[:k]]
    return out


def _eq_f64(a, b):
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    both_nan = np.isnan(a) & np.isnan(b)
    return bool(((a.view(np.int64) == b.view(np.int64)) | both_nan).all())


def check_against_brute(res, want):
    for key in ("mismatch", "cand_nan", "cand_posinf", "cand_neginf", "ref_nan",
                "ref_posinf", "ref_neginf", "n_finite_pairs", "argmax_abs", "argmax_rel",
                "flags", "passthrough_input"):
        assert res[key] == want[key], key
    for key in ("max_abs", "max_rel"):
        assert _eq_f64(res[key], want[key]), (key, res[key], want[key])
    assert abs(res["sse"] - want["sse"]) <= 1e-13 * abs(want["sse"]), (res["sse"], want["sse"])
    for key in ("tile_hist", "row_prof", "col_prof", "fk_index", "input_eq"):
        assert np.array_equal(res[key], want[key]), key
    assert _eq_f64(res["fk_cand"], want["fk_cand"])
    assert _eq_f64(res["fk_ref"], want["fk_ref"])


@pytest.mark.parametrize("seed", range(160))
def test_fuzz_against_brute_force(oracle_lib, seed):
    case = workloads.fuzz(seed)
    res = oracle_lib.validate(case["cand"], case["ref"], inputs=case["inputs"],
                              rtol=case["rtol"], atol=case["atol"], tile=case["tile"],
                              first_k=case["first_k"])
    check_against_brute(res, brute(case))
    assert res["pass"] == (res["mismatch"] == 0)
    if res["k_out"]:
        assert np.array_equal(
            np.ravel_multi_index(tuple(res["fk_coords"].T), tuple(case["cand"].shape))
            if case["cand"].dim() else np.zeros(res["k_out"], np.int64),
            res["fk_index"])


@pytest.mark.parametrize("seed", range(6))
def test_c3_shaped_cases_against_brute_force(oracle_lib, seed):
    for case in workloads.c3(seed=seed, count=6, cap=20000):
        res = oracle_lib.validate(case["cand"], case["ref"], rtol=case["rtol"],
                                  atol=case["atol"], tile=case["tile"],
                                  first_k=case["first_k"])
        check_against_brute(res, brute(case))


def test_sse_is_compensated(oracle_lib):
    """Terms of wildly different magnitude: a plain left-to-right fp64 sum
    loses the small terms; Neumaier's sum must equal math.fsum here."""
    c = torch.tensor([1e8] + [1.0] * 4000 + [-1e8], dtype=torch.float32)
    r = torch.zeros_like(c)
    res = oracle_lib.validate(c, r, rtol=0.0, atol=0.0, tile=(1, 1), first_k=0)
    terms = (c.double() ** 2).tolist()
    assert res["sse"] == math.fsum(terms)
    plain = 0.0
    for t in terms:
        plain += t
    assert plain != math.fsum(terms)
