"""Pins for the oracle's diagnostic tensor statistics (oracle.stats): closed
forms of arithmetic sequences and constants, special-value tables, and an
independent numpy brute force (np.isnan / np.isinf masks, np.min / np.max,
math.fsum for the sums, the tile grid by reshaping) on random tensors."""
import math

import numpy as np
import pytest
import torch

from paper_2608_02712_gb300 import workloads


def brute_stats(x, tile):
    """numpy restatement: returns (whole-tensor dict, per-tile dicts)."""
    shape = tuple(x.shape)
    v = x.double().reshape(-1).numpy() if x.dtype != torch.int32 else x.reshape(-1).numpy().astype(np.int64)
    numel = v.size
    m, n = (1, 1) if len(shape) == 0 else (int(np.prod(shape[:-1], dtype=np.int64)), shape[-1])
    th, tw = tile

    def one(vals, is_int):
        if is_int:
            fin = np.ones(vals.size, bool)
            cnt = [vals.size, 0, 0, 0, int((vals == 0).sum())]
            ints = [int(t) for t in vals.tolist()]
            s, q = float(sum(ints)), float(sum(t * t for t in ints))   # exact, one rounding
            f = vals.astype(np.float64)
        else:
            fin = np.isfinite(vals)
            cnt = [int(fin.sum()), int(np.isnan(vals).sum()), int(np.isposinf(vals).sum()),
                   int(np.isneginf(vals).sum()), int((vals == 0).sum())]
            f = vals[fin]
            s, q = math.fsum(f.tolist()), math.fsum((f * f).tolist())
        out = dict(zip(("n_finite", "n_nan", "n_posinf", "n_neginf", "n_zero"), cnt))
        if cnt[0]:
            mean = s / cnt[0]
            var = q / cnt[0] - mean * mean
            out.update(min=float(f.min()), max=float(f.max()), sum=s, sumsq=q, mean=mean,
                       std=math.sqrt(var) if var > 0 else 0.0)
        else:
            out.update(min=0.0, max=0.0, sum=0.0, sumsq=0.0, mean=0.0, std=0.0)
        return out

    is_int = x.dtype == torch.int32
    whole = one(v, is_int)
    gr = -(-m // th) if numel else 0
    gc = -(-n // tw) if numel else 0
    tiles = {}
    if numel:
        grid = v.reshape(m, n)
        for tr in range(gr):
            for tc in range(gc):
                tiles[(tr, tc)] = one(grid[tr * th:(tr + 1) * th, tc * tw:(tc + 1) * tw].reshape(-1), is_int)
    if is_int or numel == 0:
        fn = fi = -1
    else:
        nan_at, inf_at = np.flatnonzero(np.isnan(v)), np.flatnonzero(np.isinf(v))
        fn = int(nan_at[0]) if nan_at.size else -1
        fi = int(inf_at[0]) if inf_at.size else -1
    return whole, tiles, fn, fi


COUNTS = ("n_finite", "n_nan", "n_posinf", "n_neginf", "n_zero")


def close(a, b, scale, rel=1e-12):
    return a == b or abs(a - b) <= rel * scale


def check_stat(got, want, what):
    for k in COUNTS:
        assert got[k] == want[k], (what, k, got[k], want[k])
    for k in ("min", "max"):
        assert got[k] == want[k], (what, k, got[k], want[k])
    # the oracle's Neumaier sums against exactly rounded sums; mean and std
    # follow from them through the same formula
    assert close(got["sumsq"], want["sumsq"], abs(want["sumsq"])), (what, got["sumsq"], want["sumsq"])
    scale = max(abs(want["min"]), abs(want["max"])) * max(want["n_finite"], 1)
    assert close(got["sum"], want["sum"], scale), (what, got["sum"], want["sum"])
    assert close(got["mean"], want["mean"], scale / max(want["n_finite"], 1)), (what, "mean")
    n = max(want["n_finite"], 1)
    var_g, var_w = got["std"] ** 2, want["std"] ** 2
    assert abs(var_g - var_w) <= 1e-9 * want["sumsq"] / n + 1e-300, (what, "std", got["std"], want["std"])


def check_all(res, x, tile):
    whole, tiles, fn, fi = brute_stats(x, tile)
    check_stat(res["all"], whole, "all")
    assert (res["first_nan"], res["first_inf"]) == (fn, fi)
    gr, gc = res["grid_rows"], res["grid_cols"]
    assert gr * gc == len(tiles)
    for (tr, tc), w in tiles.items():
        got = {k: res["tiles"][k][tr, tc] for k in res["tiles"]}
        got = {k: (int(v) if k in COUNTS else float(v)) for k, v in got.items()}
        check_stat(got, w, "tile %d,%d" % (tr, tc))


@pytest.mark.parametrize("seed", range(120))
def test_stats_fuzz_against_brute_force(oracle_lib, seed):
    x, tile = workloads.stats_fuzz(seed)
    check_all(oracle_lib.stats(x, tile=tile), x, tile)


@pytest.mark.parametrize("dt", [torch.int32, torch.float32])
def test_stats_arithmetic_sequence(oracle_lib, dt):
    """x = 0, 1, ..., n-1: sum n(n-1)/2, sumsq (n-1)n(2n-1)/6, mean (n-1)/2,
    population std sqrt((n^2 - 1)/12); as tiles of 10 the sequence's pieces."""
    n = 10_000
    x = torch.arange(n, dtype=dt)
    res = oracle_lib.stats(x, tile=(1, 10))
    a = res["all"]
    assert a["n_finite"] == n and a["n_zero"] == 1 and a["min"] == 0 and a["max"] == n - 1
    assert a["sum"] == n * (n - 1) / 2 and a["sumsq"] == (n - 1) * n * (2 * n - 1) / 6
    assert a["mean"] == (n - 1) / 2
    assert abs(a["std"] - math.sqrt((n * n - 1) / 12)) <= 1e-12 * a["std"]
    assert res["grid_rows"] == 1 and res["grid_cols"] == n // 10
    t = res["tiles"]
    for j in (0, 7, n // 10 - 1):
        lo = 10 * j
        assert t["min"][0, j] == lo and t["max"][0, j] == lo + 9
        assert t["sum"][0, j] == 10 * lo + 45 and t["mean"][0, j] == lo + 4.5
        assert abs(t["std"][0, j] - math.sqrt(99 / 12)) <= 1e-9
    assert t["n_zero"][0, 0] == 1 and t["n_zero"][0, 1:].sum() == 0


def test_stats_constant_and_specials(oracle_lib):
    x = torch.full((6, 8), 3.0)
    res = oracle_lib.stats(x, tile=(3, 4))
    a = res["all"]
    assert (a["min"], a["max"], a["mean"], a["std"], a["sum"], a["sumsq"]) == (3.0, 3.0, 3.0, 0.0, 144.0, 432.0)
    assert (res["grid_rows"], res["grid_cols"]) == (2, 2)
    assert (res["tiles"]["n_finite"] == 12).all() and (res["tiles"]["std"] == 0).all()
    y = torch.tensor([[0.0, -0.0, float("nan"), 2.0],
                      [float("inf"), -1.0, float("-inf"), float("nan")]])
    res = oracle_lib.stats(y, tile=(1, 2))
    a = res["all"]
    assert (a["n_finite"], a["n_nan"], a["n_posinf"], a["n_neginf"], a["n_zero"]) == (4, 2, 1, 1, 2)
    assert (a["min"], a["max"], a["sum"], a["sumsq"]) == (-1.0, 2.0, 1.0, 5.0)
    assert (res["first_nan"], res["first_inf"]) == (2, 4)
    t = res["tiles"]
    assert t["n_zero"].tolist() == [[2, 0], [0, 0]]
    assert t["n_nan"].tolist() == [[0, 1], [0, 1]]
    assert t["n_posinf"].tolist() == [[0, 0], [1, 0]] and t["n_neginf"].tolist() == [[0, 0], [0, 1]]
    assert t["min"].tolist() == [[0.0, 2.0], [-1.0, 0.0]]     # the last tile holds no finite value
    assert t["max"].tolist() == [[0.0, 2.0], [-1.0, 0.0]]
    assert t["mean"].tolist() == [[0.0, 2.0], [-1.0, 0.0]]


def test_stats_empty_and_rank0(oracle_lib):
    res = oracle_lib.stats(torch.zeros(0, 5), tile=(2, 2))
    assert res["grid_rows"] == res["grid_cols"] == 0 and res["all"]["n_finite"] == 0
    assert res["first_nan"] == res["first_inf"] == -1 and res["all"]["std"] == 0.0
    res = oracle_lib.stats(torch.tensor(float("nan")), tile=(4, 4))
    assert res["all"]["n_nan"] == 1 and res["first_nan"] == 0 and res["grid_rows"] == res["grid_cols"] == 1


def test_stats_int32_sums_are_exact(oracle_lib):
    """int32 extremes: the exact sums differ from a plain fp64 accumulation."""
    x = torch.tensor([2 ** 31 - 1] * 3 + [-(2 ** 31)] * 2 + [1], dtype=torch.int32)
    a = oracle_lib.stats(x, tile=(1, 6))["all"]
    ints = [int(t) for t in x.tolist()]
    assert a["sum"] == float(sum(ints)) and a["sumsq"] == float(sum(t * t for t in ints))


def test_stats_float_sums_are_compensated(oracle_lib):
    """Terms far below the running sum's ulp: a plain left-to-right fp64 sum
    loses every 1.0 next to 1e20; the compensated sums keep them."""
    x = torch.tensor([1e20] + [1.0] * 4000 + [-1e20], dtype=torch.float32)
    a = oracle_lib.stats(x, tile=(1, 1))["all"]
    assert a["sum"] == 4000.0
    assert a["sumsq"] == math.fsum((x.double() ** 2).tolist())
    plain = 0.0
    for t in x.double().tolist():
        plain += t
    assert plain != 4000.0
