"""Pins of the oracle against closed forms of the planted workloads.  Each
workload plants faults whose count, positions and statistics follow from the
recipe alone (not from running any validator), at full size where the CPU
finishes in seconds and at reduced size otherwise."""
import numpy as np
import pytest
import torch

from paper_2608_02712_gb300 import workloads


def run(oracle_lib, case):
    return oracle_lib.validate(case["cand"], case["ref"], inputs=case["inputs"],
                               rtol=case["rtol"], atol=case["atol"], tile=case["tile"],
                               first_k=case["first_k"])


@pytest.mark.parametrize("numel", [1 << 16, 1 << 20])
def test_c4_closed_form(oracle_lib, numel):
    case = workloads.c4(numel=numel)
    res = run(oracle_lib, case)
    blocks = numel // 4096
    assert res["mismatch"] == blocks * 32
    assert res["max_abs"] == 1.0 and res["argmax_abs"] == 4064
    assert res["sse"] == float(blocks * 32)           # integer terms: exact
    assert res["grid_rows"] == 1 and res["grid_cols"] == blocks
    assert (res["tile_hist"] == 32).all()
    want_col = np.zeros(4096, np.int64)
    want_col[4064:] = blocks
    assert np.array_equal(res["col_prof"], want_col)
    assert res["row_prof"].tolist() == [blocks * 32]
    k = min(4096, blocks * 32)
    want_fk = np.array([t * 4096 + 4064 + j for t in range(blocks) for j in range(32)])[:k]
    assert np.array_equal(res["fk_index"], want_fk)
    assert np.array_equal(res["fk_coords"][:, 0], want_fk)
    assert (res["fk_cand"] - res["fk_ref"] == 1.0).all()
    assert res["flags"] == 0 and res["n_finite_pairs"] == numel
    assert res["cand_nan"] == res["cand_posinf"] == res["cand_neginf"] == 0
    # max_rel = 1 / min{ r_i != 0 : i mismatching }, lowest index on ties
    r = case["ref"].numpy().astype(np.int64)
    bad = np.flatnonzero(np.arange(numel) % 4096 >= 4064)
    rb = r[bad]
    nz = rb != 0
    rmin = rb[nz].min()
    assert res["max_rel"] == 1.0 / float(rmin)
    assert res["argmax_rel"] == int(bad[nz][np.argmax(rb[nz] == rmin)])


def test_c1_closed_form(oracle_lib):
    case = workloads.c1()
    res = run(oracle_lib, case)
    assert res["cand_nan"] == 4 and res["cand_posinf"] == 2 and res["cand_neginf"] == 0
    assert res["ref_nan"] == res["ref_posinf"] == res["ref_neginf"] == 0
    # rebuild the planted set P from the recipe alone
    m, n = workloads.C1_SHAPE
    g = torch.Generator().manual_seed(0)
    torch.randn(m, n, generator=g)
    torch.randn(m, n, generator=g)
    rand_idx = set(torch.randperm(m * n, generator=g)[:1049].tolist())
    zero = {i * n + j for i in range(512, 768) for j in range(n) if j % 64 >= 56}
    specials = {i * n + j for (i, j) in workloads.C1_NAN_AT + workloads.C1_INF_AT}
    P = rand_idx | zero | specials
    assert len(zero) == 32768
    # elements outside P carry relative noise 1e-6 against rtol 1e-3: all pass,
    # so the mismatch set is P minus the planted elements that happen to pass
    # (decided on P alone).
    Pl = np.array(sorted(P))
    c = case["cand"].reshape(-1)[Pl].double()
    r = case["ref"].reshape(-1)[Pl].double()
    passing = torch.isclose(c, r, rtol=1e-3, atol=1e-5).numpy()
    want_bad = Pl[~passing]
    assert res["mismatch"] == want_bad.size
    assert np.array_equal(res["fk_index"], want_bad[:256])
    # the zeroed band dominates columns 56..63 of each 64-wide tile
    assert (res["col_prof"][56:] >= 4096 - 2).all()
    assert (res["col_prof"][:56] < 100).all()
    assert (res["tile_hist"][8:12, :] >= 510).all()
    assert (res["row_prof"] > 0).all()


@pytest.mark.parametrize("shape", [(1, 1024, 4096), (2, 256, 1000)])
def test_c2_closed_form(oracle_lib, shape):
    case = workloads.c2(shape=shape)
    res = run(oracle_lib, case)
    n = shape[-1]
    m = int(np.prod(shape[:-1]))
    gc = -(-n // 128)
    c0 = (gc - 1) * 128
    rows = np.arange(m)
    odd = ((rows // 128) % 2) == 1
    fault = np.zeros((m, n), bool)
    fault[np.ix_(odd, np.arange(c0, n))] = True
    n_fault = int(fault.sum())
    # every planted element is far outside tolerance: |delta| >= 0.5 - bf16
    # rounding (<= 2^-6 below |x| < 8) - noise, versus atol + rtol * 4 < 0.066
    assert res["mismatch"] >= n_fault
    extras = res["mismatch"] - n_fault
    assert extras <= 2
    gr = -(-m // 128)
    want = np.zeros((gr, gc), np.int64)
    for t in range(gr):
        if t % 2 == 1:
            want[t, gc - 1] = int(odd[t * 128:(t + 1) * 128].sum()) * (n - c0)
    if extras == 0:
        assert np.array_equal(res["tile_hist"], want)
        first = np.flatnonzero(fault.reshape(-1))[:1024]
        assert np.array_equal(res["fk_index"], first)
    assert res["flags"] == 0


def test_c5_closed_form_reduced(oracle_lib):
    shape = (256, 1024)
    case = workloads.c5(shape=shape, first_k=4096)
    res = run(oracle_lib, case)
    numel = shape[0] * shape[1]
    half = numel // 2
    assert res["cand_nan"] == 1074 and res["cand_neginf"] == 1073
    assert res["cand_posinf"] == 0
    # rebuild S from the recipe
    gs = torch.Generator().manual_seed(4)
    draws = torch.randint(0, numel, (4096,), generator=gs).tolist()
    S = []
    for d in draws:
        if d not in S:
            S.append(d)
    S = S[:2147]
    s_first = sum(1 for s in S if s < half)
    x = case["inputs"][0].numpy().view(np.int32)
    r = case["ref"].reshape(-1).numpy().view(np.int32)
    coincide = int((x[:half] == r[:half]).sum())
    assert res["input_eq"].tolist() == [half - s_first - coincide]
    assert res["flags"] & 1 and res["passthrough_input"] == 0
    # second half: mismatches are exactly the planted specials there
    bad = res["fk_index"]
    assert bad[0] < 16
    assert res["k_out"] == 4096


def test_c3_closed_form_reduced(oracle_lib):
    cases = workloads.c3(count=24, cap=50000)
    for i, case in enumerate(cases):
        res = run(oracle_lib, case)
        n = case["cand"].numel()
        if i % 2 == 0:
            assert res["mismatch"] == 0, case["name"]
            continue
        kind = ("tail", "signflip", "scale")[(i // 2) % 3]
        if kind == "tail":
            L = min(n, 64)
            assert res["mismatch"] == L
            assert np.array_equal(res["fk_index"], np.arange(n - L, n))
        elif kind == "signflip":
            rf = case["ref"].reshape(-1).float()
            big = (rf.abs() >= 0.5).nonzero()
            if big.numel():
                assert res["mismatch"] == 1
                assert res["fk_index"].tolist() == [int(big[0])]
