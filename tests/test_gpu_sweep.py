"""GPU parity of the full-coverage escalation (nmv_sweep through the C ABI)
with the oracle's policy: the escalation decision, acceptance, pass counts,
match rates, the evidence record byte for byte, its SHA-256 digest, and every
per-case result."""
import pytest
import torch

import oracle
from _parity import assert_same
from paper_2608_02712_gb300 import sweep, workloads

pytestmark = pytest.mark.gpu


def _dev(cases):
    return [dict(c, cand=c["cand"].cuda(), ref=c["ref"].cuda(), inputs=[x.cuda() for x in c["inputs"]])
            for c in cases]


def _check(light, ext):
    got = sweep(_dev(light), _dev(ext))
    want = oracle.sweep(light, ext)
    for k in ("escalated", "accepted", "flags_any", "n_light", "n_ext", "n_run", "n_pass_light", "n_pass_ext",
              "match_rate_light", "match_rate_ext", "evidence", "digest"):
        assert got[k] == want[k], (k, got[k], want[k])
    for g, w in zip(got["results"], want["results"]):
        assert_same(g, w, "sweep case")
    return got


def _clean(n, seed):
    out = []
    for c in workloads.c3(seed=seed, count=2 * n, cap=1 << 16)[0::2]:   # even cases are clean
        out.append(c)
    return out


def test_sweep_escalates_and_rejects_a_faulted_extended_set():
    light = _clean(6, 7)
    ext = workloads.c3(seed=8, count=48, cap=1 << 18)
    rep = _check(light, ext)
    assert rep["escalated"] and not rep["accepted"] and 0 < rep["n_pass_ext"] < 48


def test_sweep_stops_after_a_failing_light_set():
    light = _clean(5, 9) + [workloads.c3(seed=9, count=2, cap=1 << 16)[1]]   # a faulted case
    rep = _check(light, workloads.c3(seed=10, count=8, cap=1 << 16))
    assert not rep["escalated"] and rep["n_run"] == len(light)


def test_sweep_accepts_clean_sets():
    rep = _check(_clean(4, 11), _clean(20, 12))
    assert rep["escalated"] and rep["accepted"] and rep["match_rate_ext"] == 1.0


def test_sweep_integrity_hazard():
    x = torch.randn(4096)
    passthrough = {"cand": x.clone(), "ref": x * (1 + 1e-7), "inputs": [x], "rtol": 1e-5, "atol": 0.0,
                   "tile": (1, 64), "first_k": 0, "name": "passthrough"}
    rep = _check(_clean(3, 13) + [passthrough], _clean(3, 14))
    assert rep["escalated"] and not rep["accepted"] and rep["flags_any"] & 1
