"""Pins for the oracle's full-coverage escalation (oracle.sweep): the
escalation decision, the acceptance rule and the evidence record, on tiny
hand-built case sets whose records are written out by hand."""
import hashlib

import torch

import oracle


def _case(c, r, rtol=1e-3, atol=0.0, inputs=()):
    return {"cand": torch.tensor(c, dtype=torch.float32), "ref": torch.tensor(r, dtype=torch.float32),
            "inputs": list(inputs), "rtol": rtol, "atol": atol, "tile": (1, 2), "first_k": 0}


def test_escalates_only_after_a_clean_light_set():
    good = _case([1.0, 2.0], [1.0, 2.0])
    bad = _case([1.0, 3.0], [1.0, 2.0])
    rep = oracle.sweep([good, bad], [good])
    assert not rep["escalated"] and not rep["accepted"] and rep["n_run"] == 2
    assert rep["n_pass_light"] == 1 and rep["match_rate_light"] == 0.5 and rep["match_rate_ext"] == 0.0
    rep = oracle.sweep([good], [good, bad])
    assert rep["escalated"] and not rep["accepted"] and rep["n_run"] == 3 and rep["n_pass_ext"] == 1
    rep = oracle.sweep([good], [good, good])
    assert rep["escalated"] and rep["accepted"] and rep["match_rate_ext"] == 1.0
    rep = oracle.sweep([good])
    assert not rep["escalated"] and rep["accepted"]


def test_integrity_hazard_blocks_acceptance():
    x = torch.tensor([1.0, 2.0, 3.0, 4.0])
    passthrough = {"cand": x.clone(), "ref": x * (1 + 1e-7), "inputs": [x], "rtol": 1e-5, "atol": 0.0,
                   "tile": (1, 4), "first_k": 0}
    rep = oracle.sweep([passthrough])
    assert rep["results"][0]["pass"] and rep["flags_any"] & 1 and not rep["accepted"]
    zeros = _case([0.0, 0.0], [0.0, 1e-9], atol=1e-6)          # all-zero candidate, reference not
    rep = oracle.sweep([zeros])
    assert rep["results"][0]["pass"] and not rep["accepted"]
    both = _case([0.0, 0.0], [0.0, 0.0])                       # all zero on both sides: no hazard
    assert oracle.sweep([both])["accepted"]


def test_evidence_record_by_hand():
    good = _case([1.0, 2.0], [1.0, 2.0])
    bad = _case([1.0, 3.0], [1.0, 2.0])
    rep = oracle.sweep([good], [bad])
    want = ("nmv-sweep v1 light=1 ext=1 escalated=1 accepted=0 pass_light=1 pass_ext=0\n"
            "L 0 dtype=0 numel=2 pass=1 mismatch=0 match=1 max_abs=0 max_rel=0 nonfinite=0 flags=0\n"
            "E 0 dtype=0 numel=2 pass=0 mismatch=1 match=0.5 max_abs=1 max_rel=0.5 nonfinite=0 flags=0\n")
    assert rep["evidence"] == want
    assert rep["digest"] == hashlib.sha256(want.encode()).hexdigest()
