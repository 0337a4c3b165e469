"""The edge-case generator reaches what it claims (CPU only): every family,
the pre-filter's switch-off tolerances, differences on both sides of |r|/4,
subnormal references, and plan edges (big tiles, wide tile grids)."""
import math

import torch

from paper_2608_02712_gb300 import workloads as W


def test_ulp_step_matches_nextafter():
    for dt in (torch.float32, torch.float16, torch.bfloat16):
        x = torch.tensor([0.0, -0.0, 1.0, -1.0, 3.5, -2.25, 1e-30, -1e-30], dtype=torch.float32).to(dt)
        up = W._ulp_step(x, torch.ones(x.shape, dtype=torch.int64))
        dn = W._ulp_step(x, -torch.ones(x.shape, dtype=torch.int64))
        inf = torch.full_like(x, float("inf"))
        assert torch.equal(up, torch.nextafter(x.float(), inf.float()).to(dt)) or dt != torch.float32
        for a, b, c in zip(x.tolist(), up.tolist(), dn.tolist()):
            assert b > a and c < a
        # two steps up then two down is the identity away from zero
        y = W._ulp_step(W._ulp_step(x, torch.full(x.shape, 2)), torch.full(x.shape, -2))
        nz = x != 0
        assert torch.equal(y[nz], x[nz])


def test_edge_families_reach_their_edges():
    fams = {}
    for s in range(60):
        c = W.edge(s)
        fam = c["name"].split("_")[2]
        if fam in ("global", "big"):
            fam = "_".join(c["name"].split("_")[2:4])
        fams.setdefault(fam, []).append(c)
    assert set(fams) == set(W.EDGE_FAMILIES)
    tol = fams["tolerance"]
    assert any(c["rtol"] > 0.5 for c in tol) and any(c["atol"] > 2.0 ** 100 for c in tol)
    assert any(c["rtol"] == 0.25 for c in tol + fams["sterbenz"])
    # sterbenz: planted differences on both sides of |r| / 4
    below = above = 0
    for c in fams["sterbenz"]:
        r, d = c["ref"].double(), (c["cand"].double() - c["ref"].double()).abs()
        fin = torch.isfinite(r) & torch.isfinite(d) & (r != 0)
        q = (d[fin] / r[fin].abs())
        below += int(((q > 0.24) & (q <= 0.25)).sum())
        above += int(((q > 0.25) & (q < 0.26)).sum())
    assert below > 0 and above > 0
    # subnormal references
    for c in fams["subnormal"]:
        r = c["ref"].float().abs()
        tiny = torch.finfo(c["ref"].dtype).tiny
        assert ((r > 0) & (r < tiny)).float().mean() > 0.9
    assert any(max(c["tile"]) > 4096 for c in fams["big_tiles"])
    for c in fams["global_hist"]:
        m, n = c["cand"].shape
        assert math.ceil(n / c["tile"][1]) * c["tile"][0] > 8192 or math.ceil(n / c["tile"][1]) > 8192 \
            or math.ceil(m / c["tile"][0]) * math.ceil(n / c["tile"][1]) > 8192
    assert all(c["cand"].numel() >= 1_900_000 for c in fams["large"])
