"""GPU parity of the deep forensics (nmv_forensics, through the C ABI) with
the oracle: every field exact (histogram, counts, the largest ulp distance
and its index, growth curve and means, marginals, flags)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_02712_gb300 import forensics, forensics_batch, workloads

pytestmark = pytest.mark.gpu


def same(got, want, what=""):
    for k, w in want.items():
        g = got[k]
        if k == "marginals":
            assert len(g) == len(w) and all(np.array_equal(a, b) for a, b in zip(g, w)), (what, k)
        elif isinstance(w, np.ndarray):
            if w.dtype == np.float64:
                assert np.array_equal(np.asarray(g).view(np.int64), w.view(np.int64)), (what, k, g, w)
            else:
                assert np.array_equal(g, w), (what, k, g, w)
        elif isinstance(w, float):
            assert np.float64(g).tobytes() == np.float64(w).tobytes(), (what, k, g, w)
        else:
            assert g == w, (what, k, g, w)


def _args(seed, rank):
    g = torch.Generator().manual_seed(seed)
    axis = int(torch.randint(-max(rank, 1), max(rank, 1), (1,), generator=g)) if rank else 0
    return dict(axis=axis, near_ulps=int(torch.randint(0, 64, (1,), generator=g)),
                near_fraction=float(torch.rand(1, generator=g)) * 0.1,
                growth_factor=1.0 + float(torch.rand(1, generator=g)) * 4)


@pytest.mark.parametrize("seed", range(200))
def test_forensics_fuzz_parity(seed):
    case = workloads.fuzz(seed)
    kw = dict(rtol=case["rtol"], atol=case["atol"], **_args(seed, case["cand"].dim()))
    got = forensics(case["cand"].cuda(), case["ref"].cuda(), **kw)
    same(got, oracle.forensics(case["cand"], case["ref"], **kw), case["name"])


@pytest.mark.parametrize("seed", range(0, 120, 4))
def test_forensics_edge_parity(seed):
    case = workloads.edge(seed)
    kw = dict(rtol=case["rtol"], atol=case["atol"], **_args(seed, case["cand"].dim()))
    got = forensics(case["cand"].cuda(), case["ref"].cuda(), **kw)
    same(got, oracle.forensics(case["cand"], case["ref"], **kw), case["name"])


def test_forensics_batch_and_unaligned():
    cases = [workloads.fuzz(s) for s in range(500, 540)]
    shift = lambda t: torch.cat([t.reshape(-1)[:1], t.reshape(-1)]).cuda()[1:].view(t.shape) if t.numel() else t.cuda()
    items = []
    for i, c in enumerate(cases):
        dev = shift if i % 2 else (lambda t: t.cuda())
        items.append(dict(cand=dev(c["cand"]), ref=dev(c["ref"]), rtol=c["rtol"], atol=c["atol"],
                          **_args(i, c["cand"].dim())))
    got = forensics_batch(items)
    for it, c, g in zip(items, cases, got):
        kw = {k: v for k, v in it.items() if k not in ("cand", "ref")}
        same(g, oracle.forensics(c["cand"], c["ref"], **kw), c["name"])


@pytest.mark.parametrize("axis", [0, 1, -1])
def test_forensics_cumsum_case(axis):
    """The cumsum of Table 1: FP32 accumulation against the per-step FP16
    reference diverges along the scan axis (flag AXIS_GROWTH on the last
    axis); the repaired candidate matches."""
    case = workloads.cumsum_fp16(device="cuda", rows=512, cols=4096)
    kw = dict(rtol=case["rtol"], atol=case["atol"], axis=axis)
    got = forensics(case["cand"], case["ref"], **kw)
    same(got, oracle.forensics(case["cand"].cpu(), case["ref"].cpu(), **kw), "cumsum")
    if axis != 0:
        assert got["flags"] & 4 and got["growth_hi"] > 10 * got["growth_lo"]
    fixed = workloads.cumsum_fp16(device="cuda", rows=512, cols=4096, repaired=True)
    got = forensics(fixed["cand"], fixed["ref"], rtol=fixed["rtol"], atol=fixed["atol"], axis=axis)
    assert got["mismatch"] == 0 and got["flags"] == 0


@pytest.mark.parametrize("shape", [(3, 5000, 7), (70000,), (2, 3, 4, 5, 6, 7, 8, 2)])
def test_forensics_large_axes_and_ranks(shape):
    """Axes longer than the shared-memory growth window (2048) and marginal
    sums above the shared-memory marginal window (4096); rank 8."""
    g = torch.Generator(device="cuda").manual_seed(13)
    ref = torch.randn(shape, generator=g, device="cuda")
    cand = ref * (1 + torch.randn(shape, generator=g, device="cuda") * 1e-3)
    for axis in range(-1, len(shape) - 1):
        kw = dict(rtol=1e-3, atol=1e-5, axis=axis)
        got = forensics(cand, ref, **kw)
        same(got, oracle.forensics(cand.cpu(), ref.cpu(), **kw), "axis %d" % axis)


def test_forensics_full_size_c5():
    """The fp32 [32768, 65536] pass-through pair (2^31 elements, 2^30 of them
    mismatching), forensics along the rows, against one oracle pass."""
    free, _ = torch.cuda.mem_get_info()
    if free < (48 << 30):
        pytest.skip("needs 48 GiB of free device memory")
    case = workloads.c5(device="cuda")
    c, r = case["cand"], case["ref"]
    kw = dict(rtol=case["rtol"], atol=case["atol"], axis=0)
    got = forensics(c, r, **kw)
    ch, rh = c.cpu(), r.cpu()
    del case, c, r
    same(got, oracle.forensics(ch, rh, **kw), "c5")


def _f32(bits):
    return torch.tensor(np.array(bits, dtype=np.uint32).view(np.float32))


@pytest.mark.parametrize("dt", [torch.float32, torch.bfloat16, torch.float16], ids=["f32", "bf16", "f16"])
def test_forensics_exact_boundaries(dt):
    """Differences at and either side of one fp16 spacing h(r) (where the
    kernel decides the fp64 comparison from an fp32 difference and its
    TwoSum remainder), differences whose fp64 rounding lands on h, fp32
    differences that overflow, subnormal and zero references, and the
    growth maximum decided by the remainder alone."""
    g = torch.Generator().manual_seed(31)
    r = (torch.randn(4096, generator=g) * torch.exp2(torch.randint(-30, 30, (4096,), generator=g).float())).to(dt).float()
    e = torch.floor(torch.log2(r.abs().clamp_min(2.0 ** -149)))
    h = torch.exp2(torch.clamp(e, min=-14) - 10)
    h = torch.where(r == 0, torch.full_like(h, 2.0 ** -24), h)
    sign = torch.where(torch.rand(4096, generator=g) < 0.5, -1.0, 1.0)
    k = torch.randint(-3, 4, (4096,), generator=g).float()
    c = (r.double() + sign.double() * h.double() * (1 + k.double() * 2.0 ** -22)).float()
    cols = [c, r]
    if dt == torch.float32:
        # fl64(2^-24 + 2^-149) = 2^-24 = h(-2^-149): within in fp64, not exactly
        extra_c = _f32([0x33800000, 0x33800000, 0x7f000000, 0x7f7fffff, 0x00000001, 0x3f800000])
        extra_r = _f32([0x80000001, 0x00000001, 0xff000000, 0xff7fffff, 0x80000001, 0x3f800001])
        cols = [torch.cat([c, extra_c]), torch.cat([r, extra_r])]
    cand, ref = cols[0].to(dt), cols[1].to(dt)
    n = cand.numel() // 64 * 64
    for shape, axis in (((n,), 0), ((n // 64, 64), 0), ((n // 64, 64), 1), ((cand.numel(),), 0)):
        cs, rs = cand[: int(np.prod(shape))].reshape(shape), ref[: int(np.prod(shape))].reshape(shape)
        kw = dict(rtol=0.0, atol=0.0, axis=axis)
        got = forensics(cs.cuda(), rs.cuda(), **kw)
        same(got, oracle.forensics(cs, rs, **kw), "boundaries %s %s axis %d" % (dt, shape, axis))


def test_forensics_int32_spacing():
    """int32 pairs around one fp16 spacing of references above and below
    2^10, and at INT32_MIN / INT32_MAX."""
    g = torch.Generator().manual_seed(32)
    r = torch.randint(-(1 << 31), (1 << 31) - 1, (3000,), generator=g, dtype=torch.int64)
    r[:1000] = torch.randint(-5000, 5000, (1000,), generator=g)
    r[:4] = torch.tensor([-(1 << 31), (1 << 31) - 1, 1024, -1024])
    mr = r.abs().clamp_min(1)
    h = torch.where(mr >= 1024, torch.exp2(torch.floor(torch.log2(mr.double())) - 10), torch.zeros_like(mr, dtype=torch.float64))
    d = (h + torch.randint(-2, 3, (3000,), generator=g).double()).clamp_min(1).long()
    c = (r + torch.where(r > 0, -d, d)).clamp(-(1 << 31), (1 << 31) - 1)
    cand, ref = c.to(torch.int32), r.to(torch.int32)
    for shape, axis in (((3000,), 0), ((60, 50), 0), ((60, 50), 1)):
        kw = dict(rtol=0.0, atol=0.0, axis=axis)
        got = forensics(cand.view(shape).cuda(), ref.view(shape).cuda(), **kw)
        same(got, oracle.forensics(cand.view(shape), ref.view(shape), **kw), "int32 %s axis %d" % (shape, axis))


@pytest.mark.parametrize("shape,axis", [((5, 70001), 0), ((5, 70001), 1), ((1, 3, 257, 129), 1),
                                        ((1, 3, 257, 129), 2), ((300, 1), 0), ((7, 9, 33), 0)])
def test_forensics_unit_geometry(shape, axis):
    """Few rows with many column windows per unit, ragged last windows,
    growth axes before the last with several rows per index, a last axis of
    length 1."""
    g = torch.Generator(device="cuda").manual_seed(17)
    ref = torch.randn(shape, generator=g, device="cuda")
    cand = torch.where(torch.rand(shape, generator=g, device="cuda") < 0.3,
                       ref * (1 + torch.randn(shape, generator=g, device="cuda") * 1e-2), ref)
    kw = dict(rtol=1e-3, atol=1e-5, axis=axis)
    got = forensics(cand, ref, **kw)
    same(got, oracle.forensics(cand.cpu(), ref.cpu(), **kw), "geometry %s axis %d" % (shape, axis))
