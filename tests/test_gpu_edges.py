"""GPU parity at the edges of the scan's fp32 proofs and of its launch plan
(workloads.edge): tolerances where the pre-filter is switched off (rtol
above 1/2, atol above 2^100) or sits at 1/4 and 1/2; differences at and
either side of |r|/4 (where c - r stops being provably exact in fp32);
subnormal references; tiles above the shared-memory profile size; tile grids
wider than the shared-memory histogram window; cases of millions of
elements.  Each case is compared with the oracle field by field, alone, in
one mixed batch, and through buffers that are not 16-byte aligned."""
import zlib

import pytest
import torch

import oracle
from _parity import assert_same
from paper_2608_02712_gb300 import validate, validate_batch, workloads

pytestmark = pytest.mark.gpu

N_EDGE = 120


def _oracle(case):
    cpu = lambda t: t.cpu()
    return oracle.validate(cpu(case["cand"]), cpu(case["ref"]),
                           inputs=[cpu(x) for x in case["inputs"]], rtol=case["rtol"],
                           atol=case["atol"], tile=case["tile"], first_k=case["first_k"])


@pytest.mark.parametrize("seed", range(N_EDGE))
def test_edge_parity(seed):
    case = workloads.edge(seed, device="cuda")
    got = validate(case["cand"], case["ref"], rtol=case["rtol"], atol=case["atol"],
                   tile=case["tile"], first_k=case["first_k"])
    assert_same(got, _oracle(case), case["name"])


def test_edge_batch():
    cases = [workloads.edge(s, device="cuda") for s in range(0, N_EDGE, 3)]
    got = validate_batch(cases)
    for c, g in zip(cases, got["results"]):
        assert_same(g, _oracle(c), c["name"] + " (batch)")


@pytest.mark.parametrize("seed", range(0, N_EDGE, 5))
def test_edge_parity_unaligned(seed):
    case = workloads.edge(seed, device="cuda")
    shift = lambda t: torch.cat([t.reshape(-1)[:1], t.reshape(-1)])[1:].view(t.shape)
    c, r = shift(case["cand"]), shift(case["ref"])
    got = validate(c, r, rtol=case["rtol"], atol=case["atol"], tile=case["tile"],
                   first_k=case["first_k"])
    assert_same(got, _oracle(case), case["name"] + " (unaligned)")


def _aligned_case(dt, tw, th, n_steps, pattern, seed):
    """A case whose last dimension is a multiple of the warp step (32 x 16
    bytes) and whose tile width divides the step: the scan's aligned
    localisation path."""
    v = 8 if dt in (torch.float16, torch.bfloat16) else 4
    n = 32 * v * n_steps
    g = torch.Generator(device="cuda").manual_seed(seed)
    m = int(torch.randint(50, 400, (1,), generator=g, device="cuda"))
    if dt == torch.int32:
        ref = torch.randint(-1000, 1000, (m, n), generator=g, device="cuda", dtype=torch.int32)
        wrong = ref + 1
    else:
        ref = torch.randn(m, n, generator=g, device="cuda").to(dt)
        wrong = (ref.float() + 1.0).to(dt)
    if pattern == "dense":
        sel = torch.rand(m, n, generator=g, device="cuda") < 0.9
    elif pattern == "sparse":
        sel = torch.rand(m, n, generator=g, device="cuda") < 0.003
    else:  # a band of columns in every other row
        sel = torch.zeros(m, n, dtype=torch.bool, device="cuda")
        sel[::2, n // 3: n // 3 + 40] = True
    cand = torch.where(sel, wrong, ref)
    rtol, atol = (0.0, 0.0) if dt == torch.int32 else (1e-2, 1e-3)
    return cand, ref, rtol, atol


@pytest.mark.parametrize("dt", [torch.float32, torch.float16, torch.bfloat16, torch.int32],
                         ids=["f32", "f16", "bf16", "i32"])
@pytest.mark.parametrize("tw_mult", [1, 2, 8, 32])
@pytest.mark.parametrize("th", [1, 7, 64, 5000])
@pytest.mark.parametrize("pattern", ["dense", "sparse", "band"])
def test_aligned_localisation(dt, tw_mult, th, pattern):
    v = 8 if dt in (torch.float16, torch.bfloat16) else 4
    tw = v * tw_mult
    seed = zlib.crc32(("%s %d %d %s" % (dt, tw_mult, th, pattern)).encode()) % 10_000
    cand, ref, rtol, atol = _aligned_case(dt, tw, th, 1 + seed % 5, pattern, seed)
    got = validate(cand, ref, rtol=rtol, atol=atol, tile=(th, tw), first_k=300)
    want = oracle.validate(cand.cpu(), ref.cpu(), rtol=rtol, atol=atol, tile=(th, tw), first_k=300)
    assert_same(got, want, "aligned %s tw=%d th=%d %s" % (dt, tw, th, pattern))


@pytest.mark.parametrize("dt", [torch.float32, torch.bfloat16], ids=["f32", "bf16"])
def test_aligned_localisation_wide_grid(dt):
    """Aligned steps whose tile grid is wider than the shared-memory
    histogram window: the histogram goes to global memory."""
    v = 8 if dt == torch.bfloat16 else 4
    cand, ref, rtol, atol = _aligned_case(dt, v, 3, 300, "dense", 77)   # N / tw = 9600 tile columns
    got = validate(cand, ref, rtol=rtol, atol=atol, tile=(3, v), first_k=50)
    want = oracle.validate(cand.cpu(), ref.cpu(), rtol=rtol, atol=atol, tile=(3, v), first_k=50)
    assert_same(got, want, "aligned wide grid %s" % dt)


@pytest.mark.parametrize("dt", [torch.float32, torch.bfloat16, torch.float16], ids=["f32", "bf16", "f16"])
@pytest.mark.parametrize("with_input", [False, True], ids=["noinput", "input"])
@pytest.mark.parametrize("n", [4096, 4099], ids=["aligned", "ragged"])
def test_dense_regime_transitions(dt, with_input, n):
    """Runs of rows that are wrong everywhere (a pass-through of the input)
    between clean runs, at several run lengths, with NaN/Inf and growing
    errors inside the dense runs: warps switch into and out of the dense
    regime, and its steps fall back to the exact path where they must."""
    g = torch.Generator(device="cuda").manual_seed(11)
    m = 700
    ref = torch.randn(m, n, generator=g, device="cuda").to(dt)
    x = torch.randn(m, n, generator=g, device="cuda").to(dt)
    cand = (ref.float() * (1 + torch.randn(m, n, generator=g, device="cuda") * 1e-4)).to(dt)
    r0 = 0
    for run in (1, 3, 17, 64, 2, 200):
        cand[r0 + 5: r0 + 5 + run] = x[r0 + 5: r0 + 5 + run]
        r0 += 5 + run + run // 2
    cf = cand.view(-1)
    for i in (6 * n + 3, 50 * n + 1000, 300 * n + 17):
        cf[i] = float("nan")
    cf[100 * n + 5] = float("-inf")
    cf[350 * n + 2] = 1e4   # a late, larger error inside a dense run (rows 159-358)
    inputs = [x.view(-1)] if with_input else []
    rtol, atol = (1e-3, 1e-5) if dt == torch.float32 else (1.6e-2, 1e-3)
    got = validate(cand, ref, inputs=inputs, rtol=rtol, atol=atol, tile=(8, 128), first_k=2000)
    want = oracle.validate(cand.cpu(), ref.cpu(), inputs=[t.cpu() for t in inputs], rtol=rtol, atol=atol,
                           tile=(8, 128), first_k=2000)
    assert_same(got, want, "dense regime %s input=%s n=%d" % (dt, with_input, n))
