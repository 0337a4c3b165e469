"""GPU parity: the CUDA path (through the C ABI) against the oracle, element
by element on the same seeded inputs."""
import numpy as np
import pytest
import torch

import oracle
from _golden import check, fixture_files, load
from _parity import assert_same
from paper_2608_02712_gb300 import validate, validate_batch, workloads

pytestmark = pytest.mark.gpu


def _gpu(case):
    dev = lambda t: t.cuda()
    return validate(dev(case["cand"]), dev(case["ref"]),
                    inputs=[dev(x) for x in case["inputs"]], rtol=case["rtol"],
                    atol=case["atol"], tile=case["tile"], first_k=case["first_k"])


def _oracle(case):
    cpu = lambda t: t.cpu()
    return oracle.validate(cpu(case["cand"]), cpu(case["ref"]),
                           inputs=[cpu(x) for x in case["inputs"]], rtol=case["rtol"],
                           atol=case["atol"], tile=case["tile"], first_k=case["first_k"])


@pytest.mark.parametrize("path", fixture_files(), ids=lambda p: p.rsplit("/", 1)[-1])
def test_golden_fixtures_on_gpu(path):
    case, expect = load(path)
    check(_gpu(case), expect)


@pytest.mark.parametrize("seed", range(300))
def test_fuzz_parity(seed):
    case = workloads.fuzz(seed)
    assert_same(_gpu(case), _oracle(case), case["name"])


@pytest.mark.parametrize("seed", range(40))
def test_fuzz_parity_unaligned(seed):
    """Views that start one element into their buffer (no 16-byte alignment)."""
    case = workloads.fuzz(1000 + seed)
    shift = lambda t: torch.cat([t.reshape(-1)[:1], t.reshape(-1)]).cuda()[1:].view(t.shape)
    c, r = shift(case["cand"]), shift(case["ref"])
    xs = [shift(x) for x in case["inputs"]]
    got = validate(c, r, inputs=xs, rtol=case["rtol"], atol=case["atol"], tile=case["tile"],
                   first_k=case["first_k"])
    assert_same(got, _oracle(case), case["name"])


def test_c1_full():
    case = workloads.c1(device="cuda")
    assert_same(_gpu(case), _oracle(case), case["name"])


@pytest.mark.parametrize("shape", [(1, 1024, 4096), (3, 1000, 4095), (8, 4096, 4096)])
def test_c2_parity(shape):
    case = workloads.c2(device="cuda", shape=shape)
    assert_same(_gpu(case), _oracle(case), case["name"])


@pytest.mark.parametrize("numel", [(1 << 20) + 77, 1 << 28])
def test_c4_parity(numel):
    case = workloads.c4(device="cuda", numel=numel)
    assert_same(_gpu(case), _oracle(case), case["name"])


@pytest.mark.parametrize("shape", [(256, 1024), (1024, 4096 + 3)])
def test_c5_parity_reduced(shape):
    case = workloads.c5(device="cuda", shape=shape, first_k=4096)
    assert_same(_gpu(case), _oracle(case), case["name"])


def test_c3_batch_parity_and_equal_to_single_calls():
    cases = workloads.c3(device="cuda", count=96, cap=1 << 20)
    got = validate_batch(cases)
    for c, g in zip(cases, got["results"]):
        assert_same(g, _oracle(c), c["name"])
        single = _gpu(c)
        assert_same(single, g, c["name"] + " (single vs batch)")
    assert got["n_pass"] == sum(int(_oracle(c)["pass"]) for c in cases)


def test_mixed_dtype_batch_with_inputs_and_empty_cases():
    cases = [workloads.fuzz(s) for s in range(60)]
    cases = [dict(c, cand=c["cand"].cuda(), ref=c["ref"].cuda(),
                  inputs=[x.cuda() for x in c["inputs"]]) for c in cases]
    got = validate_batch(cases)
    for c, g in zip(cases, got["results"]):
        assert_same(g, _oracle(c), c["name"])


def test_deterministic_bits():
    case = workloads.c2(device="cuda", shape=(2, 2048, 4096))
    a, b = _gpu(case), _gpu(case)
    for k in a:
        if isinstance(a[k], np.ndarray):
            assert np.array_equal(a[k].view(np.uint8) if a[k].dtype.kind == "f" else a[k],
                                  b[k].view(np.uint8) if b[k].dtype.kind == "f" else b[k]), k
        elif isinstance(a[k], float):
            assert np.float64(a[k]).tobytes() == np.float64(b[k]).tobytes(), k
        else:
            assert a[k] == b[k], k


def test_deterministic_sse_under_dynamic_scheduling():
    # Blocks take pieces and warps take batches in whatever order they get
    # to them; the sum of squared errors must still come out bit-identical.
    g = torch.Generator(device="cuda").manual_seed(17)
    ref = torch.randn(3000, 4099, generator=g, device="cuda")
    cand = ref * (1 + torch.randn(ref.shape, generator=g, device="cuda") * 1e-3)
    cand[::7, ::5] += 3.0
    bits = set()
    for _ in range(4):
        r = validate(cand, ref, rtol=1e-3, atol=1e-5, tile=(64, 64), first_k=64)
        bits.add(np.float64(r["sse"]).tobytes())
    assert len(bits) == 1
    want = oracle.validate(cand.cpu(), ref.cpu(), rtol=1e-3, atol=1e-5, tile=(64, 64), first_k=64)
    assert_same(r, want, "dense noisy fp32")


def test_first_k_overflowing_segment_lists():
    """Dense mismatches: every segment list overflows, first-K needs re-reads."""
    g = torch.Generator(device="cuda").manual_seed(5)
    ref = torch.randn(3, 777, 1031, generator=g, device="cuda")
    cand = ref + 1.0
    for k in (1, 127, 128, 129, 5000, 200000):
        got = validate(cand, ref, rtol=1e-3, atol=1e-5, tile=(32, 64), first_k=k)
        want = oracle.validate(cand.cpu(), ref.cpu(), rtol=1e-3, atol=1e-5, tile=(32, 64),
                               first_k=k)
        assert_same(got, want, "dense k=%d" % k)


def test_exact_tolerance_boundaries_on_gpu():
    """Elements sitting exactly on, and one ulp either side of, the fp64
    threshold: the fp32 pre-filter must hand them to the fp64 path."""
    g = torch.Generator().manual_seed(9)
    r = torch.randn(4096, generator=g, dtype=torch.float64).to(torch.float32)
    rtol, atol = 1e-3, 1e-5
    thr = atol + rtol * r.double().abs()
    c = (r.double() + thr).to(torch.float32)
    cases = [c, torch.nextafter(c, torch.full_like(c, float("inf"))),
             torch.nextafter(c, torch.full_like(c, -float("inf")))]
    for cc in cases:
        got = validate(cc.cuda(), r.cuda(), rtol=rtol, atol=atol, tile=(1, 64), first_k=4096)
        want = oracle.validate(cc, r, rtol=rtol, atol=atol, tile=(1, 64), first_k=4096)
        assert_same(got, want, "boundary")


def test_tiny_and_huge_values_sse():
    vals = torch.tensor([1e-30, -3e-38, 1e-45, 2e30, -1e38, 3.3e38, 5e-20, 0.0] * 64,
                        dtype=torch.float32)
    r = vals
    c = vals * 1.5
    got = validate(c.cuda(), r.cuda(), rtol=0.1, atol=0.0, tile=(1, 8), first_k=16)
    want = oracle.validate(c, r, rtol=0.1, atol=0.0, tile=(1, 8), first_k=16)
    assert_same(got, want, "extremes")
    small = torch.tensor([1e-42, 2e-42, 3e-41] * 100, dtype=torch.float32)
    got = validate(small.cuda() * 2, small.cuda(), rtol=0.0, atol=0.0, tile=(1, 1), first_k=5)
    want = oracle.validate(small * 2, small, rtol=0.0, atol=0.0, tile=(1, 1), first_k=5)
    assert_same(got, want, "subnormal sse")


def test_exact_equal_tensors_fast():
    x = torch.randn(1 << 22, device="cuda")
    got = validate(x, x.clone(), rtol=0, atol=0, tile=(1, 4096), first_k=8)
    assert got["pass"] and got["mismatch"] == 0 and got["max_abs"] == 0.0
    assert got["argmax_abs"] == 0 and got["argmax_rel"] == int((x != 0).nonzero()[0])


def test_repeated_call_on_rewritten_buffers():
    # The library reuses the plan of a repeated case set (same buffers,
    # shapes and parameters); the values must still be read afresh.
    case = workloads.c1()
    cand, ref = case["cand"].cuda(), case["ref"].cuda()
    args = dict(rtol=case["rtol"], atol=case["atol"], tile=case["tile"], first_k=case["first_k"])
    first = validate(cand, ref, **args)
    assert_same(first, oracle.validate(cand.cpu(), ref.cpu(), **args), "first call")
    g = torch.Generator().manual_seed(123)
    cand.copy_(ref + torch.randn(ref.shape, generator=g).cuda() * 0.5)
    second = validate(cand, ref, **args)
    assert_same(second, oracle.validate(cand.cpu(), ref.cpu(), **args), "rewritten buffers")
    assert second["mismatch"] != first["mismatch"]
    cand.copy_(ref)
    third = validate(cand, ref, **args)
    assert third["pass"] and third["k_out"] == 0 and third["tile_hist"].sum() == 0


def test_results_stay_valid_until_freed():
    import ctypes
    from paper_2608_02712_gb300 import nmv as m
    lib = m.load()
    a = workloads.c1()
    b = workloads.c4(numel=(1 << 16) + 5)
    keep = []
    outs = []
    for case in (a, b, a):
        c, k = m.make_case(case["cand"].cuda(), case["ref"].cuda(), rtol=case["rtol"], atol=case["atol"],
                           tile=case["tile"], first_k=case["first_k"])
        keep.append(k)
        out = ctypes.POINTER(m.Result)()
        assert lib.nmv_validate(ctypes.byref(c), None, ctypes.byref(out)) == 0
        outs.append(out)
    d = [m.result_to_dict(o[0]) for o in outs]
    assert_same(d[2], d[0], "same case twice")
    lib.nmv_result_free(outs[1])
    # a call after a free reuses the block; the live results do not change
    c, k = m.make_case(b["cand"].cuda(), b["ref"].cuda(), rtol=b["rtol"], atol=b["atol"], tile=b["tile"],
                       first_k=b["first_k"])
    out = ctypes.POINTER(m.Result)()
    assert lib.nmv_validate(ctypes.byref(c), None, ctypes.byref(out)) == 0
    assert_same(m.result_to_dict(out[0]), d[1], "reused block")
    assert_same(m.result_to_dict(outs[0][0]), d[0], "live result after reuse")
    for o in (outs[0], outs[2], out):
        lib.nmv_result_free(o)


def test_relative_errors_beyond_fp32_range():
    # |d| / |r| above the fp32 range (a subnormal reference): the thresholds
    # the warps share must stay finite lower bounds, or the larger of two such
    # quotients in different pieces would be skipped.
    g = torch.Generator().manual_seed(9)
    ref = torch.randn(4, 1 << 20, generator=g)
    cand = ref.clone()
    flat_r, flat_c = ref.view(-1), cand.view(-1)
    flat_r[1000], flat_c[1000] = 1e-42, 1.0
    flat_r[3_000_000], flat_c[3_000_000] = 1e-43, 4.0
    want = oracle.validate(cand, ref, rtol=1e-5, atol=1e-6, tile=(1, 4096), first_k=8)
    got = validate(cand.cuda(), ref.cuda(), rtol=1e-5, atol=1e-6, tile=(1, 4096), first_k=8)
    assert_same(got, want, "rel beyond fp32")
    assert got["argmax_rel"] == 3_000_000 and got["max_rel"] > 3.4e38


@pytest.mark.parametrize("where", [5_000, 3_000_001, (1 << 22) - 3])
def test_max_abs_tie_with_an_inexact_difference(where):
    # Every |c - r| is exactly 1 (all tie for the maximum; the lowest index
    # wins) except one whose exact difference 1 + 2^-25 rounds to 1 in fp32.
    # A warp that already holds the maximum 1 must still take that element
    # as a candidate: its fp64 |d| is the true maximum.
    g = torch.Generator().manual_seed(17)
    ref = torch.randint(-1000, 1000, (1 << 22,), generator=g).float()
    cand = ref + 1.0
    ref[where], cand[where] = -(2.0 ** -25), 1.0
    want = oracle.validate(cand, ref, rtol=0.0, atol=0.5, tile=(64, 64), first_k=16)
    got = validate(cand.cuda(), ref.cuda(), rtol=0.0, atol=0.5, tile=(64, 64), first_k=16)
    assert_same(got, want, "inexact tie")
    assert got["argmax_abs"] == where and got["max_abs"] == 1.0 + 2.0 ** -25


def test_max_abs_ties_everywhere_bf16():
    # |c - r| takes a few quantised values, the largest at many indices in
    # every piece: the argmax is the lowest of them.
    g = torch.Generator().manual_seed(23)
    ref = (torch.rand(6, 1024, 1024, generator=g) * 8 - 4).to(torch.bfloat16)
    cand = (ref.float() + 0.5).to(torch.bfloat16)
    want = oracle.validate(cand, ref, rtol=1.6e-2, atol=1e-3, tile=(128, 128), first_k=64)
    got = validate(cand.cuda(), ref.cuda(), rtol=1.6e-2, atol=1e-3, tile=(128, 128), first_k=64)
    assert_same(got, want, "bf16 ties")


def test_max_rel_tie_with_an_inexact_difference():
    # Element A (index 5) has the exact relative error 2^24 (c - r = 1 with
    # |r| = 2^-24); element B (index 15 * 1024 + 5, a later batch of the same
    # warp) has fl32(c - r) = 1 too, but its exact difference 1 + 2^-24 makes
    # its relative error 2^24 + 1: the larger, whatever the warp already holds.
    n = 1 << 24
    ref = torch.linspace(1.0, 2.0, n)
    cand = ref.clone()
    a, b = 5, 15 * 1024 + 5
    ref[a], cand[a] = -(2.0 ** -24), 1.0 - 2.0 ** -24
    ref[b], cand[b] = -(2.0 ** -24), 1.0
    want = oracle.validate(cand, ref, rtol=1e-3, atol=1e-6, tile=(1, 4096), first_k=8)
    got = validate(cand.cuda(), ref.cuda(), rtol=1e-3, atol=1e-6, tile=(1, 4096), first_k=8)
    assert_same(got, want, "inexact rel tie")
    assert got["argmax_rel"] == b and got["argmax_abs"] == b


def _closest_fractions(dt):
    """The two closest distinct relative errors |c - r| / |r| <= 1/4 over
    values c, r of type dt with r in [1, 2) (every binade alike), the
    smaller one not an fp32 value: (c, r) of each."""
    v = torch.arange(0, 1 << 16, dtype=torch.int32).to(torch.int16).view(dt).double().numpy()
    vals = np.unique(v[np.isfinite(v) & (v >= 0.75) & (v < 2.5)])
    C, R = np.meshgrid(vals, vals[(vals >= 1.0) & (vals < 2.0)])
    q = np.abs(C - R) / R
    m = (q > 0) & (np.abs(C - R) <= R / 4)
    q, C, R = q[m], C[m], R[m]
    o = np.argsort(q, kind="stable")
    q, C, R = q[o], C[o], R[o]
    gap = np.diff(q) / q[:-1]
    gap[(gap == 0) | (q[:-1].astype(np.float32).astype(np.float64) == q[:-1])] = np.inf
    i = int(np.argmin(gap))
    return (C[i], R[i]), (C[i + 1], R[i + 1])


@pytest.mark.parametrize("dt", [torch.bfloat16, torch.float16], ids=["bf16", "f16"])
@pytest.mark.parametrize("order", ["larger_late", "larger_first", "ties_only"])
def test_max_rel_closest_fractions_16bit(dt, order):
    # For 16-bit types a warp's own relative-error threshold may be the
    # maximum rounded up to fp32; the next larger relative error any pair
    # of such values can have is farther away than that rounding, so it is
    # still found.  The two closest fractions of the type, the smaller held
    # many times (also earlier in the warp that meets the larger one).
    (c1, r1), (c2, r2) = _closest_fractions(dt)
    n = 1 << 20
    ref = torch.ones(n, dtype=dt)
    cand = ref.clone()
    late = 600_000
    small_at = [3, 5000, 100_000, late - 8 * 2048, late - 8 * 1024, late - 256, late + 1, 900_000]
    for i in small_at:
        cand[i], ref[i] = c1, r1
    if order == "larger_late":
        cand[late], ref[late] = c2, r2
    elif order == "larger_first":
        cand[1], ref[1] = c2, r2
    want = oracle.validate(cand, ref, rtol=1e-3, atol=1e-3, tile=(1, 4096), first_k=16)
    got = validate(cand.cuda(), ref.cuda(), rtol=1e-3, atol=1e-3, tile=(1, 4096), first_k=16)
    assert_same(got, want, "closest fractions %s %s" % (dt, order))
    assert got["argmax_rel"] == {"larger_late": late, "larger_first": 1, "ties_only": 3}[order]


def test_c5_full_size():
    """C5 at its full size (fp32 [32768, 65536] plus a 2^31-element input,
    24 GiB), in the launch configuration the benchmark times, against one
    oracle pass over the whole tensors: every field, element by element,
    plus run-to-run bit identity and the planted closed forms."""
    free, _ = torch.cuda.mem_get_info()
    if free < (64 << 30):
        pytest.skip("needs 64 GiB of free device memory")
    case = workloads.c5(device="cuda")
    c, r, x = case["cand"], case["ref"], case["inputs"][0]
    K = case["first_k"]
    got = _gpu(case)
    again = _gpu(case)
    for k in got:
        a, b = got[k], again[k]
        if isinstance(a, np.ndarray):
            assert a.dtype == b.dtype and np.array_equal(a.view(np.uint8), b.view(np.uint8)), k
        else:
            assert a == b, k
    # planted closed forms: 2147 distinct special positions, the first 1074 NaN
    assert got["cand_nan"] == 1074 and got["cand_neginf"] == 1073 and got["cand_posinf"] == 0
    assert got["ref_nan"] == got["ref_posinf"] == got["ref_neginf"] == 0
    assert got["flags"] & 1 and got["passthrough_input"] == 0  # NMV_FLAG_CAND_EQ_INPUT
    assert got["k_out"] == K
    host = dict(case, cand=c.cpu(), ref=r.cpu(), inputs=[x.cpu()])
    del c, r, x, case
    want = _oracle(host)
    assert_same(got, want, host["name"])


def test_concurrent_calls_from_threads():
    """Four host threads, each on its own stream with its own case, call the
    library in turns that interleave: every result equals that case's
    single-threaded result, bit for bit."""
    import threading

    cases = [workloads.fuzz(5000 + i, device="cuda") for i in range(4)]
    want = [_gpu(c) for c in cases]
    errors = []

    def worker(i):
        try:
            s = torch.cuda.Stream()
            c = cases[i]
            for _ in range(10):
                got = validate(c["cand"], c["ref"], inputs=c["inputs"], rtol=c["rtol"],
                               atol=c["atol"], tile=c["tile"], first_k=c["first_k"], stream=s)
                for k, a in got.items():
                    b = want[i][k]
                    same = (a.dtype == b.dtype and np.array_equal(a.view(np.uint8), b.view(np.uint8))
                            if isinstance(a, np.ndarray) else (a == b or (a != a and b != b)))
                    if not same:
                        errors.append((i, k))
        except Exception as e:  # noqa: BLE001 - reported below
            errors.append((i, repr(e)))

    threads = [threading.Thread(target=worker, args=(i,)) for i in range(4)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors[:5]


@pytest.mark.parametrize("shape", [((1 << 32) + 4099,), (2, (1 << 31) + 4099)], ids=["1d", "2d"])
def test_indices_beyond_32_bits(shape):
    """More than 2^32 elements (bf16, 8 GiB per tensor): the scan's 64-bit
    index path.  Planted errors on both sides of 2^32 give every output in
    closed form: the records, their coordinates, the maxima and their
    indices, the histogram bins, the profiles and the SSE."""
    free, _ = torch.cuda.mem_get_info()
    if free < (40 << 30):
        pytest.skip("needs 40 GiB of free device memory")
    numel = int(np.prod(shape))
    ref = torch.ones(shape, dtype=torch.bfloat16, device="cuda")
    cand = ref.clone()
    small = [5, (1 << 32) - 1, 1 << 32, (1 << 32) + 777, numel - 1]
    big = (1 << 32) + 999
    cf = cand.view(-1)
    for i in small:
        cf[i] = 1.5
    cf[big] = 3.0
    th, tw = 2, 4096
    got = validate(cand, ref, rtol=1e-2, atol=0.0, tile=(th, tw), first_k=8)
    planted = sorted(small + [big])
    assert got["mismatch"] == 6 and not got["pass"]
    assert got["k_out"] == 6
    np.testing.assert_array_equal(got["fk_index"], planted)
    np.testing.assert_array_equal(got["fk_coords"], np.stack(np.unravel_index(planted, shape), 1))
    np.testing.assert_array_equal(got["fk_cand"], [3.0 if i == big else 1.5 for i in planted])
    np.testing.assert_array_equal(got["fk_ref"], [1.0] * 6)
    assert got["max_abs"] == 2.0 and got["argmax_abs"] == big
    assert got["max_rel"] == 2.0 and got["argmax_rel"] == big
    assert got["sse"] == 5 * 0.25 + 4.0
    assert got["n_finite_pairs"] == numel
    N = shape[-1]
    hist = np.zeros_like(got["tile_hist"])
    rowp = np.zeros(th, np.int64)
    colp = np.zeros(tw, np.int64)
    for i in planted:
        r, c = divmod(i, N)
        hist[r // th, c // tw] += 1
        rowp[r % th] += 1
        colp[c % tw] += 1
    np.testing.assert_array_equal(got["tile_hist"], hist)
    np.testing.assert_array_equal(got["row_prof"], rowp)
    np.testing.assert_array_equal(got["col_prof"], colp)
    assert got["flags"] == 16  # NMV_FLAG_REF_CONSTANT: the reference is all ones


@pytest.mark.parametrize("dt", [torch.float32, torch.bfloat16], ids=["f32", "bf16"])
def test_first_k_records_across_far_apart_pieces(dt):
    """Records in a few batches far apart (first, middle, last, and a ragged
    last batch), K larger than the mismatch count: the record pass skips the
    runs of pieces without records and still places every record."""
    n = (1 << 26) + 37
    ref = torch.ones(n, dtype=dt)
    cand = ref.clone()
    where = [0, 1, 2, 31, 4097, n // 2, n // 2 + 1, n - 40, n - 2, n - 1]
    for i in where:
        cand[i] = 3.0
    want = oracle.validate(cand, ref, rtol=1e-3, atol=0.0, tile=(1, 1024), first_k=64)
    got = validate(cand.cuda(), ref.cuda(), rtol=1e-3, atol=0.0, tile=(1, 1024), first_k=64)
    assert_same(got, want, "far-apart records %s" % dt)
    np.testing.assert_array_equal(got["fk_index"], where)


def test_workspace_grows_geometrically():
    """A rising sequence of case sizes (each 10% above the last, 40 calls)
    reallocates the device workspace O(log n) times: it grows by doubling."""
    from paper_2608_02712_gb300 import nmv as m
    m.profile_enable(m.PROFILE_TIMING)
    try:
        allocs, sizes = [], []
        n = 100_000
        for _ in range(40):
            x = torch.zeros(n, device="cuda")
            # one-element tiles: the histogram (8 bytes per element) dominates
            validate(x, x, rtol=0.0, atol=0.0, tile=(1, 1), first_k=0)
            p = m.profile_last()
            allocs.append(p["workspace_allocs"])
            sizes.append(p["workspace_bytes"])
            n = int(n * 1.1)
    finally:
        m.profile_enable(0)
    assert all(b >= a for a, b in zip(sizes, sizes[1:]))
    grew = allocs[-1] - allocs[0]
    # 1.1^40 = 45x: at most ceil(log2(45)) + 1 = 7 doublings
    assert grew <= 7, (grew, allocs)


def test_alternating_case_sets_keep_their_plans():
    """Calls that alternate among more case sets than the library keeps plans
    for (each with its own descriptors and accumulator layout in the shared
    workspace): every call equals the oracle, including after one set's
    buffers are rewritten between its calls."""
    g = torch.Generator().manual_seed(77)
    sets = []
    for k in range(6):
        cases = []
        for j in range(1 + k % 3):
            n = 1000 + 977 * k + 131 * j
            ref = torch.randn(n, generator=g)
            cand = ref + (torch.rand(n, generator=g) < 0.01).float() * (k + 1)
            cases.append(dict(cand=cand.cuda(), ref=ref.cuda(), rtol=1e-3, atol=1e-5,
                              tile=(1, 64 + 16 * k), first_k=16 + k))
        sets.append(cases)
    order = [0, 1, 0, 1, 2, 3, 4, 0, 5, 1, 2, 2, 0, 3, 5, 4, 1]
    for step, i in enumerate(order):
        if step == 9:
            c0 = sets[0][0]
            c0["cand"].copy_(c0["ref"] + 0.5)
        got = validate_batch(sets[i])["results"]
        for c, r in zip(sets[i], got):
            want = oracle.validate(c["cand"].cpu(), c["ref"].cpu(), rtol=c["rtol"], atol=c["atol"],
                                   tile=c["tile"], first_k=c["first_k"])
            assert_same(r, want, "set %d at call %d" % (i, step))
