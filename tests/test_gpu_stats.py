"""GPU parity of the diagnostic tensor statistics (nmv_stats, through the C
ABI) with the oracle, on the same seeded inputs: counts, min, max and the
first NaN/Inf indices exact; int32 sums (exact integers) and everything
derived from them bit-identical; float sums within 1e-12 of n * max|x|
(sum, mean) and relative 1e-12 (sumsq), the variance within 1e-11 of the
mean square, the bounds the float-float accumulation guarantees."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_02712_gb300 import stats, stats_batch, workloads

pytestmark = pytest.mark.gpu

COUNTS = ("n_finite", "n_nan", "n_posinf", "n_neginf", "n_zero")


def _check_level(got, want, is_int, what):
    """got / want: dicts of arrays (or scalars) of one level."""
    g = {k: np.asarray(v) for k, v in got.items()}
    w = {k: np.asarray(v) for k, v in want.items()}
    for k in COUNTS + ("min", "max"):
        assert np.array_equal(g[k], w[k]), (what, k, g[k], w[k])
    if is_int:
        for k in ("sum", "sumsq", "mean", "std"):
            assert np.array_equal(g[k].view(np.int64), w[k].view(np.int64)), (what, k, g[k], w[k])
        return
    n = np.maximum(w["n_finite"], 1).astype(np.float64)
    amax = np.maximum(np.abs(w["min"]), np.abs(w["max"]))
    assert (np.abs(g["sum"] - w["sum"]) <= 1e-12 * n * amax).all(), (what, "sum")
    assert (np.abs(g["mean"] - w["mean"]) <= 1e-12 * amax).all(), (what, "mean")
    assert (np.abs(g["sumsq"] - w["sumsq"]) <= 1e-12 * w["sumsq"]).all(), (what, "sumsq")
    var_g, var_w = g["std"] ** 2, w["std"] ** 2
    assert (np.abs(var_g - var_w) <= 1e-11 * w["sumsq"] / n).all(), (what, "std")


def check(got, want, x):
    is_int = x.dtype == torch.int32
    for k in ("numel", "rank", "grid_rows", "grid_cols", "tile_rows", "tile_cols", "first_nan", "first_inf"):
        assert got[k] == want[k], (k, got[k], want[k])
    _check_level(got["all"], want["all"], is_int, "all")
    _check_level(got["tiles"], want["tiles"], is_int, "tiles")


@pytest.mark.parametrize("seed", range(200))
def test_stats_fuzz_parity(seed):
    x, tile = workloads.stats_fuzz(seed)
    check(stats(x.cuda(), tile=tile), oracle.stats(x, tile=tile), x)


def test_stats_batch_mixed_types():
    items = [workloads.stats_fuzz(s) for s in range(300, 360)]
    got = stats_batch([(x.cuda(), t) for x, t in items])
    for (x, t), g in zip(items, got):
        check(g, oracle.stats(x, tile=t), x)


@pytest.mark.parametrize("seed", range(400, 420))
def test_stats_unaligned(seed):
    x, tile = workloads.stats_fuzz(seed)
    xs = torch.cat([x.reshape(-1)[:1], x.reshape(-1)]).cuda()[1:].view(x.shape) if x.numel() else x.cuda()
    check(stats(xs, tile=tile), oracle.stats(x, tile=tile), x)


@pytest.mark.parametrize("dt", [torch.float32, torch.bfloat16, torch.float16, torch.int32],
                         ids=["f32", "bf16", "f16", "i32"])
@pytest.mark.parametrize("tile", [(1, 1), (3, 5), (64, 64), (300, 10000), (1, 20000), (5000, 7), (100000, 100000)],
                         ids=lambda t: "%dx%d" % t)
def test_stats_tile_shapes(dt, tile):
    """Tiles of one element, odd tiles, tiles wider than a unit's columns,
    taller than a unit's rows, and one tile holding the whole tensor."""
    g = torch.Generator().manual_seed(5)
    if dt == torch.int32:
        x = torch.randint(-(1 << 31), (1 << 31) - 1, (1100, 1300), generator=g, dtype=torch.int32)
    else:
        x = (torch.randn(1100, 1300, generator=g) * 3 + 1).to(dt)
        x.view(-1)[::997] = float("nan")
        x.view(-1)[5::1009] = float("-inf")
        x.view(-1)[7::101] = 0.0
    if tile == (1, 1):
        x = x[:500, :300].contiguous()
    check(stats(x.cuda(), tile=tile), oracle.stats(x, tile=tile), x)


def test_stats_deterministic():
    g = torch.Generator(device="cuda").manual_seed(3)
    x = torch.randn(4096, 8192, generator=g, device="cuda") * 100 + 7
    a = stats(x, tile=(128, 128))
    for _ in range(3):
        b = stats(x, tile=(128, 128))
        for k, v in a["all"].items():
            assert np.float64(v).tobytes() == np.float64(b["all"][k]).tobytes(), k
        for k, v in a["tiles"].items():
            assert np.array_equal(np.ascontiguousarray(v).view(np.uint8),
                                  np.ascontiguousarray(b["tiles"][k]).view(np.uint8)), k


def test_stats_large_magnitudes_and_subnormals():
    """Values beyond 2^57 and below 2^-50 take the fp64 path per element."""
    v = torch.tensor([3e38, -3e38, 1e30, 2.0 ** 60, 1e-40, -1e-45, 2.0 ** -55, 1.0, 0.0, -0.0] * 500,
                     dtype=torch.float32)
    check(stats(v.cuda(), tile=(1, 37)), oracle.stats(v, tile=(1, 37)), v)
    b = torch.tensor([1e-40, -3e38, 2.0 ** -130, 5.0] * 300, dtype=torch.float32).to(torch.bfloat16)
    check(stats(b.cuda(), tile=(1, 16)), oracle.stats(b, tile=(1, 16)), b)


def test_stats_full_size_c5_candidate():
    """The candidate of the fp32 [32768, 65536] pass-through workload (8 GiB,
    2147 NaN/-Inf) with 128 x 128 tiles, against one oracle pass."""
    free, _ = torch.cuda.mem_get_info()
    if free < (40 << 30):
        pytest.skip("needs 40 GiB of free device memory")
    case = workloads.c5(device="cuda")
    x = case["cand"]
    del case
    got = stats(x, tile=(128, 128))
    assert got["all"]["n_nan"] == 1074 and got["all"]["n_neginf"] == 1073
    xh = x.cpu()
    del x
    check(got, oracle.stats(xh, tile=(128, 128)), xh)


@pytest.mark.parametrize("dt", [torch.float32, torch.bfloat16, torch.float16], ids=["f32", "bf16", "f16"])
def test_stats_magnitude_bands(dt):
    """Tiles whose largest magnitude lies below 2^-44 or at 2^57 and above
    (taken again element by element), tiles mixing tiny and ordinary values
    (the fast path's remainders round), subnormals, and tiles holding a NaN
    or an infinity next to tiles that hold none."""
    g = torch.Generator().manual_seed(41)
    rows, cols = 256, 384
    x = torch.randn(rows, cols, generator=g)
    scales = torch.tensor([2.0 ** -130, 2.0 ** -60, 2.0 ** -45, 2.0 ** -43, 1.0, 2.0 ** 56, 2.0 ** 58, 2.0 ** 100])
    band = scales[torch.arange(rows) // 32 % len(scales)]
    x = x * band[:, None]
    x[40, 7] = 2.0 ** -140        # one tiny value among ordinary ones
    x[130, 200] = float("nan")
    x[131, 5] = float("inf")
    x[200:203, :] = 0.0
    x = x.to(dt)
    for tile in ((32, 128), (16, 384), (5, 7), (256, 384)):
        check(stats(x.cuda(), tile=tile), oracle.stats(x, tile=tile), x)


def test_stats_result_views_outlive_later_calls():
    """The tile arrays view the library's result block: they stay valid and
    unchanged while later calls run, and the block is released with them."""
    import gc
    g = torch.Generator(device="cuda").manual_seed(3)
    x1 = torch.randn(512, 640, generator=g, device="cuda")
    x2 = torch.randn(512, 640, generator=g, device="cuda") * 5
    r1 = stats(x1, tile=(16, 32))
    keep = {k: v.copy() for k, v in r1["tiles"].items()}
    for _ in range(20):
        stats(x2, tile=(16, 32))
        gc.collect()
    for k, v in r1["tiles"].items():
        assert np.array_equal(np.ascontiguousarray(v).view(np.int64), keep[k].view(np.int64)), k
    check(r1, oracle.stats(x1.cpu(), tile=(16, 32)), x1)


def test_stats_one_tile_of_many_units():
    """A single tile over a tensor of thousands of units: merged by a whole
    block in a fixed tree."""
    g = torch.Generator(device="cuda").manual_seed(4)
    x = torch.randn(3000, 20000, generator=g, device="cuda") * 3 + 1
    x.view(-1)[123457] = float("nan")
    got = stats(x, tile=(3000, 20000))
    check(got, oracle.stats(x.cpu(), tile=(3000, 20000)), x)
    again = stats(x, tile=(3000, 20000))
    assert got["all"]["sum"] == again["all"]["sum"] and got["all"]["sumsq"] == again["all"]["sumsq"]
