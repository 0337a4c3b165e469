"""Seeded synthetic validation workloads.

These stand in for the operator test suites the paper validates against
(NPUKernelBench's lightweight and extended case sets, Sections 4.3 and 5.1,
and the 5-10 / 49-58 full-evaluation cases per operator of S6.1), which are
not available here.  Every generator is deterministic for a given seed and
device (CPU uses torch's CPU generator, CUDA uses torch's Philox generator, so
the two devices give different bytes for the same seed; each test feeds the
same bytes to both sides).

This module holds no validation arithmetic: it only draws numbers and plants
faults.  Both the CUDA path's tests and the oracle's tests consume it.

A case is a dict with keys ``cand``, ``ref``, ``inputs`` (list of tensors),
``rtol``, ``atol``, ``tile`` (rows, cols), ``first_k`` and ``name``.
"""
from __future__ import annotations

import math

import torch

# Recipes of the five headline workloads (sizes at full scale).
C1_SHAPE = (1024, 1024)
C2_SHAPE = (8, 4096, 4096)
C3_COUNT = 512
C3_CAP = 4 * 1024 * 1024
C4_NUMEL = 1 << 28
C5_SHAPE = (32768, 65536)

C1_NAN_AT = ((0, 0), (100, 300), (767, 1000), (1023, 1023))
C1_INF_AT = ((5, 5), (900, 17))

# torch.testing default tolerances per dtype (rtol, atol).
DEFAULT_TOL = {
    torch.float32: (1.3e-6, 1e-5),
    torch.float16: (1e-3, 1e-5),
    torch.bfloat16: (1.6e-2, 1e-5),
    torch.int32: (0.0, 0.0),
}

_INT_VIEW = {torch.float32: torch.int32, torch.float16: torch.int16,
             torch.bfloat16: torch.int16}


def _gen(seed: int, device) -> torch.Generator:
    return torch.Generator(device=torch.device(device)).manual_seed(seed)


def _case(name, cand, ref, rtol, atol, tile, first_k, inputs=()):
    return {"name": name, "cand": cand, "ref": ref, "inputs": list(inputs),
            "rtol": float(rtol), "atol": float(atol),
            "tile": (int(tile[0]), int(tile[1])), "first_k": int(first_k)}


def c1(seed: int = 0, device="cpu", shape=C1_SHAPE):
    """fp32 pair with three planted faults (random replacements, a zeroed
    column band in rows 512-767, fixed NaN/+Inf).  At reduced shapes the
    band covers rows [M/2, 3M/4) and the specials are skipped if out of range."""
    g = _gen(seed, device)
    m, n = shape
    ref = torch.randn(m, n, generator=g, device=device, dtype=torch.float32)
    noise = torch.randn(m, n, generator=g, device=device, dtype=torch.float32)
    cand = ref + noise * (1e-6 * ref.abs())
    numel = m * n
    n_rand = int(math.ceil(numel * 0.001))
    idx = torch.randperm(numel, generator=g, device=device)[:n_rand]
    cand.view(-1)[idx] = torch.randn(n_rand, generator=g, device=device)
    cols = (torch.arange(n, device=device) % 64) >= 56
    cand[m // 2: (3 * m) // 4, cols] = 0.0
    for (i, j) in C1_NAN_AT:
        if i < m and j < n:
            cand[i, j] = float("nan")
    for (i, j) in C1_INF_AT:
        if i < m and j < n:
            cand[i, j] = float("inf")
    return _case("c1_fp32_%dx%d" % (m, n), cand, ref, 1e-3, 1e-5, (64, 64), 256)


def c2(seed: int = 1, device="cpu", shape=C2_SHAPE):
    """bf16 pair: reference ~U(-4,4); candidate = reference with relative
    N(0, 2^-9) noise, rounded to bf16; +0.5 planted on the 128x128 tiles of the
    [M, N] view whose tile-row index is odd and whose tile column is the last."""
    g = _gen(seed, device)
    ref32 = torch.rand(shape, generator=g, device=device, dtype=torch.float32) * 8.0 - 4.0
    ref = ref32.to(torch.bfloat16)
    del ref32
    rf = ref.float()
    cand = (rf + torch.randn(shape, generator=g, device=device, dtype=torch.float32)
            * (2.0 ** -9) * rf.abs()).to(torch.bfloat16)
    del rf
    n = shape[-1]
    view = cand.view(-1, n)
    m = view.shape[0]
    gc = (n + 127) // 128
    c0 = (gc - 1) * 128
    odd_rows = ((torch.arange(m, device=device) // 128) % 2) == 1
    block = view[odd_rows, c0:]
    view[odd_rows, c0:] = (block.float() + 0.5).to(torch.bfloat16)
    return _case("c2_bf16_" + "x".join(map(str, shape)), cand, ref, 1.6e-2, 1e-3,
                 (128, 128), 1024)


def _nudge_ulp(t: torch.Tensor, g: torch.Generator) -> torch.Tensor:
    """Move each element one ulp away from or toward zero, each with
    probability 1/4 (so half the elements move)."""
    iv = _INT_VIEW[t.dtype]
    bits = t.contiguous().view(iv).to(torch.int64)
    width = 32 if t.dtype == torch.float32 else 16
    sign_bit = 1 << (width - 1)
    ubits = bits & ((1 << width) - 1)
    sign = ubits & sign_bit
    mag = ubits & (sign_bit - 1)
    u = torch.rand(t.shape, generator=g, device=t.device)
    away = u < 0.25
    toward = (u >= 0.25) & (u < 0.5)
    new_mag = torch.where(away, mag + 1, mag)
    new_mag = torch.where(toward & (mag > 0), mag - 1, new_mag)
    # toward zero from +-0 crosses to the smallest subnormal of the other sign
    cross = toward & (mag == 0)
    new_sign = torch.where(cross, sign ^ sign_bit, sign)
    new_mag = torch.where(cross, torch.ones_like(mag), new_mag)
    out = new_sign | new_mag
    if width == 16:
        out = torch.where(out >= (1 << 15), out - (1 << 16), out)
    else:
        out = torch.where(out >= (1 << 31), out - (1 << 32), out)
    return out.to(iv).view(t.dtype).reshape(t.shape)


def _c3_shape(g: torch.Generator, cap: int) -> tuple:
    rank = int(torch.randint(1, 6, (1,), generator=g))
    dims = [0] * rank
    order = torch.randperm(rank, generator=g).tolist()
    prod = 1
    for pos in order:
        hi = max(1, min(4097, cap // prod))
        tail_form = float(torch.rand(1, generator=g)) < 0.3
        if tail_form and hi >= 65:
            kmax = (hi - 1) // 64
            k = int(torch.randint(1, kmax + 1, (1,), generator=g))
            r = int(torch.randint(1, 64, (1,), generator=g))
            d = min(64 * k + r, hi)
        else:
            d = int(torch.randint(1, hi + 1, (1,), generator=g))
        dims[pos] = d
        prod *= d
    return tuple(dims)


def c3(seed: int = 2, device="cpu", count: int = C3_COUNT, cap: int = C3_CAP):
    """Full-coverage sweep: `count` pairs, rank 1-5, dims 1-4097 (30% of the
    form 64k+r), at most `cap` elements each; dtype cycles fp32/fp16/bf16;
    even-indexed pairs are clean (+-1 ulp nudges), odd-indexed pairs carry one
    fault cycling tail block / single sign flip / whole-tensor scale 1.01."""
    g = torch.Generator().manual_seed(seed)          # shapes and choices: CPU
    gd = _gen(seed + 1000, device)                   # values: on `device`
    dtypes = (torch.float32, torch.float16, torch.bfloat16)
    cases = []
    for i in range(count):
        shape = _c3_shape(g, cap)
        dt = dtypes[i % 3]
        x = torch.randn(shape, generator=gd, device=device, dtype=torch.float32) * 3.0
        ref = x.to(dt)
        if i % 2 == 0:
            cand = _nudge_ulp(ref, gd)
            kind = "clean"
        else:
            kind = ("tail", "signflip", "scale")[(i // 2) % 3]
            cand = ref.clone()
            flat = cand.view(-1)
            rflat = ref.reshape(-1).float()
            if kind == "tail":
                L = min(flat.numel(), 64)
                seg = rflat[-L:]
                flat[-L:] = (seg + 2.0 + 2.0 * seg.abs()).to(dt)
            elif kind == "signflip":
                big = (rflat.abs() >= 0.5).nonzero()
                j = int(big[0]) if big.numel() else int(rflat.abs().argmax())
                if float(rflat[j]) == 0.0:
                    flat[j] = 1.0
                else:
                    flat[j] = -ref.reshape(-1)[j]
            else:
                cand = (ref.float() * 1.01).to(dt)
        rtol, atol = DEFAULT_TOL[dt]
        cases.append(_case("c3_%03d_%s_%s_%s" % (i, str(dt).split(".")[-1], kind,
                                               "x".join(map(str, shape))),
                           cand, ref, rtol, atol, (64, 64), 256))
    return cases


def c4(seed: int = 3, device="cpu", numel: int = C4_NUMEL):
    """int32 index-output pair: reference uniform in [0, 65535]; candidate
    off by +1 wherever the linear index mod 4096 is >= 4064; exact mode."""
    g = _gen(seed, device)
    ref = torch.randint(0, 65536, (numel,), generator=g, device=device, dtype=torch.int32)
    cand = ref.clone()
    pos = torch.arange(numel, device=device, dtype=torch.int64) % 4096
    cand += (pos >= 4064).to(torch.int32)
    del pos
    return _case("c4_int32_%d" % numel, cand, ref, 0.0, 0.0, (1, 4096), 4096)


def c5(seed: int = 4, device="cpu", shape=C5_SHAPE, first_k: int = 65536):
    """fp32 pair plus one 1-D input of the same size: the first half of the
    candidate is a bitwise copy of the input (pass-through), the second half
    is reference + relative N(0, 1e-7) noise; 1074 NaN and 1073 -Inf planted
    at the first 2147 distinct positions of 4096 uniform draws."""
    g = _gen(seed, device)
    m, n = shape
    numel = m * n
    half = numel // 2
    ref = torch.randn(m, n, generator=g, device=device, dtype=torch.float32)
    x = torch.randn(numel, generator=g, device=device, dtype=torch.float32)
    cand = torch.empty(m, n, device=device, dtype=torch.float32)
    cf = cand.view(-1)
    cf[:half] = x[:half]
    rf = ref.view(-1)[half:]
    cf[half:] = rf + torch.randn(numel - half, generator=g, device=device,
                                 dtype=torch.float32) * 1e-7 * rf.abs()
    del rf
    gs = torch.Generator().manual_seed(seed)
    draws = torch.randint(0, numel, (4096,), generator=gs).tolist()
    seen, order = set(), []
    for d in draws:
        if d not in seen:
            seen.add(d)
            order.append(d)
    n_special = min(2147, len(order))
    n_nan = (n_special + 1) // 2
    nan_idx = torch.tensor(order[:n_nan], dtype=torch.int64, device=device)
    inf_idx = torch.tensor(order[n_nan:n_special], dtype=torch.int64, device=device)
    cf[nan_idx] = float("nan")
    cf[inf_idx] = float("-inf")
    return _case("c5_fp32_%dx%d_input" % (m, n), cand, ref, 1e-5, 1e-8, (128, 128),
                 first_k, inputs=[x])


SPECIALS = {
    torch.float32: [0.0, -0.0, float("inf"), float("-inf"), float("nan"),
                    1e-45, -1e-45, 1e-38, 3.4e38, -3.4e38],
    torch.float16: [0.0, -0.0, float("inf"), float("-inf"), float("nan"),
                    6e-8, -6e-8, 6.1e-5, 65504.0, -65504.0],
    torch.bfloat16: [0.0, -0.0, float("inf"), float("-inf"), float("nan"),
                     1e-40, -1e-40, 1e-38, 3.0e38, -3.0e38],
}


def fuzz(seed: int, device="cpu", max_dim: int = 300, allow_empty: bool = True):
    """One random small case: rank 0-5, dims 1-max_dim (sometimes 0), any of
    the four dtypes, sprinkled special values, random tolerances, tiles and K."""
    g = torch.Generator().manual_seed(10_000 + seed)
    gd = _gen(20_000 + seed, device)
    dtypes = (torch.float32, torch.float16, torch.bfloat16, torch.int32)
    dt = dtypes[int(torch.randint(0, 4, (1,), generator=g))]
    rank = int(torch.randint(0, 6, (1,), generator=g))
    shape = []
    budget = 1 << 18
    for _ in range(rank):
        hi = max(1, min(max_dim, budget))
        d = int(torch.randint(1, hi + 1, (1,), generator=g))
        if allow_empty and float(torch.rand(1, generator=g)) < 0.03:
            d = 0
        shape.append(d)
        budget = max(1, budget // max(d, 1))
    shape = tuple(shape)
    if dt == torch.int32:
        lo, hi = (-5, 5) if float(torch.rand(1, generator=g)) < 0.5 else (-(1 << 31), (1 << 31) - 1)
        ref = torch.randint(lo, hi, shape, generator=gd, device=device, dtype=torch.int32)
        cand = ref.clone()
        flip = torch.rand(shape, generator=gd, device=device) < 0.05
        delta = torch.randint(-3, 4, shape, generator=gd, device=device, dtype=torch.int32)
        cand = torch.where(flip, cand + delta, cand)
        if float(torch.rand(1, generator=g)) < 0.5:
            rtol, atol = 0.0, 0.0
        else:
            rtol = float(torch.rand(1, generator=g)) * 0.1
            atol = float(torch.randint(0, 3, (1,), generator=g))
    else:
        scale = 10.0 ** float(torch.randint(-3, 4, (1,), generator=g))
        ref = (torch.randn(shape, generator=gd, device=device) * scale).to(dt)
        rtol, atol = DEFAULT_TOL[dt]
        rtol *= 10.0 ** float(torch.randint(-1, 3, (1,), generator=g))
        atol *= 10.0 ** float(torch.randint(-2, 3, (1,), generator=g))
        rel = torch.randn(shape, generator=gd, device=device) * rtol * 2.0
        cand = (ref.float() * (1.0 + rel)).to(dt)
        n = cand.numel()
        if n:
            ns = int(torch.randint(0, min(n, 24) + 1, (1,), generator=g))
            pos = torch.randint(0, n, (ns,), generator=g).tolist()
            sp = SPECIALS[dt]
            which = torch.randint(0, len(sp), (ns, 2), generator=g).tolist()
            side = torch.randint(0, 3, (ns,), generator=g).tolist()
            cf, rf = cand.view(-1), ref.view(-1)
            for p, (a, b), s in zip(pos, which, side):
                if s in (0, 2):
                    cf[p] = sp[a]
                if s in (1, 2):
                    rf[p] = sp[b]
            if float(torch.rand(1, generator=g)) < 0.1:
                cand.zero_()
    n = cand.numel()
    inputs = []
    if n and float(torch.rand(1, generator=g)) < 0.3:
        x = cand.clone().view(-1)
        keep = torch.rand(n, generator=gd, device=device) < 0.5
        other = ref.reshape(-1)
        x = torch.where(keep, x, other)
        inputs.append(x)
        if float(torch.rand(1, generator=g)) < 0.5:
            inputs.append(torch.zeros(max(n - 1, 1), dtype=dt, device=device))
    th = int(torch.randint(1, 70, (1,), generator=g))
    tw = int(torch.randint(1, 70, (1,), generator=g))
    k = int(torch.randint(0, 300, (1,), generator=g))
    return _case("fuzz_%d" % seed, cand, ref, rtol, atol, (th, tw), k, inputs)


# Tolerances at the edges of the scan's fp32 proofs: rtol around 1/4 and
# 1/2 (the exactness and pre-filter limits), atol from 0 up past 2^100.
EDGE_RTOL = (0.0, 0.25, 0.5, math.nextafter(0.5, 1.0), 2.0)
EDGE_ATOL = (0.0, 1e-50, 2.0 ** 100, 2.0 ** 101, 1e300)
EDGE_FAMILIES = ("tolerance", "sterbenz", "subnormal", "big_tiles", "global_hist", "large")


def _bits_of(t: torch.Tensor) -> torch.Tensor:
    return t.contiguous().view(_INT_VIEW[t.dtype]).to(torch.int64)


def _from_bits(b: torch.Tensor, dt) -> torch.Tensor:
    width = 32 if dt == torch.float32 else 16
    b = b & ((1 << width) - 1)
    b = torch.where(b >= (1 << (width - 1)), b - (1 << width), b)
    return b.to(_INT_VIEW[dt]).view(dt)


def _ulp_step(t: torch.Tensor, k: torch.Tensor) -> torch.Tensor:
    """Move each element k[i] representable values up (k > 0) or down, in
    the order of the real line (through zero)."""
    width = 32 if t.dtype == torch.float32 else 16
    b = _bits_of(t) & ((1 << width) - 1)
    sign = b >> (width - 1)
    mag = b & ((1 << (width - 1)) - 1)
    key = torch.where(sign == 1, -mag, mag)          # ordered integer key (-0 -> 0)
    key = key + k
    nb = torch.where(key < 0, (1 << (width - 1)) | (-key), key)
    return _from_bits(nb, t.dtype).reshape(t.shape)


def edge(seed: int, device="cpu"):
    """One case at an edge of the fast path's proofs or of the launch plan,
    by family (seed % 6):

    * tolerance: rtol in {0, 1/4, 1/2, the double after 1/2, 2} and atol in
      {0, 1e-50, 2^100, 2^101, 1e300} (the pre-filter is off above rtol 1/2
      or atol 2^100);
    * sterbenz: differences planted at |c - r| = |r|/4 and 1-2 values either
      side (c near 5r/4 and 3r/4), where c - r stops being provably exact;
    * subnormal: references (and candidates) in the subnormal range of the
      type, a few representable values apart;
    * big_tiles: row or column tiles above 4096 (profiles not privatised in
      shared memory);
    * global_hist: a tile grid wider than the shared-memory histogram window
      (8192 bins), with mismatches;
    * large: 2-6 million elements, so the case spans many pieces and blocks.
    """
    g = torch.Generator().manual_seed(50_000 + seed)
    gd = _gen(60_000 + seed, device)
    fam = EDGE_FAMILIES[seed % len(EDGE_FAMILIES)]
    floats = (torch.float32, torch.float16, torch.bfloat16)
    pick = lambda seq: seq[int(torch.randint(0, len(seq), (1,), generator=g))]
    dt = pick(floats)
    rtol, atol = DEFAULT_TOL[dt]
    tile = (int(torch.randint(1, 70, (1,), generator=g)), int(torch.randint(1, 70, (1,), generator=g)))
    k = int(torch.randint(0, 600, (1,), generator=g))
    if fam == "big_tiles":
        m, n = pick(((300, 10000), (5001, 600), (700, 4099)))
        tile = pick(((5000, 10000), (4097, 64), (64, 4097), (m, n), (4096, 4096)))
    elif fam == "global_hist":
        m, n = pick(((40, 100000), (20, 65536 + 3), (2000, 3000)))
        tile = pick(((1, 8), (1, 1), (2, 4)))
    elif fam == "large":
        numel = int(torch.randint(2_000_000, 6_000_000, (1,), generator=g))
        n = pick((1, 7, 4096, 4099, 65536))
        m = max(1, numel // n)
        dt = pick(floats + (torch.int32,))
        k = int(torch.randint(0, 5000, (1,), generator=g))
    else:
        m = int(torch.randint(1, 600, (1,), generator=g))
        n = int(torch.randint(1, 3000, (1,), generator=g))
    shape = (m, n)
    if dt == torch.int32:
        ref = torch.randint(-(1 << 20), 1 << 20, shape, generator=gd, device=device, dtype=torch.int32)
        cand = ref.clone()
        hit = torch.rand(shape, generator=gd, device=device) < 0.01
        cand = torch.where(hit, cand + torch.randint(-2, 3, shape, generator=gd, device=device,
                                                     dtype=torch.int32), cand)
        rtol, atol = pick(((0.0, 0.0), (1e-6, 1.0), (0.5, 0.0)))
        return _case("edge_%d_%s_int32" % (seed, fam), cand, ref, rtol, atol, tile, k)

    x = torch.randn(shape, generator=gd, device=device)
    if fam == "subnormal":
        width = 32 if dt == torch.float32 else 16
        mant = (1 << 23) if dt == torch.float32 else (1 << 10 if dt == torch.float16 else 1 << 7)
        mag = torch.randint(0, mant, shape, generator=gd, device=device, dtype=torch.int64)
        sgn = torch.randint(0, 2, shape, generator=gd, device=device, dtype=torch.int64)
        ref = _from_bits((sgn << (width - 1)) | mag, dt).reshape(shape)
        steps = torch.randint(-3, 4, shape, generator=gd, device=device, dtype=torch.int64)
        steps = torch.where(torch.rand(shape, generator=gd, device=device) < 0.7, 0 * steps, steps)
        cand = _ulp_step(ref, steps)
        atol = pick((0.0, 1e-50, 1e-45, 6e-8, 1e-40, 1e-39))
        rtol = pick((0.0, rtol, 0.25, 0.5))
    else:
        ref = (x * 10.0 ** float(torch.randint(-2, 3, (1,), generator=g))).to(dt)
        if fam == "tolerance":
            rtol, atol = pick(EDGE_RTOL), pick(EDGE_ATOL)
            rel = torch.randn(shape, generator=gd, device=device) * pick((1e-3, 0.3, 1.0, 3.0))
            cand = (ref.float() * (1.0 + rel)).to(dt)
        elif fam == "sterbenz":
            rtol = pick((0.2, 0.25, 0.3, 0.5, math.nextafter(0.5, 1.0)))
            atol = pick((0.0, 1e-8, 1e-3))
            f = torch.where(torch.rand(shape, generator=gd, device=device) < 0.5,
                            torch.full(shape, 1.25, device=device), torch.full(shape, 0.75, device=device))
            near = (ref.double() * f.double()).to(dt)
            steps = torch.randint(-2, 3, shape, generator=gd, device=device, dtype=torch.int64)
            near = _ulp_step(near, steps)
            noisy = (ref.float() * (1.0 + torch.randn(shape, generator=gd, device=device) * 1e-3)).to(dt)
            cand = torch.where(torch.rand(shape, generator=gd, device=device) < 0.3, near, noisy)
        else:
            rel = torch.randn(shape, generator=gd, device=device) * rtol * 2.0
            cand = (ref.float() * (1.0 + rel)).to(dt)
            if fam == "global_hist":
                band = torch.rand(shape, generator=gd, device=device) < 0.2
                cand = torch.where(band, (cand.float() + 1.0).to(dt), cand)
            elif fam == "large":
                r0 = int(torch.randint(0, m, (1,), generator=g))
                cand.view(m, n)[r0: r0 + max(1, m // 50)] += 1
    cf, rf = cand.view(-1), ref.view(-1)
    nsp = int(torch.randint(0, 9, (1,), generator=g))
    sp = SPECIALS[dt]
    for _ in range(nsp):
        p = int(torch.randint(0, cf.numel(), (1,), generator=g))
        cf[p] = sp[int(torch.randint(0, len(sp), (1,), generator=g))]
    return _case("edge_%d_%s_%s_%dx%d" % (seed, fam, str(dt).split(".")[-1], m, n), cand, ref,
                 rtol, atol, tile, k)


def stats_fuzz(seed: int, device="cpu", max_dim: int = 200):
    """One random tensor for the diagnostic statistics: rank 0-4, any of the
    four dtypes, values of a random scale and offset, sprinkled NaN/Inf and
    zeros, a random tile.  Returns (tensor, tile)."""
    g = torch.Generator().manual_seed(70_000 + seed)
    gd = _gen(80_000 + seed, device)
    dtypes = (torch.float32, torch.float16, torch.bfloat16, torch.int32)
    dt = dtypes[int(torch.randint(0, 4, (1,), generator=g))]
    rank = int(torch.randint(0, 5, (1,), generator=g))
    shape, budget = [], 1 << 16
    for _ in range(rank):
        d = int(torch.randint(1, max(2, min(max_dim, budget)) + 1, (1,), generator=g))
        if float(torch.rand(1, generator=g)) < 0.03:
            d = 0
        shape.append(d)
        budget = max(1, budget // max(d, 1))
    shape = tuple(shape)
    if dt == torch.int32:
        hi = (1 << 31) - 1 if float(torch.rand(1, generator=g)) < 0.5 else 1000
        x = torch.randint(-hi, hi, shape, generator=gd, device=device, dtype=torch.int32)
    else:
        scale = 10.0 ** float(torch.randint(-3, 4, (1,), generator=g))
        offset = float(torch.randn(1, generator=g)) * scale * 5
        x = (torch.randn(shape, generator=gd, device=device) * scale + offset).to(dt)
        n = x.numel()
        if n:
            ns = int(torch.randint(0, min(n, 16) + 1, (1,), generator=g))
            pos = torch.randint(0, n, (ns,), generator=g).tolist()
            sp = SPECIALS[dt]
            which = torch.randint(0, len(sp), (ns,), generator=g).tolist()
            xf = x.view(-1)
            for p, w in zip(pos, which):
                xf[p] = sp[w]
    if x.numel() and float(torch.rand(1, generator=g)) < 0.3:
        x.view(-1)[torch.rand(x.numel(), generator=gd, device=device) < 0.2] = 0
    tile = (int(torch.randint(1, 70, (1,), generator=g)), int(torch.randint(1, 70, (1,), generator=g)))
    return x, tile


def cumsum_fp16(seed: int = 5, device="cpu", rows: int = 256, cols: int = 4096, repaired: bool = False):
    """The cumsum case of the paper's Table 1: the reference accumulates a
    running sum along the last axis in FP16 arithmetic with per-step
    rounding (the vendor reference), the candidate in pure FP32 (the
    near-miss baseline), whose divergence compounds along the axis; with
    repaired=True the candidate rounds every step to FP16 too (the fix) and
    matches.  Inputs x ~ fp16(N(0, 0.1) + 0.05); both outputs are stored as
    fp32.  Tolerances: torch.testing's fp16 defaults."""
    g = _gen(seed, device)
    x = (torch.randn(rows, cols, generator=g, device=device) * 0.1 + 0.05).to(torch.float16)
    xf = x.float()
    ref = torch.empty(rows, cols, device=device)
    acc = torch.zeros(rows, device=device, dtype=torch.float16)
    for j in range(cols):  # per-step fp16 rounding of the running sum
        acc = (acc.float() + xf[:, j]).to(torch.float16)
        ref[:, j] = acc.float()
    cand = ref.clone() if repaired else torch.cumsum(xf, dim=1)
    rtol, atol = DEFAULT_TOL[torch.float16]
    return _case("cumsum_fp16_%dx%d%s" % (rows, cols, "_repaired" if repaired else ""), cand, ref,
                 rtol, atol, (16, 256), 256)
