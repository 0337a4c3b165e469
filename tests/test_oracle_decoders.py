"""Pins for the oracle's own fp16 / bf16 / fp32 decoders (exhaustive for the
16-bit formats) against torch's and numpy's bit reinterpretation."""
import math
import struct

import numpy as np
import torch


def _same(a: float, b: float) -> bool:
    if math.isnan(a) or math.isnan(b):
        return math.isnan(a) and math.isnan(b)
    return struct.pack("<d", a) == struct.pack("<d", b)


def test_decode_f16_exhaustive(oracle_lib):
    bits = torch.arange(65536, dtype=torch.int32).to(torch.int16)
    want = bits.view(torch.float16).double().tolist()
    for b in range(65536):
        got = oracle_lib.decode(b, torch.float16)
        assert _same(got, want[b]), (hex(b), got, want[b])


def test_decode_bf16_exhaustive(oracle_lib):
    bits = torch.arange(65536, dtype=torch.int32).to(torch.int16)
    want = bits.view(torch.bfloat16).double().tolist()
    for b in range(65536):
        got = oracle_lib.decode(b, torch.bfloat16)
        assert _same(got, want[b]), (hex(b), got, want[b])


def test_decode_f32_sampled(oracle_lib):
    rng = np.random.default_rng(7)
    pats = list(rng.integers(0, 1 << 32, 200_000, dtype=np.uint64))
    # every exponent with edge fractions, both signs
    for s in (0, 1):
        for e in range(256):
            for f in (0, 1, 0x400000, 0x7FFFFF):
                pats.append((s << 31) | (e << 23) | f)
    arr = np.array(pats, dtype=np.uint32)
    with np.errstate(invalid="ignore"):
        want = arr.view(np.float32).astype(np.float64)
    for b, w in zip(arr.tolist(), want.tolist()):
        assert _same(oracle_lib.decode(b, torch.float32), w), hex(b)
