"""Reader for the hand-built fixtures under tests/golden/."""
import glob
import os

import numpy as np
import torch

GOLDEN_DIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
_DT = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16, "i32": torch.int32}
_IV = {torch.float32: torch.int32, torch.float16: torch.int16, torch.bfloat16: torch.int16}


def _tensor(tokens, dtype, shape):
    if tokens and tokens[0] == "bits":
        vals = [int(t, 16) for t in tokens[1:]]
        iv = _IV[dtype]
        width = 16 if iv == torch.int16 else 32
        vals = [v - (1 << width) if v >= (1 << (width - 1)) else v for v in vals]
        t = torch.tensor(vals, dtype=iv).view(dtype)
    elif dtype == torch.int32:
        t = torch.tensor([int(v) for v in tokens], dtype=torch.int32)
    else:
        t = torch.tensor([float(v) for v in tokens], dtype=dtype)
    return t.reshape(shape)


def load(path):
    spec, expect = {}, {}
    for raw in open(path):
        line = raw.split("#", 1)[0].split()
        if not line:
            continue
        if line[0] == "expect":
            expect[line[1]] = line[2:]
        else:
            spec.setdefault(line[0], []).append(line[1:])
    dtype = _DT[spec["dtype"][0][0]]
    shape = tuple(int(s) for s in spec["shape"][0])
    case = {
        "name": os.path.basename(path),
        "cand": _tensor(spec["cand"][0], dtype, shape),
        "ref": _tensor(spec["ref"][0], dtype, shape),
        "inputs": [_tensor(v[1:], _DT[v[0]], (len(v) - 1 - (v[1] == "bits"),))
                   for v in spec.get("input", [])],
        "rtol": float(spec["rtol"][0][0]), "atol": float(spec["atol"][0][0]),
        "tile": tuple(int(t) for t in spec["tile"][0]),
        "first_k": int(spec["first_k"][0][0]),
    }
    return case, expect


def all_fixtures():
    return sorted(glob.glob(os.path.join(GOLDEN_DIR, "*.txt")))


def fixture_files():
    return [p for p in all_fixtures() if not p.endswith("README.txt")]


def check(res, expect):
    """Compare a result dict with the expected tokens of one fixture."""
    for key, toks in expect.items():
        got = res[key]
        if isinstance(got, (bool, np.bool_)):
            assert int(got) == int(toks[0]), key
        elif isinstance(got, (int, np.integer)):
            assert got == int(toks[0]), (key, got, toks)
        elif isinstance(got, float):
            want = float(toks[0])
            assert (np.isnan(got) and np.isnan(want)) or got == want, (key, got, want)
        else:
            arr = np.asarray(got).reshape(-1)
            if arr.dtype.kind == "f":
                want = np.array([float(t) for t in toks])
                same = (arr == want) | (np.isnan(arr) & np.isnan(want))
                assert arr.size == want.size and same.all(), (key, arr, want)
            else:
                want = np.array([int(t) for t in toks], np.int64)
                assert np.array_equal(arr, want), (key, arr, want)
