"""The C-ABI library without a GPU: it builds, loads, exports every symbol
include/nmv.h declares, its structs have the header's layout, and argument
checks reject bad calls before any CUDA work."""
import ctypes
import os
import re
import subprocess

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "nmv.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_02712_gb300 import _build, nmv
    _build.build()
    return nmv.load()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^(?:int|void|const char \*)\s*\*?(nmv_\w+)\(", text, re.M)))


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert {"nmv_validate", "nmv_validate_batch", "nmv_result_free", "nmv_status_string",
            "nmv_last_error"} <= set(names)
    for name in names:
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", os.path.join(
        ROOT, "paper_2608_02712_gb300", "libnmv.so")], capture_output=True, text=True).stdout
    for name in names:
        assert re.search(r"\bT %s$" % name, out, re.M), name


def test_struct_layout_matches_header(tmp_path):
    from paper_2608_02712_gb300 import nmv
    prog = tmp_path / "layout.c"
    fields = {"nmv_tensor": nmv.Tensor, "nmv_case": nmv.Case, "nmv_result": nmv.Result,
              "nmv_profile": nmv.Profile, "nmv_stats_case": nmv.StatsCase, "nmv_stat": nmv.Stat,
              "nmv_stats_result": nmv.StatsResult, "nmv_forensics_case": nmv.ForensicsCase,
              "nmv_forensics_result": nmv.ForensicsResult, "nmv_sweep_report": nmv.SweepReport}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "nmv.h"', 'int main(void){']
    for cname, py in fields.items():
        lines.append('printf("%s sizeof %%zu\\n", sizeof(%s));' % (cname, cname))
        for fname, _ in py._fields_:
            cf = "pass" if fname == "pass_" else fname
            lines.append('printf("%s %s %%zu\\n", offsetof(%s, %s));' % (cname, fname, cname, cf))
    lines.append("return 0;}")
    prog.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(prog), "-o",
                    str(exe)], check=True)
    got = {}
    for line in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n"):
        if line:
            a, b, v = line.split()
            got[(a, b)] = int(v)
    for cname, py in fields.items():
        assert got[(cname, "sizeof")] == ctypes.sizeof(py), cname
        for fname, _ in py._fields_:
            assert got[(cname, fname)] == getattr(py, fname).offset, (cname, fname)


def test_profile_last_without_a_profiled_call(lib):
    from paper_2608_02712_gb300 import nmv
    assert lib.nmv_profile_last(None) == -1
    nmv.profile_enable(False)
    out = nmv.Profile()
    assert lib.nmv_profile_last(ctypes.byref(out)) == -1


def test_status_strings(lib):
    assert lib.nmv_status_string(0) == b"ok"
    assert lib.nmv_status_string(-1) == b"invalid argument"
    assert lib.nmv_status_string(-3) == b"CUDA error"
    assert lib.nmv_status_string(-4) == b"unsupported device"
    assert lib.nmv_status_string(-5) == b"kernel wait limit reached"
    assert lib.nmv_status_string(12345) == b"unknown status"


def test_status_codes_match_header():
    from paper_2608_02712_gb300 import nmv
    text = open(HEADER).read()
    codes = {m.group(1): int(m.group(2)) for m in
             re.finditer(r"#define (NMV_E\w+|NMV_OK) \(?(-?\d+)\)?", text)}
    assert codes == {"NMV_OK": 0, "NMV_EINVAL": -1, "NMV_ENOMEM": -2, "NMV_ECUDA": -3,
                     "NMV_EUNSUPPORTED": -4, "NMV_ETIMEOUT": -5}
    for name, v in codes.items():
        assert getattr(nmv, name) == v, name


def _host_case(nmv, n=16, dtype=0, **over):
    shape = (ctypes.c_int64 * 1)(n)
    buf = (ctypes.c_float * max(n, 1))()
    t = nmv.Tensor(ctypes.cast(buf, ctypes.c_void_p), dtype, 1, ctypes.cast(shape, ctypes.POINTER(ctypes.c_int64)))
    c = nmv.Case()
    c.cand = t
    c.ref = nmv.Tensor(t.data, t.dtype, t.rank, t.shape)
    c.n_inputs = 0
    c.rtol, c.atol = 1e-3, 1e-5
    c.tile_rows, c.tile_cols, c.first_k = 1, 4, 3
    for k, v in over.items():
        setattr(c, k, v)
    return c, (shape, buf)


@pytest.mark.parametrize("bad", [
    {"rtol": -1.0}, {"atol": float("nan")}, {"rtol": float("inf")}, {"tile_rows": 0},
    {"tile_cols": (1 << 24) + 1}, {"first_k": -1}, {"first_k": (1 << 24) + 1},
    {"n_inputs": 9}, {"n_inputs": 1}, {"reserved": 1},
])
def test_invalid_arguments_rejected(lib, bad):
    from paper_2608_02712_gb300 import nmv
    c, keep = _host_case(nmv, **bad)
    out = ctypes.POINTER(nmv.Result)()
    rc = lib.nmv_validate(ctypes.byref(c), None, ctypes.byref(out))
    assert rc == nmv.NMV_EINVAL
    assert not out
    assert lib.nmv_last_error()


def test_invalid_tensors_rejected(lib):
    from paper_2608_02712_gb300 import nmv
    out = ctypes.POINTER(nmv.Result)()
    c, keep = _host_case(nmv)
    c.ref.dtype = 1                                   # dtype mismatch
    assert lib.nmv_validate(ctypes.byref(c), None, ctypes.byref(out)) == nmv.NMV_EINVAL
    c, keep = _host_case(nmv)
    c.cand.dtype = 7                                  # unknown dtype
    assert lib.nmv_validate(ctypes.byref(c), None, ctypes.byref(out)) == nmv.NMV_EINVAL
    c, keep = _host_case(nmv)
    c.cand.rank = 9                                   # rank too large
    assert lib.nmv_validate(ctypes.byref(c), None, ctypes.byref(out)) == nmv.NMV_EINVAL
    c, keep = _host_case(nmv)
    c.cand.data = None                                # NULL data, numel > 0
    assert lib.nmv_validate(ctypes.byref(c), None, ctypes.byref(out)) == nmv.NMV_EINVAL
    shape2 = (ctypes.c_int64 * 1)(17)
    c, keep = _host_case(nmv)
    c.ref.shape = ctypes.cast(shape2, ctypes.POINTER(ctypes.c_int64))   # shape mismatch
    assert lib.nmv_validate(ctypes.byref(c), None, ctypes.byref(out)) == nmv.NMV_EINVAL
    assert lib.nmv_validate(None, None, ctypes.byref(out)) == nmv.NMV_EINVAL
    assert lib.nmv_validate(ctypes.byref(c), None, None) == nmv.NMV_EINVAL


def test_batch_names_the_bad_case(lib):
    from paper_2608_02712_gb300 import nmv
    good, k1 = _host_case(nmv)
    bad, k2 = _host_case(nmv, first_k=-5)
    arr = (nmv.Case * 3)(good, good, bad)
    out = ctypes.POINTER(nmv.Result)()
    rc = lib.nmv_validate_batch(arr, 3, None, ctypes.byref(out))
    assert rc == nmv.NMV_EINVAL and not out
    assert lib.nmv_last_error().startswith(b"case 2:")
    assert lib.nmv_validate_batch(arr, -1, None, ctypes.byref(out)) == nmv.NMV_EINVAL
    assert lib.nmv_validate_batch(arr, 0, None, ctypes.byref(out)) == nmv.NMV_OK and not out


def test_result_free_accepts_null(lib):
    lib.nmv_result_free(None)


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-device error path")
def test_no_device_reports_cuda_error(lib):
    from paper_2608_02712_gb300 import nmv
    c, keep = _host_case(nmv)
    out = ctypes.POINTER(nmv.Result)()
    rc = lib.nmv_validate(ctypes.byref(c), None, ctypes.byref(out))
    assert rc == nmv.NMV_ECUDA and not out
    assert lib.nmv_last_error()


def test_binding_refuses_host_tensors():
    from paper_2608_02712_gb300 import validate
    with pytest.raises(ValueError):
        validate(torch.zeros(4), torch.zeros(4), rtol=0, atol=0)


def test_stats_rejects_bad_cases(lib):
    from paper_2608_02712_gb300 import nmv
    shape = (ctypes.c_int64 * 2)(4, 4)
    buf = (ctypes.c_float * 16)()
    t = nmv.Tensor(ctypes.cast(buf, ctypes.c_void_p), 0, 2, ctypes.cast(shape, ctypes.POINTER(ctypes.c_int64)))
    good = nmv.StatsCase(t, 2, 2)
    out = ctypes.POINTER(nmv.StatsResult)()
    for bad in (nmv.StatsCase(t, 0, 2), nmv.StatsCase(t, 2, (1 << 24) + 1),
                nmv.StatsCase(nmv.Tensor(t.data, 9, 2, t.shape), 2, 2),
                nmv.StatsCase(nmv.Tensor(None, 0, 2, t.shape), 2, 2)):
        arr = (nmv.StatsCase * 2)(good, bad)
        assert lib.nmv_stats(arr, 2, None, ctypes.byref(out)) == nmv.NMV_EINVAL and not out
        assert lib.nmv_last_error().startswith(b"case 1:")
    big = (ctypes.c_int64 * 2)(1 << 12, 1 << 12)
    huge = nmv.StatsCase(nmv.Tensor(t.data, 0, 2, ctypes.cast(big, ctypes.POINTER(ctypes.c_int64))), 1, 1)
    assert lib.nmv_stats(ctypes.byref(huge), 1, None, ctypes.byref(out)) == nmv.NMV_EINVAL   # 2^24 tiles
    assert lib.nmv_stats(None, 1, None, ctypes.byref(out)) == nmv.NMV_EINVAL
    assert lib.nmv_stats(ctypes.byref(good), 1, None, None) == nmv.NMV_EINVAL
    assert lib.nmv_stats(ctypes.byref(good), 0, None, ctypes.byref(out)) == nmv.NMV_OK and not out


def test_forensics_rejects_bad_cases(lib):
    from paper_2608_02712_gb300 import nmv
    shape = (ctypes.c_int64 * 2)(4, 4)
    buf = (ctypes.c_float * 16)()
    t = nmv.Tensor(ctypes.cast(buf, ctypes.c_void_p), 0, 2, ctypes.cast(shape, ctypes.POINTER(ctypes.c_int64)))

    def case(**over):
        c = nmv.ForensicsCase(t, t, 1e-3, 1e-5, -1, 0, 4, 0.01, 4.0)
        for k, v in over.items():
            setattr(c, k, v)
        return c

    out = ctypes.POINTER(nmv.ForensicsResult)()
    for bad in ({"axis": 2}, {"axis": -3}, {"rtol": -1.0}, {"atol": float("nan")}, {"reserved": 1},
                {"near_ulps": -1}, {"near_fraction": float("inf")}, {"growth_factor": -2.0}):
        arr = (nmv.ForensicsCase * 2)(case(), case(**bad))
        assert lib.nmv_forensics(arr, 2, None, ctypes.byref(out)) == nmv.NMV_EINVAL and not out, bad
        assert lib.nmv_last_error().startswith(b"case 1:"), bad
    c = case()
    c.ref = nmv.Tensor(t.data, 1, 2, t.shape)
    assert lib.nmv_forensics(ctypes.byref(c), 1, None, ctypes.byref(out)) == nmv.NMV_EINVAL
    assert lib.nmv_forensics(ctypes.byref(case()), 0, None, ctypes.byref(out)) == nmv.NMV_OK and not out


@pytest.mark.parametrize("n", [0, 1, 55, 56, 63, 64, 65, 119, 120, 1000, 100_000])
def test_sha256_matches_hashlib(lib, n):
    import hashlib
    import random
    from paper_2608_02712_gb300 import sha256
    data = random.Random(n).randbytes(n)
    assert sha256(data) == hashlib.sha256(data).hexdigest()


def test_sweep_rejects_empty_light_set(lib):
    from paper_2608_02712_gb300 import nmv
    out = ctypes.POINTER(nmv.SweepReport)()
    assert lib.nmv_sweep(None, 0, None, 0, None, ctypes.byref(out)) == nmv.NMV_EINVAL and not out
    lib.nmv_sweep_free(None)
