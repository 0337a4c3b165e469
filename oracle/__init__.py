"""CPU oracle for numerical validation with failure forensics.

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg and reference arm of ``bench.py`` are the only callers.  The product path (the
CUDA library and its binding in ``paper_2608_02712_gb300``) never imports this
package, and this package imports nothing from it.

The arithmetic lives in ``nmv_oracle.c`` (one ordered fp64 loop per pair,
following the definitions P1-P6 written out at its top, which read the paper's
Validate(K_fixed, R, T_ext, tau) check of Section 3.2, Eq. 1, and the
forensic evidence of Sections 4.2-4.3).  This module only compiles it,
marshals buffers and shapes the outputs into a dict.  P7 (a batch is n
independent cases; the batch pass count is the sum of the per-case pass bits,
the "x% matched cases" of Table S4) is ``validate_batch`` below.

Every function here is pinned by tests in ``tests/test_oracle_*.py``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "nmv_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

DTYPE_CODES = {torch.float32: 0, torch.float16: 1, torch.bfloat16: 2, torch.int32: 3}
FLAG_NAMES = {
    1: "CAND_EQ_INPUT",
    2: "CAND_ALL_ZERO",
    4: "CAND_CONSTANT",
    8: "REF_ALL_ZERO",
    16: "REF_CONSTANT",
}


def build(force: bool = False, src: str = _SRC, out: str = _LIB) -> str:
    """Compile the oracle source into a shared library (no FMA contraction)."""
    if (not force and os.path.exists(out)
            and os.path.getmtime(out) >= os.path.getmtime(src)):
        return out
    tmp = out + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", "-o", tmp, src, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def _bind(path: str):
    lib = ctypes.CDLL(path)
    i64p = ctypes.POINTER(ctypes.c_int64)
    f64p = ctypes.POINTER(ctypes.c_double)
    lib.oracle_validate.restype = ctypes.c_int
    lib.oracle_validate.argtypes = [
        ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int, ctypes.c_int64,
        ctypes.c_int64, ctypes.c_int, ctypes.POINTER(ctypes.c_void_p),
        ctypes.POINTER(ctypes.c_int), i64p,
        ctypes.c_double, ctypes.c_double, ctypes.c_int64, ctypes.c_int64,
        ctypes.c_int64, i64p, f64p, i64p, i64p, i64p, i64p, i64p, f64p,
        f64p, i64p, ctypes.POINTER(ctypes.c_uint32),
        ctypes.POINTER(ctypes.c_int32)]
    for name in ("oracle_decode_f16", "oracle_decode_bf16", "oracle_decode_f32"):
        fn = getattr(lib, name)
        fn.restype = ctypes.c_double
        fn.argtypes = [ctypes.c_uint32]
    lib.oracle_pass.restype = ctypes.c_int
    lib.oracle_pass.argtypes = [ctypes.c_double] * 4
    lib.oracle_forensics.restype = ctypes.c_int
    lib.oracle_forensics.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int, ctypes.c_int, i64p,
                                     ctypes.c_double, ctypes.c_double, ctypes.c_int, ctypes.c_int64,
                                     ctypes.c_double, ctypes.c_double, i64p, i64p, f64p, f64p, i64p,
                                     ctypes.POINTER(ctypes.c_uint32)]
    lib.oracle_stats.restype = ctypes.c_int
    lib.oracle_stats.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_int64,
                                 ctypes.c_int64, ctypes.c_int64, i64p, f64p, i64p, i64p, f64p]
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            _lib = _bind(_LIB)
    return _lib


class Oracle:
    """The oracle bound to one compiled library (the default one, or a copy
    built from another source file, e.g. a deliberately broken one in a test
    that checks the pins catch the breakage)."""

    def __init__(self, lib_path: str):
        self.lib = _bind(lib_path)

    def decode(self, bits, dtype):
        return _decode(self.lib, bits, dtype)

    def pass_predicate(self, c, r, rtol, atol):
        return bool(self.lib.oracle_pass(c, r, rtol, atol))

    def validate(self, cand, ref, **kw):
        return _validate(self.lib, cand, ref, **kw)

    def validate_batch(self, cases):
        return _validate_batch(self.validate, cases)

    def stats(self, x, **kw):
        return _stats(self.lib, x, **kw)

    def forensics(self, cand, ref, **kw):
        return _forensics(self.lib, cand, ref, **kw)


def _decode(lib, bits: int, dtype: torch.dtype) -> float:
    if dtype == torch.float16:
        return lib.oracle_decode_f16(bits)
    if dtype == torch.bfloat16:
        return lib.oracle_decode_bf16(bits)
    if dtype == torch.float32:
        return lib.oracle_decode_f32(bits)
    raise ValueError(dtype)


def decode(bits: int, dtype: torch.dtype) -> float:
    """Decode one stored bit pattern to its exact fp64 value."""
    return _decode(_load(), bits, dtype)


def pass_predicate(c: float, r: float, rtol: float, atol: float) -> bool:
    """P1 on two fp64 values."""
    return bool(_load().oracle_pass(c, r, rtol, atol))


def view_2d(shape) -> tuple[int, int]:
    """[M, N] of the 2-D view: M = prod(shape[:-1]), N = shape[-1]; rank 0 -> [1, 1]."""
    shape = tuple(int(s) for s in shape)
    if len(shape) == 0:
        return 1, 1
    m = 1
    for s in shape[:-1]:
        m *= s
    return m, shape[-1]


def _ptr(a: np.ndarray, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def validate(cand: torch.Tensor, ref: torch.Tensor, **kw) -> dict:
    """Run the oracle on one pair of CPU tensors (same dtype and shape)."""
    return _validate(_load(), cand, ref, **kw)


def _validate(lib, cand: torch.Tensor, ref: torch.Tensor, *, inputs=(), rtol: float,
              atol: float, tile=(64, 64), first_k: int = 256) -> dict:
    if cand.dtype != ref.dtype or tuple(cand.shape) != tuple(ref.shape):
        raise ValueError("cand and ref must share dtype and shape")
    if cand.dtype not in DTYPE_CODES:
        raise ValueError("unsupported dtype %s" % cand.dtype)
    cand = cand.detach().cpu().contiguous()
    ref = ref.detach().cpu().contiguous()
    inputs = [x.detach().cpu().contiguous() for x in inputs]
    shape = tuple(cand.shape)
    numel = cand.numel()
    m, n = view_2d(shape)
    th, tw = int(tile[0]), int(tile[1])
    ncols = max(n, 1)
    gr = -(-m // th) if numel else 0
    gc = -(-n // tw) if numel else 0
    k = int(first_k)

    counts = np.zeros(9, np.int64)
    fstats = np.zeros(3, np.float64)
    argmax = np.zeros(2, np.int64)
    hist = np.zeros(max(gr * gc, 1), np.int64)
    row_prof = np.zeros(th, np.int64)
    col_prof = np.zeros(tw, np.int64)
    fk_index = np.zeros(max(k, 1), np.int64)
    fk_cand = np.zeros(max(k, 1), np.float64)
    fk_ref = np.zeros(max(k, 1), np.float64)
    n_in = len(inputs)
    input_eq = np.zeros(max(n_in, 1), np.int64)
    flags = np.zeros(1, np.uint32)
    passthrough = np.zeros(1, np.int32)
    in_ptrs = (ctypes.c_void_p * max(n_in, 1))(*[x.data_ptr() for x in inputs])
    in_dt = (ctypes.c_int * max(n_in, 1))(*[DTYPE_CODES.get(x.dtype, -1) for x in inputs])
    in_n = (ctypes.c_int64 * max(n_in, 1))(*[x.numel() for x in inputs])

    rc = lib.oracle_validate(
        ctypes.c_void_p(cand.data_ptr()), ctypes.c_void_p(ref.data_ptr()),
        DTYPE_CODES[cand.dtype], numel, ncols, n_in, in_ptrs, in_dt, in_n,
        float(rtol), float(atol), th, tw, k,
        _ptr(counts, ctypes.c_int64), _ptr(fstats, ctypes.c_double),
        _ptr(argmax, ctypes.c_int64), _ptr(hist, ctypes.c_int64),
        _ptr(row_prof, ctypes.c_int64), _ptr(col_prof, ctypes.c_int64),
        _ptr(fk_index, ctypes.c_int64), _ptr(fk_cand, ctypes.c_double),
        _ptr(fk_ref, ctypes.c_double), _ptr(input_eq, ctypes.c_int64),
        _ptr(flags, ctypes.c_uint32), _ptr(passthrough, ctypes.c_int32))
    if rc != 0:
        raise ValueError("oracle rejected the arguments")
    k_out = int(counts[8])
    idx = fk_index[:k_out].copy()
    if len(shape) == 0:
        coords = np.zeros((k_out, 0), np.int64)
    else:
        coords = np.stack(np.unravel_index(idx, shape), axis=1).astype(np.int64) \
            if k_out else np.zeros((0, len(shape)), np.int64)
    mismatch = int(counts[0])
    return {
        "pass": mismatch == 0,
        "numel": numel,
        "rank": len(shape),
        "mismatch": mismatch,
        "match_fraction": 1.0 if numel == 0 else (numel - mismatch) / numel,
        "cand_nan": int(counts[1]), "cand_posinf": int(counts[2]),
        "cand_neginf": int(counts[3]), "ref_nan": int(counts[4]),
        "ref_posinf": int(counts[5]), "ref_neginf": int(counts[6]),
        "n_finite_pairs": int(counts[7]),
        "max_abs": float(fstats[0]), "argmax_abs": int(argmax[0]),
        "max_rel": float(fstats[1]), "argmax_rel": int(argmax[1]),
        "sse": float(fstats[2]),
        "grid_rows": gr, "grid_cols": gc, "tile_rows": th, "tile_cols": tw,
        "tile_hist": hist[:gr * gc].reshape(gr, gc),
        "row_prof": row_prof, "col_prof": col_prof,
        "k_out": k_out, "fk_index": idx, "fk_coords": coords,
        "fk_cand": fk_cand[:k_out].copy(), "fk_ref": fk_ref[:k_out].copy(),
        "flags": int(flags[0]),
        "input_eq": input_eq[:n_in].copy(),
        "passthrough_input": int(passthrough[0]),
    }


def _validate_batch(fn, cases) -> dict:
    results = [fn(c["cand"], c["ref"], inputs=c.get("inputs", ()),
                  rtol=c["rtol"], atol=c["atol"], tile=c["tile"],
                  first_k=c["first_k"]) for c in cases]
    return {"results": results, "n_pass": sum(int(r["pass"]) for r in results)}


def validate_batch(cases) -> dict:
    """P7: each case validated independently; the batch pass count is the sum."""
    return _validate_batch(validate, cases)


STAT_COUNTS = ("n_finite", "n_nan", "n_posinf", "n_neginf", "n_zero")
STAT_VALUES = ("min", "max", "sum", "sumsq", "mean", "std")


def _stat_dict(cnt, f):
    d = {k: int(v) for k, v in zip(STAT_COUNTS, cnt)}
    d.update({k: float(v) for k, v in zip(STAT_VALUES, f)})
    return d


def stats(x: torch.Tensor, *, tile=(64, 64)) -> dict:
    """Diagnostic tensor statistics of one CPU tensor (see oracle_stats in
    nmv_oracle.c): the whole tensor, and every tile of the [M, N] view."""
    return _stats(_load(), x, tile=tile)


def _stats(lib, x: torch.Tensor, *, tile=(64, 64)) -> dict:
    if x.dtype not in DTYPE_CODES:
        raise ValueError("unsupported dtype %s" % x.dtype)
    x = x.detach().cpu().contiguous()
    shape = tuple(x.shape)
    numel = x.numel()
    m, n = view_2d(shape)
    th, tw = int(tile[0]), int(tile[1])
    gr = -(-m // th) if numel else 0
    gc = -(-n // tw) if numel else 0
    counts = np.zeros(5, np.int64)
    f = np.zeros(6, np.float64)
    first = np.zeros(2, np.int64)
    tcnt = np.zeros(max(gr * gc, 1) * 5, np.int64)
    tf = np.zeros(max(gr * gc, 1) * 6, np.float64)
    rc = lib.oracle_stats(ctypes.c_void_p(x.data_ptr()), DTYPE_CODES[x.dtype], numel, max(n, 1),
                          th, tw, _ptr(counts, ctypes.c_int64), _ptr(f, ctypes.c_double),
                          _ptr(first, ctypes.c_int64), _ptr(tcnt, ctypes.c_int64),
                          _ptr(tf, ctypes.c_double))
    if rc != 0:
        raise ValueError("oracle rejected the arguments")
    tiles = {k: tcnt[i:gr * gc * 5:5].reshape(gr, gc).copy() for i, k in enumerate(STAT_COUNTS)}
    tiles.update({k: tf[i:gr * gc * 6:6].reshape(gr, gc).copy() for i, k in enumerate(STAT_VALUES)})
    return {"numel": numel, "rank": len(shape), "all": _stat_dict(counts, f),
            "first_nan": int(first[0]), "first_inf": int(first[1]),
            "grid_rows": gr, "grid_cols": gc, "tile_rows": th, "tile_cols": tw, "tiles": tiles}


FX_FLAGS = {"NEAR_PASS": 1, "F16_CEILING": 2, "AXIS_GROWTH": 4}
ULP_BINS = 34


def forensics(cand: torch.Tensor, ref: torch.Tensor, **kw) -> dict:
    """Deep forensics of one pair of CPU tensors (see oracle_forensics in
    nmv_oracle.c): ulp distances, fp16-ceiling counts, error growth along an
    axis, mismatch marginals of every axis and the scheduling flags."""
    return _forensics(_load(), cand, ref, **kw)


def _forensics(lib, cand, ref, *, rtol, atol, axis=-1, near_ulps=4, near_fraction=0.01,
               growth_factor=4.0) -> dict:
    if cand.dtype != ref.dtype or tuple(cand.shape) != tuple(ref.shape):
        raise ValueError("cand and ref must share dtype and shape")
    cand = cand.detach().cpu().contiguous()
    ref = ref.detach().cpu().contiguous()
    shape = tuple(int(s) for s in cand.shape)
    rank = len(shape)
    ax = (axis % rank) if rank else 0
    length = shape[ax] if rank else 1
    counts = np.zeros(6, np.int64)
    hist = np.zeros(ULP_BINS, np.int64)
    growth = np.zeros(max(length, 1), np.float64)
    gmean = np.zeros(2, np.float64)
    marg = np.zeros(max(sum(shape), 1), np.int64)
    flags = np.zeros(1, np.uint32)
    shp = (ctypes.c_int64 * max(rank, 1))(*shape)
    rc = lib.oracle_forensics(ctypes.c_void_p(cand.data_ptr()), ctypes.c_void_p(ref.data_ptr()),
                              DTYPE_CODES[cand.dtype], rank, shp, float(rtol), float(atol), ax,
                              int(near_ulps), float(near_fraction), float(growth_factor),
                              _ptr(counts, ctypes.c_int64), _ptr(hist, ctypes.c_int64),
                              _ptr(growth, ctypes.c_double), _ptr(gmean, ctypes.c_double),
                              _ptr(marg, ctypes.c_int64), _ptr(flags, ctypes.c_uint32))
    if rc != 0:
        raise ValueError("oracle rejected the arguments")
    offs = np.concatenate([[0], np.cumsum(shape)]).astype(np.int64) if rank else np.zeros(1, np.int64)
    return {"numel": cand.numel(), "rank": rank, "mismatch": int(counts[0]),
            "n_finite_pairs": int(counts[1]), "ulp_hist": hist,
            "max_ulp_mismatch": int(counts[2]), "argmax_ulp_mismatch": int(counts[3]),
            "mism_nonfinite": int(counts[4]), "mism_within_f16": int(counts[5]),
            "flags": int(flags[0]), "axis": ax, "axis_len": length, "growth": growth[:length].copy(),
            "growth_lo": float(gmean[0]), "growth_hi": float(gmean[1]),
            "marginals": [marg[offs[a]:offs[a + 1]].copy() for a in range(rank)]}


# ---- full-coverage escalation (Section 4.3; Figure 3, bottom-right; S6.1)
def _hazard(flags: int) -> bool:
    """An integrity hazard: the candidate passes an input through, or is
    constant / all zero while the reference is not."""
    if flags & 1:
        return True
    if (flags & 4) and not (flags & 16):
        return True
    if (flags & 2) and not (flags & 8):
        return True
    return False


def sweep(light, extended=()) -> dict:
    """The escalation policy written out: validate the lightweight set; only
    if every case passes, validate the extended set; accept when every case
    of both sets passed and none raised an integrity hazard.  The evidence
    is one header line and one line per validated case (the format of
    nmv_sweep in nmv.h), sealed with its SHA-256 digest."""
    import hashlib
    codes = DTYPE_CODES

    def run(cases):
        return [validate(c["cand"], c["ref"], inputs=c.get("inputs", ()), rtol=c["rtol"], atol=c["atol"],
                         tile=c["tile"], first_k=c["first_k"]) for c in cases]

    rl = run(light)
    pass_l = sum(int(r["pass"]) for r in rl)
    escalate = pass_l == len(light) and len(extended) > 0
    re_ = run(extended) if escalate else []
    pass_e = sum(int(r["pass"]) for r in re_)
    hazard = any(_hazard(r["flags"]) for r in rl + re_)
    accepted = pass_l == len(light) and (len(extended) == 0 or (escalate and pass_e == len(extended))) \
        and not hazard
    lines = ["nmv-sweep v1 light=%d ext=%d escalated=%d accepted=%d pass_light=%d pass_ext=%d"
             % (len(light), len(extended), int(escalate), int(accepted), pass_l, pass_e)]

    def line(tag, i, r, c):
        nonfin = (r["cand_nan"] + r["cand_posinf"] + r["cand_neginf"] + r["ref_nan"] + r["ref_posinf"]
                  + r["ref_neginf"])
        return ("%s %d dtype=%d numel=%d pass=%d mismatch=%d match=%.17g max_abs=%.17g max_rel=%.17g "
                "nonfinite=%d flags=%d" % (tag, i, codes[c["cand"].dtype], r["numel"], int(r["pass"]),
                                           r["mismatch"], r["match_fraction"], r["max_abs"], r["max_rel"],
                                           nonfin, r["flags"]))

    lines += [line("L", i, r, c) for i, (r, c) in enumerate(zip(rl, light))]
    lines += [line("E", i, r, c) for i, (r, c) in enumerate(zip(re_, extended))]
    evidence = "".join(ln + "\n" for ln in lines)
    flags_any = 0
    for r in rl + re_:
        flags_any |= r["flags"]
    return {"escalated": escalate, "accepted": accepted, "flags_any": flags_any,
            "n_light": len(light), "n_ext": len(extended), "n_run": len(rl) + len(re_),
            "n_pass_light": pass_l, "n_pass_ext": pass_e,
            "match_rate_light": pass_l / len(light),
            "match_rate_ext": pass_e / len(extended) if escalate else 0.0,
            "evidence": evidence, "digest": hashlib.sha256(evidence.encode()).hexdigest(),
            "results": rl + re_}
