"""ctypes binding of libnmv.so (include/nmv.h): argument marshalling only.

Every step of the validation runs in the library's CUDA kernels; this module
turns torch CUDA tensors into ``nmv_tensor`` / ``nmv_case`` structs, calls the
C ABI, and copies the returned ``nmv_result`` into a dict.  It raises if the
library is missing: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libnmv.so")

NMV_OK, NMV_EINVAL, NMV_ENOMEM, NMV_ECUDA, NMV_EUNSUPPORTED, NMV_ETIMEOUT = 0, -1, -2, -3, -4, -5
MAX_RANK, MAX_INPUTS = 8, 8
DTYPES = {torch.float32: 0, torch.float16: 1, torch.bfloat16: 2, torch.int32: 3}
FLAGS = {"CAND_EQ_INPUT": 1, "CAND_ALL_ZERO": 2, "CAND_CONSTANT": 4,
         "REF_ALL_ZERO": 8, "REF_CONSTANT": 16}

_i64p = ctypes.POINTER(ctypes.c_int64)
_f64p = ctypes.POINTER(ctypes.c_double)


class Tensor(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("dtype", ctypes.c_int32),
                ("rank", ctypes.c_int32), ("shape", _i64p)]


class Profile(ctypes.Structure):
    _fields_ = [("scan_ms", ctypes.c_double), ("finalize_ms", ctypes.c_double),
                ("kernel_launches", ctypes.c_int64), ("h2d_bytes", ctypes.c_int64),
                ("d2h_bytes", ctypes.c_int64), ("slow_steps", ctypes.c_int64),
                ("light_steps", ctypes.c_int64),
                ("exact_abs", ctypes.c_int64), ("exact_rel", ctypes.c_int64),
                ("exact_pred", ctypes.c_int64), ("slow_cycles", ctypes.c_int64),
                ("light_cycles", ctypes.c_int64), ("dense_steps", ctypes.c_int64),
                ("dense_cycles", ctypes.c_int64), ("workspace_allocs", ctypes.c_int64),
                ("workspace_bytes", ctypes.c_int64)]


class Case(ctypes.Structure):
    _fields_ = [("cand", Tensor), ("ref", Tensor), ("inputs", ctypes.POINTER(Tensor)),
                ("n_inputs", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("rtol", ctypes.c_double), ("atol", ctypes.c_double),
                ("tile_rows", ctypes.c_int64), ("tile_cols", ctypes.c_int64),
                ("first_k", ctypes.c_int64)]


class Result(ctypes.Structure):
    _fields_ = [("status", ctypes.c_int32), ("rank", ctypes.c_int32), ("numel", ctypes.c_int64),
                ("pass_", ctypes.c_int32), ("flags", ctypes.c_uint32),
                ("mismatch", ctypes.c_int64), ("cand_nan", ctypes.c_int64),
                ("cand_posinf", ctypes.c_int64), ("cand_neginf", ctypes.c_int64),
                ("ref_nan", ctypes.c_int64), ("ref_posinf", ctypes.c_int64),
                ("ref_neginf", ctypes.c_int64), ("n_finite_pairs", ctypes.c_int64),
                ("max_abs", ctypes.c_double), ("max_rel", ctypes.c_double),
                ("sse", ctypes.c_double), ("argmax_abs", ctypes.c_int64),
                ("argmax_rel", ctypes.c_int64), ("grid_rows", ctypes.c_int64),
                ("grid_cols", ctypes.c_int64), ("tile_rows", ctypes.c_int64),
                ("tile_cols", ctypes.c_int64), ("tile_hist", _i64p), ("row_prof", _i64p),
                ("col_prof", _i64p), ("k_out", ctypes.c_int64), ("fk_index", _i64p),
                ("fk_coords", _i64p), ("fk_cand", _f64p), ("fk_ref", _f64p),
                ("n_inputs", ctypes.c_int32), ("passthrough_input", ctypes.c_int32),
                ("input_eq", _i64p), ("match_fraction", ctypes.c_double)]


class StatsCase(ctypes.Structure):
    _fields_ = [("x", Tensor), ("tile_rows", ctypes.c_int64), ("tile_cols", ctypes.c_int64)]


STAT_COUNTS = ("n_finite", "n_nan", "n_posinf", "n_neginf", "n_zero")
STAT_VALUES = ("min", "max", "sum", "sumsq", "mean", "std")


class Stat(ctypes.Structure):
    _fields_ = [(k, ctypes.c_int64) for k in STAT_COUNTS] + [(k, ctypes.c_double) for k in STAT_VALUES]


class StatsResult(ctypes.Structure):
    _fields_ = [("status", ctypes.c_int32), ("rank", ctypes.c_int32), ("numel", ctypes.c_int64),
                ("all", Stat), ("first_nan", ctypes.c_int64), ("first_inf", ctypes.c_int64),
                ("grid_rows", ctypes.c_int64), ("grid_cols", ctypes.c_int64),
                ("tile_rows", ctypes.c_int64), ("tile_cols", ctypes.c_int64),
                ("tiles", ctypes.POINTER(Stat))]


ULP_BINS = 34
FX_FLAGS = {"NEAR_PASS": 1, "F16_CEILING": 2, "AXIS_GROWTH": 4}


class ForensicsCase(ctypes.Structure):
    _fields_ = [("cand", Tensor), ("ref", Tensor), ("rtol", ctypes.c_double), ("atol", ctypes.c_double),
                ("axis", ctypes.c_int32), ("reserved", ctypes.c_int32), ("near_ulps", ctypes.c_int64),
                ("near_fraction", ctypes.c_double), ("growth_factor", ctypes.c_double)]


class ForensicsResult(ctypes.Structure):
    _fields_ = [("status", ctypes.c_int32), ("rank", ctypes.c_int32), ("numel", ctypes.c_int64),
                ("mismatch", ctypes.c_int64), ("n_finite_pairs", ctypes.c_int64),
                ("ulp_hist", ctypes.c_int64 * ULP_BINS), ("max_ulp_mismatch", ctypes.c_int64),
                ("argmax_ulp_mismatch", ctypes.c_int64), ("mism_nonfinite", ctypes.c_int64),
                ("mism_within_f16", ctypes.c_int64), ("flags", ctypes.c_uint32), ("axis", ctypes.c_int32),
                ("axis_len", ctypes.c_int64), ("growth_lo", ctypes.c_double), ("growth_hi", ctypes.c_double),
                ("growth", _f64p), ("marg_off", ctypes.c_int64 * (MAX_RANK + 1)), ("marginals", _i64p)]


class SweepReport(ctypes.Structure):
    _fields_ = [("status", ctypes.c_int32), ("escalated", ctypes.c_int32), ("accepted", ctypes.c_int32),
                ("flags_any", ctypes.c_uint32), ("n_light", ctypes.c_int64), ("n_ext", ctypes.c_int64),
                ("n_run", ctypes.c_int64), ("n_pass_light", ctypes.c_int64), ("n_pass_ext", ctypes.c_int64),
                ("match_rate_light", ctypes.c_double), ("match_rate_ext", ctypes.c_double),
                ("digest", ctypes.c_uint8 * 32), ("evidence", ctypes.c_char_p),
                ("evidence_len", ctypes.c_int64), ("results", ctypes.POINTER(Result)),
                ("blocks", ctypes.POINTER(Result) * 2)]


_lock = threading.Lock()
_lib = None


def load() -> ctypes.CDLL:
    """Load libnmv.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(
                    "libnmv.so is not built (run __graft_entry__.build() or "
                    "python -m paper_2608_02712_gb300._build); there is no fallback")
            lib = ctypes.CDLL(LIB_PATH)
            lib.nmv_validate.restype = ctypes.c_int
            lib.nmv_validate.argtypes = [ctypes.POINTER(Case), ctypes.c_void_p,
                                         ctypes.POINTER(ctypes.POINTER(Result))]
            lib.nmv_validate_batch.restype = ctypes.c_int
            lib.nmv_validate_batch.argtypes = [ctypes.POINTER(Case), ctypes.c_int64,
                                               ctypes.c_void_p,
                                               ctypes.POINTER(ctypes.POINTER(Result))]
            lib.nmv_result_free.restype = None
            lib.nmv_result_free.argtypes = [ctypes.c_void_p]
            lib.nmv_forensics.restype = ctypes.c_int
            lib.nmv_forensics.argtypes = [ctypes.POINTER(ForensicsCase), ctypes.c_int64, ctypes.c_void_p,
                                          ctypes.POINTER(ctypes.POINTER(ForensicsResult))]
            lib.nmv_sweep.restype = ctypes.c_int
            lib.nmv_sweep.argtypes = [ctypes.POINTER(Case), ctypes.c_int64, ctypes.POINTER(Case),
                                      ctypes.c_int64, ctypes.c_void_p,
                                      ctypes.POINTER(ctypes.POINTER(SweepReport))]
            lib.nmv_sweep_free.restype = None
            lib.nmv_sweep_free.argtypes = [ctypes.POINTER(SweepReport)]
            lib.nmv_sha256.restype = None
            lib.nmv_sha256.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.POINTER(ctypes.c_uint8)]
            lib.nmv_stats.restype = ctypes.c_int
            lib.nmv_stats.argtypes = [ctypes.POINTER(StatsCase), ctypes.c_int64, ctypes.c_void_p,
                                      ctypes.POINTER(ctypes.POINTER(StatsResult))]
            lib.nmv_status_string.restype = ctypes.c_char_p
            lib.nmv_status_string.argtypes = [ctypes.c_int]
            lib.nmv_last_error.restype = ctypes.c_char_p
            lib.nmv_last_error.argtypes = []
            lib.nmv_profile_enable.restype = None
            lib.nmv_profile_enable.argtypes = [ctypes.c_int]
            lib.nmv_profile_last.restype = ctypes.c_int
            lib.nmv_profile_last.argtypes = [ctypes.POINTER(Profile)]
            lib.nmv_validate_noalloc.restype = ctypes.c_int
            lib.nmv_validate_noalloc.argtypes = [ctypes.POINTER(Case), ctypes.c_void_p,
                                                 ctypes.POINTER(Result)]
            _lib = lib
    return _lib


class NmvError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__("nmv status %d: %s" % (status, message))
        self.status = status


def _raise(lib, rc):
    raise NmvError(rc, (lib.nmv_last_error() or b"").decode() or
                   lib.nmv_status_string(rc).decode())


class _Keep:
    """Holds the ctypes objects a Case points into."""

    def __init__(self):
        self.items = []


def _tensor(t: torch.Tensor, keep: _Keep, device_only: bool = True) -> Tensor:
    if t.dtype not in DTYPES:
        raise TypeError("unsupported dtype %s" % t.dtype)
    if device_only and not t.is_cuda:
        raise ValueError("tensors must live on the CUDA device")
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    shape = (ctypes.c_int64 * max(t.dim(), 1))(*t.shape)
    keep.items.append(shape)
    return Tensor(ctypes.c_void_p(t.data_ptr() if t.numel() else 0), DTYPES[t.dtype],
                  t.dim(), ctypes.cast(shape, _i64p))


def make_case(cand, ref, *, inputs=(), rtol, atol, tile=(64, 64), first_k=256,
              keep: _Keep | None = None) -> tuple[Case, _Keep]:
    keep = keep or _Keep()
    c = Case()
    c.cand = _tensor(cand, keep)
    c.ref = _tensor(ref, keep)
    if inputs:
        arr = (Tensor * len(inputs))(*[_tensor(x, keep) for x in inputs])
        keep.items.append(arr)
        c.inputs = ctypes.cast(arr, ctypes.POINTER(Tensor))
    c.n_inputs = len(inputs)
    c.reserved = 0
    c.rtol, c.atol = float(rtol), float(atol)
    c.tile_rows, c.tile_cols = int(tile[0]), int(tile[1])
    c.first_k = int(first_k)
    keep.items.extend([cand, ref, *inputs])
    return c, keep


def _arr(ptr, n, dtype):
    if n == 0:
        return np.zeros(0, dtype)
    return np.ctypeslib.as_array(ptr, shape=(n,)).astype(dtype, copy=True)


def result_to_dict(r: Result) -> dict:
    numel, mismatch = int(r.numel), int(r.mismatch)
    gr, gc = int(r.grid_rows), int(r.grid_cols)
    k = int(r.k_out)
    return {
        "pass": bool(r.pass_), "numel": numel, "rank": int(r.rank), "mismatch": mismatch,
        "match_fraction": float(r.match_fraction),
        "cand_nan": int(r.cand_nan), "cand_posinf": int(r.cand_posinf),
        "cand_neginf": int(r.cand_neginf), "ref_nan": int(r.ref_nan),
        "ref_posinf": int(r.ref_posinf), "ref_neginf": int(r.ref_neginf),
        "n_finite_pairs": int(r.n_finite_pairs),
        "max_abs": float(r.max_abs), "argmax_abs": int(r.argmax_abs),
        "max_rel": float(r.max_rel), "argmax_rel": int(r.argmax_rel), "sse": float(r.sse),
        "grid_rows": gr, "grid_cols": gc, "tile_rows": int(r.tile_rows),
        "tile_cols": int(r.tile_cols),
        "tile_hist": _arr(r.tile_hist, gr * gc, np.int64).reshape(gr, gc),
        "row_prof": _arr(r.row_prof, int(r.tile_rows), np.int64),
        "col_prof": _arr(r.col_prof, int(r.tile_cols), np.int64),
        "k_out": k, "fk_index": _arr(r.fk_index, k, np.int64),
        "fk_coords": _arr(r.fk_coords, k * int(r.rank), np.int64).reshape(k, int(r.rank)),
        "fk_cand": _arr(r.fk_cand, k, np.float64), "fk_ref": _arr(r.fk_ref, k, np.float64),
        "flags": int(r.flags), "input_eq": _arr(r.input_eq, int(r.n_inputs), np.int64),
        "passthrough_input": int(r.passthrough_input),
    }


def _stream_handle(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def validate(cand: torch.Tensor, ref: torch.Tensor, *, inputs=(), rtol: float, atol: float,
             tile=(64, 64), first_k: int = 256, stream=None) -> dict:
    """Validate one candidate/reference pair on the GPU (nmv_validate)."""
    lib = load()
    case, keep = make_case(cand, ref, inputs=inputs, rtol=rtol, atol=atol, tile=tile,
                           first_k=first_k)
    out = ctypes.POINTER(Result)()
    rc = lib.nmv_validate(ctypes.byref(case), _stream_handle(stream), ctypes.byref(out))
    if rc != NMV_OK:
        _raise(lib, rc)
    try:
        return result_to_dict(out[0])
    finally:
        lib.nmv_result_free(out)
        del keep


def validate_batch(cases, stream=None) -> dict:
    """Validate many pairs in one call (nmv_validate_batch).  `cases` holds
    dicts with keys cand, ref, rtol, atol, tile, first_k and optional inputs."""
    lib = load()
    keep = _Keep()
    structs = [make_case(c["cand"], c["ref"], inputs=c.get("inputs", ()), rtol=c["rtol"],
                         atol=c["atol"], tile=c["tile"], first_k=c["first_k"], keep=keep)[0]
               for c in cases]
    arr = (Case * max(len(structs), 1))(*structs)
    out = ctypes.POINTER(Result)()
    rc = lib.nmv_validate_batch(arr, len(structs), _stream_handle(stream), ctypes.byref(out))
    if rc != NMV_OK:
        _raise(lib, rc)
    try:
        results = [result_to_dict(out[i]) for i in range(len(structs))]
    finally:
        if out:
            lib.nmv_result_free(out)
    return {"results": results, "n_pass": sum(int(r["pass"]) for r in results)}


def validate_noalloc(cand: torch.Tensor, ref: torch.Tensor, *, inputs=(), rtol: float,
                     atol: float, tile=(64, 64), first_k: int = 256, stream=None) -> dict:
    """Validate one pair through nmv_validate_noalloc, the entry point that
    allocates no device or pinned memory (its scratch is a fixed array in the
    library; see nmv.h).  The output arrays are host arrays owned here."""
    lib = load()
    case, keep = make_case(cand, ref, inputs=inputs, rtol=rtol, atol=atol, tile=tile,
                           first_k=first_k)
    shape = list(cand.shape)
    n = cand.shape[-1] if cand.dim() else 1
    m = cand.numel() // n if (cand.dim() and n) else (0 if cand.numel() == 0 else 1)
    if cand.numel() == 0:
        gr = gc = 0
    else:
        gr, gc = -(-m // int(tile[0])), -(-n // int(tile[1]))
    k = int(first_k)
    bufs = {
        "tile_hist": np.zeros(max(gr * gc, 1), np.int64),
        "row_prof": np.zeros(int(tile[0]), np.int64),
        "col_prof": np.zeros(int(tile[1]), np.int64),
        "fk_index": np.zeros(max(k, 1), np.int64),
        "fk_coords": np.zeros(max(k * len(shape), 1), np.int64),
        "fk_cand": np.zeros(max(k, 1), np.float64),
        "fk_ref": np.zeros(max(k, 1), np.float64),
        "input_eq": np.zeros(max(len(inputs), 1), np.int64),
    }
    r = Result()
    for name, arr in bufs.items():
        ctype = ctypes.c_double if arr.dtype == np.float64 else ctypes.c_int64
        setattr(r, name, arr.ctypes.data_as(ctypes.POINTER(ctype)))
    rc = lib.nmv_validate_noalloc(ctypes.byref(case), _stream_handle(stream), ctypes.byref(r))
    if rc != NMV_OK:
        _raise(lib, rc)
    out = result_to_dict(r)
    del keep, bufs
    return out


class Prepared:
    """A case marshalled once and called many times (benchmark loops): each
    call() runs nmv_validate / nmv_validate_batch and frees the result."""

    def __init__(self, cases, stream=None):
        self.lib = load()
        self.keep = _Keep()
        self.structs = [make_case(c["cand"], c["ref"], inputs=c.get("inputs", ()),
                                  rtol=c["rtol"], atol=c["atol"], tile=c["tile"],
                                  first_k=c["first_k"], keep=self.keep)[0] for c in cases]
        self.arr = (Case * len(self.structs))(*self.structs)
        self.n = len(self.structs)
        self.stream = _stream_handle(stream)
        self.out = ctypes.POINTER(Result)()

    def call(self) -> int:
        if self.n == 1:
            rc = self.lib.nmv_validate(self.arr, self.stream, ctypes.byref(self.out))
        else:
            rc = self.lib.nmv_validate_batch(self.arr, self.n, self.stream, ctypes.byref(self.out))
        if rc != NMV_OK:
            _raise(self.lib, rc)
        self.lib.nmv_result_free(self.out)
        return rc

    def call_dicts(self) -> list:
        if self.n == 1:
            rc = self.lib.nmv_validate(self.arr, self.stream, ctypes.byref(self.out))
        else:
            rc = self.lib.nmv_validate_batch(self.arr, self.n, self.stream, ctypes.byref(self.out))
        if rc != NMV_OK:
            _raise(self.lib, rc)
        try:
            return [result_to_dict(self.out[i]) for i in range(self.n)]
        finally:
            self.lib.nmv_result_free(self.out)


def _stat_dict(st: Stat) -> dict:
    return {k: getattr(st, k) for k, _ in Stat._fields_}


class _ResultBlock:
    """Owns a result block of the library (a batch's records and arrays);
    the block is released when the last array viewing it is gone."""

    def __init__(self, lib, ptr):
        self._lib, self._ptr = lib, ptr

    def __del__(self):
        if self._ptr:
            self._lib.nmv_result_free(self._ptr)
            self._ptr = None


def _block_view(owner: _ResultBlock, addr: int, nbytes: int) -> np.ndarray:
    """nbytes of host memory at addr as a uint8 array that keeps owner alive."""
    buf = (ctypes.c_uint8 * nbytes).from_address(addr)
    buf._owner = owner
    return np.frombuffer(buf, dtype=np.uint8)


STAT_RECORD = np.dtype([(k, np.int64) for k in STAT_COUNTS] + [(k, np.float64) for k in STAT_VALUES])


def stats_result_to_dict(r: StatsResult, owner: "_ResultBlock | None" = None) -> dict:
    """One case's statistics.  With owner, the tile arrays are views of the
    library's result block (no copy); without, copies."""
    gr, gc = int(r.grid_rows), int(r.grid_cols)
    n = gr * gc
    tiles = {}
    if n:
        addr = ctypes.cast(r.tiles, ctypes.c_void_p).value
        if owner is not None:
            rec = _block_view(owner, addr, n * ctypes.sizeof(Stat)).view(STAT_RECORD)
            tiles = {k: rec[k].reshape(gr, gc) for k in STAT_COUNTS + STAT_VALUES}
        else:
            raw = np.ctypeslib.as_array(ctypes.cast(r.tiles, ctypes.POINTER(ctypes.c_uint8)),
                                        shape=(n * ctypes.sizeof(Stat),))
            rec = raw.view(STAT_RECORD)
            tiles = {k: rec[k].reshape(gr, gc).copy() for k in STAT_COUNTS + STAT_VALUES}
    else:
        tiles = {k: np.zeros((gr, gc), np.int64 if k in STAT_COUNTS else np.float64)
                 for k in STAT_COUNTS + STAT_VALUES}
    return {"numel": int(r.numel), "rank": int(r.rank), "all": _stat_dict(r.all),
            "first_nan": int(r.first_nan), "first_inf": int(r.first_inf), "grid_rows": gr,
            "grid_cols": gc, "tile_rows": int(r.tile_rows), "tile_cols": int(r.tile_cols),
            "tiles": tiles}


def stats_batch(items, stream=None) -> list:
    """Diagnostic statistics of several buffers in one call (nmv_stats);
    `items` holds (tensor, (tile_rows, tile_cols)) pairs."""
    lib = load()
    keep = _Keep()
    structs = []
    for x, tile in items:
        c = StatsCase()
        c.x = _tensor(x, keep)
        c.tile_rows, c.tile_cols = int(tile[0]), int(tile[1])
        keep.items.append(x)
        structs.append(c)
    arr = (StatsCase * max(len(structs), 1))(*structs)
    out = ctypes.POINTER(StatsResult)()
    rc = lib.nmv_stats(arr, len(structs), _stream_handle(stream), ctypes.byref(out))
    if rc != NMV_OK:
        _raise(lib, rc)
    owner = _ResultBlock(lib, ctypes.cast(out, ctypes.c_void_p).value)
    return [stats_result_to_dict(out[i], owner) for i in range(len(structs))]


def stats(x: torch.Tensor, *, tile=(64, 64), stream=None) -> dict:
    """Diagnostic statistics of one buffer (nmv_stats): the whole tensor and
    every tile of its [M, N] view.  The per-tile arrays are views of the
    library's result records (strided, no copy), valid as long as they are
    referenced."""
    return stats_batch([(x, tile)], stream=stream)[0]


def forensics_result_to_dict(r: ForensicsResult) -> dict:
    rank = int(r.rank)
    offs = [int(r.marg_off[a]) for a in range(rank + 1)]
    n_m = offs[-1] if rank else 0
    marg = _arr(r.marginals, n_m, np.int64)
    return {"numel": int(r.numel), "rank": rank, "mismatch": int(r.mismatch),
            "n_finite_pairs": int(r.n_finite_pairs),
            "ulp_hist": np.array(list(r.ulp_hist), np.int64),
            "max_ulp_mismatch": int(r.max_ulp_mismatch),
            "argmax_ulp_mismatch": int(r.argmax_ulp_mismatch),
            "mism_nonfinite": int(r.mism_nonfinite), "mism_within_f16": int(r.mism_within_f16),
            "flags": int(r.flags), "axis": int(r.axis), "axis_len": int(r.axis_len),
            "growth": _arr(r.growth, int(r.axis_len), np.float64),
            "growth_lo": float(r.growth_lo), "growth_hi": float(r.growth_hi),
            "marginals": [marg[offs[a]:offs[a + 1]].copy() for a in range(rank)]}


def forensics_batch(items, stream=None) -> list:
    """Deep forensics of several pairs in one call (nmv_forensics); each item
    is a dict with cand, ref, rtol, atol and optional axis, near_ulps,
    near_fraction, growth_factor."""
    lib = load()
    keep = _Keep()
    structs = []
    for it in items:
        c = ForensicsCase()
        c.cand = _tensor(it["cand"], keep)
        c.ref = _tensor(it["ref"], keep)
        c.rtol, c.atol = float(it["rtol"]), float(it["atol"])
        c.axis = int(it.get("axis", -1))
        c.reserved = 0
        c.near_ulps = int(it.get("near_ulps", 4))
        c.near_fraction = float(it.get("near_fraction", 0.01))
        c.growth_factor = float(it.get("growth_factor", 4.0))
        keep.items.extend([it["cand"], it["ref"]])
        structs.append(c)
    arr = (ForensicsCase * max(len(structs), 1))(*structs)
    out = ctypes.POINTER(ForensicsResult)()
    rc = lib.nmv_forensics(arr, len(structs), _stream_handle(stream), ctypes.byref(out))
    if rc != NMV_OK:
        _raise(lib, rc)
    try:
        return [forensics_result_to_dict(out[i]) for i in range(len(structs))]
    finally:
        if out:
            lib.nmv_result_free(out)


def forensics(cand: torch.Tensor, ref: torch.Tensor, *, rtol: float, atol: float, axis: int = -1,
              near_ulps: int = 4, near_fraction: float = 0.01, growth_factor: float = 4.0,
              stream=None) -> dict:
    """Deep forensics of one pair (nmv_forensics): ulp distances, the fp16
    ceiling, error growth along an axis, per-axis mismatch marginals."""
    return forensics_batch([dict(cand=cand, ref=ref, rtol=rtol, atol=atol, axis=axis, near_ulps=near_ulps,
                                 near_fraction=near_fraction, growth_factor=growth_factor)], stream=stream)[0]


def sha256(data: bytes) -> str:
    """The library's SHA-256 (the sweep evidence digest) of `data`, as hex."""
    lib = load()
    out = (ctypes.c_uint8 * 32)()
    buf = ctypes.create_string_buffer(data, len(data))
    lib.nmv_sha256(buf, len(data), out)
    return bytes(out).hex()


def sweep(light, extended=(), stream=None) -> dict:
    """Full-coverage escalation (nmv_sweep): the lightweight cases first, the
    extended ones only if every lightweight case passed.  Cases are dicts as
    for validate_batch.  Returns the report with its evidence text, SHA-256
    digest and the per-case results."""
    lib = load()
    keep = _Keep()

    def arr(cases):
        structs = [make_case(c["cand"], c["ref"], inputs=c.get("inputs", ()), rtol=c["rtol"], atol=c["atol"],
                             tile=c["tile"], first_k=c["first_k"], keep=keep)[0] for c in cases]
        return (Case * max(len(structs), 1))(*structs), len(structs)

    la, nl = arr(light)
    ea, ne = arr(extended)
    out = ctypes.POINTER(SweepReport)()
    rc = lib.nmv_sweep(la, nl, ea, ne, _stream_handle(stream), ctypes.byref(out))
    if rc != NMV_OK:
        _raise(lib, rc)
    try:
        r = out[0]
        return {"escalated": bool(r.escalated), "accepted": bool(r.accepted), "flags_any": int(r.flags_any),
                "n_light": int(r.n_light), "n_ext": int(r.n_ext), "n_run": int(r.n_run),
                "n_pass_light": int(r.n_pass_light), "n_pass_ext": int(r.n_pass_ext),
                "match_rate_light": float(r.match_rate_light), "match_rate_ext": float(r.match_rate_ext),
                "digest": bytes(r.digest).hex(),
                "evidence": ctypes.string_at(r.evidence, int(r.evidence_len)).decode(),
                "results": [result_to_dict(r.results[i]) for i in range(int(r.n_run))]}
    finally:
        lib.nmv_sweep_free(out)


class PreparedSweep:
    """A sweep's case sets marshalled once and run many times (benchmark
    loops): each call() runs nmv_sweep and releases the report."""

    def __init__(self, light, extended=(), stream=None):
        self.lib = load()
        self.keep = _Keep()

        def arr(cases):
            structs = [make_case(c["cand"], c["ref"], inputs=c.get("inputs", ()), rtol=c["rtol"],
                                 atol=c["atol"], tile=c["tile"], first_k=c["first_k"], keep=self.keep)[0]
                       for c in cases]
            return (Case * max(len(structs), 1))(*structs), len(structs)

        self.la, self.nl = arr(light)
        self.ea, self.ne = arr(extended)
        self.stream = _stream_handle(stream)

    def call(self) -> int:
        out = ctypes.POINTER(SweepReport)()
        rc = self.lib.nmv_sweep(self.la, self.nl, self.ea, self.ne, self.stream, ctypes.byref(out))
        if rc != NMV_OK:
            _raise(self.lib, rc)
        self.lib.nmv_sweep_free(out)
        return rc


PROFILE_TIMING = 1
PROFILE_COUNTERS = 2


def profile_enable(mode: int = PROFILE_TIMING) -> None:
    """Profile every following call: PROFILE_TIMING records CUDA events
    around the kernels, PROFILE_COUNTERS counts the scan's exact-path work
    (and slows it down); 0 or False turns profiling off."""
    load().nmv_profile_enable(int(mode))


def profile_last() -> dict:
    """Launch profile of the last profiled call (see nmv_profile in nmv.h)."""
    lib = load()
    p = Profile()
    rc = lib.nmv_profile_last(ctypes.byref(p))
    if rc != NMV_OK:
        _raise(lib, rc)
    return {name: getattr(p, name) for name, _ in Profile._fields_}
