"""Field-by-field comparison of a GPU result with the oracle's.

Every integer, index, flag and map must be equal; max_abs / max_rel and the
first-K values must be bit-identical (NaN matches NaN); the sum of squared
errors must agree to a relative 1e-9 (the tolerance the validation contract
states for it)."""
import numpy as np

SSE_RTOL = 1e-9


def _f64_same(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    if a.shape != b.shape:
        return False
    return bool(((a.view(np.int64) == b.view(np.int64)) | (np.isnan(a) & np.isnan(b))).all())


def diff(got, want):
    bad = []
    for key, w in want.items():
        g = got[key]
        if key == "sse":
            ok = g == w or abs(g - w) <= SSE_RTOL * abs(w)
        elif key in ("max_abs", "max_rel", "fk_cand", "fk_ref", "match_fraction"):
            ok = _f64_same(g, w)
        elif isinstance(w, np.ndarray):
            ok = isinstance(g, np.ndarray) and g.shape == w.shape and bool((g == w).all())
        else:
            ok = g == w
        if not ok:
            bad.append(key)
    return bad


def assert_same(got, want, name=""):
    bad = diff(got, want)
    if bad:
        lines = ["%s: GPU and oracle differ in %s" % (name, bad)]
        for k in bad[:6]:
            g, w = got[k], want[k]
            if isinstance(w, np.ndarray) and w.size > 8:
                idx = np.flatnonzero(np.asarray(g).reshape(-1) != np.asarray(w).reshape(-1))[:5] \
                    if np.asarray(g).shape == w.shape else []
                lines.append("  %s: shapes %s/%s first diffs at %s" % (
                    k, np.asarray(g).shape, w.shape, list(idx)))
            else:
                lines.append("  %s: gpu=%r oracle=%r" % (k, g, w))
        raise AssertionError("\n".join(lines))
