/*
 * nmv_oracle.c -- plain, slow, single-threaded CPU oracle for numerical
 * validation with failure forensics.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg and reference arm may load this library.  The product path
 * (the CUDA library and its Python binding) never calls it, includes it or
 * shares a line of code, a header or a table with it.
 *
 * What it computes comes from the paper's problem statement (Section 3.2,
 * Eq. 1 and the constraint Validate(K_fixed, R, T_ext, tau) = true): a
 * candidate output is checked against a reference output within a numerical
 * tolerance tau, and the diagnostic evidence D given to the repair agent
 * includes "numerical-deviation metrics" (Section 3.2).  The paper gives no
 * formula for the check, so every definition below is a written-out reading:
 *
 *   P1 pass predicate (allclose form, equal_nan = false), per element i,
 *      after widening both stored values to fp64 exactly:
 *         pass(i) = (c == r)  OR  (c, r finite AND
 *                   fl(|fl(c - r)|) <= fl(atol + fl(rtol * |r|)))
 *      NaN never passes; an infinity passes only against the same infinity.
 *   P2 counts: mismatch = #!pass; NaN/+Inf/-Inf counts of c and of r;
 *      n_finite_pairs = #{both finite}.  The match rate of Table S4 /
 *      Section 4.3 ("per-case pass/fail, numerical match rates") is
 *      (numel - mismatch) / numel.
 *   P3 error statistics over the both-finite set: d = fl(c - r), a = |d|,
 *      max a with the lowest index attaining it; rel = fl(a / |r|) for r != 0,
 *      max rel with the lowest index; sse = sum of fl(d * d) accumulated with
 *      Neumaier's compensated summation (Neumaier 1974).  No eligible
 *      element: max = 0.0, argmax = -1.
 *   P4 localisation (the "localize" step of the forensics, Section 4.2 and
 *      S2.2): 2-D view [M = prod(shape[:-1]), N = shape[-1]], row = i / N,
 *      col = i % N; for every mismatch tile_hist[(row/th)*GC + col/tw] += 1,
 *      row_prof[row % th] += 1, col_prof[col % tw] += 1.
 *   P5 first-K: the K lowest mismatching linear indices in ascending order,
 *      each with c and r widened to fp64.
 *   P6 degenerate-output flags (the "repair by degeneration" and bypass
 *      hazards, Sections 1, 2.2 and 4.3): see oracle_validate below.
 *
 * Build: gcc -std=c11 -O2 -ffp-contract=off -fPIC -shared (no FMA
 * contraction: every rounding above happens exactly where it is written).
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

enum { OR_F32 = 0, OR_F16 = 1, OR_BF16 = 2, OR_I32 = 3 };

/* Flag bits of the degenerate-output mask (interface format). */
#define OR_FLAG_CAND_EQ_INPUT 1u
#define OR_FLAG_CAND_ALL_ZERO 2u
#define OR_FLAG_CAND_CONSTANT 4u
#define OR_FLAG_REF_ALL_ZERO 8u
#define OR_FLAG_REF_CONSTANT 16u

/* ---- decoders: stored bit pattern -> exact fp64 value ------------------ */

/* IEEE 754 binary16: 1 sign bit, 5 exponent bits (bias 15), 10 fraction. */
double oracle_decode_f16(uint32_t bits)
{
    uint32_t sign = (bits >> 15) & 1u;
    uint32_t expo = (bits >> 10) & 31u;
    uint32_t frac = bits & 1023u;
    double v;
    if (expo == 0) {
        v = ldexp((double)frac, -24); /* subnormal: frac * 2^(1-15-10) */
    } else if (expo == 31) {
        v = (frac == 0) ? INFINITY : NAN;
    } else {
        v = ldexp((double)(1024u + frac), (int)expo - 25);
    }
    return sign ? -v : v;
}

/* bfloat16: 1 sign bit, 8 exponent bits (bias 127), 7 fraction bits. */
double oracle_decode_bf16(uint32_t bits)
{
    uint32_t sign = (bits >> 15) & 1u;
    uint32_t expo = (bits >> 7) & 255u;
    uint32_t frac = bits & 127u;
    double v;
    if (expo == 0) {
        v = ldexp((double)frac, -133); /* subnormal: frac * 2^(1-127-7) */
    } else if (expo == 255) {
        v = (frac == 0) ? INFINITY : NAN;
    } else {
        v = ldexp((double)(128u + frac), (int)expo - 134);
    }
    return sign ? -v : v;
}

/* IEEE 754 binary32: 1 sign bit, 8 exponent bits (bias 127), 23 fraction. */
double oracle_decode_f32(uint32_t bits)
{
    uint32_t sign = bits >> 31;
    uint32_t expo = (bits >> 23) & 255u;
    uint32_t frac = bits & 0x7fffffu;
    double v;
    if (expo == 0) {
        v = ldexp((double)frac, -149);
    } else if (expo == 255) {
        v = (frac == 0) ? INFINITY : NAN;
    } else {
        v = ldexp((double)(0x800000u + frac), (int)expo - 150);
    }
    return sign ? -v : v;
}

static int elem_size(int dtype)
{
    return (dtype == OR_F16 || dtype == OR_BF16) ? 2 : 4;
}

/* Raw stored bit pattern of element i (zero-extended to 32 bits). */
static uint32_t load_bits(const void *p, int dtype, int64_t i)
{
    if (elem_size(dtype) == 2) {
        uint16_t h;
        memcpy(&h, (const char *)p + 2 * i, 2);
        return h;
    }
    uint32_t w;
    memcpy(&w, (const char *)p + 4 * i, 4);
    return w;
}

static double decode(uint32_t bits, int dtype)
{
    switch (dtype) {
    case OR_F32: return oracle_decode_f32(bits);
    case OR_F16: return oracle_decode_f16(bits);
    case OR_BF16: return oracle_decode_bf16(bits);
    default: return (double)(int32_t)bits;
    }
}

/* P1: the pass predicate, exactly as written (no contraction). */
int oracle_pass(double c, double r, double rtol, double atol)
{
    if (c == r) return 1;
    if (!isfinite(c) || !isfinite(r)) return 0;
    double diff = c - r;
    double err = fabs(diff);
    double scaled = rtol * fabs(r);
    double allowed = atol + scaled;
    return err <= allowed;
}

/*
 * Validate one candidate/reference pair.
 *
 *   cand, ref      host buffers of numel elements of `dtype`, row-major.
 *   ncols          N = the last dimension (the 2-D view is [numel/N, N]);
 *                  for numel == 0 any value >= 1 is accepted.
 *   inputs[j]      optional operator inputs with input_dtype[j] and
 *                  input_numel[j]; only those with the candidate's dtype and
 *                  numel take part in the pass-through check.
 *
 * Outputs (all caller-allocated):
 *   counts[9]   mismatch, cand_nan, cand_posinf, cand_neginf, ref_nan,
 *               ref_posinf, ref_neginf, n_finite_pairs, k_out
 *   fstats[3]   max_abs, max_rel, sse
 *   argmax[2]   argmax_abs, argmax_rel
 *   tile_hist[GR*GC], row_prof[th], col_prof[tw]   (zeroed here)
 *   fk_index[K], fk_cand[K], fk_ref[K]
 *   input_eq[n_inputs]   pass-through count, or -1 when not eligible
 *   flags[1], passthrough[1]
 *
 * P6, the degenerate-output flags (our reading; the paper implements its
 * anti-cheat check on source code and gives no numeric rule):
 *   input_eq[j] = #{i : bits(c_i) == bits(x_ij) and bits(r_i) != bits(x_ij)}
 *   CAND_EQ_INPUT  some eligible j has input_eq[j] >= max(1, ceil(numel/100))
 *   CAND_ALL_ZERO  numel >= 1 and every c_i == 0 by value (+0 and -0)
 *   CAND_CONSTANT  numel >= 2 and every bits(c_i) == bits(c_0)
 *   REF_ALL_ZERO, REF_CONSTANT  the same two rules applied to r
 *   passthrough = the lowest flagged j, else -1.
 */
int oracle_validate(const void *cand, const void *ref, int dtype, int64_t numel,
                    int64_t ncols, int n_inputs, const void *const *inputs,
                    const int *input_dtype, const int64_t *input_numel,
                    double rtol, double atol, int64_t tile_rows,
                    int64_t tile_cols, int64_t first_k, int64_t *counts,
                    double *fstats, int64_t *argmax, int64_t *tile_hist,
                    int64_t *row_prof, int64_t *col_prof, int64_t *fk_index,
                    double *fk_cand, double *fk_ref, int64_t *input_eq,
                    uint32_t *flags, int32_t *passthrough)
{
    if (ncols < 1 || tile_rows < 1 || tile_cols < 1 || first_k < 0) return -1;
    if (n_inputs < 0 || n_inputs > 64) return -1;
    int64_t nrows = numel / ncols;
    int64_t grid_rows = (nrows + tile_rows - 1) / tile_rows;
    int64_t grid_cols = (ncols + tile_cols - 1) / tile_cols;
    if (numel == 0) grid_rows = grid_cols = 0;

    for (int64_t t = 0; t < grid_rows * grid_cols; ++t) tile_hist[t] = 0;
    for (int64_t t = 0; t < tile_rows; ++t) row_prof[t] = 0;
    for (int64_t t = 0; t < tile_cols; ++t) col_prof[t] = 0;

    int64_t mismatch = 0, cand_nan = 0, cand_posinf = 0, cand_neginf = 0;
    int64_t ref_nan = 0, ref_posinf = 0, ref_neginf = 0, n_finite = 0;
    int64_t k_out = 0;
    double max_abs = 0.0, max_rel = 0.0;
    int64_t arg_abs = -1, arg_rel = -1;
    double sse_sum = 0.0, sse_comp = 0.0; /* Neumaier: running sum + correction */

    int eligible[64];
    for (int j = 0; j < n_inputs; ++j) {
        eligible[j] = (input_dtype[j] == dtype && input_numel[j] == numel);
        input_eq[j] = eligible[j] ? 0 : -1;
    }

    int cand_all_zero = 1, cand_constant = 1, ref_all_zero = 1, ref_constant = 1;
    uint32_t c0 = 0, r0 = 0;
    if (numel > 0) {
        c0 = load_bits(cand, dtype, 0);
        r0 = load_bits(ref, dtype, 0);
    }

    for (int64_t i = 0; i < numel; ++i) {
        uint32_t cb = load_bits(cand, dtype, i);
        uint32_t rb = load_bits(ref, dtype, i);
        double c = decode(cb, dtype);
        double r = decode(rb, dtype);

        /* P2: classes of each side. */
        if (isnan(c)) cand_nan++;
        else if (isinf(c)) { if (c > 0) cand_posinf++; else cand_neginf++; }
        if (isnan(r)) ref_nan++;
        else if (isinf(r)) { if (r > 0) ref_posinf++; else ref_neginf++; }

        /* P1 + P4 + P5 */
        if (!oracle_pass(c, r, rtol, atol)) {
            mismatch++;
            int64_t row = i / ncols;
            int64_t col = i % ncols;
            tile_hist[(row / tile_rows) * grid_cols + col / tile_cols] += 1;
            row_prof[row % tile_rows] += 1;
            col_prof[col % tile_cols] += 1;
            if (k_out < first_k) {
                fk_index[k_out] = i;
                fk_cand[k_out] = c;
                fk_ref[k_out] = r;
                k_out++;
            }
        }

        /* P3 over the both-finite set, in ascending index order. */
        if (isfinite(c) && isfinite(r)) {
            n_finite++;
            double d = c - r;
            double a = fabs(d);
            if (arg_abs < 0 || a > max_abs) { max_abs = a; arg_abs = i; }
            if (r != 0.0) {
                double rel = a / fabs(r);
                if (arg_rel < 0 || rel > max_rel) { max_rel = rel; arg_rel = i; }
            }
            double term = d * d;
            double t = sse_sum + term;
            if (fabs(sse_sum) >= fabs(term)) sse_comp += (sse_sum - t) + term;
            else sse_comp += (term - t) + sse_sum;
            sse_sum = t;
        }

        /* P6 */
        if (!(c == 0.0)) cand_all_zero = 0;
        if (!(r == 0.0)) ref_all_zero = 0;
        if (cb != c0) cand_constant = 0;
        if (rb != r0) ref_constant = 0;
        for (int j = 0; j < n_inputs; ++j) {
            if (!eligible[j]) continue;
            uint32_t xb = load_bits(inputs[j], dtype, i);
            if (cb == xb && rb != xb) input_eq[j] += 1;
        }
    }

    uint32_t f = 0;
    int32_t pt = -1;
    int64_t threshold = (numel + 99) / 100; /* ceil(numel / 100) */
    if (threshold < 1) threshold = 1;
    for (int j = 0; j < n_inputs; ++j) {
        if (eligible[j] && input_eq[j] >= threshold) {
            f |= OR_FLAG_CAND_EQ_INPUT;
            if (pt < 0) pt = j;
        }
    }
    if (numel >= 1 && cand_all_zero) f |= OR_FLAG_CAND_ALL_ZERO;
    if (numel >= 2 && cand_constant) f |= OR_FLAG_CAND_CONSTANT;
    if (numel >= 1 && ref_all_zero) f |= OR_FLAG_REF_ALL_ZERO;
    if (numel >= 2 && ref_constant) f |= OR_FLAG_REF_CONSTANT;

    counts[0] = mismatch;
    counts[1] = cand_nan;
    counts[2] = cand_posinf;
    counts[3] = cand_neginf;
    counts[4] = ref_nan;
    counts[5] = ref_posinf;
    counts[6] = ref_neginf;
    counts[7] = n_finite;
    counts[8] = k_out;
    fstats[0] = max_abs;
    fstats[1] = max_rel;
    fstats[2] = sse_sum + sse_comp;
    argmax[0] = arg_abs;
    argmax[1] = arg_rel;
    flags[0] = f;
    passthrough[0] = pt;
    return 0;
}

/*
 * ---- diagnostic tensor statistics (the instrumentation probe) -----------
 *
 * The engine's diagnostic instrumentation (Section 4.2, "Diagnostic
 * instrumentation"; Figure 3 bottom-left; S5.1 "tensor-statistic
 * instrumentation") records multi-level tensor statistics at pipeline
 * boundaries so that diffuse precision failures can be localised.  The paper
 * gives no list of statistics and no formula; the reading written out here:
 *
 *   levels: the whole tensor, and every tile of the same [M, N] view and
 *           tile grid as the localisation maps (P4);
 *   per level, over its elements x_i (widened to fp64 exactly):
 *     n_finite, n_nan, n_posinf, n_neginf   class counts (int32: all finite)
 *     n_zero                                #{x_i == 0 by value} (+0 and -0)
 *     min, max                              over the finite x_i (0.0 if none)
 *     sum   = sum of the finite x_i
 *     sumsq = sum of x_i^2 over the finite x_i
 *     mean  = sum / n_finite                (0.0 if n_finite == 0)
 *     std   = sqrt(max(0, sumsq / n_finite - mean^2))   (0.0 if none)
 *             (the population standard deviation written with the two
 *             sums; each operation one fp64 rounding)
 *   tensor level only: first_nan / first_inf = the lowest index holding a
 *           NaN / an infinity of either sign, -1 if none.
 *
 * Sums: int32 elements are summed exactly (integers; x^2 in 128 bits) and
 * rounded once to fp64; float elements with Neumaier's compensated
 * summation in index order.
 *
 * Output layout: stat[11] = {n_finite, n_nan, n_posinf, n_neginf, n_zero}
 * as int64 in counts[5] and {min, max, sum, sumsq, mean, std} as fp64 in
 * f[6]; tile t (row-major on the tile grid) at counts + 5 t, f + 6 t.
 */
static void or_stat_finish(const int64_t *cnt, double *f)
{
    double n = (double)cnt[0];
    if (cnt[0] == 0) {
        f[0] = f[1] = f[2] = f[3] = f[4] = f[5] = 0.0;
        return;
    }
    double mean = f[2] / n;
    double ex2 = f[3] / n;
    double var = ex2 - mean * mean;
    f[4] = mean;
    f[5] = var > 0.0 ? sqrt(var) : 0.0;
}

typedef struct {
    int64_t cnt[5];
    double mn, mx;
    int have;
    /* float sums: Neumaier (running value + correction) */
    double s, sc, q, qc;
    /* int32 sums: exact */
    __int128 is, iq;
} or_acc;

static void or_acc_init(or_acc *a)
{
    memset(a, 0, sizeof(*a));
}

static void neumaier(double *sum, double *comp, double term)
{
    double t = *sum + term;
    if (fabs(*sum) >= fabs(term)) *comp += (*sum - t) + term;
    else *comp += (term - t) + *sum;
    *sum = t;
}

static void or_acc_add(or_acc *a, uint32_t bits, int dtype)
{
    if (dtype == OR_I32) {
        int64_t v = (int64_t)(int32_t)bits;
        a->cnt[0]++;
        if (v == 0) a->cnt[4]++;
        double d = (double)v;
        if (!a->have || d < a->mn) a->mn = d;
        if (!a->have || d > a->mx) a->mx = d;
        a->have = 1;
        a->is += v;
        a->iq += (__int128)(v * v);
        return;
    }
    double x = decode(bits, dtype);
    if (isnan(x)) { a->cnt[1]++; return; }
    if (isinf(x)) { if (x > 0) a->cnt[2]++; else a->cnt[3]++; return; }
    a->cnt[0]++;
    if (x == 0.0) a->cnt[4]++;
    if (!a->have || x < a->mn) a->mn = x;
    if (!a->have || x > a->mx) a->mx = x;
    a->have = 1;
    neumaier(&a->s, &a->sc, x);
    neumaier(&a->q, &a->qc, x * x);
}

static void or_acc_out(const or_acc *a, int dtype, int64_t *cnt, double *f)
{
    for (int k = 0; k < 5; ++k) cnt[k] = a->cnt[k];
    f[0] = a->have ? a->mn : 0.0;
    f[1] = a->have ? a->mx : 0.0;
    if (dtype == OR_I32) {
        f[2] = (double)a->is;   /* one rounding of the exact integer */
        f[3] = (double)a->iq;
    } else {
        f[2] = a->s + a->sc;
        f[3] = a->q + a->qc;
    }
    or_stat_finish(cnt, f);
}

int oracle_stats(const void *x, int dtype, int64_t numel, int64_t ncols, int64_t tile_rows,
                 int64_t tile_cols, int64_t *counts, double *f, int64_t *first,
                 int64_t *tile_counts, double *tile_f)
{
    if (ncols < 1 || tile_rows < 1 || tile_cols < 1 || numel < 0) return -1;
    int64_t nrows = numel / ncols;
    int64_t gr = numel ? (nrows + tile_rows - 1) / tile_rows : 0;
    int64_t gc = numel ? (ncols + tile_cols - 1) / tile_cols : 0;
    or_acc all;
    or_acc_init(&all);
    int64_t first_nan = -1, first_inf = -1;
    /* whole tensor, in index order */
    for (int64_t i = 0; i < numel; ++i) {
        uint32_t b = load_bits(x, dtype, i);
        or_acc_add(&all, b, dtype);
        if (dtype != OR_I32) {
            double v = decode(b, dtype);
            if (isnan(v) && first_nan < 0) first_nan = i;
            if (isinf(v) && first_inf < 0) first_inf = i;
        }
    }
    or_acc_out(&all, dtype, counts, f);
    first[0] = first_nan;
    first[1] = first_inf;
    /* every tile, its elements in index order */
    for (int64_t tr = 0; tr < gr; ++tr) {
        for (int64_t tc = 0; tc < gc; ++tc) {
            or_acc a;
            or_acc_init(&a);
            for (int64_t r = tr * tile_rows; r < nrows && r < (tr + 1) * tile_rows; ++r)
                for (int64_t c = tc * tile_cols; c < ncols && c < (tc + 1) * tile_cols; ++c)
                    or_acc_add(&a, load_bits(x, dtype, r * ncols + c), dtype);
            int64_t t = tr * gc + tc;
            or_acc_out(&a, dtype, tile_counts + 5 * t, tile_f + 6 * t);
        }
    }
    return 0;
}

/*
 * ---- deep forensics: per-axis maps, ulp distances, error growth ---------
 *
 * The evidence behind the adaptive-scheduling rules "near-pass and
 * fp16-ceiling detection" (Section 4.4) and behind localising a divergence
 * that "compounds along the reduction axis" (Section 3.2, the cumsum of
 * Table 1), plus mismatch counts at every index of every axis.  The paper
 * states no formula; the reading written out here, over the pairs of P1:
 *
 *   ord(x)    the order-preserving integer of a float's bits: +m for a
 *             positive sign, -m for a negative one (m = the magnitude bits),
 *             so +0 and -0 are both 0 and consecutive floats differ by 1;
 *             int32: the value itself
 *   u(i)      = |ord(c_i) - ord(r_i)|, the distance in representable values
 *   ulp_hist  both-finite pairs by u: bin 0 holds u = 0, bin k (1..33) holds
 *             2^(k-1) <= u < 2^k (bin 33 also everything above)
 *   max_ulp_mismatch / argmax   the largest u over finite mismatches
 *             (both values finite) and the lowest index attaining it (-1, -1)
 *   mism_nonfinite   mismatches where c or r is NaN or infinite
 *   mism_within_f16  finite mismatches with fl(|c - r|) <= h(r), h(r) the
 *             spacing of an 11-bit significand at |r|: 2^(max(e, -14) - 10)
 *             with e = floor(log2 |r|), and 2^-24 for r = 0 (one fp16 ulp,
 *             its exponent range unbounded above)
 *   growth[j] max fl(|c - r|) over both-finite pairs whose coordinate on the
 *             chosen axis is j (0.0 if none)
 *   growth_lo / growth_hi   the mean of growth[] over its first / last
 *             q = max(1, floor(len / 4)) entries: a left-to-right fp64 sum
 *             divided by q (0.0 for an empty axis)
 *   marginals mismatches at each index of each axis (axis 0 first)
 *   flags     NEAR_PASS (1): mismatch > 0, no non-finite mismatch,
 *               max_ulp_mismatch <= near_ulps and mismatch <= near_fraction
 *               * numel (fp64 product);
 *             F16_CEILING (2): mismatch > 0, no non-finite mismatch and
 *               mism_within_f16 == mismatch;
 *             AXIS_GROWTH (4): len >= 4, growth_hi > 0 and growth_hi >=
 *               growth_factor * growth_lo.
 */
#define OR_FX_NEAR_PASS 1u
#define OR_FX_F16_CEILING 2u
#define OR_FX_AXIS_GROWTH 4u
#define OR_ULP_BINS 34

static int64_t or_ord(uint32_t bits, int dtype)
{
    if (dtype == OR_I32) return (int64_t)(int32_t)bits;
    int width = elem_size(dtype) * 8;
    uint32_t sign = (bits >> (width - 1)) & 1u;
    int64_t mag = (int64_t)(bits & ((width == 32) ? 0x7fffffffu : 0x7fffu));
    return sign ? -mag : mag;
}

static double or_f16_spacing(double r)
{
    double a = fabs(r);
    if (a == 0.0) return ldexp(1.0, -24);
    int e;
    frexp(a, &e);          /* a = m * 2^e with 0.5 <= m < 1, so floor(log2 a) = e - 1 */
    int fl = e - 1;
    if (fl < -14) fl = -14;
    return ldexp(1.0, fl - 10);
}

int oracle_forensics(const void *cand, const void *ref, int dtype, int rank, const int64_t *shape,
                     double rtol, double atol, int axis, int64_t near_ulps, double near_fraction,
                     double growth_factor, int64_t *counts, int64_t *ulp_hist, double *growth,
                     double *growth_mean, int64_t *marginals, uint32_t *flags)
{
    if (rank < 0 || rank > 8) return -1;
    int64_t numel = 1;
    for (int a = 0; a < rank; ++a) numel *= shape[a];
    if (rank > 0 && (axis < 0 || axis >= rank)) return -1;
    int64_t len = rank > 0 ? shape[axis] : 1;
    int64_t stride = 1;                       /* elements between consecutive indices of the axis */
    for (int a = rank - 1; a > axis; --a) stride *= shape[a];
    int64_t moff[9];
    moff[0] = 0;
    for (int a = 0; a < rank; ++a) moff[a + 1] = moff[a] + shape[a];
    for (int64_t t = 0; t < moff[rank]; ++t) marginals[t] = 0;
    for (int k = 0; k < OR_ULP_BINS; ++k) ulp_hist[k] = 0;
    for (int64_t j = 0; j < len; ++j) growth[j] = 0.0;
    int64_t mismatch = 0, n_finite = 0, max_ulp = -1, arg_ulp = -1, nonfin = 0, within = 0;
    for (int64_t i = 0; i < numel; ++i) {
        uint32_t cb = load_bits(cand, dtype, i);
        uint32_t rb = load_bits(ref, dtype, i);
        double c = decode(cb, dtype);
        double r = decode(rb, dtype);
        int fin = isfinite(c) && isfinite(r);
        int64_t u = or_ord(cb, dtype) - or_ord(rb, dtype);
        if (u < 0) u = -u;
        if (fin) {
            n_finite++;
            int k = 0;
            if (u > 0) {
                k = 1;
                while (k < OR_ULP_BINS - 1 && u >= ((int64_t)1 << k)) k++;
            }
            ulp_hist[k]++;
            double d = fabs(c - r);
            int64_t j = rank > 0 ? (i / stride) % len : 0;
            if (d > growth[j]) growth[j] = d;
        }
        if (!oracle_pass(c, r, rtol, atol)) {
            mismatch++;
            if (!fin) {
                nonfin++;
            } else {
                if (u > max_ulp) { max_ulp = u; arg_ulp = i; }
                if (fabs(c - r) <= or_f16_spacing(r)) within++;
            }
            int64_t rest = i;
            for (int a = rank - 1; a >= 0; --a) {
                int64_t coord = rest % shape[a];
                rest /= shape[a];
                marginals[moff[a] + coord]++;
            }
        }
    }
    int64_t q = len / 4;
    if (q < 1) q = 1;
    double lo = 0.0, hi = 0.0;
    if (len > 0) {
        for (int64_t j = 0; j < q && j < len; ++j) lo += growth[j];
        for (int64_t j = len - q; j < len; ++j) if (j >= 0) hi += growth[j];
        lo /= (double)q;
        hi /= (double)q;
    }
    uint32_t f = 0;
    if (mismatch > 0 && nonfin == 0 && max_ulp <= near_ulps &&
        (double)mismatch <= near_fraction * (double)numel) f |= OR_FX_NEAR_PASS;
    if (mismatch > 0 && nonfin == 0 && within == mismatch) f |= OR_FX_F16_CEILING;
    if (len >= 4 && hi > 0.0 && hi >= growth_factor * lo) f |= OR_FX_AXIS_GROWTH;
    counts[0] = mismatch;
    counts[1] = n_finite;
    counts[2] = max_ulp;
    counts[3] = arg_ulp;
    counts[4] = nonfin;
    counts[5] = within;
    growth_mean[0] = lo;
    growth_mean[1] = hi;
    flags[0] = f;
    return 0;
}
