/*
 * nmv.h -- numerical validation with failure forensics on one NVIDIA GB300
 * (sm_103a).  C ABI of libnmv.so.
 *
 * The operation is the engine's validation step of the paper (Section 3.2,
 * Eq. 1: a repaired operator must satisfy Validate(K_fixed, R, T_ext, tau) =
 * true, i.e. its outputs must match the reference outputs within the
 * numerical tolerance tau over the extended test suite), together with the
 * numerical-deviation evidence the engine hands to the repair agent (Section
 * 3.2, "numerical-deviation metrics"; Section 4.2, localisation of diffuse
 * deviation; S2.2, NaN/Inf forensics), the per-case pass/fail and match-rate
 * evidence of full-coverage evaluation (Section 4.3, Table S4 "x% matched
 * cases"), and value-level flags for the degeneration / bypass hazards the
 * integrity layer guards against (Sections 1, 2.2, 4.3).
 *
 * The paper gives no formula for the check.  This library implements the
 * following reading (the same one the CPU oracle of the test suite writes
 * out), element by element after widening both stored values to fp64
 * exactly:
 *
 *   pass(i) = (c == r) OR (c, r finite AND
 *             fl(|fl(c - r)|) <= fl(atol + fl(rtol * |r|)))
 *
 * so NaN never passes and an infinity passes only against the same infinity.
 * Results are bit-identical to that fp64 arithmetic (the sum of squared
 * errors to a relative 1e-9), and bit-identical from run to run.
 *
 * Threading: every entry point may be called from any host thread; calls
 * are serialised on an internal lock (the device workspace is shared).
 */
#ifndef NMV_H
#define NMV_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- limits ------------------------------------------------------------ */
#define NMV_MAX_RANK 8
#define NMV_MAX_INPUTS 8
#define NMV_MAX_TILE (1LL << 24)      /* tile_rows, tile_cols <= this        */
#define NMV_MAX_HIST_BINS (1LL << 26) /* grid_rows * grid_cols <= this       */
#define NMV_MAX_FIRST_K (1LL << 24)   /* first_k <= this                     */
#define NMV_MAX_CASES (1LL << 20)     /* cases per nmv_validate_batch call   */

/* ---- status codes (return values and nmv_result.status) --------------- */
#define NMV_OK 0
#define NMV_EINVAL (-1)       /* an argument breaks a rule stated here      */
#define NMV_ENOMEM (-2)       /* host or device allocation failed           */
#define NMV_ECUDA (-3)        /* a CUDA call failed (no device, bad stream,
                                 a kernel error); see nmv_last_error()      */
#define NMV_EUNSUPPORTED (-4) /* the device is not sm_103                   */
#define NMV_ETIMEOUT (-5)     /* a kernel gave up waiting (its bulk copies into
                                 shared memory did not complete within its
                                 2 s wait limit); the call's results are void,
                                 nothing stays allocated and the CUDA context
                                 remains usable                             */

/* ---- element types ----------------------------------------------------- */
typedef enum nmv_dtype {
    NMV_F32 = 0,  /* IEEE binary32                                        */
    NMV_F16 = 1,  /* IEEE binary16                                        */
    NMV_BF16 = 2, /* bfloat16                                             */
    NMV_I32 = 3   /* two's-complement int32 (never NaN or infinite)       */
} nmv_dtype;

/* ---- degenerate-output flags (nmv_result.flags) ------------------------ */
/* Value-level stand-ins for the integrity hazards of Sections 1 and 4.3
 * (host-fallback bypass, "repair by degeneration").  The paper checks
 * integrity on source code; these numeric rules are this library's. */
#define NMV_FLAG_CAND_EQ_INPUT 1u  /* some input j with the candidate's dtype
                                      and numel has input_eq[j] >=
                                      max(1, ceil(numel / 100)), where
                                      input_eq[j] = #{i : bits(c_i) ==
                                      bits(x_j,i) and bits(r_i) != bits(x_j,i)} */
#define NMV_FLAG_CAND_ALL_ZERO 2u  /* numel >= 1, every c_i == 0 by value   */
#define NMV_FLAG_CAND_CONSTANT 4u  /* numel >= 2, every bits(c_i) == bits(c_0) */
#define NMV_FLAG_REF_ALL_ZERO 8u   /* the same rules applied to the reference */
#define NMV_FLAG_REF_CONSTANT 16u

/* One tensor: a device buffer of prod(shape) elements, contiguous row-major.
 * `data` must be readable by the current CUDA device (device memory, or
 * host memory the device can address).  It is borrowed, never written, and
 * must stay valid until the call returns.  `shape` is host memory with
 * `rank` entries, each >= 0 (it may be NULL when rank == 0; a rank-0 tensor
 * has one element). */
typedef struct nmv_tensor {
    const void *data;
    int32_t dtype;        /* nmv_dtype */
    int32_t rank;         /* 0 .. NMV_MAX_RANK */
    const int64_t *shape;
} nmv_tensor;

/* One validation case: the check Validate(K, R, T, tau) of Section 3.2 on
 * one output pair.  The forensics view the tensors as the 2-D matrix
 * [M, N] with M = prod(shape[:-1]) and N = shape[-1] (rank 1: M = 1; rank 0:
 * [1, 1]); element i sits at row i / N, column i % N. */
typedef struct nmv_case {
    nmv_tensor cand;            /* candidate output (the repaired kernel's) */
    nmv_tensor ref;             /* reference output; same dtype and shape   */
    const nmv_tensor *inputs;   /* operator inputs for the pass-through
                                   check; may be NULL when n_inputs == 0    */
    int32_t n_inputs;           /* 0 .. NMV_MAX_INPUTS                       */
    int32_t reserved;           /* must be 0                                */
    double rtol, atol;          /* tau: finite and >= 0                     */
    int64_t tile_rows;          /* localisation tile, 1 .. NMV_MAX_TILE     */
    int64_t tile_cols;
    int64_t first_k;            /* mismatch records to return, 0 .. NMV_MAX_FIRST_K */
} nmv_case;

/* Result of one case.  All arrays live in one host block owned by the
 * library until nmv_result_free(). */
typedef struct nmv_result {
    int32_t status;             /* NMV_OK                                   */
    int32_t rank;
    int64_t numel;
    int32_t pass;               /* 1 iff mismatch == 0 (torch.allclose)     */
    uint32_t flags;             /* NMV_FLAG_* bits                          */
    int64_t mismatch;           /* #{i : !pass(i)}; match rate = 1 - mismatch/numel */
    int64_t cand_nan, cand_posinf, cand_neginf;
    int64_t ref_nan, ref_posinf, ref_neginf;
    int64_t n_finite_pairs;     /* #{i : c_i and r_i both finite}           */
    /* Over the both-finite pairs, with d = fl64(c - r):                    */
    double max_abs;             /* max |d|; 0.0 when there is no such pair  */
    double max_rel;             /* max fl64(|d| / |r|) over r != 0          */
    double sse;                 /* sum of d^2 (relative error <= 1e-9)      */
    int64_t argmax_abs;         /* lowest index attaining max_abs, or -1    */
    int64_t argmax_rel;         /* lowest index attaining max_rel, or -1    */
    /* Localisation of the mismatches on the [M, N] view:                   */
    int64_t grid_rows, grid_cols;   /* ceil(M/tile_rows), ceil(N/tile_cols); 0 when numel == 0 */
    int64_t tile_rows, tile_cols;
    int64_t *tile_hist;         /* [grid_rows * grid_cols] row-major: mismatches per tile */
    int64_t *row_prof;          /* [tile_rows]: mismatches per (row % tile_rows) */
    int64_t *col_prof;          /* [tile_cols]: mismatches per (col % tile_cols) */
    /* The first min(first_k, mismatch) mismatches in ascending index order: */
    int64_t k_out;
    int64_t *fk_index;          /* [k_out] linear indices                  */
    int64_t *fk_coords;         /* [k_out * rank] row-major coordinates      */
    double *fk_cand;            /* [k_out] candidate values widened to fp64  */
    double *fk_ref;             /* [k_out] reference values widened to fp64  */
    /* Pass-through check:                                                  */
    int32_t n_inputs;
    int32_t passthrough_input;  /* lowest input that raised CAND_EQ_INPUT, or -1 */
    int64_t *input_eq;          /* [n_inputs]; -1 for an input of another dtype or numel */
    /* The numerical match rate of full-coverage evaluation (Section 4.3,
     * Table S4 "x% matched cases" per case): (numel - mismatch) / numel,
     * one fp64 division of the two exact integers; 1.0 when numel == 0.    */
    double match_fraction;
} nmv_result;

/* Validate one case on `cuda_stream` (a cudaStream_t; NULL = the legacy
 * default stream).  Synchronous: returns after the stream has produced the
 * result.  On NMV_OK, *out points to one nmv_result to be released with
 * nmv_result_free().  On any error, *out is NULL, nothing stays allocated
 * and nmv_last_error() describes the failure. */
int nmv_validate(const nmv_case *c, void *cuda_stream, nmv_result **out);

/* Validate n independent cases (a full-coverage sweep, Section 4.3) in one
 * call: one descriptor upload, one launch of the scan kernel per element
 * type and input class present, one launch of the finalize kernel, the
 * results written by the finalize kernel straight into mapped host memory.
 * Results are identical, bit for bit, to n nmv_validate calls.  Every case
 * is checked before any work starts; an invalid case fails the whole call
 * (the message names its index).  On NMV_OK, *out points to an array of n
 * results released by ONE nmv_result_free(*out) call. */
int nmv_validate_batch(const nmv_case *cases, int64_t n, void *cuda_stream,
                       nmv_result **out);

/* ---- validation without allocation --------------------------------------
 * The paper has no counterpart of this entry point; it is a service of this
 * library.  nmv_validate may allocate: it grows a cached device workspace
 * with cudaMalloc and a pinned staging block with cudaHostAlloc when a case
 * needs more than earlier calls did.  Some callers cannot allow that: a
 * process whose framework allocator has reserved (nearly) all device memory
 * up front, so that a library's own cudaMalloc fails or fragments it, and
 * latency-critical code that must not meet cudaMalloc/cudaFree's implicit
 * device-wide synchronisation.  nmv_validate_noalloc validates one case like
 * nmv_validate, with the same kernels and bit-identical results, but calls
 * no cudaMalloc, cudaFree, cudaHostAlloc or other allocating routine:
 *
 *  - its device scratch is one fixed array of NMV_NOALLOC_SCRATCH_BYTES in
 *    the library's module; every GPU that loads the library holds it until
 *    the process exits;
 *  - the caller owns the output: before the call it points out->tile_hist
 *    [grid_rows * grid_cols], row_prof [tile_rows], col_prof [tile_cols],
 *    fk_index, fk_cand, fk_ref [first_k], fk_coords [first_k * rank] and
 *    input_eq [n_inputs] at host arrays of at least those sizes (grid_rows =
 *    ceil(M / tile_rows), grid_cols = ceil(N / tile_cols), see nmv_case; an
 *    array whose size is 0 may be NULL).  The call fills them and every
 *    scalar field of *out, and leaves the pointers as they were.
 *
 * A case needs about: 4 bytes per batch of 2048 (16-bit types) or 1024
 * (32-bit types) elements, 8 bytes per histogram bin, 8 * (tile_rows +
 * tile_cols) + 24 * first_k bytes, and under 1 MiB of descriptors and
 * partials.  A case that
 * does not fit fails with NMV_EINVAL and a message giving the bytes it needs
 * (nmv_validate has no such limit).
 *
 * The first call on each device looks up the scratch array's device address
 * (cudaGetSymbolAddress, with that device current).  All calls share the
 * one array and find the previous call's contents in it; each call clears
 * what must start at zero.
 * Calls made through this library are serialised by its lock and return
 * only after their stream work has finished, also when they fail; calls
 * that did overlap on the
 * GPU would race on the array.  Profiling (nmv_profile_enable) does not
 * apply to this entry point.  On error *out's scalar fields are unspecified.
 */
#define NMV_NOALLOC_SCRATCH_BYTES (32LL << 20)

int nmv_validate_noalloc(const nmv_case *c, void *cuda_stream, nmv_result *out);

/* ---- diagnostic tensor statistics ---------------------------------------
 * The engine's diagnostic instrumentation (Section 4.2, "Diagnostic
 * instrumentation"; Figure 3, bottom-left; S5.1): when a repair attempt fails
 * on diffuse numerical deviation, the engine records multi-level tensor
 * statistics of the buffers at the kernel's pipeline boundaries and re-runs
 * forensics.  The paper gives no list of statistics; this library's reading:
 * two levels, the whole tensor and every tile of the same [M, N] view and
 * tile grid as the localisation maps, each with the statistics of nmv_stat.
 * One call instruments n buffers (one per boundary).
 *
 * Values are widened to fp64 exactly.  Counts, min, max, first_nan and
 * first_inf are exact.  int32 sums are exact integers rounded once to fp64,
 * so every int32 field is bit-identical to that definition.  Float sums
 * are accumulated in float-float pairs and fp64 and lie within 1e-12 of
 * the sum of |x| (sum) and relative 1e-12 (sumsq) of the exact sums; mean
 * and std are computed from them as stated in nmv_stat.  Results are
 * bit-identical from run to run. */
#define NMV_MAX_STAT_TILES (1LL << 22)  /* grid_rows * grid_cols per buffer  */

typedef struct nmv_stats_case {
    nmv_tensor x;               /* the buffer (borrowed, device-readable)    */
    int64_t tile_rows;          /* tile of the [M, N] view, 1 .. NMV_MAX_TILE */
    int64_t tile_cols;
} nmv_stats_case;

/* Statistics of one region (the tensor, or one tile), over its elements x:
 * every element is finite for int32.  With no finite element, min, max,
 * sum, sumsq, mean and std are 0.0. */
typedef struct nmv_stat {
    int64_t n_finite, n_nan, n_posinf, n_neginf;
    int64_t n_zero;             /* x == 0 by value (+0 and -0)              */
    double min, max;            /* over the finite x                        */
    double sum, sumsq;          /* sum of x and of x^2 over the finite x    */
    double mean;                /* sum / n_finite                            */
    double std;                 /* sqrt(max(0, sumsq / n_finite - mean^2)),
                                   each operation one fp64 rounding          */
} nmv_stat;

typedef struct nmv_stats_result {
    int32_t status;             /* NMV_OK                                   */
    int32_t rank;
    int64_t numel;
    nmv_stat all;               /* the whole tensor                         */
    int64_t first_nan;          /* lowest index of a NaN, or -1             */
    int64_t first_inf;          /* lowest index of +-Inf, or -1             */
    int64_t grid_rows, grid_cols;   /* ceil(M/tile_rows), ceil(N/tile_cols); 0 when numel == 0 */
    int64_t tile_rows, tile_cols;
    nmv_stat *tiles;            /* [grid_rows * grid_cols] row-major        */
} nmv_stats_result;

/* Statistics of n buffers on `cuda_stream`, synchronous like nmv_validate.
 * Every case is checked first (the message names a bad case's index).  On
 * NMV_OK, *out points to an array of n results released by ONE
 * nmv_result_free(*out) call; on error *out is NULL and nothing stays
 * allocated. */
int nmv_stats(const nmv_stats_case *cases, int64_t n, void *cuda_stream, nmv_stats_result **out);

/* ---- deep forensics: per-axis maps, ulp distances, error growth -------
 * The evidence the engine's adaptive-scheduling rules read ("near-pass and
 * fp16-ceiling detection", Section 4.4) and the localisation of a divergence
 * that compounds along a reduction axis (Section 3.2, the cumsum of Table 1),
 * plus mismatch counts at every index of every axis.  An on-demand second
 * pass over a pair (the engine instruments only after a failed attempt,
 * Section 4.2).  The paper gives no formula; this library's reading, over the
 * pairs and the predicate of nmv_validate:
 *
 *   ord(x)   the order-preserving integer of a float's bits (+m for a
 *            positive sign, -m for a negative one, m the magnitude bits: +0
 *            and -0 are both 0, consecutive floats differ by 1); int32: x
 *   u        = |ord(c) - ord(r)|, the distance in representable values
 *   h(r)     one fp16 spacing at |r|: 2^(max(floor(log2 |r|), -14) - 10),
 *            2^-24 for r = 0 (the exponent range unbounded above)
 *
 * Every field is exact; growth_lo / growth_hi are left-to-right fp64 sums
 * divided by q, the same operations as the definition. */
#define NMV_ULP_BINS 34
#define NMV_FX_NEAR_PASS 1u    /* mismatch > 0, no non-finite mismatch,
                                  max_ulp_mismatch <= near_ulps and mismatch
                                  <= near_fraction * numel (fp64 product)   */
#define NMV_FX_F16_CEILING 2u  /* mismatch > 0, no non-finite mismatch and
                                  every mismatch within one fp16 spacing h(r)
                                  (the candidate sits at fp16 precision)    */
#define NMV_FX_AXIS_GROWTH 4u  /* axis_len >= 4, growth_hi > 0 and growth_hi
                                  >= growth_factor * growth_lo (the error
                                  compounds along the axis)                  */

typedef struct nmv_forensics_case {
    nmv_tensor cand, ref;       /* as nmv_case: same dtype and shape        */
    double rtol, atol;          /* the predicate's tolerance                */
    int32_t axis;               /* growth axis, -rank .. rank-1 (negative
                                   counts from the last); rank 0: ignored   */
    int32_t reserved;           /* must be 0                                */
    int64_t near_ulps;          /* NMV_FX_NEAR_PASS, >= 0                   */
    double near_fraction;       /* NMV_FX_NEAR_PASS, finite, >= 0           */
    double growth_factor;       /* NMV_FX_AXIS_GROWTH, finite, >= 0         */
} nmv_forensics_case;

typedef struct nmv_forensics_result {
    int32_t status;             /* NMV_OK                                   */
    int32_t rank;
    int64_t numel;
    int64_t mismatch;           /* as nmv_result.mismatch                   */
    int64_t n_finite_pairs;
    int64_t ulp_hist[NMV_ULP_BINS];  /* both-finite pairs by u: bin 0: u = 0,
                                        bin k: 2^(k-1) <= u < 2^k (bin 33 also
                                        every larger u)                     */
    int64_t max_ulp_mismatch;   /* largest u over mismatches with both values
                                   finite, -1 if none                        */
    int64_t argmax_ulp_mismatch;    /* lowest index attaining it, -1        */
    int64_t mism_nonfinite;     /* mismatches with a NaN or infinite value  */
    int64_t mism_within_f16;    /* finite mismatches with fl64|c - r| <= h(r) */
    uint32_t flags;             /* NMV_FX_* bits                            */
    int32_t axis;               /* the growth axis, 0 .. rank-1             */
    int64_t axis_len;           /* its extent (1 for rank 0)                */
    double growth_lo;           /* mean of growth over its first q entries,
                                   q = max(1, floor(axis_len / 4))          */
    double growth_hi;           /* ... and over its last q entries          */
    double *growth;             /* [axis_len]: max fl64|c - r| over the
                                   both-finite pairs at each index of the
                                   axis (0.0 if none)                        */
    int64_t marg_off[NMV_MAX_RANK + 1];  /* axis a's marginal is
                                   marginals[marg_off[a] .. marg_off[a+1])  */
    int64_t *marginals;         /* mismatches at each index of each axis    */
} nmv_forensics_result;

/* Deep forensics of n pairs on `cuda_stream`, synchronous.  sum(shape) of a
 * case may be at most NMV_MAX_HIST_BINS.  Every case is checked first (the
 * message names a bad case's index).  On NMV_OK, *out points to an array of
 * n results released by ONE nmv_result_free(*out) call; on error *out is
 * NULL and nothing stays allocated. */
int nmv_forensics(const nmv_forensics_case *cases, int64_t n, void *cuda_stream,
                  nmv_forensics_result **out);

/* ---- full-coverage escalation --------------------------------------------
 * The engine's validation escalation (Section 4.3, "Full-coverage
 * evaluation"; Figure 3, bottom-right; S6.1): the lightweight case set is
 * validated first (one nmv_validate_batch call), and only when every one of
 * its cases passes does the extended set run (a second call).  A repair is
 * accepted when every case of both sets passes and no case raises an
 * integrity hazard (NMV_FLAG_CAND_EQ_INPUT, or CAND_CONSTANT / CAND_ALL_ZERO
 * without the matching REF_* flag).  The per-case evidence (pass/fail and
 * numerical match rate, the "x% matched cases" of Table S4) is written as a
 * canonical text record, one header line and one line per validated case:
 *
 *   nmv-sweep v1 light=<n> ext=<n> escalated=<0|1> accepted=<0|1>
 *       pass_light=<n> pass_ext=<n>
 *   <L|E> <index> dtype=<d> numel=<n> pass=<0|1> mismatch=<n> match=<%.17g>
 *       max_abs=<%.17g> max_rel=<%.17g> nonfinite=<n> flags=<u>
 *
 * (each record is one line; nonfinite counts NaN/Inf on both sides) and
 * sealed with its SHA-256 digest (FIPS 180-4), so the evidence behind an
 * acceptance cannot change unnoticed. */
typedef struct nmv_sweep_report {
    int32_t status;             /* NMV_OK                                   */
    int32_t escalated;          /* 1: the extended set ran                  */
    int32_t accepted;           /* 1: every case of both sets passed, no hazard */
    uint32_t flags_any;         /* OR of the NMV_FLAG_* bits of the cases run */
    int64_t n_light, n_ext;     /* cases in each set                        */
    int64_t n_run;              /* cases validated: n_light (+ n_ext when escalated) */
    int64_t n_pass_light, n_pass_ext;
    double match_rate_light;    /* n_pass_light / n_light                    */
    double match_rate_ext;      /* n_pass_ext / n_ext when escalated, else 0 */
    uint8_t digest[32];         /* SHA-256 of evidence[0 .. evidence_len)   */
    char *evidence;             /* the canonical record (NUL-terminated)    */
    int64_t evidence_len;
    nmv_result *results;        /* [n_run]: the light cases, then the extended */
    nmv_result *blocks[2];      /* the result blocks the records point into
                                   (owned by the report)                     */
} nmv_sweep_report;

/* Run the escalation on `cuda_stream` (synchronous): light[0 .. n_light),
 * n_light >= 1, then ext[0 .. n_ext) if every light case passed.  Cases are
 * checked as in nmv_validate_batch (the message names the set and the
 * case).  On NMV_OK, *out is released with nmv_sweep_free(). */
int nmv_sweep(const nmv_case *light, int64_t n_light, const nmv_case *ext, int64_t n_ext,
              void *cuda_stream, nmv_sweep_report **out);
void nmv_sweep_free(nmv_sweep_report *r);   /* NULL is accepted */

/* SHA-256 (FIPS 180-4) of len bytes, the digest of the sweep's evidence. */
void nmv_sha256(const void *data, int64_t len, uint8_t out[32]);

/* Release what one nmv_validate / nmv_validate_batch / nmv_stats /
 * nmv_forensics call returned.  NULL is accepted.  (The block is mapped pinned host memory, which the library
 * keeps for reuse by later calls.) */
void nmv_result_free(void *r);

/* Static text for a status code. */
const char *nmv_status_string(int status);

/* Text of the last failure on the calling thread ("" if none). */
const char *nmv_last_error(void);

/* Launch profile, for measuring the kernels against their roofline (the
 * paper's forensics "compiles and profiles" a kernel, Section 4; this is the
 * library's own profile).  nmv_profile_enable(mode) applies to every
 * following call on any thread; mode is a set of NMV_PROFILE_* bits (0 =
 * off).  NMV_PROFILE_TIMING records CUDA events on the call's stream around
 * its scan-kernel launches and around its finalize launch.
 * NMV_PROFILE_COUNTERS makes the scan kernel count its exact-path work
 * (atomic counters and clock reads, which slow it down; the counter fields
 * are 0 without it).  nmv_profile_last() fills *out for the last successful
 * profiled call; it returns NMV_EINVAL if there is none since the last
 * nmv_profile_enable() or out is NULL. */
#define NMV_PROFILE_TIMING 1
#define NMV_PROFILE_COUNTERS 2

typedef struct nmv_profile {
    double scan_ms;            /* scan-kernel launches, stream time          */
    double finalize_ms;        /* finalize launch, stream time               */
    int64_t kernel_launches;   /* kernels the call launched                  */
    int64_t h2d_bytes;         /* bytes the library copied host to device    */
    int64_t d2h_bytes;         /* bytes the library copied device to host    */
    int64_t slow_steps;        /* warp steps that took the exact path        */
    int64_t light_steps;       /* warp steps that only updated the maxima    */
    int64_t exact_abs;         /* fp64 evaluations of a max |d| candidate    */
    int64_t exact_rel;         /* fp64 evaluations of a max |d|/|r| candidate */
    int64_t exact_pred;        /* fp64 evaluations of the predicate          */
    int64_t slow_cycles;       /* SM clock cycles warps spent in exact steps  */
    int64_t light_cycles;      /* SM clock cycles warps spent in light steps  */
    int64_t dense_steps;       /* warp steps that only counted and localised
                                  mismatches (no maximum candidates)         */
    int64_t dense_cycles;      /* SM clock cycles warps spent in those steps */
    int64_t workspace_allocs;  /* device workspace allocations on this device
                                  since the library was loaded (the workspace
                                  grows by doubling, so a rising sequence of
                                  case sizes allocates O(log n) times)       */
    int64_t workspace_bytes;   /* the device workspace's current size        */
} nmv_profile;

void nmv_profile_enable(int mode);
int nmv_profile_last(nmv_profile *out);

#ifdef __cplusplus
}
#endif

#endif /* NMV_H */
