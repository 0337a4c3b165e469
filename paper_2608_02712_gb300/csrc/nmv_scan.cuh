// nmv_scan.cuh -- the streaming validation pass (one kernel per element type
// and input class; instantiated by nmv_scan_<dtype>.cu).
//
// One pass over candidate, reference (and the inputs of the pass-through
// check) computes, per piece of a case: the pass predicate of the tolerance
// check (Section 3.2, Eq. 1, read as allclose in fp64), NaN/Inf counts, the
// maximum absolute and relative errors with their lowest indices, the sum of
// squared errors, the tile-histogram and row/column profiles of the
// mismatches (localisation evidence, Sections 4.2 and S2.2), the mismatch
// count of every batch (for the first-K records) and the degenerate-output
// accumulators (Sections 1 and 4.3).
//
// Exactness without fp64 throughput.  GB300 has very little fp64
// throughput, so the sweep works in fp32 wherever a margin or an exact
// transformation proves the fp64 result.  A warp takes an out-of-line path
// for a step only when some lane holds an element the fast proof does not
// cover.  An element (float types) is on the fast path when, with
// s = fl32(c - r):
//     |s| <= min(fma_rz(lo_r, |r|, lo_a), mul_rz(min(tR, 1/4), |r|), tA)
//  * predicate: lo_* are the fp32 round-down of (1 - 2^-20) {rtol, atol}; the
//    margin absorbs every fp32 rounding, so the element provably passes the
//    fp64 test fl(|fl(c-r)|) <= fl(atol + fl(rtol |r|)).
//  * max |d|/|r|: no fraction |d|/|r| of such an element lies between tR
//    and the best relative error held, so the element provably is no new
//    maximum (strictly below a maximum published by any warp of the case,
//    or not above one held earlier in this warp's ascending sweep, whose
//    index is lower).
//  * max |d|: the same with tA, which is also capped at 2^56 (SSE range).
//  * |s| <= |r|/4 gives |c - r| < min(|c|, |r|), so c - r is exact in fp32
//    (Sterbenz's lemma): d = s exactly and d^2 = p + pe with p = fl(s*s),
//    pe = fma(s, s, -p).
// Out of the fast path, a "light" step handles steps that only hold
// candidates for a new maximum, and the exact step everything else (NaN/Inf,
// mismatches, inexact differences, the undecided predicate band).  Maxima
// are kept exactly in fp32 terms where possible: |d| when c - r is exact, and
// |d|/|r| as the fraction of two fp32 values, compared by exact
// cross-products (Dekker's TwoProduct with fma).  Two quotients of 24-bit
// values that differ, differ by more than 2^-48 relative, so their order is
// the order of their fp64 roundings; only inexact differences fall back to
// fp64 arithmetic.
// The SSE is accumulated per lane as two float-float pairs (even and odd
// elements of each vector) with Knuth's TwoSum; the exact step feeds the same
// pairs with the same arithmetic (plus 2 s e for an inexact c - r, e from
// TwoSum), so the result does not depend on which path an element takes.
// A warp's batches within a piece follow a fixed schedule and the lane,
// warp and piece sums are combined in a fixed order, so the SSE does not
// depend on which block took which piece either: it is bit-identical run to
// run.  Terms with |s| > 2^56 are
// squared in fp64.  When max |d| < 2^-38 the fp32 squares may lose tiny
// terms; the host then recomputes that case's SSE in fp64 (sse64 kernels).
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "nmv_internal.h"

namespace nmv {

constexpr float kHuge = 0x1p56f;
constexpr float kMarginLo = 1.0f - 0x1p-20f;

// ------------------------------------------------------------------ utils
__device__ __forceinline__ uint64_t div_q(uint64_t n, uint64_t d, uint64_t m) {
  uint64_t q = __umul64hi(n, m);
  if (n - q * d >= d) q += 1;
  return q;
}

// n / d for n < 2^32 with m = floor((2^32 - 1) / d): the product's high
// word is the quotient or one below it.
__device__ __forceinline__ uint32_t div_q32(uint32_t n, uint32_t d, uint32_t m) {
  uint32_t q = __umulhi(n, m);
  if (n - q * d >= d) q += 1;
  return q;
}

__device__ __forceinline__ uint4 ld_v4(const void *p) {
  uint4 v;
  asm("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
      : "l"(p));
  return v;
}

template <int EB>
__device__ __forceinline__ uint32_t ld_one(const void *base, int64_t i) {
  if constexpr (EB == 2) {
    unsigned short h;
    asm("ld.global.nc.u16 %0, [%1];" : "=h"(h) : "l"((const char *)base + 2 * i));
    return h;
  } else {
    uint32_t w;
    asm("ld.global.nc.u32 %0, [%1];" : "=r"(w) : "l"((const char *)base + 4 * i));
    return w;
  }
}

__device__ __forceinline__ uint64_t ld_relaxed64(const uint32_t *p) {
  uint64_t v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p));
  return v;
}

__device__ __forceinline__ float min3f(float a, float b, float c) {
  float r;
  asm("min.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Atomic updates whose result is not used, with the state space explicit:
// the localisation maps and class counters sit in shared memory behind
// pointers kept in PieceSh, which a plain atomicAdd would reach through a
// generic (slow) atomic.  No memory clobber: these words are read only
// after a block barrier, and the reductions may be reordered among
// themselves.
__device__ __forceinline__ void sh_add_at(uint32_t addr, int v) {
  asm volatile("red.shared.add.u32 [%0], %1;" ::"r"(addr), "r"(v));
}
__device__ __forceinline__ void sh_add(int32_t *p, int v) { sh_add_at((uint32_t)__cvta_generic_to_shared(p), v); }
__device__ __forceinline__ void gl_add(unsigned long long *p, unsigned long long v) {
  asm volatile("red.global.add.u64 [%0], %1;" ::"l"(p), "l"(v));
}
__device__ __forceinline__ void sh_max(uint32_t *p, uint32_t v) {
  asm volatile("red.shared.max.u32 [%0], %1;" ::"r"((uint32_t)__cvta_generic_to_shared(p)), "r"(v));
}
__device__ __forceinline__ uint32_t sh_max_old(uint32_t *p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.shared.max.u32 %0, [%1], %2;"
               : "=r"(old)
               : "r"((uint32_t)__cvta_generic_to_shared(p)), "r"(v)
               : "memory");
  return old;
}

// ---------------------------------------------------------- dtype traits
template <int DT>
struct Tr {
  static constexpr int V = (DT == NMV_F16 || DT == NMV_BF16) ? 8 : 4;
  static constexpr int EB = (DT == NMV_F16 || DT == NMV_BF16) ? 2 : 4;
  static constexpr bool kInt = DT == NMV_I32;
  static constexpr uint32_t kElemMask = EB == 2 ? 0xffffu : 0xffffffffu;
};

template <int DT>
__device__ __forceinline__ uint32_t vbits(const uint4 &v, int k) {
  const uint32_t w = (&v.x)[Tr<DT>::EB == 2 ? (k >> 1) : k];
  if constexpr (Tr<DT>::EB == 2) return (k & 1) ? (w >> 16) : (w & 0xffffu);
  return w;
}

// Stored bits -> fp32 (exact for the float formats, rounded for int32).
template <int DT>
__device__ __forceinline__ float to_f32(uint32_t b) {
  if constexpr (DT == NMV_F32) return __uint_as_float(b);
  if constexpr (DT == NMV_BF16) return __uint_as_float(b << 16);
  if constexpr (DT == NMV_F16) return __half2float(__ushort_as_half((unsigned short)b));
  return __int2float_rn((int32_t)b);
}

// Element k of a 16-byte vector -> fp32, straight from the packed word.
template <int DT>
__device__ __forceinline__ float vdec(const uint4 &v, int k) {
  if constexpr (DT == NMV_BF16) {
    const uint32_t w = (&v.x)[k >> 1];
    return __uint_as_float((k & 1) ? (w & 0xffff0000u) : (w << 16));
  }
  return to_f32<DT>(vbits<DT>(v, k));
}

template <int DT>
__device__ __forceinline__ double to_f64(uint32_t b) {
  if constexpr (DT == NMV_I32) return (double)(int32_t)b;
  return (double)to_f32<DT>(b);
}

// The predicate in fp64, written out: (c == r) or (both finite and
// fl(|fl(c - r)|) <= fl(atol + fl(rtol * |r|))).  No contraction.
__device__ __forceinline__ bool pass64_inl(double c, double r, double rtol, double atol) {
  if (c == r) return true;
  if (!(isfinite(c) && isfinite(r))) return false;
  const double err = fabs(__dsub_rn(c, r));
  const double allowed = __dadd_rn(atol, __dmul_rn(rtol, fabs(r)));
  return err <= allowed;
}

// The same, out of line (the scan's exact path keeps its code small).
static __device__ __noinline__ bool pass64(double c, double r, double rtol, double atol) {
  return pass64_inl(c, r, rtol, atol);
}

// --------------------------------------------------------------- the SSE
// Two float-float accumulators per lane (slot x: even elements of each
// vector, slot y: odd elements) plus an fp64 total.
struct SseAcc {
  float2 hi, lo;
  double acc;
};

// The canonical term: d = s + e exactly; add d^2 = p + pe + 2se (e*e is
// below 2^-48 relative and dropped) to (hi, lo) with Knuth's TwoSum.
__device__ __forceinline__ void ff_term(float &hi, float &lo, float s, float e) {
  const float p = __fmul_rn(s, s);
  const float pe = __fmaf_rn(s, s, -p);
  const float q = __fmaf_rn(__fadd_rn(s, s), e, pe);
  const float t = __fadd_rn(hi, p);
  const float bp = __fsub_rn(t, hi);
  const float err = __fadd_rn(__fsub_rn(hi, __fsub_rn(t, bp)), __fsub_rn(p, bp));
  hi = t;
  lo = __fadd_rn(lo, __fadd_rn(err, q));
}

// The same arithmetic on an even/odd pair with e = 0, in packed f32x2 form.
// For 16-bit inputs on the fast path s has at most 12 significant bits, so
// s*s is exact and pe = q = +0 (kPe = false); otherwise q = pe.
template <bool kPe>
__device__ __forceinline__ void ff_pair(SseAcc &a, float2 s) {
  const float2 m1 = make_float2(-1.f, -1.f);
  const float2 p = __fmul2_rn(s, s);
  float2 q = make_float2(0.f, 0.f);
  if constexpr (kPe) q = __ffma2_rn(s, s, __fmul2_rn(p, m1));
  const float2 t = __fadd2_rn(a.hi, p);
  const float2 bp = __ffma2_rn(a.hi, m1, t);
  const float2 x1 = __ffma2_rn(bp, m1, t);
  const float2 x2 = __ffma2_rn(x1, m1, a.hi);
  const float2 x3 = __ffma2_rn(bp, m1, p);
  const float2 err = __fadd2_rn(x2, x3);
  // (kPe false: q is +0, and lo + err equals lo + (err + 0): lo starts at +0
  // and a rounded sum is never -0, so only err = -0 could tell them apart,
  // and lo + -0 = lo for every lo that is not -0)
  if constexpr (kPe) a.lo = __fadd2_rn(a.lo, __fadd2_rn(err, q));
  else a.lo = __fadd2_rn(a.lo, err);
  a.hi = t;
}

// ------------------------------------------------------------ reductions
// Best (value, index): the larger value wins, equal values go to the lower
// index.  Values are >= 0 or -1 (none), so their bit patterns order as
// int64 the way the values do: no fp64 comparisons are needed.
struct Best {
  double v;
  int64_t i;
};

__device__ __forceinline__ bool beats(double v, int64_t i, double bv, int64_t bi) {
  const long long a = __double_as_longlong(v), b = __double_as_longlong(bv);
  return a > b || (a == b && i < bi);
}

__device__ __forceinline__ void best_offer(Best &b, double v, int64_t i) {
  if (beats(v, i, b.v, b.i)) {
    b.v = v;
    b.i = i;
  }
}

__device__ __forceinline__ Best best_warp(Best b) {
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const double v = __shfl_xor_sync(0xffffffffu, b.v, o);
    const int64_t i = __shfl_xor_sync(0xffffffffu, b.i, o);
    best_offer(b, v, i);
  }
  return b;
}

template <typename T, typename Op>
__device__ __forceinline__ T warp_reduce(T v, Op op) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// (h, l) += (h2, l2) for float-float pairs: TwoSum of the high parts (its
// error is exact, so the result does not depend on the operand order).
__device__ __forceinline__ void ff_add(float &h, float &l, float h2, float l2) {
  const float t = __fadd_rn(h, h2);
  const float bp = __fsub_rn(t, h);
  const float err = __fadd_rn(__fsub_rn(h, __fsub_rn(t, bp)), __fsub_rn(h2, bp));
  h = t;
  l = __fadd_rn(__fadd_rn(l, l2), err);
}

// ----------------------------------------------------------------- state
// Piece-constant data, in shared memory.
struct PieceSh {
  CaseDesc cd;
  int64_t piece;   // the piece's index in the launch
  int64_t pbegin;  // the piece's first element
  int64_t tr0, tc0;
  int32_t wr, wc, prof_smem;
  int32_t rel_ru;  // 16-bit element type: exact fractions up to 1/4 round up (rel_thr)
  int32_t *sh_cls, *sh_row, *sh_col, *sh_hist;
  unsigned long long *g_hist, *g_row, *g_col;
  uint32_t *g_thr;
  uint32_t *cta_thr;  // [2] the block's view of the case-wide maxima (float bits), in shared memory
  int32_t *sh_eq;  // [kThreads][NMV_MAX_INPUTS] pass-through counts of the exact paths (inputs only)
  uint32_t lcol_sa;  // shared address of the lanes' private column counters ([kThreads][V], aligned mode)
  unsigned long long *stats;  // [exact steps, exact abs, exact rel, exact predicate, light steps,
                              //  SM cycles in exact steps, SM cycles in light steps,
                              //  dense steps, SM cycles in dense steps]
};

// The maxima one lane holds, in shared memory.
//  |d|:      a_f (an fp32 that is exactly the fp64 value) when a_x, else a_v.
//  |d|/|r|:  the exact fraction r_n / r_d of two fp32 values when r_x, else
//            the fp64 quotient r_v.
// An index of INT64_MAX means "none held".
struct LaneSh {
  double a_v, r_v;
  int64_t a_i, r_i;
  float a_f, r_n, r_d;
  float r_lo;  // an fp32 strictly below the held |d|/|r| by the 2^-20 margin (-1: none)
  int32_t a_x, r_x;
  uint32_t cacc, racc;
};

// Warp-uniform state of a batch sweep, in shared memory.
struct WarpSh {
  float tA, tR;       // thresholds in force
  float wA, wR;       // the warp's own part of them (-1: no maximum held yet)
  float cA, cR;       // the part carried from the warp's earlier pieces of the case
  float ga, gr;       // the case-wide part at the last merge (-1: none)
  uint32_t pubA, pubR;
  int64_t mism;       // mismatches so far in this batch
  uint32_t sbits;     // steps of this batch that hold mismatches (bit u: warp step u)
  int64_t mism_tot;   // mismatches in the warp's batches of this piece
  uint32_t stage_b[4];  // batch held by each ring stage (kNoBatch: none)
  unsigned long long st[9];  // the warp's profile counters (layout of PieceSh::stats)
};

__device__ __forceinline__ float pub_thr(uint32_t bits) {
  const float f = __uint_as_float(bits);
  return f > 0.f ? __fmul_rz(f, kMarginLo) : -1.f;
}

__device__ __forceinline__ void merge_thr(float wA, float wR, float ga, float gr, float &tA, float &tR) {
  tA = fminf(fmaxf(wA, ga), kHuge);
  tR = fmaxf(wR, gr);
}

// fl32(|s| / |r|) for |r| != 0, within 2^-22 of the quotient: a fast
// reciprocal in the normal range, an IEEE division otherwise.
__device__ __forceinline__ float rel32(float as, float ar) {
  if (ar > 0x1p-125f && ar < 0x1p125f) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(ar));
    return __fmul_rn(as, r);
  }
  return __fdiv_rn(as, ar);
}

// A strict fp32 lower bound of n / d (n >= 0, d > 0): rel32 is within 2^-22.
// A quotient beyond the fp32 range (d subnormal, say) gives the largest
// finite float, still a lower bound; an infinite bound would make every
// warp skip the larger quotients it cannot tell apart.
__device__ __forceinline__ float quot_lb(float n, float d) {
  return __fmul_rz(fminf(rel32(n, d), 0x1.fffffep127f), 1.0f - 0x1p-21f);
}

// fp32 lower bounds of a lane's maxima (-1 when none held).
__device__ __forceinline__ float abs_lb(const LaneSh *L) {
  if (L->a_i == INT64_MAX) return -1.f;
  return L->a_x ? L->a_f : __double2float_rd(L->a_v);
}

// The warp's own threshold from a lane's maximum |d|/|r| (-1 when none
// held): a value t such that an element whose exact fraction is at most t
// is at most the maximum.  An exact fraction n/d is rounded down (the
// maximum itself when fp32 holds it exactly), an fp64 quotient, itself
// rounded, gets the 2^-20 margin.  For fp16 and bf16 an exact fraction
// q = n/d <= 1/4 is rounded up instead: with |c - r| <= |r|/4, c lies within
// one binade of r, so q = M / (2R) for integers R < 2^11 (r's significand)
// and M <= R/2; two such fractions q < q' differ by q' - q >= 1 / (2 R R'),
// i.e. by more than 2^-21 q relative, while (q, ru(q)] is narrower than one
// fp32 ulp of q (2^-23 q).  So no element the fast path can pass (|s| <=
// |r|/4, c - r exact) has a fraction in (q, ru(q)], and ties with the
// maximum stay on the fast path.
__device__ __forceinline__ float rel_thr(const PieceSh *P, const LaneSh *L) {
  if (L->r_i == INT64_MAX) return -1.f;
  if (!L->r_x) return __fmul_rz(__double2float_rd(L->r_v), kMarginLo);
  return P->rel_ru && L->r_n <= 0.25f * L->r_d ? __fdiv_ru(L->r_n, L->r_d) : __fdiv_rd(L->r_n, L->r_d);
}

// The lane's maximum |d| as fp64 (for the reduction at the end of a piece).
__device__ __forceinline__ Best abs_best64(const LaneSh *L) {
  if (L->a_i == INT64_MAX) return {-1.0, INT64_MAX};
  return {L->a_x ? (double)L->a_f : L->a_v, L->a_i};
}

// Offer |d| of element idx: as = |fl32(c - r)|, exact when e == 0; a64 is
// fl64(|c - r|) and is read only when !exact.
__device__ __forceinline__ bool offer_abs(LaneSh *L, float as, bool exact, double a64, int64_t idx) {
  if (L->a_i == INT64_MAX) {
    L->a_x = exact;
    L->a_f = as;
    L->a_v = exact ? 0.0 : a64;
    L->a_i = idx;
    return true;
  }
  if (exact && L->a_x) {
    if (as > L->a_f || (as == L->a_f && idx < L->a_i)) {
      L->a_f = as;
      L->a_i = idx;
      return true;
    }
    return false;
  }
  const double v = exact ? (double)as : a64;
  const double bv = L->a_x ? (double)L->a_f : L->a_v;
  if (beats(v, idx, bv, L->a_i)) {
    L->a_x = exact;
    L->a_f = as;
    L->a_v = v;
    L->a_i = idx;
    return true;
  }
  return false;
}

// Compare n1/d1 with n2/d2 (n >= 0, d > 0, fp32 values) exactly through the
// cross products n1*d2 and n2*d1, each as an exact float-float pair; returns
// 1, 0, -1, or 2 when a product leaves the range where that is exact.
__device__ __forceinline__ int frac_cmp(float n1, float d1, float n2, float d2) {
  const float p1 = __fmul_rn(n1, d2), p2 = __fmul_rn(n2, d1);
  const bool ok1 = p1 == 0.f ? n1 == 0.f : (p1 >= 0x1p-100f && p1 < 0x1p126f);
  const bool ok2 = p2 == 0.f ? n2 == 0.f : (p2 >= 0x1p-100f && p2 < 0x1p126f);
  if (!(ok1 && ok2)) return 2;
  if (p1 != p2) return p1 > p2 ? 1 : -1;
  const float e1 = __fmaf_rn(n1, d2, -p1), e2 = __fmaf_rn(n2, d1, -p2);
  if (e1 != e2) return e1 > e2 ? 1 : -1;
  return 0;
}

// The warp's best |d|/|r| (largest, lowest index on ties) from the lanes'
// maxima, comparing exact fractions through frac_cmp and anything else
// through fp64 quotients, so that an fp64 division is needed only for
// inexact maxima and for the result; every lane returns the result.
__device__ __forceinline__ Best rel_best_warp(const LaneSh *L) {
  int64_t i = L->r_i;
  int x = L->r_x;
  float n = L->r_n, d = L->r_d;
  double v = L->r_v;
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const int64_t i2 = __shfl_xor_sync(0xffffffffu, i, o);
    const int x2 = __shfl_xor_sync(0xffffffffu, x, o);
    const float n2 = __shfl_xor_sync(0xffffffffu, n, o), d2 = __shfl_xor_sync(0xffffffffu, d, o);
    const double v2 = __shfl_xor_sync(0xffffffffu, v, o);
    bool take;
    if (i2 == INT64_MAX) {
      take = false;
    } else if (i == INT64_MAX) {
      take = true;
    } else {
      const int c = (x && x2) ? frac_cmp(n2, d2, n, d) : 2;
      if (c != 2) {
        take = c > 0 || (c == 0 && i2 < i);
      } else {
        const double q = x ? __ddiv_rn((double)n, (double)d) : v;
        const double q2 = x2 ? __ddiv_rn((double)n2, (double)d2) : v2;
        take = beats(q2, i2, q, i);
      }
    }
    if (take) {
      i = i2;
      x = x2;
      n = n2;
      d = d2;
      v = v2;
    }
  }
  if (i == INT64_MAX) return {-1.0, INT64_MAX};
  return {x ? __ddiv_rn((double)n, (double)d) : v, i};
}

// Offer |d|/|r| of element idx (q32: its fp32 quotient for screening;
// exact: |d| = as is exact and |r| = ar is exact; otherwise a64 = fl64(|d|)
// and r64 = |r| in fp64).
__device__ __forceinline__ bool offer_rel(LaneSh *L, float as, float ar, bool exact, double a64, double r64,
                                          float q32, int64_t idx, unsigned &n_fp64) {
  if (q32 < L->r_lo) return false;
  bool win;
  const bool none = L->r_i == INT64_MAX;
  if (exact && (none || L->r_x)) {
    int c = none ? 1 : frac_cmp(as, ar, L->r_n, L->r_d);
    if (c != 2) {
      win = c > 0 || (c == 0 && idx < L->r_i);
      if (win) {
        L->r_x = 1;
        L->r_n = as;
        L->r_d = ar;
        L->r_i = idx;
        L->r_lo = __fmul_rz(quot_lb(as, ar), kMarginLo);
      }
      return win;
    }
  }
  ++n_fp64;
  const double q = __ddiv_rn(exact ? (double)as : a64, exact ? (double)ar : r64);
  const double bq = none ? -1.0 : (L->r_x ? __ddiv_rn((double)L->r_n, (double)L->r_d) : L->r_v);
  win = beats(q, idx, bq, none ? INT64_MAX : L->r_i);
  if (win) {
    L->r_x = 0;
    L->r_v = q;
    L->r_i = idx;
    L->r_lo = __fmul_rz(__double2float_rd(q), kMarginLo);
  }
  return win;
}

// Order of two candidates for the maximum of |d|/|r| (true when the first,
// at a higher index, is strictly larger): exact fractions compared exactly,
// otherwise the fp64 quotients.
__device__ __forceinline__ bool rel_gt(float as1, float ar1, bool ex1, double a1, double r1, float as2, float ar2,
                                       bool ex2, double a2, double r2, unsigned &n_fp64) {
  if (ex1 && ex2) {
    const int c = frac_cmp(as1, ar1, as2, ar2);
    if (c != 2) return c > 0;
  }
  ++n_fp64;
  const double q1 = __ddiv_rn(ex1 ? (double)as1 : a1, ex1 ? (double)ar1 : r1);
  const double q2 = __ddiv_rn(ex2 ? (double)as2 : a2, ex2 ? (double)ar2 : r2);
  return __double_as_longlong(q1) > __double_as_longlong(q2);
}

// ------------------------------------------------------------- slow path
static __device__ __noinline__ void record_lane(const PieceSh *P, uint32_t mask, uint64_t row, uint64_t col,
                                                uint64_t tr, uint64_t rp, uint64_t tc, uint64_t cp);

// Localisation maps and the batch's mismatch count for one step: bit k of
// `mask` is element idx0 + k of this lane.  When every lane's mismatches lie
// in one row and one tile, and all lanes' in the same ones, the warp adds
// its total to that histogram bin and row bin with one atomic each;
// otherwise each lane walks its elements, merging runs of equal bins.
__device__ __forceinline__ void record_step(const PieceSh *P, WarpSh *W, uint32_t mask, int64_t idx0, int V) {
  const int lane = threadIdx.x & 31;
  const int total = __reduce_add_sync(0xffffffffu, (unsigned)__popc(mask));
  if (total == 0) return;
  const int64_t mism0 = W->mism;
  __syncwarp();
  if (lane == 0) {
    // lane 0's element is the step's first: its warp step within the batch
    // (32 V elements per warp step: V is 4 or 8; batch_steps is a power of two)
    const int64_t step = (idx0 - P->pbegin) >> (V == 8 ? 8 : 7);
    W->mism = mism0 + total;
    W->sbits |= 1u << (uint32_t)(step & (batch_steps(nin_class_of(P->cd.n_elig)) - 1));
  }
  const CaseDesc &cd = P->cd;
  const uint64_t N = cd.dN.d, th = cd.dth.d, tw = cd.dtw.d;
  if (cd.idx32) {
    // The first element of the first lane holding a mismatch, computed by
    // every lane alike: when the lanes from it to the last one holding a
    // mismatch lie in one row and one tile, the maps need no further vote.
    const unsigned act = __ballot_sync(0xffffffffu, mask != 0);
    const int lead = __ffs(act) - 1, span = 32 - __clz(act) - lead;
    const uint32_t b0 = (uint32_t)idx0 + (uint32_t)((lead - lane) * V);
    const uint32_t r0 = div_q32(b0, (uint32_t)N, cd.m32N);
    const uint32_t c0 = b0 - r0 * (uint32_t)N;
    const uint32_t tc0 = div_q32(c0, (uint32_t)tw, cd.m32tw);
    const uint32_t cp0 = c0 - tc0 * (uint32_t)tw;
    if ((uint64_t)c0 + span * V <= N && (uint64_t)cp0 + span * V <= tw) {
      if (lane == lead) {
        const uint32_t tr0 = div_q32(r0, (uint32_t)th, cd.m32th);
        const uint32_t rp0 = r0 - tr0 * (uint32_t)th;
        const int64_t hb = P->wr > 0 ? ((int64_t)tr0 - P->tr0) * P->wc + ((int64_t)tc0 - P->tc0)
                                     : (int64_t)((uint64_t)tr0 * (uint64_t)cd.GC + tc0);
        if (P->wr > 0) sh_add(&P->sh_hist[hb], total);
        else gl_add(&P->g_hist[hb], (unsigned long long)total);
        if (P->prof_smem) sh_add(&P->sh_row[rp0], total);
        else gl_add(&P->g_row[rp0], (unsigned long long)total);
      }
      if (mask) {
        const uint32_t cp = cp0 + (uint32_t)((lane - lead) * V);  // lane >= lead here
        if (P->prof_smem) {
          const uint32_t base = (uint32_t)__cvta_generic_to_shared(P->sh_col + cp);
#pragma unroll
          for (int k = 0; k < 8; ++k)
            if (k < V && ((mask >> k) & 1u)) sh_add_at(base + 4 * k, 1);
        } else {
          for (uint32_t m = mask; m; m &= m - 1) gl_add(&P->g_col[cp + __ffs(m) - 1], 1ull);
        }
      }
      return;
    }
  }
  uint64_t row = 0, col = 0, tr = 0, rp = 0, tc = 0, cp = 0;
  int64_t hbin = -1;
  bool single = false;
  if (mask) {
    if (cd.idx32) {
      const uint32_t r32 = div_q32((uint32_t)idx0, (uint32_t)N, cd.m32N);
      const uint32_t c32 = (uint32_t)idx0 - r32 * (uint32_t)N;
      const uint32_t tr32 = div_q32(r32, (uint32_t)th, cd.m32th), tc32 = div_q32(c32, (uint32_t)tw, cd.m32tw);
      row = r32;
      col = c32;
      tr = tr32;
      rp = r32 - tr32 * (uint32_t)th;
      tc = tc32;
      cp = c32 - tc32 * (uint32_t)tw;
    } else {
      row = div_q((uint64_t)idx0, N, cd.dN.m);
      col = (uint64_t)idx0 - row * N;
      tr = div_q(row, th, cd.dth.m);
      rp = row - tr * th;
      tc = div_q(col, tw, cd.dtw.m);
      cp = col - tc * tw;
    }
    hbin = P->wr > 0 ? ((int64_t)tr - P->tr0) * P->wc + ((int64_t)tc - P->tc0) : (int64_t)(tr * (uint64_t)cd.GC + tc);
    single = col + V <= N && cp + V <= tw;
  }
  const unsigned act = __ballot_sync(0xffffffffu, mask != 0);
  const int lead = __ffs(act) - 1;
  const int64_t hb_l = __shfl_sync(0xffffffffu, hbin, lead);
  const uint64_t rp_l = __shfl_sync(0xffffffffu, rp, lead);
  if (__all_sync(0xffffffffu, mask == 0 || (single && hbin == hb_l && rp == rp_l))) {
    if (lane == lead) {
      if (P->wr > 0) sh_add(&P->sh_hist[hbin], total);
      else gl_add(&P->g_hist[hbin], (unsigned long long)total);
      if (P->prof_smem) sh_add(&P->sh_row[rp], total);
      else gl_add(&P->g_row[rp], (unsigned long long)total);
    }
    if (P->prof_smem) {
      const uint32_t base = (uint32_t)__cvta_generic_to_shared(P->sh_col + cp);
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if (k < V && ((mask >> k) & 1u)) sh_add_at(base + 4 * k, 1);
    } else {
      for (uint32_t m = mask; m; m &= m - 1) gl_add(&P->g_col[cp + __ffs(m) - 1], 1ull);
    }
    return;
  }
  if (mask) record_lane(P, mask, row, col, tr, rp, tc, cp);
}

// Localisation and the batch's mismatch count for one step of a case with
// aligned geometry (CaseDesc::amode): the step (32 V elements from s0, a
// multiple of the step) lies in one row, and lane l's elements lie in tile
// column (s0 mod N) / tw + (l >> a_shift) at column offsets
// (l mod 2^a_shift) V + k.  Every lane computes the row and tile from s0
// alike (no vote), the first lane of each tile adds the tile's count to its
// histogram bin, lane 0 adds the step's count to the row bin, and each lane
// adds its column bits to its private counters in shared memory, which are
// added to the column profile at the end of the piece.
template <int V>
__device__ __forceinline__ void record_step_aligned(const PieceSh *P, WarpSh *W, uint32_t mask, int64_t idx0) {
  const int lane = threadIdx.x & 31;
  const int cnt = __popc(mask);
  const int total = __reduce_add_sync(0xffffffffu, (unsigned)cnt);
  if (total == 0) return;
  const CaseDesc &cd = P->cd;
  const uint32_t N = (uint32_t)cd.dN.d, th = (uint32_t)cd.dth.d, tw = (uint32_t)cd.dtw.d;
  const uint32_t s0 = (uint32_t)idx0 - (uint32_t)(lane * V);
  const uint32_t row = div_q32(s0, N, cd.m32N);
  const uint32_t col0 = s0 - row * N;
  const uint32_t tr = div_q32(row, th, cd.m32th);
  const uint32_t rp = row - tr * th;
  const int sh = cd.a_shift;
  const uint32_t tc = div_q32(col0, tw, cd.m32tw) + (uint32_t)(lane >> sh);
  int gsum = cnt;
  if (sh == 5) {
    gsum = total;
  } else {
    for (int o = 1; o < (1 << sh); o <<= 1) gsum += __shfl_xor_sync(0xffffffffu, gsum, o);
  }
  if (gsum != 0 && (lane & ((1 << sh) - 1)) == 0) {
    if (P->wr > 0) sh_add(&P->sh_hist[((int64_t)tr - P->tr0) * P->wc + ((int64_t)tc - P->tc0)], gsum);
    else gl_add(&P->g_hist[(int64_t)tr * cd.GC + tc], (unsigned long long)gsum);
  }
  if (lane == 0) {
    if (P->prof_smem) sh_add(&P->sh_row[rp], total);
    else gl_add(&P->g_row[rp], (unsigned long long)total);
    W->mism += total;
    W->sbits |= 1u << (((s0 - (uint32_t)P->pbegin) >> (V == 8 ? 8 : 7)) & (batch_steps(nin_class_of(cd.n_elig)) - 1));
  }
  if (mask) {
    const uint32_t a = P->lcol_sa + (uint32_t)threadIdx.x * (V * 4);
#pragma unroll
    for (int j = 0; j < V; j += 4) {
      int x, y, z, w;
      asm volatile("ld.shared.v4.s32 {%0,%1,%2,%3}, [%4];" : "=r"(x), "=r"(y), "=r"(z), "=r"(w) : "r"(a + 4 * j));
      x += (mask >> j) & 1u;
      y += (mask >> (j + 1)) & 1u;
      z += (mask >> (j + 2)) & 1u;
      w += (mask >> (j + 3)) & 1u;
      asm volatile("st.shared.v4.s32 [%0], {%1,%2,%3,%4};" ::"r"(a + 4 * j), "r"(x), "r"(y), "r"(z), "r"(w));
    }
  }
}

// The general case of record_step for one lane: walk its mismatches from
// the coordinates of its first element, merging runs of equal bins.
static __device__ __noinline__ void record_lane(const PieceSh *P, uint32_t mask, uint64_t row, uint64_t col,
                                                uint64_t tr, uint64_t rp, uint64_t tc, uint64_t cp) {
  const CaseDesc &cd = P->cd;
  const uint64_t N = cd.dN.d, th = cd.dth.d, tw = cd.dtw.d;
  uint32_t m = mask;
  int kprev = 0;
  int64_t hb_cur = -1, rbin = -1;
  int hcnt = 0, rcnt = 0;
  while (m) {
    const int k = __ffs(m) - 1;
    m &= m - 1;
    for (int st = k - kprev; st > 0; --st) {  // advance one element
      ++col;
      ++cp;
      if (cp == tw) {
        cp = 0;
        ++tc;
      }
      if (col == N) {
        col = cp = tc = 0;
        ++row;
        if (++rp == th) {
          rp = 0;
          ++tr;
        }
      }
    }
    kprev = k;
    const int64_t hb = P->wr > 0 ? ((int64_t)tr - P->tr0) * P->wc + ((int64_t)tc - P->tc0)
                                 : (int64_t)(tr * (uint64_t)cd.GC + tc);
    if (hb != hb_cur) {
      if (hcnt) {
        if (P->wr > 0) sh_add(&P->sh_hist[hb_cur], hcnt);
        else gl_add(&P->g_hist[hb_cur], (unsigned long long)hcnt);
      }
      hb_cur = hb;
      hcnt = 0;
    }
    ++hcnt;
    if ((int64_t)rp != rbin) {
      if (rcnt) {
        if (P->prof_smem) sh_add(&P->sh_row[rbin], rcnt);
        else gl_add(&P->g_row[rbin], (unsigned long long)rcnt);
      }
      rbin = (int64_t)rp;
      rcnt = 0;
    }
    ++rcnt;
    if (P->prof_smem) sh_add(&P->sh_col[cp], 1);
    else gl_add(&P->g_col[cp], 1ull);
  }
  if (P->wr > 0) sh_add(&P->sh_hist[hb_cur], hcnt);
  else gl_add(&P->g_hist[hb_cur], (unsigned long long)hcnt);
  if (P->prof_smem) sh_add(&P->sh_row[rbin], rcnt);
  else gl_add(&P->g_row[rbin], (unsigned long long)rcnt);
}

// After a step in which some lane's maximum changed: the warp's own
// thresholds from the lanes' maxima (fp32 lower bounds, so no fp64 is
// needed), publication of improvements to the case, the merged thresholds.
//   abs: fl_rd(max), which is max itself when max is exact in fp32: an
//        element whose exact |d| is not above it is not larger than a
//        maximum held at a lower index of this warp (the warp sweeps its
//        batches of a piece in ascending order), so ties with the warp's
//        own maximum leave the fast path alone.  An inexact difference whose
//        rounded |s| equals it may exceed it and stays a candidate;
//   rel: rel_thr of the largest fraction held (rounded down, or for fp16
//        and bf16 up where no other fraction can fall in between), by the
//        same argument; an inexact difference whose rounded |s| meets the
//        threshold may lie above it, so the exact and dense steps compare
//        those against the threshold less 2^-20.
static __device__ __noinline__ void refresh(const PieceSh *P, const LaneSh *L, WarpSh *W) {
  const int lane = threadIdx.x & 31;
  const float fa = warp_reduce(abs_lb(L), [](float x, float y) { return fmaxf(x, y); });
  const float fr = warp_reduce(rel_thr(P, L), [](float x, float y) { return fmaxf(x, y); });
  __syncwarp();
  if (lane == 0) {
    W->wA = fmaxf(W->cA, fa < 0.f ? -1.f : fa);
    W->wR = fmaxf(W->cR, fr < 0.f ? -1.f : fr);
    // Publish improvements to the block, and to the case when they raise
    // the block's value (the block's value came from the case or from a
    // warp that published it there).
    if (fa > 0.f && __float_as_uint(fa) > W->pubA) {
      if (sh_max_old(&P->cta_thr[0], __float_as_uint(fa)) < __float_as_uint(fa))
        atomicMax(&P->g_thr[0], __float_as_uint(fa));
      W->pubA = __float_as_uint(fa);
    }
    if (fr > 0.f && __float_as_uint(fr) > W->pubR) {
      if (sh_max_old(&P->cta_thr[1], __float_as_uint(fr)) < __float_as_uint(fr))
        atomicMax(&P->g_thr[1], __float_as_uint(fr));
      W->pubR = __float_as_uint(fr);
    }
    merge_thr(W->wA, W->wR, W->ga, W->gr, W->tA, W->tR);
  }
  __syncwarp();
}

// Profile counters of one exact (slot 0), light (slot 1) or dense (slot 2)
// step, kept per warp and added to the call's counters once per piece.
__device__ __forceinline__ void count_stats(WarpSh *W, int slot, long long t0, unsigned n_abs, unsigned n_rel,
                                            unsigned n_pred) {
  n_abs = __reduce_add_sync(0xffffffffu, n_abs);
  n_rel = __reduce_add_sync(0xffffffffu, n_rel);
  n_pred = __reduce_add_sync(0xffffffffu, n_pred);
  if ((threadIdx.x & 31) == 0) {
    W->st[slot == 0 ? 0 : (slot == 1 ? 4 : 7)] += 1;
    W->st[slot == 0 ? 5 : (slot == 1 ? 6 : 8)] += (unsigned long long)(clock64() - t0);
    W->st[1] += n_abs;
    W->st[2] += n_rel;
    W->st[3] += n_pred;
  }
}

// The exact path for one step: this lane's n (<= V) elements idx0 ..
// idx0+n-1, whose stored bits sit in cv / rv (vector layout).  Called by
// the whole warp.  Candidates for a new maximum are screened within the
// step in fp32 (only the lane's near-largest values go on).
template <int DT>
__device__ __noinline__ SseAcc slow_step(const PieceSh *P, LaneSh *L, WarpSh *W, uint4 cv, uint4 rv,
                                         int64_t idx0, int n, SseAcc sse) {
  constexpr int V = Tr<DT>::V;
  const long long t_start = P->stats ? clock64() : 0;
  const CaseDesc &cd = P->cd;
  const float tA = W->tA, tR = W->tR;
  uint32_t mask = 0, candA = 0, candR = 0;
  float s[V], e[V], rel[V];
  float mA = -1.f, mR = -1.f;
  unsigned n_abs = 0, n_rel = 0, n_pred = 0;
#pragma unroll 1
  for (int k = 0; k < V; ++k) {
    s[k] = 0.f;
    e[k] = 0.f;
    rel[k] = 0.f;
    if (k >= n) continue;
    const uint32_t cb = vbits<DT>(cv, k), rb = vbits<DT>(rv, k);
    const float cf = to_f32<DT>(cb), rf = to_f32<DT>(rb);
    bool cfin = true, rfin = true, equal;
    if constexpr (Tr<DT>::kInt) {
      const long long d = (long long)(int32_t)cb - (long long)(int32_t)rb;
      s[k] = __ll2float_rn(d);
      e[k] = __ll2float_rn(d - __float2ll_rn(s[k]));
      equal = cb == rb;
    } else {
      s[k] = __fsub_rn(cf, rf);
      const float bb = __fsub_rn(s[k], cf);
      e[k] = __fsub_rn(__fsub_rn(cf, __fsub_rn(s[k], bb)), __fadd_rn(rf, bb));  // TwoSum(c, -r)
      cfin = isfinite(cf);
      rfin = isfinite(rf);
      equal = cf == rf;
      if (!cfin) sh_add(&P->sh_cls[isnan(cf) ? 0 : (cf > 0.f ? 1 : 2)], 1);
      if (!rfin) sh_add(&P->sh_cls[isnan(rf) ? 3 : (rf > 0.f ? 4 : 5)], 1);
    }
    const float as = fabsf(s[k]), ar = fabsf(rf);
    const bool fin = cfin && rfin;
    bool pass;
    if (equal) {
      pass = true;
    } else if (!fin) {
      pass = false;
    } else if (as <= __fmaf_rz(cd.lo_r, ar, cd.lo_a)) {
      pass = true;
    } else if (as > __fmaf_ru(cd.hi_r, ar, cd.hi_a)) {
      pass = false;
    } else {
      pass = pass64(to_f64<DT>(cb), to_f64<DT>(rb), cd.rtol, cd.atol);
      ++n_pred;
    }
    if (!pass) mask |= 1u << k;
    if (fin) {
      // an inexact difference rounded onto the threshold may lie above it
      if (!(as <= tA) || (as == tA && e[k] != 0.f)) {
        candA |= 1u << k;
        mA = fmaxf(mA, as);
      }
      // (an inexact difference may lie above its rounded as: a margin)
      if (ar != 0.f && !(as <= __fmul_rz(e[k] == 0.f ? tR : __fmul_rz(tR, kMarginLo), ar))) {
        candR |= 1u << k;
        rel[k] = rel32(as, ar);
        mR = fmaxf(mR, rel[k]);
      }
      if (as <= kHuge) {
        if (k & 1) ff_term(sse.hi.y, sse.lo.y, s[k], e[k]);
        else ff_term(sse.hi.x, sse.lo.x, s[k], e[k]);
      } else {
        const double d = __dsub_rn(to_f64<DT>(cb), to_f64<DT>(rb));
        sse.acc = __dadd_rn(sse.acc, __dmul_rn(d, d));
      }
    } else {
      sh_add(&P->sh_cls[6], 1);
    }
  }
  // Exact evaluation of the screened candidates.  abs: values below the
  // fp32 predecessor of the step's largest |s| are strictly smaller than it.
  // rel: fl32(|s| / |r|) is within 2^-22 of the quotient, so values below
  // (1 - 2^-20) of the largest are strictly smaller.  The lane's best of
  // each kind (largest, lowest index on ties) is chosen in registers and
  // offered once.
  bool changed = false;
  if (candA | candR) {
    const float fA = mA > 0.f ? __uint_as_float(__float_as_uint(mA) - 1u) : mA;
    const float fR = __fmul_rz(mR, kMarginLo);
    int kA = -1, kR = -1;
    float bA = 0.f, bRn = 0.f, bRd = 1.f, bRq = 0.f;
    bool xA = true, xR = true;
    double aA = 0.0, aR = 0.0, rR = 0.0;
#pragma unroll 1
    for (int k = 0; k < V; ++k) {
      const bool ca = ((candA >> k) & 1u) && fabsf(s[k]) >= fA;
      const bool cr = ((candR >> k) & 1u) && rel[k] >= fR;
      if (!(ca || cr)) continue;
      const float as = fabsf(s[k]);
      const uint32_t rb = vbits<DT>(rv, k);
      const float ar = fabsf(to_f32<DT>(rb));
      bool exact = e[k] == 0.f;
      if constexpr (Tr<DT>::kInt) exact = exact && as < 0x1p24f && ar < 0x1p24f;
      // fl64(|c - r|) from the widened values when c - r is not exact in
      // fp32 (this also covers an fp32 overflow of c - r).
      double a64 = (double)as;
      if (!exact) {
        ++n_abs;
        a64 = fabs(__dsub_rn(to_f64<DT>(vbits<DT>(cv, k)), to_f64<DT>(rb)));
      }
      if (ca) {
        const bool better = kA < 0 || ((exact && xA) ? as > bA
                                                      : __double_as_longlong(a64) > __double_as_longlong(aA));
        if (better) {
          kA = k;
          bA = as;
          xA = exact;
          aA = a64;
        }
      }
      if (cr) {
        const double r64 = fabs(to_f64<DT>(rb));
        if (kR < 0 || rel_gt(as, ar, exact, a64, r64, bRn, bRd, xR, aR, rR, n_rel)) {
          kR = k;
          bRn = as;
          bRd = ar;
          bRq = rel[k];
          xR = exact;
          aR = a64;
          rR = r64;
        }
      }
    }
    if (kA >= 0) changed |= offer_abs(L, bA, xA, aA, idx0 + kA);
    if (kR >= 0) changed |= offer_rel(L, bRn, bRd, xR, aR, rR, bRq, idx0 + kR, n_rel);
  }
  if (__any_sync(0xffffffffu, mask != 0)) {
    if (P->cd.amode) record_step_aligned<V>(P, W, mask, idx0);
    else record_step(P, W, mask, idx0, V);
  }
  if (__any_sync(0xffffffffu, changed)) refresh(P, L, W);
  if (P->stats) count_stats(W, 0, t_start, n_abs, n_rel, n_pred);
  return sse;
}

// A step whose only reason to leave the fast path is a possible new
// maximum: every element is finite, provably passes, and c - r is exact in
// fp32 (the fast path's conditions other than the thresholds tA, tR).  The
// maxima are updated as in slow_step; the SSE takes the fast path's
// arithmetic.
template <int DT>
__device__ __noinline__ SseAcc light_step(const PieceSh *P, LaneSh *L, WarpSh *W, uint4 cv, uint4 rv,
                                          int64_t idx0, SseAcc sse) {
  constexpr int V = Tr<DT>::V;
  const long long t_start = P->stats ? clock64() : 0;
  const float tA = W->tA, tR = W->tR;
  float s[V], rel[V];
  uint32_t candA = 0, candR = 0;
  float mA = -1.f, mR = -1.f;
#pragma unroll 1
  for (int k = 0; k < V; ++k) {
    const float cf = vdec<DT>(cv, k), rf = vdec<DT>(rv, k);
    if constexpr (Tr<DT>::kInt) {
      s[k] = 0.f;  // int32 light steps are bitwise-equal steps
    } else {
      s[k] = __fsub_rn(cf, rf);
    }
    const float as = fabsf(s[k]), ar = fabsf(rf);
    rel[k] = 0.f;
    if (!(as <= tA)) {
      candA |= 1u << k;
      mA = fmaxf(mA, as);
    }
    if (ar != 0.f && !(as <= __fmul_rz(tR, ar))) {
      candR |= 1u << k;
      rel[k] = rel32(as, ar);
      mR = fmaxf(mR, rel[k]);
    }
  }
  bool changed = false;
  unsigned n_rel = 0;
  if (candA | candR) {
    // every element here is finite with c - r exact: the lane's best of
    // each kind is chosen in registers (exact comparisons) and offered once
    const float fA = mA > 0.f ? __uint_as_float(__float_as_uint(mA) - 1u) : mA;
    const float fR = __fmul_rz(mR, kMarginLo);
    int kA = -1, kR = -1;
    float bA = 0.f, bRn = 0.f, bRd = 1.f, bRq = 0.f;
    bool xR = true;
    double rR = 0.0;
#pragma unroll 1
    for (int k = 0; k < V; ++k) {
      const float as = fabsf(s[k]);
      if (((candA >> k) & 1u) && as >= fA && (kA < 0 || as > bA)) {
        kA = k;
        bA = as;
      }
      if (((candR >> k) & 1u) && rel[k] >= fR) {
        const uint32_t rb = vbits<DT>(rv, k);
        const float ar = fabsf(to_f32<DT>(rb));
        const bool exact = !Tr<DT>::kInt || ar < 0x1p24f;
        const double r64 = fabs(to_f64<DT>(rb));
        if (kR < 0 || rel_gt(as, ar, exact, (double)as, r64, bRn, bRd, xR, (double)bRn, rR, n_rel)) {
          kR = k;
          bRn = as;
          bRd = ar;
          bRq = rel[k];
          xR = exact;
          rR = r64;
        }
      }
    }
    if (kA >= 0) changed |= offer_abs(L, bA, true, 0.0, idx0 + kA);
    if (kR >= 0) changed |= offer_rel(L, bRn, bRd, xR, (double)bRn, rR, bRq, idx0 + kR, n_rel);
  }
  if constexpr (!Tr<DT>::kInt) {
#pragma unroll
    for (int k = 0; k < V; k += 2) ff_pair<Tr<DT>::EB == 4>(sse, make_float2(s[k], s[k + 1]));
  }
  if (__any_sync(0xffffffffu, changed)) refresh(P, L, W);
  if (P->stats) count_stats(W, 1, t_start, 0, n_rel, 0);
  return sse;
}

// A float step that needs more than a maximum update: one classification
// pass over the lane's elements decides for the warp between
//  * dense: every element finite, its predicate decided by the fp32 bounds
//    and no candidate for a maximum (|s| <= tA and |s| <= tR |r|, tR
//    uncapped): only the mismatch count, the maps and the SSE remain, done
//    here; the SSE terms take the exact path's arithmetic (c - r as s + e by
//    TwoSum, d^2 = p + pe + 2se), so the result does not depend on which path
//    an element took;
//  * a light step when every element provably passes, is finite and has an
//    exact fp32 difference (only candidates for a maximum);
//  * otherwise the exact step.
template <int DT>
__device__ __noinline__ SseAcc hard_step(const PieceSh *P, LaneSh *L, WarpSh *W, uint4 cv, uint4 rv,
                                         int64_t idx0, SseAcc sse) {
  constexpr int V = Tr<DT>::V;
  const long long t_start = P->stats ? clock64() : 0;
  const float2 m1 = make_float2(-1.f, -1.f);
  const float2 lo_r2 = make_float2(P->cd.lo_r, P->cd.lo_r), lo_a2 = make_float2(P->cd.lo_a, P->cd.lo_a);
  const float2 hi_r2 = make_float2(P->cd.hi_r, P->cd.hi_r), hi_a2 = make_float2(P->cd.hi_a, P->cd.hi_a);
  const float tA = W->tA, tR = W->tR;
  const float2 tR2 = make_float2(tR, tR);
  float2 s[V / 2], e[V / 2];
  bool dense = true;
  uint32_t mask = 0;
#pragma unroll
  for (int j = 0; j < V / 2; ++j) {
    const float2 c2 = make_float2(vdec<DT>(cv, 2 * j), vdec<DT>(cv, 2 * j + 1));
    const float2 r2 = make_float2(vdec<DT>(rv, 2 * j), vdec<DT>(rv, 2 * j + 1));
    // TwoSum(c, -r): s + e = c - r exactly when both are finite
    const float2 s2 = __ffma2_rn(r2, m1, c2);
    const float2 bb = __ffma2_rn(c2, m1, s2);
    const float2 y = __ffma2_rn(__ffma2_rn(bb, m1, s2), m1, c2);
    s[j] = s2;
    e[j] = __ffma2_rn(__fadd2_rn(r2, bb), m1, y);
    const float2 ar2 = make_float2(fabsf(r2.x), fabsf(r2.y));
    const float2 a2 = __ffma2_rz(ar2, lo_r2, lo_a2);
    const float2 h2 = __ffma2_ru(ar2, hi_r2, hi_a2);
    const float2 t2 = __fmul2_rz(ar2, tR2);
    const float as0 = fabsf(s2.x), as1 = fabsf(s2.y);
    // (an inexact difference rounded onto tA may lie above it)
    // (and one rounded onto tR |r|: a margin)
    dense &= (as0 <= a2.x || as0 > h2.x) && (as0 < tA || (as0 == tA && e[j].x == 0.f)) &&
             as0 <= (e[j].x == 0.f ? t2.x : __fmul_rz(t2.x, kMarginLo));
    dense &= (as1 <= a2.y || as1 > h2.y) && (as1 < tA || (as1 == tA && e[j].y == 0.f)) &&
             as1 <= (e[j].y == 0.f ? t2.y : __fmul_rz(t2.y, kMarginLo));
    if (!(as0 <= a2.x)) mask |= 1u << (2 * j);
    if (!(as1 <= a2.y)) mask |= 2u << (2 * j);
  }
  if (!__all_sync(0xffffffffu, dense)) {
    // Light or exact: a light step needs every element provably passing,
    // finite and exact in fp32 (|s| <= min(fma_rz(lo_r, |r|, lo_a), |r|/4);
    // the finite cap keeps infinities out).
    bool other = false;
#pragma unroll
    for (int j = 0; j < V / 2; ++j) {
      const float2 r2 = make_float2(vdec<DT>(rv, 2 * j), vdec<DT>(rv, 2 * j + 1));
      const float2 ar2 = make_float2(fabsf(r2.x), fabsf(r2.y));
      const float2 a2 = __ffma2_rz(ar2, lo_r2, lo_a2);
      other |= !(fabsf(s[j].x) <= min3f(a2.x, __fmul_rz(0.25f, ar2.x), kHuge));
      other |= !(fabsf(s[j].y) <= min3f(a2.y, __fmul_rz(0.25f, ar2.y), kHuge));
    }
    if (__any_sync(0xffffffffu, other)) return slow_step<DT>(P, L, W, cv, rv, idx0, V, sse);
    return light_step<DT>(P, L, W, cv, rv, idx0, sse);
  }
#pragma unroll
  for (int j = 0; j < V / 2; ++j) {
    const float2 p = __fmul2_rn(s[j], s[j]);
    const float2 pe = __ffma2_rn(s[j], s[j], __fmul2_rn(p, m1));
    const float2 q = __ffma2_rn(__fadd2_rn(s[j], s[j]), e[j], pe);
    const float2 t = __fadd2_rn(sse.hi, p);
    const float2 bp = __ffma2_rn(sse.hi, m1, t);
    const float2 x2 = __ffma2_rn(__ffma2_rn(bp, m1, t), m1, sse.hi);
    const float2 err = __fadd2_rn(x2, __ffma2_rn(bp, m1, p));
    sse.lo = __fadd2_rn(sse.lo, __fadd2_rn(err, q));
    sse.hi = t;
  }
  if (__any_sync(0xffffffffu, mask != 0)) {
    if (P->cd.amode) record_step_aligned<V>(P, W, mask, idx0);
    else record_step(P, W, mask, idx0, V);
  }
  if (P->stats) count_stats(W, 2, t_start, 0, 0, 0);
  return sse;
}

// A ragged step: this lane's n (0..V) elements from idx0, loaded one by one.
template <int DT, int NIN>
__device__ __noinline__ SseAcc tail_step(const PieceSh *P, LaneSh *L, WarpSh *W, int64_t idx0, int n,
                                         SseAcc sse) {
  constexpr int EB = Tr<DT>::EB;
  const CaseDesc &cd = P->cd;
  uint32_t cw[4] = {0, 0, 0, 0}, rw[4] = {0, 0, 0, 0};
  const uint32_t c0 = ld_one<EB>(cd.cand, 0), r0 = ld_one<EB>(cd.ref, 0);
  for (int k = 0; k < n; ++k) {
    const int64_t i = idx0 + k;
    const uint32_t cb = ld_one<EB>(cd.cand, i), rb = ld_one<EB>(cd.ref, i);
    L->cacc |= cb ^ c0;
    L->racc |= rb ^ r0;
    if constexpr (NIN != 0) {
      for (int j = 0; j < cd.n_elig; ++j) {
        const uint32_t xb = ld_one<EB>(cd.in_ptr[j], i);
        P->sh_eq[threadIdx.x * NMV_MAX_INPUTS + j] += (cb == xb) & (rb != xb);
      }
    }
    if constexpr (EB == 2) {
      cw[k >> 1] |= cb << (16 * (k & 1));
      rw[k >> 1] |= rb << (16 * (k & 1));
    } else {
      cw[k] = cb;
      rw[k] = rb;
    }
  }
  return slow_step<DT>(P, L, W, make_uint4(cw[0], cw[1], cw[2], cw[3]), make_uint4(rw[0], rw[1], rw[2], rw[3]),
                       idx0, n, sse);
}

// Pass-through counts of one step for the generic input path (n_elig >= 2).
template <int DT>
__device__ __noinline__ void eq_generic(const PieceSh *P, LaneSh *L, const uint4 cv, const uint4 rv,
                                        int64_t e) {
  const CaseDesc &cd = P->cd;
  for (int j = 0; j < cd.n_elig; ++j) {
    const uint4 x = ld_v4((const char *)cd.in_ptr[j] + e * Tr<DT>::EB);
    int add = 0;
#pragma unroll
    for (int k = 0; k < Tr<DT>::V; ++k) {
      const uint32_t xb = vbits<DT>(x, k);
      add += (vbits<DT>(cv, k) == xb) & (vbits<DT>(rv, k) != xb);
    }
    P->sh_eq[threadIdx.x * NMV_MAX_INPUTS + j] += add;
  }
}

// -------------------------------------------------- the shared-memory ring
// Each warp streams its own batches into a private ring of shared-memory
// stages with bulk copies (cp.async.bulk, completion counted in bytes on an
// mbarrier per stage), kRingStages(nin) - 1 batches ahead of the one it is
// checking.  Memory parallelism then needs no registers, and the checking
// loop stays small.
__device__ __forceinline__ uint32_t smem_addr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t *bar) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// The same at a 32-bit shared address.
__device__ __forceinline__ bool mbar_try_wait_at(uint32_t bar_sa, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(bar_sa), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Wait for a stage's copies; gives up after kWaitNs (then the call reports
// an error instead of hanging the GPU).
constexpr uint64_t kWaitNs = 2000000000ull;

// try_wait with a suspend-time hint: the thread sleeps until the phase
// completes or hint_ns elapse, instead of re-polling (a waiting warp then
// takes no issue slots from the warps that compute).
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t *bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

static __device__ __noinline__ bool mbar_wait_slow(uint64_t *bar, uint32_t parity) {
  const uint64_t t0 = global_ns();
  while (!mbar_try_wait_sleep(bar, parity, 100000u))  // at most 0.1 ms per try
    if (global_ns() - t0 > kWaitNs) return false;
  return true;
}

// The streamed tensors are read once: their L2 lines are marked
// evict-first, so they do not push out what is reused (kernel code,
// descriptors, counters, the next call's metadata).
__device__ __forceinline__ uint64_t evict_first_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// One lane of the (converged) warp, chosen by the hardware.
__device__ __forceinline__ bool elect_one() {
  uint32_t e;
  asm volatile("{\n .reg .pred p;\n elect.sync _|p, 0xffffffff;\n selp.u32 %0, 1, 0, p;\n}" : "=r"(e));
  return e != 0;
}

// A bulk copy into shared memory at a 32-bit shared address, completing on
// the mbarrier at bar_sa.
__device__ __forceinline__ void bulk_load_sa(uint32_t dst_sa, const void *src, uint32_t bytes, uint32_t bar_sa,
                                             uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          dst_sa),
      "l"(src), "r"(bytes), "r"(bar_sa), "l"(pol)
      : "memory");
}

__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(pol)
      : "memory");
}

__device__ __forceinline__ uint4 lds_v4(const void *p) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(smem_addr(p)));
  return v;
}

// The same from a 32-bit shared address plus a byte offset.
__device__ __forceinline__ uint4 lds_v4_off(uint32_t sa, uint32_t off) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(sa + off));
  return v;
}

// ------------------------------------------------------------- fast step
// Lane registers carried through a piece.
template <int NIN>
struct Regs {
  SseAcc sse;
  uint32_t cacc, racc, cpat, rpat;
  int eq[NIN > 0 ? NIN : 1];
  float tA, tR;
  float tRq;     // min(tR, 1/4): also proves c - r exact (see the file comment)
  float ga, gr;  // copy of WarpSh::ga / gr
  float lo_r, lo_a;
  bool track_c, track_r;  // warp-uniform: the constant / all-zero accumulators still matter
};

template <int NIN>
__device__ __forceinline__ void reload_thr(Regs<NIN> &R, const WarpSh *W) {
  R.tA = W->tA;
  R.tR = W->tR;
  R.tRq = fminf(R.tR, 0.25f);
}

template <int DT, int NIN>
__device__ __forceinline__ void step(const PieceSh *P, LaneSh *L, WarpSh *W, Regs<NIN> &R, const uint4 &cv,
                                     const uint4 &rv, const uint4 &xv, uint32_t erel) {
  constexpr int V = Tr<DT>::V;
  if (R.track_c) R.cacc |= (cv.x ^ R.cpat) | (cv.y ^ R.cpat) | (cv.z ^ R.cpat) | (cv.w ^ R.cpat);
  if (R.track_r) R.racc |= (rv.x ^ R.rpat) | (rv.y ^ R.rpat) | (rv.z ^ R.rpat) | (rv.w ^ R.rpat);
  if constexpr (NIN == 1) {
#pragma unroll
    for (int k = 0; k < V; ++k) {
      const uint32_t xb = vbits<DT>(xv, k);
      R.eq[0] += (vbits<DT>(cv, k) == xb) & (vbits<DT>(rv, k) != xb);
    }
  } else if constexpr (NIN < 0) {
    eq_generic<DT>(P, L, cv, rv, P->pbegin + erel);
  }
  bool hard, other = false;
  if constexpr (Tr<DT>::kInt) {
    // int32: the fast path covers bitwise-equal steps (d = 0 everywhere,
    // which adds nothing to the SSE), once both maxima are held; everything
    // else takes the exact integer path.
    other = (cv.x != rv.x) | (cv.y != rv.y) | (cv.z != rv.z) | (cv.w != rv.w);
    hard = other | (R.tA < 0.f) | (R.tR < 0.f);
    if (!__any_sync(0xffffffffu, hard)) return;
  } else {
    float s[V];
    hard = false;
    const float2 m1 = make_float2(-1.f, -1.f);
#pragma unroll
    for (int k = 0; k < V; k += 2) {
      const float2 c2 = make_float2(vdec<DT>(cv, k), vdec<DT>(cv, k + 1));
      const float2 r2 = make_float2(vdec<DT>(rv, k), vdec<DT>(rv, k + 1));
      const float2 s2 = __ffma2_rn(r2, m1, c2);  // fl(c - r), one rounding
      s[k] = s2.x;
      s[k + 1] = s2.y;
      const float2 ar2 = make_float2(fabsf(r2.x), fabsf(r2.y));
      float2 a2, b2;
      if constexpr (Tr<DT>::EB == 2) {
        // the bounds in packed form (the same roundings as the scalar ones)
        a2 = __ffma2_rz(ar2, make_float2(R.lo_r, R.lo_r), make_float2(R.lo_a, R.lo_a));
        b2 = __fmul2_rz(ar2, make_float2(R.tRq, R.tRq));
      } else {
        a2 = make_float2(__fmaf_rz(R.lo_r, ar2.x, R.lo_a), __fmaf_rz(R.lo_r, ar2.y, R.lo_a));
        b2 = make_float2(__fmul_rz(R.tRq, ar2.x), __fmul_rz(R.tRq, ar2.y));
      }
      hard |= !(fabsf(s2.x) <= min3f(a2.x, b2.x, R.tA));
      hard |= !(fabsf(s2.y) <= min3f(a2.y, b2.y, R.tA));
    }
    if (!__any_sync(0xffffffffu, hard)) {
#pragma unroll
      for (int k = 0; k < V; k += 2) ff_pair<Tr<DT>::EB == 4>(R.sse, make_float2(s[k], s[k + 1]));
      return;
    }
    // dense, light or exact: decided out of line
    R.sse = hard_step<DT>(P, L, W, cv, rv, P->pbegin + erel, R.sse);
    reload_thr(R, W);
    return;
  }
  if (__any_sync(0xffffffffu, other)) R.sse = slow_step<DT>(P, L, W, cv, rv, P->pbegin + erel, V, R.sse);
  else R.sse = light_step<DT>(P, L, W, cv, rv, P->pbegin + erel, R.sse);
  reload_thr(R, W);
}

// The bins of a batch in the dense regime, when the batch lies in one row
// of the [M, N] view (aligned localisation and N a multiple of the batch):
// its row bin and the histogram bin of its first tile, computed once per
// batch; the batch's mismatch count, row total and step bits accumulate in
// registers and are added at the end of the batch.
struct DenseBins {
  int32_t ok;        // 0: not used this batch; 1: histogram window in shared memory; 2: global histogram
  int32_t sh;        // the case's a_shift (tile width V 2^sh)
  bool prof;         // the call counts profile statistics
  int32_t rp;        // row bin
  uint32_t hbin;     // the batch's first tile bin: shared address (ok 1) or global index (ok 2, < 2^26)
  int32_t rowsum;    // mismatches recorded this way in this batch
  uint32_t sbits;    // their warp steps
  int32_t lc0, lc1, lc2, lc3;  // this lane's column counts in the batch (fp32: V = 4 columns)
  int32_t ht;                  // one tile per step (sh = 5): lane u holds step u's count
  float hr, ha;                // the case's sure-fail bound terms (hi_r, hi_a)
};

// A float step of a warp in the dense regime (its last batch was mostly
// mismatches, as where a candidate passes an input through): one inline
// pass classifies every element with the TwoSum of c - r, the sure-pass and
// sure-fail bounds, and the maximum thresholds shrunk by the 2^-20 margin
// (|d| <= |s| (1 + 2^-24), so |s| <= tA (1 - 2^-20) proves |d| < tA, and
// |s| <= rz(|r| tR (1 - 2^-20)) proves |d| / |r| < tR: no new maximum,
// whether or not c - r is exact).  When every element of the warp is dense
// (finite, decided by the fp32 bounds, no candidate for a maximum) the SSE
// terms (the hard step's arithmetic), the mismatch count and the maps are
// done here too; any other step goes out of line as usual.  A clean step
// takes this path's SSE arithmetic with e = 0, which is the fast path's, so
// results do not depend on the regime.
template <int DT, int NIN>
__device__ __forceinline__ void step_dense(const PieceSh *P, LaneSh *L, WarpSh *W, Regs<NIN> &R, DenseBins &B,
                                           const uint4 &cv, const uint4 &rv, const uint4 &xv, uint32_t erel,
                                           int u) {
  constexpr int V = Tr<DT>::V;
  const long long t_start = B.prof ? clock64() : 0;
  if (R.track_c) R.cacc |= (cv.x ^ R.cpat) | (cv.y ^ R.cpat) | (cv.z ^ R.cpat) | (cv.w ^ R.cpat);
  if (R.track_r) R.racc |= (rv.x ^ R.rpat) | (rv.y ^ R.rpat) | (rv.z ^ R.rpat) | (rv.w ^ R.rpat);
  if constexpr (NIN == 1) {
#pragma unroll
    for (int k = 0; k < V; ++k) {
      const uint32_t xb = vbits<DT>(xv, k);
      R.eq[0] += (vbits<DT>(cv, k) == xb) & (vbits<DT>(rv, k) != xb);
    }
  } else if constexpr (NIN < 0) {
    eq_generic<DT>(P, L, cv, rv, P->pbegin + erel);
  }
  const float2 m1 = make_float2(-1.f, -1.f);
  const float2 lo_r2 = make_float2(R.lo_r, R.lo_r), lo_a2 = make_float2(R.lo_a, R.lo_a);
  const float hr = B.hr, ha = B.ha;
  const float2 hi_r2 = make_float2(hr, hr), hi_a2 = make_float2(ha, ha);
  const float tAm = __fmul_rz(R.tA, kMarginLo);
  const float tRm = __fmul_rz(R.tR, kMarginLo);
  const float2 tR2 = make_float2(tRm, tRm);
  float2 s[V / 2], e[V / 2];
  bool dense = true;
  uint32_t mask = 0;
#pragma unroll
  for (int j = 0; j < V / 2; ++j) {
    const float2 c2 = make_float2(vdec<DT>(cv, 2 * j), vdec<DT>(cv, 2 * j + 1));
    const float2 r2 = make_float2(vdec<DT>(rv, 2 * j), vdec<DT>(rv, 2 * j + 1));
    const float2 s2 = __ffma2_rn(r2, m1, c2);
    const float2 bb = __ffma2_rn(c2, m1, s2);
    const float2 y = __ffma2_rn(__ffma2_rn(bb, m1, s2), m1, c2);
    s[j] = s2;
    e[j] = __ffma2_rn(__fadd2_rn(r2, bb), m1, y);
    const float2 ar2 = make_float2(fabsf(r2.x), fabsf(r2.y));
    const float2 a2 = __ffma2_rz(ar2, lo_r2, lo_a2);
    const float2 h2 = __ffma2_ru(ar2, hi_r2, hi_a2);
    const float2 t2 = __fmul2_rz(ar2, tR2);
    const float as0 = fabsf(s2.x), as1 = fabsf(s2.y);
    const bool p0 = as0 <= a2.x, p1 = as1 <= a2.y;
    dense &= (p0 || as0 > h2.x) && as0 <= tAm && as0 <= t2.x;
    dense &= (p1 || as1 > h2.y) && as1 <= tAm && as1 <= t2.y;
    if (!p0) mask |= 1u << (2 * j);
    if (!p1) mask |= 2u << (2 * j);
  }
  if (!__all_sync(0xffffffffu, dense)) {
    R.sse = hard_step<DT>(P, L, W, cv, rv, P->pbegin + erel, R.sse);
    reload_thr(R, W);
    return;
  }
#pragma unroll
  for (int j = 0; j < V / 2; ++j) {
    const float2 p = __fmul2_rn(s[j], s[j]);
    const float2 pe = __ffma2_rn(s[j], s[j], __fmul2_rn(p, m1));
    const float2 q = __ffma2_rn(__fadd2_rn(s[j], s[j]), e[j], pe);
    const float2 t = __fadd2_rn(R.sse.hi, p);
    const float2 bp = __ffma2_rn(R.sse.hi, m1, t);
    const float2 x2 = __ffma2_rn(__ffma2_rn(bp, m1, t), m1, R.sse.hi);
    const float2 err = __fadd2_rn(x2, __ffma2_rn(bp, m1, p));
    R.sse.lo = __fadd2_rn(R.sse.lo, __fadd2_rn(err, q));
    R.sse.hi = t;
  }
  if (B.ok) {
    // the batch's bins: the step's tiles follow the batch's first one
    const int lane = threadIdx.x & 31;
    const int cnt = __popc(mask);
    const int total = __reduce_add_sync(0xffffffffu, (unsigned)cnt);
    if (total) {
      const int sh = B.sh;
      if (sh == 5) {
        // the step is one tile: lane u keeps its count for the batch's end
        if (lane == u) B.ht = total;
      } else {
        int gsum = cnt;
        for (int o = 1; o < (1 << sh); o <<= 1) gsum += __shfl_xor_sync(0xffffffffu, gsum, o);
        if (gsum != 0 && (lane & ((1 << sh) - 1)) == 0) {
          // the step holds 32 >> sh tiles (STEP / tw with tw = V 2^sh)
          const uint32_t t = (uint32_t)u * (32u >> sh) + (uint32_t)(lane >> sh);
          if (B.ok == 1) sh_add_at(B.hbin + 4 * t, gsum);
          else gl_add(P->g_hist + (B.hbin + t), (unsigned long long)gsum);
        }
      }
      B.rowsum += total;
      B.sbits |= 1u << u;
      static_assert(V == 4, "the dense regime is fp32 only");
      B.lc0 += (int32_t)(mask & 1u);  // added to the lanes' column counters at the batch's end
      B.lc1 += (int32_t)((mask >> 1) & 1u);
      B.lc2 += (int32_t)((mask >> 2) & 1u);
      B.lc3 += (int32_t)((mask >> 3) & 1u);
    }
  } else if (__any_sync(0xffffffffu, mask != 0)) {
    if (P->cd.amode) record_step_aligned<V>(P, W, mask, P->pbegin + erel);
    else record_step(P, W, mask, P->pbegin + erel, V);
  }
  if (B.prof) count_stats(W, 2, t_start, 0, 0, 0);
}

// Issue the copies of one stage (half a batch), at byte offset `off` of the
// piece and with `bytes` (whole steps only) per tensor (lane 0 only).  A
// ragged rest and the buffers of a case that is not 16-byte aligned
// (bytes = 0) are read from global memory by tail_step.
// The same from 32-bit shared addresses (the warp's elected lane).
template <int NIN>
__device__ __forceinline__ void ring_issue_sa(const char *c, const char *r, const char *x, uint32_t off,
                                              uint32_t bytes, uint32_t stage_sa, uint32_t bar_sa, bool stall) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar_sa),
               "r"(bytes * (NIN == 1 ? 3u : 2u))
               : "memory");
  if (bytes && !stall) {
    const uint64_t pol = evict_first_policy();
    bulk_load_sa(stage_sa, c + off, bytes, bar_sa, pol);
    bulk_load_sa(stage_sa + stage_bytes(NIN), r + off, bytes, bar_sa, pol);
    if constexpr (NIN == 1) bulk_load_sa(stage_sa + 2 * stage_bytes(NIN), x + off, bytes, bar_sa, pol);
  }
}

template <int NIN>
__device__ __forceinline__ void ring_issue(const char *c, const char *r, const char *x, uint32_t off,
                                           uint32_t bytes, uint8_t *stage, uint64_t *bar, bool stall) {
  mbar_arrive_tx(bar, bytes * (NIN == 1 ? 3u : 2u));
  // (stall: the test hook of the wait limit announces the bytes and issues
  // no copy, so the stage never completes and nothing is in flight)
  if (bytes && !stall) {
    const uint64_t pol = evict_first_policy();
    bulk_load(stage, c + off, bytes, bar, pol);
    bulk_load(stage + stage_bytes(NIN), r + off, bytes, bar, pol);
    if constexpr (NIN == 1) bulk_load(stage + 2 * stage_bytes(NIN), x + off, bytes, bar, pol);
  }
}

// Position of a warp in its ring: the stage it checks next and that
// stage's mbarrier phase.  Carried across pieces.
struct RingPos {
  uint32_t stage, phase;
};

constexpr uint32_t kNoBatch = 0xffffffffu;
// The SSE's float-float pairs go to fp64 every kFlushBatches batches of a
// lane (at most 128 terms per pair in between).
constexpr int kFlushBatches = 2;

// Number of batches warp w takes in a piece of nb batches (the j with
// j * kWarps + ((w - j) mod kWarps) < nb).
__device__ __forceinline__ uint32_t warp_batches(uint32_t nb, int warp) {
  const uint32_t J = nb / kWarps;
  const uint32_t last = (uint32_t)(((warp - (int)(J % kWarps)) % kWarps + kWarps) % kWarps);
  return J + (last < nb % kWarps ? 1u : 0u);
}

__device__ __forceinline__ void sse_flush(SseAcc &a) {
  // TwoSum of the two slots' high parts, then two fp64 additions.
  float h = a.hi.x, l = a.lo.x;
  ff_add(h, l, a.hi.y, a.lo.y);
  a.acc = __dadd_rn(a.acc, __dadd_rn((double)h, (double)l));
  a.hi = a.lo = make_float2(0.f, 0.f);
}

// Sweep this warp's batches of a piece (each batch_elems elements; only a
// case's last batch may be shorter) through its ring, one stage (half a
// batch) of copies ahead of the check, writing each batch's mismatch count.
// Offsets within the piece are 32-bit (a piece holds at most kMaxPiece
// elements).
template <int DT, int NIN>
__device__ __forceinline__ bool sweep(PieceSh *P, LaneSh *L, WarpSh *W, Regs<NIN> &R, const Piece &pc,
                                      int32_t *batch_count, uint8_t *ring, uint64_t *bars, RingPos &rp,
                                      uint32_t *err) {
  constexpr int V = Tr<DT>::V;
  constexpr int EB = Tr<DT>::EB;
  constexpr int STEP = 32 * V;
  constexpr int KS = batch_steps(NIN);
  constexpr int HS = stage_steps(NIN);
  constexpr int BATCH = STEP * KS;
  constexpr uint32_t BB = BATCH * EB;          // bytes of one tensor's batch
  constexpr uint32_t HB = stage_bytes(NIN);    // bytes of one tensor's stage
  constexpr uint32_t NSB = KS / HS;            // stages per batch
  constexpr uint32_t NST = ring_stages(NIN);
  constexpr int STAGE = ring_streams(NIN) * stage_bytes(NIN);
  constexpr int kPoll = kWarps;  // batches between a warp's readings of the case-wide maxima
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t *g_thr = P->g_thr;
  const uint32_t nb = __shfl_sync(0xffffffffu, (uint32_t)((pc.end - pc.begin + BATCH - 1) / BATCH), 0);
  const uint32_t mag = Tr<DT>::kInt ? 0xffffffffu : (Tr<DT>::EB == 2 ? 0x7fff7fffu : 0x7fffffffu);
  const uint32_t pbytes = __shfl_sync(0xffffffffu, (uint32_t)((pc.end - pc.begin) * EB), 0);
  const bool vec_ok = __shfl_sync(0xffffffffu, P->cd.vec_ok != 0 ? 1 : 0, 0) != 0;
  const char *src_c = (const char *)P->cd.cand + pc.begin * EB;
  const char *src_r = (const char *)P->cd.ref + pc.begin * EB;
  const char *src_x = NIN == 1 ? (const char *)P->cd.in_ptr[0] + pc.begin * EB : nullptr;
  int32_t *bcount = batch_count + pc.batch_base;
  // lane 0: issue the copies of the warp's next stage into ring stage st_i.
  // The j-th batch of warp w is j * kWarps + ((w - j) mod kWarps): in round j
  // the block's warps take batches j * kWarps .. j * kWarps + kWarps - 1, a
  // warp's batches stay in ascending order, and a pattern that repeats every
  // few batches (a faulty column band) spreads over all warps.  The schedule
  // is fixed, so each lane's sums do not depend on timing.
  // The issue state is kept by every lane alike, from values broadcast from
  // lane 0 (so the copies' operands are warp-uniform), and one elected lane
  // issues the copies.
  const uint32_t warp_u = (uint32_t)__shfl_sync(0xffffffffu, warp, 0);
  const uint32_t nj = warp_batches(nb, (int)warp_u);
  const uint32_t ring_sa = (uint32_t)__shfl_sync(0xffffffffu, smem_addr(ring), 0);
  const uint32_t bars_sa = (uint32_t)__shfl_sync(0xffffffffu, smem_addr(bars), 0);
  const char *isrc_c = (const char *)__shfl_sync(0xffffffffu, (unsigned long long)src_c, 0);
  const char *isrc_r = (const char *)__shfl_sync(0xffffffffu, (unsigned long long)src_r, 0);
  const char *isrc_x = (const char *)__shfl_sync(0xffffffffu, (unsigned long long)src_x, 0);
  const bool stall = P->cd.test_stall != 0;
  uint32_t st_i = rp.stage, j_i = 0, h_i = 0, rot_i = warp_u;
  bool live = true;  // the end of the piece has not been marked yet
  auto issue_next = [&]() {  // the whole warp, converged
    if (j_i >= nj) {
      if (lane == 0) W->stage_b[st_i] = kNoBatch;
      live = false;
      return;
    }
    const uint32_t b = j_i * kWarps + rot_i;
    if (lane == 0) W->stage_b[st_i] = b;
    const uint32_t off = b * BB + h_i * HB;
    uint32_t bytes = 0;
    if (vec_ok && off < pbytes) bytes = pbytes - off >= HB ? HB : (pbytes - off) / (STEP * EB) * (STEP * EB);
    if (elect_one()) {
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      ring_issue_sa<NIN>(isrc_c, isrc_r, isrc_x, off, bytes, ring_sa + st_i * STAGE, bars_sa + st_i * 8u, stall);
    }
    st_i = st_i + 1 == NST ? 0 : st_i + 1;
    if (++h_i == NSB) {
      h_i = 0;
      ++j_i;
      rot_i = (rot_i + kWarps - 1) & (kWarps - 1);
    }
  };
  for (uint32_t i = 0; i < NST - 1 && live; ++i) issue_next();
  if (lane == 0) W->mism_tot = 0;
  __syncwarp();
  // The block's view of the case-wide maxima is read every batch; the case's
  // own value is read by one warp of the block per batch round (each warp
  // every kPoll batches, its load kPoll batches ahead of its use, so the L2
  // latency hides and the hot word sees few readers).
  uint64_t gAR = ld_relaxed64(g_thr);
  const uint32_t lane_off = (uint32_t)lane * V;
  int flush = 0;
  // warp-uniform: the warp's last batch was mostly mismatches (float types)
  bool dmode = false;
  // the batch's bins can be computed once when every batch lies in one row
  const bool bins_ok = __shfl_sync(0xffffffffu, P->cd.amode && P->cd.dN.d % (uint64_t)BATCH == 0 ? 1 : 0, 0) != 0;
  DenseBins B;
  B.ok = 0;
  const int32_t a_shift_u = __shfl_sync(0xffffffffu, P->cd.a_shift, 0);
  const bool prof_u = __shfl_sync(0xffffffffu, P->stats != nullptr ? 1 : 0, 0) != 0;
  const bool bins_smem = __shfl_sync(0xffffffffu, P->wr > 0 ? 1 : 0, 0) != 0;
  B.sh = a_shift_u;
  B.prof = prof_u;
  B.hr = __shfl_sync(0xffffffffu, P->cd.hi_r, 0);
  B.ha = __shfl_sync(0xffffffffu, P->cd.hi_a, 0);
  for (uint32_t j = 0;; ++j) {
    const uint32_t b = __shfl_sync(0xffffffffu, W->stage_b[rp.stage], 0);  // warp-uniform, and known so
    if (b == kNoBatch) break;
    const uint32_t erel = b * BATCH;  // element offset of the batch in the piece
    __syncwarp();
    if (lane == 0) {
      W->mism = 0;
      W->sbits = 0;
    }
    B.ok = 0;
    if (Tr<DT>::EB == 4 && !Tr<DT>::kInt && dmode && bins_ok) {
      // row, row bin and first tile of the batch (all lanes alike)
      const CaseDesc &cd = P->cd;
      const uint32_t s0 = (uint32_t)P->pbegin + erel;
      const uint32_t N = (uint32_t)cd.dN.d, th = (uint32_t)cd.dth.d, tw = (uint32_t)cd.dtw.d;
      const uint32_t row = div_q32(s0, N, cd.m32N);
      const uint32_t tr = div_q32(row, th, cd.m32th);
      const uint32_t tc = div_q32(s0 - row * N, tw, cd.m32tw);
      B.rp = (int32_t)(row - tr * th);
      if (bins_smem) {
        B.ok = 1;
        B.hbin = smem_addr(P->sh_hist + (((int64_t)tr - P->tr0) * P->wc + ((int64_t)tc - P->tc0)));
      } else {
        B.ok = 2;
        B.hbin = (uint32_t)((int64_t)tr * cd.GC + tc);
      }
      B.rp = __shfl_sync(0xffffffffu, B.rp, 0);
      B.hbin = __shfl_sync(0xffffffffu, B.hbin, 0);
      B.sh = a_shift_u;
      B.prof = prof_u;
      B.rowsum = 0;
      B.sbits = 0;
      B.lc0 = B.lc1 = B.lc2 = B.lc3 = 0;
      B.ht = 0;
    }
    if ((j + warp_u) % kPoll == 0) {
      if (lane == 0) {
        sh_max(&P->cta_thr[0], (uint32_t)gAR);
        sh_max(&P->cta_thr[1], (uint32_t)(gAR >> 32));
      }
      gAR = ld_relaxed64(g_thr);
    }
    {
      // lane 0's reading of the block's value, so the branch is uniform
      uint64_t v = 0;
      if (lane == 0) v = *(volatile const uint64_t *)P->cta_thr;
      v = __shfl_sync(0xffffffffu, v, 0);
      const float ga = pub_thr((uint32_t)v), gr = pub_thr((uint32_t)(v >> 32));
      if (ga > R.ga || gr > R.gr) {
        __syncwarp();
        if (lane == 0) {
          W->ga = fmaxf(W->ga, ga);
          W->gr = fmaxf(W->gr, gr);
          merge_thr(W->wA, W->wR, W->ga, W->gr, W->tA, W->tR);
        }
        __syncwarp();
        R.ga = W->ga;
        R.gr = W->gr;
        reload_thr(R, W);
      }
    }
#pragma unroll 1
    for (int h = 0; h < (int)NSB; ++h) {
      if (live) issue_next();  // refills the stage released before this one
      __syncwarp();
      const uint8_t *stage = ring + rp.stage * STAGE + lane * 16;
      const uint32_t ssa = ring_sa + rp.stage * STAGE + lane * 16;  // the same, as a shared address
      bool ok = mbar_try_wait_at(bars_sa + rp.stage * 8u, rp.phase);
      if (!__all_sync(0xffffffffu, ok)) ok = mbar_wait_slow(bars + rp.stage, rp.phase);
      if (!__all_sync(0xffffffffu, ok)) {
        // A stage's copies did not complete within the wait limit: report
        // (the data of this call is void), wait again, with the same limit,
        // for this warp's copies still in flight (this stage's and those of
        // the stage issued ahead of it), so none lands in shared memory after
        // the block has stopped, mark the warp's remaining batches empty,
        // and stop.
        if (lane == 0) atomicOr(err, 1u);
        mbar_wait_slow(bars + rp.stage, rp.phase);
        uint32_t nx = rp.stage, nph = rp.phase;
        for (uint32_t q = 1; q < NST; ++q) {  // the stages issued ahead, up to the piece's end mark
          if (++nx == NST) {
            nx = 0;
            nph ^= 1u;
          }
          if (W->stage_b[nx] == kNoBatch) break;
          mbar_wait_slow(bars + nx, nph);
        }
        if (lane == 0) {
          for (uint32_t jj = j; jj < nj; ++jj) bcount[jj * kWarps + (((uint32_t)warp + kWarps - jj % kWarps) % kWarps)] = 0;
        }
        __syncwarp();
        return true;
      }
      if (++rp.stage == NST) {
        rp.stage = 0;
        rp.phase ^= 1u;
      }
      const uint32_t hoff = b * BB + h * HB;
      const uint32_t hrel = erel + h * (HS * STEP);
      if (vec_ok && hoff < pbytes && pbytes - hoff >= HB) {
        if (Tr<DT>::EB == 4 && !Tr<DT>::kInt && dmode) {
#pragma unroll
          for (int u = 0; u < HS; ++u) {
            const uint4 cv = lds_v4_off(ssa, u * 512);
            const uint4 rv = lds_v4_off(ssa, HB + u * 512);
            uint4 xv = make_uint4(0, 0, 0, 0);
            if constexpr (NIN == 1) xv = lds_v4_off(ssa, 2 * HB + u * 512);
            if constexpr (Tr<DT>::EB == 4 && !Tr<DT>::kInt)
              step_dense<DT, NIN>(P, L, W, R, B, cv, rv, xv, hrel + u * STEP + lane_off, h * HS + u);
          }
        } else {
#pragma unroll 2
          for (int u = 0; u < HS; ++u) {
            const uint4 cv = lds_v4_off(ssa, u * 512);
            const uint4 rv = lds_v4_off(ssa, HB + u * 512);
            uint4 xv = make_uint4(0, 0, 0, 0);
            if constexpr (NIN == 1) xv = lds_v4_off(ssa, 2 * HB + u * 512);
            step<DT, NIN>(P, L, W, R, cv, rv, xv, hrel + u * STEP + lane_off);
          }
        }
      } else {
        // part of the case's last batch, or a case that is not 16-byte aligned
        const uint32_t pel = pbytes / EB;  // elements in the piece
        const uint32_t nfull = vec_ok && hrel < pel ? (pel - hrel) / STEP : 0u;
        for (int u = 0; u < HS; ++u) {
          const uint32_t e = hrel + u * STEP + lane_off;
          if ((uint32_t)u < nfull) {
            const uint4 cv = lds_v4(stage + u * 512);
            const uint4 rv = lds_v4(stage + HB + u * 512);
            uint4 xv = make_uint4(0, 0, 0, 0);
            if constexpr (NIN == 1) xv = lds_v4(stage + 2 * HB + u * 512);
            step<DT, NIN>(P, L, W, R, cv, rv, xv, e);
          } else if (hrel + u * STEP < pel) {
            const int n = e >= pel ? 0 : (pel - e > (uint32_t)V ? V : (int)(pel - e));
            R.sse = tail_step<DT, NIN>(P, L, W, P->pbegin + e, n, R.sse);
            reload_thr(R, W);
          }
        }
      }
      __syncwarp();  // every lane is done with the stage before it is refilled
    }
    if (B.ok && B.ht != 0) {  // one tile per step: lane u adds step u's count to its tile
      if (B.ok == 1) sh_add_at(B.hbin + 4u * (uint32_t)lane, B.ht);
      else gl_add(P->g_hist + (B.hbin + (uint32_t)lane), (unsigned long long)B.ht);
    }
    if (B.ok && (B.lc0 | B.lc1 | B.lc2 | B.lc3)) {
      // this lane's column counts of the batch's dense steps
      const uint32_t a = P->lcol_sa + (uint32_t)threadIdx.x * 16u;
      int x, y, z, w;
      asm volatile("ld.shared.v4.s32 {%0,%1,%2,%3}, [%4];" : "=r"(x), "=r"(y), "=r"(z), "=r"(w) : "r"(a));
      asm volatile("st.shared.v4.s32 [%0], {%1,%2,%3,%4};" ::"r"(a), "r"(x + B.lc0), "r"(y + B.lc1), "r"(z + B.lc2),
                   "r"(w + B.lc3));
    }
    if (B.ok && B.rowsum) {
      // the dense steps' row total and counts (all lanes hold them)
      if (lane == 0) {
        if (P->prof_smem) sh_add(&P->sh_row[B.rp], B.rowsum);
        else gl_add(&P->g_row[B.rp], (unsigned long long)B.rowsum);
        W->mism += B.rowsum;
        W->sbits |= B.sbits;
      }
      __syncwarp();
    }
    if (lane == 0) {
      bcount[b] = (int32_t)((uint32_t)W->mism | (W->sbits << kStepBitsShift));
      W->mism_tot += W->mism;
    }
    if constexpr (Tr<DT>::EB == 4 && !Tr<DT>::kInt) {
      // the next batch's regime (fp32): dense when at least half of this one
      // mismatched (16-bit types keep the plain loop: their scan is bound by
      // instruction issue on clean data, where every extra branch costs)
      __syncwarp();
      dmode = __shfl_sync(0xffffffffu, 2 * W->mism >= (int64_t)BATCH ? 1 : 0, 0) != 0;
    }
    if (R.track_c | R.track_r) {
      R.track_c = R.track_c && !__any_sync(0xffffffffu, (R.cacc & mag) != 0u);
      R.track_r = R.track_r && !__any_sync(0xffffffffu, (R.racc & mag) != 0u);
    }
    if (++flush == kFlushBatches) {
      sse_flush(R.sse);
      flush = 0;
    }
  }
  sse_flush(R.sse);
  return false;
}

// ------------------------------------------------------------ seeding
// Lower bounds of |d| and |d|/|r| of one element from its stored bits (fp32
// values rounded down from its fp64 error; nothing for a non-finite pair),
// folded into ma, mr.
template <int DT>
__device__ __forceinline__ void seed_bits(uint32_t cb, uint32_t rb, float &ma, float &mr) {
  float as, ar;
  if constexpr (Tr<DT>::kInt) {
    const long long d = (long long)(int32_t)cb - (long long)(int32_t)rb;
    as = __ll2float_rd(d < 0 ? -d : d);
    const long long r = (long long)(int32_t)rb;
    ar = __ll2float_ru(r < 0 ? -r : r);
  } else {
    const float c = to_f32<DT>(cb), r = to_f32<DT>(rb);
    if (!(isfinite(c) && isfinite(r))) return;
    as = __fsub_rd(fmaxf(c, r), fminf(c, r));  // <= |c - r|
    ar = fabsf(r);
  }
  ma = fmaxf(ma, as);
  if (ar > 0.f) mr = fmaxf(mr, quot_lb(as, ar));
}

template <int DT>
__device__ __forceinline__ void seed_elem(const CaseDesc &cd, int64_t i, float &ma, float &mr) {
  constexpr int EB = Tr<DT>::EB;
  seed_bits<DT>(ld_one<EB>(cd.cand, i), ld_one<EB>(cd.ref, i), ma, mr);
}

// The same for the V elements e .. e + V - 1 of one lane (e a multiple of
// V): one vector load per tensor when the case is 16-byte aligned.
template <int DT>
__device__ __forceinline__ void seed_step(const CaseDesc &cd, int64_t e, float &ma, float &mr) {
  constexpr int V = Tr<DT>::V;
  if (!cd.vec_ok) {
    for (int k = 0; k < V; ++k) seed_elem<DT>(cd, e + k, ma, mr);
    return;
  }
  const uint4 cv = ld_v4((const char *)cd.cand + e * Tr<DT>::EB);
  const uint4 rv = ld_v4((const char *)cd.ref + e * Tr<DT>::EB);
#pragma unroll
  for (int k = 0; k < V; ++k) seed_bits<DT>(vbits<DT>(cv, k), vbits<DT>(rv, k), ma, mr);
}

// ------------------------------------------------------------ the kernel
// Dynamic shared memory: the warps' rings (ring_bytes(NIN): stage data, then
// one mbarrier per stage), then int32 words: [0, 8) class counters
// (NaN/+Inf/-Inf of c, of r, non-finite pairs), [8, 16) unused, the row
// profile [th], the column profile [tw] and the histogram window.
constexpr int kShHead = 16;

template <int DT, int NIN>
__global__ void __launch_bounds__(kThreads, 2)
    scan_kernel(const CaseDesc *__restrict__ cases, const Piece *__restrict__ pieces,
                unsigned long long *piece_ctr, int64_t n_pieces, int64_t piece_base, Partial *partials,
                int32_t *batch_count, uint8_t *out, uint32_t *g_thr, unsigned long long *stats, uint32_t *err) {
  constexpr int EB = Tr<DT>::EB;
  constexpr int NST = ring_stages(NIN);
  constexpr int STAGE = ring_streams(NIN) * stage_bytes(NIN);
  // the finalize kernel, launched as this launch's programmatic dependent,
  // may be scheduled as blocks of this one finish (it waits for the whole
  // grid before it reads anything this kernel writes)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  extern __shared__ __align__(128) uint8_t dsm[];
  __shared__ PieceSh P;
  __shared__ LaneSh lanes[kThreads];
  __shared__ WarpSh warps[kWarps];
  __shared__ Partial red[kWarps];
  __shared__ int32_t sh_eq[NIN != 0 ? kThreads * NMV_MAX_INPUTS : 1];
  __shared__ __align__(8) uint32_t cta_thr[2];
  // each lane's column counters of an aligned case (record_step_aligned)
  __shared__ __align__(16) int32_t lcol[kThreads * Tr<DT>::V];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  LaneSh *L = &lanes[threadIdx.x];
  WarpSh *W = &warps[warp];
  uint8_t *ring = dsm + (size_t)warp * NST * STAGE;
  uint64_t *bars = (uint64_t *)(dsm + (size_t)kWarps * NST * STAGE) + warp * NST;
  int32_t *smem = (int32_t *)(dsm + ring_bytes(NIN));
  if (lane == 0) {
    for (int s = 0; s < NST; ++s) mbar_init(bars + s);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();
  RingPos rpos = {0u, 0u};
  bool tr_first = true;  // the block's first piece seeds the published maxima
  // Blocks take pieces from the launch's counter as they finish the last
  // one, so pieces of uneven cost (a region wrong everywhere next to a clean
  // one) balance over the blocks.  The next piece is claimed, and its
  // descriptor fetched, by the first warp of the block to finish its sweep
  // of the current one, behind the other warps' work.
  __shared__ int64_t sh_piece;
  __shared__ Piece sh_pc;
  __shared__ int32_t sh_case;    // case whose descriptor P holds (-1: none)
  __shared__ int32_t sh_done;    // warps done with the current sweep
  __shared__ int32_t sh_newcase;  // the current piece starts a case for this block
  __shared__ uint32_t sh_pat[2];  // the case's first stored words (replicated for 16-bit types)
  __shared__ int32_t sh_abort;    // a warp gave up waiting for its copies: the block stops
  if (threadIdx.x == 0) {
    const int64_t p0 = (int64_t)atomicAdd(piece_ctr, 1ull);
    sh_piece = p0;
    if (p0 < n_pieces) sh_pc = pieces[p0];
    sh_case = -1;
    sh_abort = 0;
  }
  for (;;) {
    __syncthreads();
    const int64_t p = sh_piece;
    if (p >= n_pieces || sh_abort) break;
    const Piece pc = sh_pc;
    const bool newcase = sh_case != pc.case_id;
    if (newcase) {
      // a new case: its descriptor, copied by the block in 8-byte words
      static_assert(sizeof(CaseDesc) % 8 == 0, "CaseDesc copy");
      const uint64_t *src = (const uint64_t *)&cases[pc.case_id];
      for (int w = threadIdx.x; w < (int)(sizeof(CaseDesc) / 8); w += kThreads) ((uint64_t *)&P.cd)[w] = src[w];
      __syncthreads();
      if (threadIdx.x == 0) {
        uint8_t *o = out + P.cd.out_off;
        P.g_hist = (unsigned long long *)(o + P.cd.hist_off);
        P.g_row = (unsigned long long *)(o + P.cd.rowp_off);
        P.g_col = (unsigned long long *)(o + P.cd.colp_off);
        P.g_thr = g_thr + 2 * pc.case_id;
        P.sh_cls = smem;
        P.sh_eq = sh_eq;
        P.lcol_sa = smem_addr(lcol);
        P.cta_thr = cta_thr;
        P.stats = stats;
        // the block's view starts from what the case has published so far
        const uint64_t g = ld_relaxed64(P.g_thr);
        cta_thr[0] = (uint32_t)g;
        cta_thr[1] = (uint32_t)(g >> 32);
        const uint32_t c0 = ld_one<EB>(P.cd.cand, 0), r0 = ld_one<EB>(P.cd.ref, 0);
        sh_pat[0] = EB == 2 ? (c0 | (c0 << 16)) : c0;
        sh_pat[1] = EB == 2 ? (r0 | (r0 << 16)) : r0;
        sh_case = pc.case_id;
      }
    }
    if (threadIdx.x == 0) {
      P.piece = p;
      sh_newcase = newcase ? 1 : 0;
      P.pbegin = pc.begin;
      P.tr0 = pc.tr0;
      P.tc0 = pc.tc0;
      P.wr = pc.wr;
      P.wc = pc.wc;
      P.prof_smem = pc.prof_smem;
      P.rel_ru = EB == 2 && !Tr<DT>::kInt;
      P.sh_row = smem + kShHead;
      P.sh_col = P.sh_row + (pc.prof_smem ? P.cd.th : 0);
      P.sh_hist = P.sh_col + (pc.prof_smem ? P.cd.tw : 0);
      sh_done = 0;
    }
    __syncthreads();
    if (tr_first) {
      // A sample of the case seeds the published maxima, so warps start near
      // the final thresholds instead of establishing them one light step at
      // a time: each warp of every block reads one warp step (32 vectors,
      // coalesced) at its own place, spread over the whole case.  Every
      // value is a lower bound of an actual element's error, published like
      // the scan's own (lanes -> the block's view -> once to the case).
      constexpr int V = Tr<DT>::V;
      const int64_t nsteps = P.cd.numel / (32 * V);
      const int64_t slots = (int64_t)gridDim.x * kWarps;
      if (nsteps > 0) {
        const int64_t slot = (int64_t)blockIdx.x * kWarps + warp;
        const int64_t st = nsteps > slots ? (nsteps / slots) * slot : slot % nsteps;
        float ma = -1.f, mr = -1.f;
        seed_step<DT>(P.cd, st * (32 * V) + lane * V, ma, mr);
        ma = warp_reduce(ma, [](float x, float y) { return fmaxf(x, y); });
        mr = warp_reduce(mr, [](float x, float y) { return fmaxf(x, y); });
        if (lane == 0) {
          if (ma > 0.f) atomicMax(&cta_thr[0], __float_as_uint(ma));
          if (mr > 0.f) atomicMax(&cta_thr[1], __float_as_uint(mr));
        }
      }
    }
    const int64_t used = (int64_t)(P.sh_hist - smem) + (int64_t)pc.wr * pc.wc;
    for (int64_t t = threadIdx.x; t < used; t += kThreads) smem[t] = 0;
    L->a_i = L->r_i = INT64_MAX;
    L->a_v = L->r_v = 0.0;
    L->a_f = L->r_n = 0.f;
    L->r_d = 1.f;
    L->a_x = L->r_x = 1;
    L->r_lo = -1.f;
    L->cacc = 0;
    L->racc = 0;
    if (P.cd.amode) {
#pragma unroll
      for (int k = 0; k < Tr<DT>::V; ++k) lcol[threadIdx.x * Tr<DT>::V + k] = 0;
    }
    if constexpr (NIN != 0) {
      for (int j = 0; j < NMV_MAX_INPUTS; ++j) sh_eq[threadIdx.x * NMV_MAX_INPUTS + j] = 0;
    }
    if (lane == 0) {
      // A block takes the pieces of a case in ascending order, so the
      // warp's own thresholds from its earlier pieces of the case bound
      // maxima held at lower indices and carry over; a new case starts
      // from nothing.
      if (sh_newcase) W->wA = W->wR = -1.f;
      W->cA = W->wA;
      W->cR = W->wR;
      W->ga = W->gr = -1.f;
      merge_thr(W->wA, W->wR, W->ga, W->gr, W->tA, W->tR);
      W->pubA = W->pubR = 0;
      W->mism = 0;
      for (int k = 0; k < 9; ++k) W->st[k] = 0;
    }
    __syncthreads();
    if (tr_first) {
      if (threadIdx.x == 0) {
        if (cta_thr[0] != 0u) atomicMax(&P.g_thr[0], cta_thr[0]);
        if (cta_thr[1] != 0u) atomicMax(&P.g_thr[1], cta_thr[1]);
      }
      tr_first = false;
    }

    Regs<NIN> R;
    R.sse.hi = R.sse.lo = make_float2(0.f, 0.f);
    R.sse.acc = 0.0;
    R.cacc = R.racc = 0;
#pragma unroll
    for (int j = 0; j < (NIN > 0 ? NIN : 1); ++j) R.eq[j] = 0;
    R.cpat = sh_pat[0];
    R.rpat = sh_pat[1];
    R.ga = R.gr = -1.f;
    reload_thr(R, W);
    R.lo_r = P.cd.lo_r;
    R.lo_a = P.cd.lo_a;
    R.track_c = R.track_r = true;
    if (sweep<DT, NIN>(&P, L, W, R, pc, batch_count, ring, bars, rpos, err) && lane == 0) sh_abort = 1;
    if (P.cd.amode) {
      // this lane's column counters into the column profile
      constexpr int V = Tr<DT>::V;
      const int cp0 = (lane & ((1 << P.cd.a_shift) - 1)) * V;
#pragma unroll
      for (int k = 0; k < V; ++k) {
        const int v = lcol[threadIdx.x * V + k];
        if (v) {
          if (P.prof_smem) sh_add(&P.sh_col[cp0 + k], v);
          else gl_add(&P.g_col[cp0 + k], (unsigned long long)v);
        }
      }
    }
    __syncwarp();
    if (lane == 0 && atomicAdd(&sh_done, 1) == 0) {
      // the first warp done claims the block's next piece
      const int64_t nx = (int64_t)atomicAdd(piece_ctr, 1ull);
      sh_piece = nx;
      if (nx < n_pieces) sh_pc = pieces[nx];
    }
    if (stats && lane == 0)
      for (int k = 0; k < 9; ++k)
        if (W->st[k]) atomicAdd(&stats[k], W->st[k]);

    // ---- lanes -> warps -> the piece's partial
    const Best a = best_warp(abs_best64(L)), r = rel_best_warp(L);
    const double sse = warp_reduce(R.sse.acc, [](double x, double y) { return __dadd_rn(x, y); });
    const uint32_t cacc = warp_reduce(R.cacc | L->cacc, [](uint32_t x, uint32_t y) { return x | y; });
    const uint32_t racc = warp_reduce(R.racc | L->racc, [](uint32_t x, uint32_t y) { return x | y; });
    int eqs[NMV_MAX_INPUTS];
#pragma unroll
    for (int j = 0; j < NMV_MAX_INPUTS; ++j) {
      eqs[j] = 0;
      if constexpr (NIN != 0) {
        int v = sh_eq[threadIdx.x * NMV_MAX_INPUTS + j];
        if constexpr (NIN > 0) {
          if (j < NIN) v += R.eq[j < NIN ? j : 0];
        }
        eqs[j] = warp_reduce(v, [](int x, int y) { return x + y; });
      }
    }
    if (lane == 0) {
      Partial &w = red[warp];
      w.cnt[0] = W->mism_tot;
      w.best_abs = a.v;
      w.arg_abs = a.i;
      w.best_rel = r.v;
      w.arg_rel = r.i;
      w.sse = sse;
      w.cacc = cacc;
      w.racc = racc;
#pragma unroll
      for (int j = 0; j < NMV_MAX_INPUTS; ++j) w.eq[j] = eqs[j];
    }
    __syncthreads();
    if (warp != 0) {
      // warps 1.. flush the localisation maps to the case's arrays
      const int tid = threadIdx.x - 32, nt = kThreads - 32;
      if (P.wr > 0) {
        for (int64_t t = tid; t < (int64_t)P.wr * P.wc; t += nt) {
          const int v = P.sh_hist[t];
          if (v) {
            const int64_t tr = P.tr0 + t / P.wc, tc = P.tc0 + t % P.wc;
            gl_add(&P.g_hist[tr * P.cd.GC + tc], (unsigned long long)v);
          }
        }
      }
      if (P.prof_smem) {
        for (int64_t t = tid; t < P.cd.th; t += nt)
          if (P.sh_row[t]) gl_add(&P.g_row[t], (unsigned long long)P.sh_row[t]);
        for (int64_t t = tid; t < P.cd.tw; t += nt)
          if (P.sh_col[t]) gl_add(&P.g_col[t], (unsigned long long)P.sh_col[t]);
      }
    } else {
      // warp 0 combines the warps' parts: lanes 0..kWarps-1 hold one each,
      // then a fixed tree (the same on every run)
      int64_t m = 0;
      Best ba = {-1.0, INT64_MAX}, br = {-1.0, INT64_MAX};
      double s = 0.0;
      uint32_t ca = 0, ra = 0;
      int64_t eq[NMV_MAX_INPUTS];
#pragma unroll
      for (int j = 0; j < NMV_MAX_INPUTS; ++j) eq[j] = 0;
      if (lane < kWarps) {
        const Partial &w = red[lane];
        m = w.cnt[0];
        ba = {w.best_abs, w.arg_abs};
        br = {w.best_rel, w.arg_rel};
        s = w.sse;
        ca = w.cacc;
        ra = w.racc;
        if constexpr (NIN != 0) {
#pragma unroll
          for (int j = 0; j < NMV_MAX_INPUTS; ++j) eq[j] = w.eq[j];
        }
      }
      static_assert(kWarps == 8, "three rounds");
#pragma unroll
      for (int o = kWarps / 2; o; o >>= 1) {
        m += __shfl_xor_sync(0xffffffffu, m, o);
        best_offer(ba, __shfl_xor_sync(0xffffffffu, ba.v, o), __shfl_xor_sync(0xffffffffu, ba.i, o));
        best_offer(br, __shfl_xor_sync(0xffffffffu, br.v, o), __shfl_xor_sync(0xffffffffu, br.i, o));
        // lanes below the partner add the partner's value second, lanes
        // above first, so both hold the same bits
        const double s2 = __shfl_xor_sync(0xffffffffu, s, o);
        s = (lane & o) ? __dadd_rn(s2, s) : __dadd_rn(s, s2);
        ca |= __shfl_xor_sync(0xffffffffu, ca, o);
        ra |= __shfl_xor_sync(0xffffffffu, ra, o);
        if constexpr (NIN != 0) {
#pragma unroll
          for (int j = 0; j < NMV_MAX_INPUTS; ++j) eq[j] += __shfl_xor_sync(0xffffffffu, eq[j], o);
        }
      }
      if (lane == 0) {
        Partial Q;
        Q.cnt[0] = m;
        for (int k = 1; k < 8; ++k) Q.cnt[k] = smem[k - 1];
        Q.best_abs = ba.v;
        Q.arg_abs = ba.i;
        Q.best_rel = br.v;
        Q.arg_rel = br.i;
        Q.sse = s;
        Q.cacc = ca;
        Q.racc = ra;
        for (int j = 0; j < NMV_MAX_INPUTS; ++j) Q.eq[j] = eq[j];
        partials[piece_base + P.piece] = Q;
      }
    }
  }
  // A later launch of a batch call (another element type) may run as this
  // grid's programmatic dependent, overlapping its drain; each grid then
  // ends only after the one before it, so the finalize kernel, which waits
  // for the last, sees all of them (a no-op for a grid launched normally).
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

// Launch helpers of one element type (defined in nmv_scan_<dtype>.cu).  The
// `smem` they take is the localisation part of the dynamic shared memory;
// they add the rings (ring_bytes).
template <int DT>
struct ScanOps {
  static cudaError_t prepare(int nin, size_t smem);
  static int occupancy(int nin, size_t smem);
  static cudaError_t launch(int nin, int grid, size_t smem, cudaStream_t st, bool pdl, const CaseDesc *cases,
                            const Piece *pieces, unsigned long long *piece_ctr, int64_t n_pieces, int64_t piece_base,
                            Partial *partials, int32_t *batch_count, uint8_t *out, uint32_t *g_thr,
                            unsigned long long *stats, uint32_t *err);
};

#define NMV_SCAN_FN(DT, NIN) scan_kernel<DT, NIN>
#define NMV_SCAN_SMEM(NIN, smem) ((int)((smem) + ring_bytes(NIN)))
#define NMV_DEFINE_SCAN_OPS(DT)                                                                          \
  template <>                                                                                            \
  cudaError_t ScanOps<DT>::prepare(int nin, size_t smem) {                                               \
    const cudaFuncAttribute A = cudaFuncAttributeMaxDynamicSharedMemorySize;                             \
    if (nin == 0) return cudaFuncSetAttribute(NMV_SCAN_FN(DT, 0), A, NMV_SCAN_SMEM(0, smem));            \
    if (nin == 1) return cudaFuncSetAttribute(NMV_SCAN_FN(DT, 1), A, NMV_SCAN_SMEM(1, smem));            \
    return cudaFuncSetAttribute(NMV_SCAN_FN(DT, -1), A, NMV_SCAN_SMEM(-1, smem));                        \
  }                                                                                                      \
  template <>                                                                                            \
  int ScanOps<DT>::occupancy(int nin, size_t smem) {                                                     \
    int n = 0;                                                                                           \
    cudaError_t e;                                                                                       \
    if (nin == 0)                                                                                        \
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, NMV_SCAN_FN(DT, 0), kThreads, NMV_SCAN_SMEM(0, smem)); \
    else if (nin == 1)                                                                                   \
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, NMV_SCAN_FN(DT, 1), kThreads, NMV_SCAN_SMEM(1, smem)); \
    else                                                                                                 \
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, NMV_SCAN_FN(DT, -1), kThreads, NMV_SCAN_SMEM(-1, smem)); \
    return e == cudaSuccess ? n : 0;                                                                     \
  }                                                                                                      \
  template <>                                                                                            \
  cudaError_t ScanOps<DT>::launch(int nin, int grid, size_t smem, cudaStream_t st, bool pdl,             \
                                  const CaseDesc *cases, const Piece *pieces, unsigned long long *piece_ctr, \
                                  int64_t n_pieces, int64_t piece_base, Partial *partials,                \
                                  int32_t *batch_count, uint8_t *out, uint32_t *g_thr,                    \
                                  unsigned long long *stats, uint32_t *err) {                            \
    cudaLaunchConfig_t cfg = {};                                                                         \
    cfg.gridDim = dim3(grid);                                                                            \
    cfg.blockDim = dim3(kThreads);                                                                       \
    cfg.stream = st;                                                                                     \
    cudaLaunchAttribute attr[1];                                                                         \
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;                                     \
    attr[0].val.programmaticStreamSerializationAllowed = 1;                                              \
    cfg.attrs = attr;                                                                                    \
    cfg.numAttrs = pdl ? 1 : 0;                                                                          \
    cudaError_t e;                                                                                       \
    if (nin == 0) {                                                                                      \
      cfg.dynamicSmemBytes = NMV_SCAN_SMEM(0, smem);                                                     \
      e = cudaLaunchKernelEx(&cfg, NMV_SCAN_FN(DT, 0), cases, pieces, piece_ctr, n_pieces, piece_base,   \
                             partials, batch_count, out, g_thr, stats, err);                             \
    } else if (nin == 1) {                                                                               \
      cfg.dynamicSmemBytes = NMV_SCAN_SMEM(1, smem);                                                     \
      e = cudaLaunchKernelEx(&cfg, NMV_SCAN_FN(DT, 1), cases, pieces, piece_ctr, n_pieces, piece_base,   \
                             partials, batch_count, out, g_thr, stats, err);                             \
    } else {                                                                                             \
      cfg.dynamicSmemBytes = NMV_SCAN_SMEM(-1, smem);                                                    \
      e = cudaLaunchKernelEx(&cfg, NMV_SCAN_FN(DT, -1), cases, pieces, piece_ctr, n_pieces, piece_base,  \
                             partials, batch_count, out, g_thr, stats, err);                             \
    }                                                                                                    \
    if (e != cudaSuccess) return e;                                                                      \
    return cudaGetLastError();                                                                           \
  }

}  // namespace nmv
