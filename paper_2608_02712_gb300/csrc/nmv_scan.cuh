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
//  * max |d|/|r|: tR lies below the best relative error held, so the element
//    provably is no new maximum (strictly below a maximum published by any
//    warp of the case, or not above one held earlier in this warp's
//    ascending sweep, whose index is lower).
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
// elements of each vector) with Knuth's TwoSum, flushed to fp64 every few
// batches; the exact step feeds the same pairs with the same arithmetic
// (plus 2 s e for an inexact c - r, e from TwoSum), so the result is
// bit-identical whichever path an element takes.  Terms with |s| > 2^56 are
// squared in fp64.  When max |d| < 2^-38 the fp32 squares may lose tiny
// terms; the host then recomputes that case's SSE in fp64 (sse64 kernels).
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "nmv_internal.h"

namespace nmv {

constexpr int kFlushBatches = 8;
constexpr float kHuge = 0x1p56f;
constexpr float kMarginLo = 1.0f - 0x1p-20f;

// ------------------------------------------------------------------ utils
__device__ __forceinline__ uint64_t div_q(uint64_t n, uint64_t d, uint64_t m) {
  uint64_t q = __umul64hi(n, m);
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

__device__ __forceinline__ uint32_t ld_relaxed(const uint32_t *p) {
  uint32_t v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}

__device__ __forceinline__ float min3f(float a, float b, float c) {
  float r;
  asm("min.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
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
__device__ __forceinline__ bool pass64(double c, double r, double rtol, double atol) {
  if (c == r) return true;
  if (!(isfinite(c) && isfinite(r))) return false;
  const double err = fabs(__dsub_rn(c, r));
  const double allowed = __dadd_rn(atol, __dmul_rn(rtol, fabs(r)));
  return err <= allowed;
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
  a.lo = __fadd2_rn(a.lo, __fadd2_rn(err, q));
  a.hi = t;
}

__device__ __forceinline__ void sse_flush(SseAcc &a) {
  // TwoSum of the two slots' high parts, then two fp64 additions.
  const float h = __fadd_rn(a.hi.x, a.hi.y);
  const float hb = __fsub_rn(h, a.hi.x);
  const float herr = __fadd_rn(__fsub_rn(a.hi.x, __fsub_rn(h, hb)), __fsub_rn(a.hi.y, hb));
  const float l = __fadd_rn(__fadd_rn(a.lo.x, a.lo.y), herr);
  a.acc = __dadd_rn(a.acc, __dadd_rn((double)h, (double)l));
  a.hi = make_float2(0.f, 0.f);
  a.lo = make_float2(0.f, 0.f);
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

// ----------------------------------------------------------------- state
// Piece-constant data, in shared memory.
struct PieceSh {
  CaseDesc cd;
  int64_t tr0, tc0;
  int32_t wr, wc, prof_smem, pad;
  int32_t *sh_cls, *sh_row, *sh_col, *sh_hist;
  unsigned long long *g_hist, *g_row, *g_col;
  uint32_t *g_thr;
  unsigned long long *stats;  // [exact steps, exact abs, exact rel, exact predicate, light steps,
                              //  SM cycles in exact steps, SM cycles in light steps]
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
  int32_t eq[NMV_MAX_INPUTS];
};

// Warp-uniform state of a batch sweep, in shared memory.
struct WarpSh {
  float tA, tR;       // thresholds in force
  float wA, wR;       // the warp's own part of them (-1: no maximum held yet)
  float ga, gr;       // the case-wide part at the last merge (-1: none)
  uint32_t pubA, pubR;
  int64_t mism;       // mismatches so far in this batch
};

__device__ __forceinline__ float pub_thr(uint32_t bits) {
  const float f = __uint_as_float(bits);
  return f > 0.f ? __fmul_rz(f, kMarginLo) : -1.f;
}

__device__ __forceinline__ void merge_thr(float wA, float wR, float ga, float gr, float &tA, float &tR) {
  tA = fminf(fmaxf(wA, ga), kHuge);
  tR = fmaxf(wR, gr);
}

// fl32 round-down lower bounds of a lane's maxima (-1 when none held).
__device__ __forceinline__ float abs_lb(const LaneSh *L) {
  if (L->a_i == INT64_MAX) return -1.f;
  return L->a_x ? L->a_f : __double2float_rd(L->a_v);
}

__device__ __forceinline__ float rel_lb(const LaneSh *L) {
  if (L->r_i == INT64_MAX) return -1.f;
  return L->r_x ? __fdiv_rd(L->r_n, L->r_d) : __double2float_rd(L->r_v);
}

// The lane's maxima as fp64 (for the reduction at the end of a piece).
__device__ __forceinline__ Best abs_best64(const LaneSh *L) {
  if (L->a_i == INT64_MAX) return {-1.0, INT64_MAX};
  return {L->a_x ? (double)L->a_f : L->a_v, L->a_i};
}

__device__ __forceinline__ Best rel_best64(const LaneSh *L) {
  if (L->r_i == INT64_MAX) return {-1.0, INT64_MAX};
  return {L->r_x ? __ddiv_rn((double)L->r_n, (double)L->r_d) : L->r_v, L->r_i};
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
        L->r_lo = __fmul_rz(__fdiv_rd(as, ar), kMarginLo);
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

// fl32(|s| / |r|) for |r| != 0, within 2^-23 of the quotient: a fast
// reciprocal in the normal range, an IEEE division otherwise.
__device__ __forceinline__ float rel32(float as, float ar) {
  if (ar > 0x1p-125f && ar < 0x1p125f) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(ar));
    return __fmul_rn(as, r);
  }
  return __fdiv_rn(as, ar);
}

// ------------------------------------------------------------- slow path
// Localisation maps and the batch's mismatch count for one step: bit k of
// `mask` is element idx0 + k of this lane.  Row, column and tile
// coordinates are found once per lane and then advanced element by element.
__device__ __forceinline__ void record_step(const PieceSh *P, WarpSh *W, uint32_t mask, int64_t idx0) {
  const int lane = threadIdx.x & 31;
  const int total = __reduce_add_sync(0xffffffffu, (unsigned)__popc(mask));
  if (total == 0) return;
  const int64_t mism0 = W->mism;
  __syncwarp();
  if (lane == 0) W->mism = mism0 + total;
  if (mask == 0) return;
  const CaseDesc &cd = P->cd;
  const uint64_t N = cd.dN.d, th = cd.dth.d, tw = cd.dtw.d;
  uint64_t row = div_q((uint64_t)idx0, N, cd.dN.m);
  uint64_t col = (uint64_t)idx0 - row * N;
  uint64_t tr = div_q(row, th, cd.dth.m);
  uint64_t rp = row - tr * th;
  uint64_t tc = div_q(col, tw, cd.dtw.m);
  uint64_t cp = col - tc * tw;
  uint32_t m = mask;
  int kprev = 0;
  int64_t hbin = -1, rbin = -1;
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
    if (hb != hbin) {
      if (hcnt) {
        if (P->wr > 0) atomicAdd(&P->sh_hist[hbin], hcnt);
        else atomicAdd(&P->g_hist[hbin], (unsigned long long)hcnt);
      }
      hbin = hb;
      hcnt = 0;
    }
    ++hcnt;
    if ((int64_t)rp != rbin) {
      if (rcnt) {
        if (P->prof_smem) atomicAdd(&P->sh_row[rbin], rcnt);
        else atomicAdd(&P->g_row[rbin], (unsigned long long)rcnt);
      }
      rbin = (int64_t)rp;
      rcnt = 0;
    }
    ++rcnt;
    if (P->prof_smem) atomicAdd(&P->sh_col[cp], 1);
    else atomicAdd(&P->g_col[cp], 1ull);
  }
  if (P->wr > 0) atomicAdd(&P->sh_hist[hbin], hcnt);
  else atomicAdd(&P->g_hist[hbin], (unsigned long long)hcnt);
  if (P->prof_smem) atomicAdd(&P->sh_row[rbin], rcnt);
  else atomicAdd(&P->g_row[rbin], (unsigned long long)rcnt);
}

// After a step in which some lane's maximum changed: the warp's own
// thresholds from the lanes' maxima (fp32 lower bounds, so no fp64 is
// needed), publication of improvements to the case, the merged thresholds.
//   abs: the largest fp32 strictly below fl_rd(max), or 0 when max == 0
//        (elements not above it are not larger than a maximum at a lower
//        index of this warp);
//   rel: fl_rd(max) (1 - 2^-20) rounded toward zero.
__device__ __forceinline__ void refresh(const PieceSh *P, const LaneSh *L, WarpSh *W) {
  const int lane = threadIdx.x & 31;
  const float fa = warp_reduce(abs_lb(L), [](float x, float y) { return fmaxf(x, y); });
  const float fr = warp_reduce(rel_lb(L), [](float x, float y) { return fmaxf(x, y); });
  __syncwarp();
  if (lane == 0) {
    W->wA = fa < 0.f ? -1.f : (fa > 0.f ? __uint_as_float(__float_as_uint(fa) - 1u) : 0.f);
    W->wR = fr < 0.f ? -1.f : __fmul_rz(fr, kMarginLo);
    if (fa > 0.f && __float_as_uint(fa) > W->pubA) {
      atomicMax(&P->g_thr[0], __float_as_uint(fa));
      W->pubA = __float_as_uint(fa);
    }
    if (fr > 0.f && __float_as_uint(fr) > W->pubR) {
      atomicMax(&P->g_thr[1], __float_as_uint(fr));
      W->pubR = __float_as_uint(fr);
    }
    merge_thr(W->wA, W->wR, W->ga, W->gr, W->tA, W->tR);
  }
  __syncwarp();
}

__device__ __forceinline__ void count_stats(const PieceSh *P, int slot, long long t0, unsigned n_abs,
                                            unsigned n_rel, unsigned n_pred) {
  n_abs = __reduce_add_sync(0xffffffffu, n_abs);
  n_rel = __reduce_add_sync(0xffffffffu, n_rel);
  n_pred = __reduce_add_sync(0xffffffffu, n_pred);
  if ((threadIdx.x & 31) == 0) {
    atomicAdd(&P->stats[slot == 0 ? 0 : 4], 1ull);
    atomicAdd(&P->stats[slot == 0 ? 5 : 6], (unsigned long long)(clock64() - t0));
    atomicAdd(&P->stats[1], (unsigned long long)n_abs);
    atomicAdd(&P->stats[2], (unsigned long long)n_rel);
    atomicAdd(&P->stats[3], (unsigned long long)n_pred);
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
#pragma unroll
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
      if (!cfin) atomicAdd(&P->sh_cls[isnan(cf) ? 0 : (cf > 0.f ? 1 : 2)], 1);
      if (!rfin) atomicAdd(&P->sh_cls[isnan(rf) ? 3 : (rf > 0.f ? 4 : 5)], 1);
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
      if (!(as <= tA)) {
        candA |= 1u << k;
        mA = fmaxf(mA, as);
      }
      if (ar != 0.f && !(as <= __fmul_rz(tR, ar))) {
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
      atomicAdd(&P->sh_cls[6], 1);
    }
  }
  // Exact evaluation of the screened candidates.  abs: values below the
  // fp32 predecessor of the step's largest |s| are strictly smaller than it.
  // rel: fl32(|s| / |r|) is within 2^-22 of the quotient, so values below
  // (1 - 2^-20) of the largest are strictly smaller.
  bool changed = false;
  if (candA | candR) {
    const float fA = mA > 0.f ? __uint_as_float(__float_as_uint(mA) - 1u) : mA;
    const float fR = __fmul_rz(mR, kMarginLo);
#pragma unroll
    for (int k = 0; k < V; ++k) {
      const bool ca = ((candA >> k) & 1u) && fabsf(s[k]) >= fA;
      const bool cr = ((candR >> k) & 1u) && rel[k] >= fR;
      if (!(ca || cr)) continue;
      const int64_t idx = idx0 + k;
      const float as = fabsf(s[k]);
      const uint32_t rb = vbits<DT>(rv, k);
      const float ar = fabsf(to_f32<DT>(rb));
      bool exact = e[k] == 0.f;
      if constexpr (Tr<DT>::kInt) exact = exact && as < 0x1p24f && ar < 0x1p24f;
      // fl64(|c - r|) from the widened values when c - r is not exact in
      // fp32 (this also covers an fp32 overflow of c - r).
      double a64 = 0.0;
      if (!exact) {
        ++n_abs;
        a64 = fabs(__dsub_rn(to_f64<DT>(vbits<DT>(cv, k)), to_f64<DT>(rb)));
      }
      if (ca) changed |= offer_abs(L, as, exact, a64, idx);
      if (cr) changed |= offer_rel(L, as, ar, exact, a64, fabs(to_f64<DT>(rb)), rel[k], idx, n_rel);
    }
  }
  if (__any_sync(0xffffffffu, mask != 0)) record_step(P, W, mask, idx0);
  if (__any_sync(0xffffffffu, changed)) refresh(P, L, W);
  if (P->stats) count_stats(P, 0, t_start, n_abs, n_rel, n_pred);
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
#pragma unroll
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
    const float fA = mA > 0.f ? __uint_as_float(__float_as_uint(mA) - 1u) : mA;
    const float fR = __fmul_rz(mR, kMarginLo);
#pragma unroll
    for (int k = 0; k < V; ++k) {
      const float as = fabsf(s[k]);
      const bool ca = ((candA >> k) & 1u) && as >= fA;
      const bool cr = ((candR >> k) & 1u) && rel[k] >= fR;
      const int64_t idx = idx0 + k;
      if (ca) changed |= offer_abs(L, as, true, 0.0, idx);
      if (cr) {
        const uint32_t rb = vbits<DT>(rv, k);
        const float ar = fabsf(to_f32<DT>(rb));
        const bool exact = !Tr<DT>::kInt || ar < 0x1p24f;
        changed |= offer_rel(L, as, ar, exact, (double)as, fabs(to_f64<DT>(rb)), rel[k], idx, n_rel);
      }
    }
  }
  if constexpr (!Tr<DT>::kInt) {
#pragma unroll
    for (int k = 0; k < V; k += 2) ff_pair<Tr<DT>::EB == 4>(sse, make_float2(s[k], s[k + 1]));
  }
  if (__any_sync(0xffffffffu, changed)) refresh(P, L, W);
  if (P->stats) count_stats(P, 1, t_start, 0, n_rel, 0);
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
        L->eq[j] += (cb == xb) & (rb != xb);
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
    L->eq[j] += add;
  }
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
};

template <int NIN>
__device__ __forceinline__ void reload_thr(Regs<NIN> &R, const WarpSh *W) {
  R.tA = W->tA;
  R.tR = W->tR;
  R.tRq = fminf(R.tR, 0.25f);
}

template <int DT, int NIN>
__device__ __forceinline__ void step(const PieceSh *P, LaneSh *L, WarpSh *W, Regs<NIN> &R, const uint4 &cv,
                                     const uint4 &rv, const uint4 *xv, int64_t e) {
  constexpr int V = Tr<DT>::V;
  R.cacc |= (cv.x ^ R.cpat) | (cv.y ^ R.cpat) | (cv.z ^ R.cpat) | (cv.w ^ R.cpat);
  R.racc |= (rv.x ^ R.rpat) | (rv.y ^ R.rpat) | (rv.z ^ R.rpat) | (rv.w ^ R.rpat);
  if constexpr (NIN > 0) {
#pragma unroll
    for (int j = 0; j < NIN; ++j) {
#pragma unroll
      for (int k = 0; k < V; ++k) {
        const uint32_t xb = vbits<DT>(xv[j], k);
        R.eq[j] += (vbits<DT>(cv, k) == xb) & (vbits<DT>(rv, k) != xb);
      }
    }
  } else if constexpr (NIN < 0) {
    eq_generic<DT>(P, L, cv, rv, e);
  }
  bool hard, other;
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
#pragma unroll
    for (int k = 0; k < V; ++k) {
      const float cf = vdec<DT>(cv, k), rf = vdec<DT>(rv, k);
      s[k] = __fsub_rn(cf, rf);
      const float a = __fmaf_rz(R.lo_r, fabsf(rf), R.lo_a);
      const float b = __fmul_rz(R.tRq, fabsf(rf));
      hard |= !(fabsf(s[k]) <= min3f(a, b, R.tA));
    }
    if (!__any_sync(0xffffffffu, hard)) {
#pragma unroll
      for (int k = 0; k < V; k += 2) ff_pair<Tr<DT>::EB == 4>(R.sse, make_float2(s[k], s[k + 1]));
      return;
    }
    // Which steps need the exact path (a mismatch, a non-finite value, an
    // inexact c - r, an undecided predicate) and which only a maximum update
    // (the finite cap keeps infinities out of the light path).
    other = false;
#pragma unroll
    for (int k = 0; k < V; ++k) {
      const float rf = vdec<DT>(rv, k);
      const float a = __fmaf_rz(R.lo_r, fabsf(rf), R.lo_a);
      other |= !(fabsf(s[k]) <= min3f(a, __fmul_rz(0.25f, fabsf(rf)), kHuge));
    }
  }
  if (__any_sync(0xffffffffu, other)) R.sse = slow_step<DT>(P, L, W, cv, rv, e, V, R.sse);
  else R.sse = light_step<DT>(P, L, W, cv, rv, e, R.sse);
  reload_thr(R, W);
}

// Sweep this warp's batches of a piece (each batch_elems elements; the last
// one may be shorter), writing each batch's mismatch count.  In round r the
// block's warps take batches r*kWarps .. r*kWarps + kWarps - 1, warp w the
// one at offset (w - r) mod kWarps: a warp's batches stay in ascending order,
// and a pattern that repeats every few batches (a faulty column band, say)
// spreads over all warps instead of landing on the same ones.
template <int DT, int NIN>
__device__ __forceinline__ void sweep(const PieceSh *P, LaneSh *L, WarpSh *W, Regs<NIN> &R, const Piece &pc,
                                      int32_t *batch_count) {
  constexpr int V = Tr<DT>::V;
  constexpr int EB = Tr<DT>::EB;
  constexpr int STEP = 32 * V;
  constexpr int BATCH = STEP * kUnroll;
  constexpr int NX = NIN > 0 ? NIN : 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const CaseDesc &cd = P->cd;
  const char *cp = (const char *)cd.cand;
  const char *rp = (const char *)cd.ref;
  const char *xp[NX];
#pragma unroll
  for (int j = 0; j < NX; ++j) xp[j] = (const char *)cd.in_ptr[j];
  const uint32_t *g_thr = P->g_thr;
  const bool vec_ok = cd.vec_ok != 0;
  const int64_t nb = (pc.end - pc.begin + BATCH - 1) / BATCH;
  int flush = 0;
  for (int64_t r = 0; r * kWarps < nb; ++r) {
    const int64_t b = r * kWarps + ((warp - r) % kWarps + kWarps) % kWarps;
    if (b >= nb) continue;
    const int64_t lo = pc.begin + b * BATCH;
    const int64_t hi = lo + BATCH < pc.end ? lo + BATCH : pc.end;
    const uint32_t gA = ld_relaxed(&g_thr[0]);
    const uint32_t gR = ld_relaxed(&g_thr[1]);
    if (lane == 0) W->mism = 0;
    {
      // Case-wide maxima published since the last batch: lane 0's reading,
      // compared with the warp's register copy, so the branch is uniform.
      const float ga = __shfl_sync(0xffffffffu, pub_thr(gA), 0);
      const float gr = __shfl_sync(0xffffffffu, pub_thr(gR), 0);
      if (__any_sync(0xffffffffu, ga > R.ga || gr > R.gr)) {
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
    __syncwarp();
    if (vec_ok && hi - lo == BATCH) {
      uint4 cv[kUnroll], rv[kUnroll];
      uint4 xv[NIN > 0 ? kUnroll : 1][NX];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t e = lo + (int64_t)u * STEP + lane * V;
        cv[u] = ld_v4(cp + e * EB);
        rv[u] = ld_v4(rp + e * EB);
        if constexpr (NIN > 0) {
#pragma unroll
          for (int j = 0; j < NIN; ++j) xv[u][j] = ld_v4(xp[j] + e * EB);
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u)
        step<DT, NIN>(P, L, W, R, cv[u], rv[u], xv[NIN > 0 ? u : 0], lo + (int64_t)u * STEP + lane * V);
    } else {
      int64_t base = lo;
      if (vec_ok) {
        for (; base + STEP <= hi; base += STEP) {
          const int64_t e = base + lane * V;
          const uint4 cv = ld_v4(cp + e * EB), rv = ld_v4(rp + e * EB);
          uint4 xv[NX];
          if constexpr (NIN > 0) {
#pragma unroll
            for (int j = 0; j < NIN; ++j) xv[j] = ld_v4(xp[j] + e * EB);
          }
          step<DT, NIN>(P, L, W, R, cv, rv, xv, e);
        }
      }
      for (; base < hi; base += STEP) {
        const int64_t e = base + lane * V;
        int64_t n = hi - e;
        n = n < 0 ? 0 : (n > V ? V : n);
        R.sse = tail_step<DT, NIN>(P, L, W, e, (int)n, R.sse);
        reload_thr(R, W);
      }
    }
    __syncwarp();
    if (lane == 0) batch_count[pc.batch_base + b] = (int32_t)W->mism;
    if (++flush == kFlushBatches) {
      sse_flush(R.sse);
      flush = 0;
    }
  }
  sse_flush(R.sse);
}

// ------------------------------------------------------------ the kernel
// Dynamic shared memory (int32 words): [0, 8) class counters (NaN/+Inf/-Inf
// of c, of r, non-finite pairs), [8, 16) unused, then the row profile [th],
// the column profile [tw] and the histogram window.
constexpr int kShHead = 16;

template <int DT, int NIN>
__global__ void __launch_bounds__(kThreads, 2)
    scan_kernel(const CaseDesc *__restrict__ cases, const Piece *__restrict__ pieces,
                const int64_t *__restrict__ block_piece, int64_t piece_base, Partial *partials,
                int32_t *batch_count, uint8_t *out, uint32_t *g_thr, unsigned long long *stats) {
  constexpr int EB = Tr<DT>::EB;
  extern __shared__ int32_t smem[];
  __shared__ PieceSh P;
  __shared__ LaneSh lanes[kThreads];
  __shared__ WarpSh warps[kWarps];
  __shared__ Partial red[kWarps];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  LaneSh *L = &lanes[threadIdx.x];
  WarpSh *W = &warps[warp];
  const int64_t p0 = block_piece[blockIdx.x], p1 = block_piece[blockIdx.x + 1];
  for (int64_t p = p0; p < p1; ++p) {
    const Piece pc = pieces[p];
    if (threadIdx.x == 0) {
      P.cd = cases[pc.case_id];
      P.tr0 = pc.tr0;
      P.tc0 = pc.tc0;
      P.wr = pc.wr;
      P.wc = pc.wc;
      P.prof_smem = pc.prof_smem;
      P.sh_cls = smem;
      P.sh_row = smem + kShHead;
      P.sh_col = P.sh_row + (pc.prof_smem ? P.cd.th : 0);
      P.sh_hist = P.sh_col + (pc.prof_smem ? P.cd.tw : 0);
      uint8_t *o = out + P.cd.out_off;
      P.g_hist = (unsigned long long *)(o + P.cd.hist_off);
      P.g_row = (unsigned long long *)(o + P.cd.rowp_off);
      P.g_col = (unsigned long long *)(o + P.cd.colp_off);
      P.g_thr = g_thr + 2 * pc.case_id;
      P.stats = stats;
    }
    __syncthreads();
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
    for (int j = 0; j < NMV_MAX_INPUTS; ++j) L->eq[j] = 0;
    if (lane == 0) {
      W->tA = W->tR = W->wA = W->wR = W->ga = W->gr = -1.f;
      W->pubA = W->pubR = 0;
      W->mism = 0;
    }
    __syncthreads();

    Regs<NIN> R;
    R.sse.hi = R.sse.lo = make_float2(0.f, 0.f);
    R.sse.acc = 0.0;
    R.cacc = R.racc = 0;
#pragma unroll
    for (int j = 0; j < (NIN > 0 ? NIN : 1); ++j) R.eq[j] = 0;
    {
      const uint32_t c0 = ld_one<EB>(P.cd.cand, 0), r0 = ld_one<EB>(P.cd.ref, 0);
      R.cpat = EB == 2 ? (c0 | (c0 << 16)) : c0;
      R.rpat = EB == 2 ? (r0 | (r0 << 16)) : r0;
    }
    R.tA = R.tR = R.tRq = R.ga = R.gr = -1.f;
    R.lo_r = P.cd.lo_r;
    R.lo_a = P.cd.lo_a;
    sweep<DT, NIN>(&P, L, W, R, pc, batch_count);
    __syncwarp();

    // ---- lanes -> warps -> the piece's partial
    const Best a = best_warp(abs_best64(L)), r = best_warp(rel_best64(L));
    const double sse = warp_reduce(R.sse.acc, [](double x, double y) { return __dadd_rn(x, y); });
    const uint32_t cacc = warp_reduce(R.cacc | L->cacc, [](uint32_t x, uint32_t y) { return x | y; });
    const uint32_t racc = warp_reduce(R.racc | L->racc, [](uint32_t x, uint32_t y) { return x | y; });
    int eqs[NMV_MAX_INPUTS];
#pragma unroll
    for (int j = 0; j < NMV_MAX_INPUTS; ++j) {
      int v = L->eq[j];
      if constexpr (NIN > 0) {
        if (j < NIN) v += R.eq[j < NIN ? j : 0];
      }
      eqs[j] = warp_reduce(v, [](int x, int y) { return x + y; });
    }
    int64_t mism = 0;
    if (lane == 0) {
      const int64_t nb = piece_batches(pc.begin, pc.end, DT);
      for (int64_t rr = 0; rr * kWarps < nb; ++rr) {
        const int64_t b = rr * kWarps + ((warp - rr) % kWarps + kWarps) % kWarps;
        if (b < nb) mism += batch_count[pc.batch_base + b];
      }
      Partial &w = red[warp];
      w.cnt[0] = mism;
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
    if (pc.wr > 0) {
      for (int64_t t = threadIdx.x; t < (int64_t)pc.wr * pc.wc; t += kThreads) {
        const int v = P.sh_hist[t];
        if (v) {
          const int64_t tr = pc.tr0 + t / pc.wc, tc = pc.tc0 + t % pc.wc;
          atomicAdd(&P.g_hist[tr * P.cd.GC + tc], (unsigned long long)v);
        }
      }
    }
    if (pc.prof_smem) {
      for (int64_t t = threadIdx.x; t < P.cd.th; t += kThreads)
        if (P.sh_row[t]) atomicAdd(&P.g_row[t], (unsigned long long)P.sh_row[t]);
      for (int64_t t = threadIdx.x; t < P.cd.tw; t += kThreads)
        if (P.sh_col[t]) atomicAdd(&P.g_col[t], (unsigned long long)P.sh_col[t]);
    }
    if (threadIdx.x == 0) {
      Partial Q;
      Q.cnt[0] = 0;
      for (int k = 1; k < 8; ++k) Q.cnt[k] = smem[k - 1];
      Best ba = {-1.0, INT64_MAX}, br = {-1.0, INT64_MAX};
      Q.sse = 0.0;
      Q.cacc = 0;
      Q.racc = 0;
      for (int j = 0; j < NMV_MAX_INPUTS; ++j) Q.eq[j] = 0;
      for (int w = 0; w < kWarps; ++w) {
        Q.cnt[0] += red[w].cnt[0];
        best_offer(ba, red[w].best_abs, red[w].arg_abs);
        best_offer(br, red[w].best_rel, red[w].arg_rel);
        Q.sse = __dadd_rn(Q.sse, red[w].sse);
        Q.cacc |= red[w].cacc;
        Q.racc |= red[w].racc;
        for (int j = 0; j < NMV_MAX_INPUTS; ++j) Q.eq[j] += red[w].eq[j];
      }
      Q.best_abs = ba.v;
      Q.arg_abs = ba.i;
      Q.best_rel = br.v;
      Q.arg_rel = br.i;
      partials[piece_base + p] = Q;
    }
    __syncthreads();
  }
}

// Launch helpers of one element type (defined in nmv_scan_<dtype>.cu).
template <int DT>
struct ScanOps {
  static cudaError_t prepare(int nin, size_t smem);
  static int occupancy(int nin, size_t smem);
  static cudaError_t launch(int nin, int grid, size_t smem, cudaStream_t st, const CaseDesc *cases,
                            const Piece *pieces, const int64_t *block_piece, int64_t piece_base,
                            Partial *partials, int32_t *batch_count, uint8_t *out, uint32_t *g_thr,
                            unsigned long long *stats);
};

#define NMV_DEFINE_SCAN_OPS(DT)                                                                     \
  template <>                                                                                       \
  cudaError_t ScanOps<DT>::prepare(int nin, size_t smem) {                                          \
    if (nin == 0) return cudaFuncSetAttribute(scan_kernel<DT, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
    if (nin == 1) return cudaFuncSetAttribute(scan_kernel<DT, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
    return cudaFuncSetAttribute(scan_kernel<DT, -1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
  }                                                                                                 \
  template <>                                                                                       \
  int ScanOps<DT>::occupancy(int nin, size_t smem) {                                                \
    int n = 0;                                                                                      \
    cudaError_t e;                                                                                  \
    if (nin == 0) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, scan_kernel<DT, 0>, kThreads, smem); \
    else if (nin == 1) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, scan_kernel<DT, 1>, kThreads, smem); \
    else e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, scan_kernel<DT, -1>, kThreads, smem); \
    return e == cudaSuccess ? n : 0;                                                                \
  }                                                                                                 \
  template <>                                                                                       \
  cudaError_t ScanOps<DT>::launch(int nin, int grid, size_t smem, cudaStream_t st, const CaseDesc *cases, \
                                  const Piece *pieces, const int64_t *block_piece, int64_t piece_base, \
                                  Partial *partials, int32_t *batch_count, uint8_t *out, uint32_t *g_thr, \
                                  unsigned long long *stats) {                                      \
    if (nin == 0)                                                                                   \
      scan_kernel<DT, 0><<<grid, kThreads, smem, st>>>(cases, pieces, block_piece, piece_base, partials, \
                                                       batch_count, out, g_thr, stats);             \
    else if (nin == 1)                                                                              \
      scan_kernel<DT, 1><<<grid, kThreads, smem, st>>>(cases, pieces, block_piece, piece_base, partials, \
                                                       batch_count, out, g_thr, stats);             \
    else                                                                                            \
      scan_kernel<DT, -1><<<grid, kThreads, smem, st>>>(cases, pieces, block_piece, piece_base, partials, \
                                                        batch_count, out, g_thr, stats);            \
    return cudaGetLastError();                                                                      \
  }

}  // namespace nmv
