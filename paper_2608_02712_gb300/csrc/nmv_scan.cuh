// nmv_scan.cuh -- the streaming validation pass (one kernel per element type
// and input count; instantiated by nmv_scan_<dtype>.cu).
//
// One pass over candidate, reference (and the inputs of the pass-through
// check) computes, per piece of a case: the pass predicate of the tolerance
// check (Section 3.2, Eq. 1, read as allclose in fp64), NaN/Inf counts, the
// maximum absolute and relative errors with their lowest indices, the sum of
// squared errors, the tile-histogram and row/column profiles of the
// mismatches (localisation evidence, Sections 4.2 and S2.2), the first
// mismatch offsets of each warp segment (for the first-K records) and the
// degenerate-output accumulators (Sections 1 and 4.3).
//
// Exactness without fp64 throughput.  GB300 has very little fp64
// throughput, so each element is handled in fp32 where a margin proves the
// fp64 result; only elements inside the margin, non-finite elements and
// candidates for a new maximum take the fp64 path (the "slow" path, taken by
// the whole warp for a step when any lane needs it):
//  * predicate: sure-pass if |s| <= fma_rz(lo_r, |r|, lo_a) with s = fl32(c-r)
//    and lo_* = fp32 round-down of (1 - 2^-20) * {rtol, atol}; sure-fail if
//    |s| > fma_ru(hi_r, |r|, hi_a) with hi_* the round-up of
//    (1 + 2^-20) * {rtol, atol}; otherwise fl64(|c-r|) <= fl64(atol +
//    fl64(rtol*|r|)) is evaluated.  The margin absorbs every fp32 rounding
//    (|s| vs |c-r|, the fp32 coefficients, |r| of an int32), so the decision
//    equals the fp64 one.
//  * max |d| and max |d|/|r|: an element is skipped only when its fp32 values
//    prove its fp64 value is below a maximum already held: strictly (margin
//    2^-20, thresholds shared through the case's published maxima), or equal
//    at a higher index within the warp's own ascending sweep.
//  * SSE: d = s + e exactly (Knuth's TwoSum; int32: exact remainder), d^2 =
//    p + pe + 2se with p = fl(s*s), pe = fma(s, s, -p) (Dekker's product via
//    fma), accumulated as a float-float pair per lane and flushed to an fp64
//    sum after every unrolled batch.  Terms with |s| outside [2^-40, 2^60)
//    are squared in fp64.  Every element takes the same SSE arithmetic on
//    the fast and the slow path, so results are bit-identical run to run.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "nmv_internal.h"

namespace nmv {

constexpr int kUnroll = 4;
constexpr float kTiny = 0x1p-40f;
constexpr float kHuge = 0x1p60f;
constexpr float kMarginLo = 1.0f - 0x1p-20f;
constexpr float kMinSub = 0x1p-149f;

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

// d = c - r = s + e exactly (s = fl32(d)), as = |s|, ar = |r| in fp32.
struct Diff {
  float s, e, as, ar;
};

template <int DT>
__device__ __forceinline__ Diff make_diff(uint32_t cb, uint32_t rb, float cf, float rf) {
  Diff x;
  if constexpr (Tr<DT>::kInt) {
    const long long d = (long long)(int32_t)cb - (long long)(int32_t)rb;
    x.s = __ll2float_rn(d);
    x.e = __ll2float_rn(d - __float2ll_rn(x.s));
  } else {
    // Knuth's TwoSum of c and -r.
    const float s = __fsub_rn(cf, rf);
    const float bb = __fsub_rn(s, cf);
    x.e = __fsub_rn(__fsub_rn(cf, __fsub_rn(s, bb)), __fadd_rn(rf, bb));
    x.s = s;
  }
  x.ar = fabsf(rf);
  x.as = fabsf(x.s);
  return x;
}

// Float-float SSE accumulator of one lane.
struct Sse {
  float hi, lo;
  double acc;
};

__device__ __forceinline__ void sse_add_ff(Sse &a, float s, float e) {
  const float p = __fmul_rn(s, s);
  const float pe = __fmaf_rn(s, s, -p);                 // s*s - p, exact
  const float q = __fmaf_rn(__fadd_rn(s, s), e, pe);    // + 2 s e (e*e dropped)
  const float t = __fadd_rn(a.hi, p);                   // TwoSum(hi, p)
  const float bp = __fsub_rn(t, a.hi);
  const float err = __fadd_rn(__fsub_rn(a.hi, __fsub_rn(t, bp)), __fsub_rn(p, bp));
  a.hi = t;
  a.lo = __fadd_rn(a.lo, __fadd_rn(err, q));
}

__device__ __forceinline__ void sse_flush(Sse &a) {
  a.acc = __dadd_rn(a.acc, __dadd_rn((double)a.hi, (double)a.lo));
  a.hi = 0.f;
  a.lo = 0.f;
}

// One both-finite element's d^2: float-float when the fp32 square is safe,
// otherwise the fp64 square of fl64(c - r) (which also covers an fp32
// overflow of c - r).
template <int DT>
__device__ __forceinline__ void sse_term(Sse &a, const Diff &x, uint32_t cb, uint32_t rb) {
  if (x.as == 0.f) return;
  if (x.as >= kTiny && x.as < kHuge) {
    sse_add_ff(a, x.s, x.e);
  } else {
    const double d = __dsub_rn(to_f64<DT>(cb), to_f64<DT>(rb));
    a.acc = __dadd_rn(a.acc, __dmul_rn(d, d));
  }
}

// Best (value, index): larger value wins, equal values go to the lower index.
struct Best {
  double v;  // -1 when none
  int64_t i;
};

__device__ __forceinline__ void best_offer(Best &b, double v, int64_t i) {
  if (v > b.v || (v == b.v && i < b.i)) {
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

// -------------------------------------------------------------- state
// Piece-constant data of the slow path, read from shared memory.
struct PieceSh {
  CaseDesc cd;
  int64_t tr0, tc0;
  int32_t wr, wc, prof_smem;
  int32_t *sh_cls, *sh_row, *sh_col, *sh_hist;
  unsigned long long *g_hist, *g_row, *g_col;
  uint32_t *g_thr;
};

// Per-lane state carried through a segment.
template <int NIN>
struct Lane {
  Best babs, brel;
  Sse sse;
  uint32_t cacc, racc;
  int eq[NIN > 0 ? NIN : 1];
  uint32_t cpat, rpat;  // element-0 bits replicated over a 32-bit word
};

// Warp-uniform state of a segment sweep.
struct WarpSt {
  float tA, tR;         // current skip thresholds
  float wA, wR;         // the warp's own part of them
  uint32_t pubA, pubR;  // last maxima this warp published to the case
  int64_t mism;         // mismatches so far in this segment
  uint32_t *seg_list;   // kFirstR slots of this segment
  int64_t seg_lo;
};

__device__ __forceinline__ void count_maps(const PieceSh &P, int64_t idx) {
  const CaseDesc &cd = P.cd;
  const uint64_t row = div_q((uint64_t)idx, cd.dN.d, cd.dN.m);
  const uint64_t col = (uint64_t)idx - row * cd.dN.d;
  const uint64_t tr = div_q(row, cd.dth.d, cd.dth.m);
  const uint64_t tc = div_q(col, cd.dtw.d, cd.dtw.m);
  const int64_t rp = (int64_t)(row - tr * cd.dth.d);
  const int64_t cp = (int64_t)(col - tc * cd.dtw.d);
  if (P.wr > 0) {
    atomicAdd(&P.sh_hist[((int64_t)tr - P.tr0) * P.wc + ((int64_t)tc - P.tc0)], 1);
  } else {
    atomicAdd(&P.g_hist[tr * (uint64_t)cd.GC + tc], 1ull);
  }
  if (P.prof_smem) {
    atomicAdd(&P.sh_row[rp], 1);
    atomicAdd(&P.sh_col[cp], 1);
  } else {
    atomicAdd(&P.g_row[rp], 1ull);
    atomicAdd(&P.g_col[cp], 1ull);
  }
}

// Exact treatment of one element (slow path).  Returns true on mismatch.
template <int DT, int NIN>
__device__ __forceinline__ bool slow_elem(const PieceSh &P, Lane<NIN> &L, const WarpSt &W,
                                          uint32_t cb, uint32_t rb, int64_t idx) {
  const CaseDesc &cd = P.cd;
  const float cf = to_f32<DT>(cb), rf = to_f32<DT>(rb);
  const Diff x = make_diff<DT>(cb, rb, cf, rf);
  bool cfin = true, rfin = true, equal;
  if constexpr (Tr<DT>::kInt) {
    equal = cb == rb;
  } else {
    cfin = isfinite(cf);
    rfin = isfinite(rf);
    equal = cf == rf;
    if (!cfin) atomicAdd(&P.sh_cls[isnan(cf) ? 0 : (cf > 0.f ? 1 : 2)], 1);
    if (!rfin) atomicAdd(&P.sh_cls[isnan(rf) ? 3 : (rf > 0.f ? 4 : 5)], 1);
  }
  const bool fin = cfin && rfin;
  bool pass;
  if (equal) {
    pass = true;
  } else if (!fin) {
    pass = false;
  } else if (x.as <= __fmaf_rz(cd.lo_r, x.ar, cd.lo_a)) {
    pass = true;
  } else if (x.as > __fmaf_ru(cd.hi_r, x.ar, cd.hi_a)) {
    pass = false;
  } else {
    pass = pass64(to_f64<DT>(cb), to_f64<DT>(rb), cd.rtol, cd.atol);
  }
  if (fin) {
    if (!(x.as < W.tA)) {
      const double a64 = fabs(__dsub_rn(to_f64<DT>(cb), to_f64<DT>(rb)));
      best_offer(L.babs, a64, idx);
    }
    if (x.ar != 0.f && x.as >= __fmul_rn(W.tR, x.ar)) {
      const double r64 = to_f64<DT>(rb);
      if (r64 != 0.0) {
        const double a64 = fabs(__dsub_rn(to_f64<DT>(cb), r64));
        best_offer(L.brel, __ddiv_rn(a64, fabs(r64)), idx);
      }
    }
    sse_term<DT>(L.sse, x, cb, rb);
  } else {
    atomicAdd(&P.sh_cls[6], 1);
  }
  return !pass;
}

// Refresh the warp's thresholds from the lanes' bests and publish
// improvements to the case (for the other warps).
template <int NIN>
__device__ __forceinline__ void refresh_thresholds(const PieceSh &P, const Lane<NIN> &L, WarpSt &W) {
  const Best a = best_warp(L.babs);
  const Best r = best_warp(L.brel);
  if (a.v >= 0.0) {
    const float f = __double2float_rd(a.v);
    W.wA = fminf(fmaxf(f, kMinSub), kHuge);
    const uint32_t u = __float_as_uint(f);
    if (u > W.pubA) {
      if ((threadIdx.x & 31) == 0) atomicMax(&P.g_thr[0], u);
      W.pubA = u;
    }
  }
  if (r.v >= 0.0) {
    const float f = __double2float_rd(r.v);
    W.wR = fmaxf(__fmul_rn(f, kMarginLo), kMinSub);
    const uint32_t u = __float_as_uint(f);
    if (u > W.pubR) {
      if ((threadIdx.x & 31) == 0) atomicMax(&P.g_thr[1], u);
      W.pubR = u;
    }
  }
  W.tA = fminf(fmaxf(W.tA, W.wA), kHuge);
  W.tR = fmaxf(W.tR, W.wR);
}

// Combine the warp's own thresholds with the case-wide published maxima.
__device__ __forceinline__ void merge_thresholds(WarpSt &W, uint32_t gA, uint32_t gR) {
  const float ga = __fmul_rn(__uint_as_float(gA), kMarginLo);
  const float gr = __fmul_rn(__uint_as_float(gR), kMarginLo);
  W.tA = fminf(fmaxf(W.wA, ga), kHuge);
  W.tR = fmaxf(W.wR, gr);
}

// Record this lane's mismatches of one step (bit k of `mask` = element
// idx0 + k) in ascending index order: segment list, then the maps.
__device__ __forceinline__ void record_step(const PieceSh &P, WarpSt &W, uint32_t mask, int64_t idx0) {
  const int lane = threadIdx.x & 31;
  const int cnt = __popc(mask);
  int incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  const int total = __shfl_sync(0xffffffffu, incl, 31);
  if (total == 0) return;
  int64_t pos = W.mism + (incl - cnt);
  uint32_t m = mask;
  while (m) {
    const int k = __ffs(m) - 1;
    m &= m - 1;
    const int64_t idx = idx0 + k;
    if (pos < kFirstR) W.seg_list[pos] = (uint32_t)(idx - W.seg_lo);
    ++pos;
    count_maps(P, idx);
  }
  W.mism += total;
}

// The slow path of one step: lane elements idx0 .. idx0 + n - 1 with the
// stored bits held in (c0..c3, r0..r3) for the vector form; words are
// consumed by shifting so the loop needs no dynamic register indexing.
template <int DT, int NIN>
__device__ __forceinline__ void slow_step(const PieceSh &P, Lane<NIN> &L, WarpSt &W, uint4 cv, uint4 rv,
                                       int64_t idx0, int n) {
  constexpr int EB = Tr<DT>::EB;
  uint32_t mask = 0;
#pragma unroll 1
  for (int k = 0; k < n; ++k) {
    const uint32_t cb = cv.x & Tr<DT>::kElemMask, rb = rv.x & Tr<DT>::kElemMask;
    if (slow_elem<DT, NIN>(P, L, W, cb, rb, idx0 + k)) mask |= 1u << k;
    if constexpr (EB == 2) {
      cv.x = __funnelshift_r(cv.x, cv.y, 16);
      cv.y = __funnelshift_r(cv.y, cv.z, 16);
      cv.z = __funnelshift_r(cv.z, cv.w, 16);
      cv.w >>= 16;
      rv.x = __funnelshift_r(rv.x, rv.y, 16);
      rv.y = __funnelshift_r(rv.y, rv.z, 16);
      rv.z = __funnelshift_r(rv.z, rv.w, 16);
      rv.w >>= 16;
    } else {
      cv = make_uint4(cv.y, cv.z, cv.w, 0u);
      rv = make_uint4(rv.y, rv.z, rv.w, 0u);
    }
  }
  record_step(P, W, mask, idx0);
  refresh_thresholds<NIN>(P, L, W);
}

// ----------------------------------------------------------- one step
template <int DT, int NIN>
__device__ __forceinline__ void eq_vec(Lane<NIN> &L, const uint4 &cv, const uint4 &rv, const uint4 &xv,
                                       int j) {
#pragma unroll
  for (int k = 0; k < Tr<DT>::V; ++k) {
    const uint32_t xb = vbits<DT>(xv, k);
    L.eq[j] += (vbits<DT>(cv, k) == xb) & (vbits<DT>(rv, k) != xb);
  }
}

// One full step: this lane owns the V elements idx0 .. idx0 + V - 1.
template <int DT, int NIN>
__device__ __forceinline__ void step_vec(const PieceSh &P, Lane<NIN> &L, WarpSt &W, float lo_r, float lo_a,
                                         const uint4 &cv, const uint4 &rv, int64_t idx0) {
  constexpr int V = Tr<DT>::V;
  L.cacc |= (cv.x ^ L.cpat) | (cv.y ^ L.cpat) | (cv.z ^ L.cpat) | (cv.w ^ L.cpat);
  L.racc |= (rv.x ^ L.rpat) | (rv.y ^ L.rpat) | (rv.z ^ L.rpat) | (rv.w ^ L.rpat);
  bool hard = false;
#pragma unroll
  for (int k = 0; k < V; ++k) {
    const float cf = vdec<DT>(cv, k), rf = vdec<DT>(rv, k);
    float as, ar;
    if constexpr (Tr<DT>::kInt) {
      const Diff x = make_diff<DT>(vbits<DT>(cv, k), vbits<DT>(rv, k), cf, rf);
      as = x.as;
      ar = x.ar;
    } else {
      as = fabsf(__fsub_rn(cf, rf));
      ar = fabsf(rf);
    }
    const bool sure = as <= __fmaf_rz(lo_r, ar, lo_a);
    const bool skipA = as < W.tA;
    const bool candR = (as >= __fmul_rn(W.tR, ar)) && (ar != 0.f);
    const bool tiny = (as < kTiny) && (as != 0.f);
    hard |= !(sure && skipA) || candR || tiny;
  }
  if (!__any_sync(0xffffffffu, hard)) {
#pragma unroll
    for (int k = 0; k < V; ++k) {
      const Diff x = make_diff<DT>(vbits<DT>(cv, k), vbits<DT>(rv, k), vdec<DT>(cv, k), vdec<DT>(rv, k));
      if (x.as != 0.f) sse_add_ff(L.sse, x.s, x.e);
    }
    return;
  }
  slow_step<DT, NIN>(P, L, W, cv, rv, idx0, V);
}

// Ragged part: this lane owns n (0..V) elements from idx0, loaded one by one.
template <int DT, int NIN>
__device__ __forceinline__ void step_tail(const PieceSh &P, Lane<NIN> &L, WarpSt &W, int64_t idx0, int n) {
  constexpr int EB = Tr<DT>::EB;
  const CaseDesc &cd = P.cd;
  uint32_t cw[4] = {0, 0, 0, 0}, rw[4] = {0, 0, 0, 0};
  for (int k = 0; k < n; ++k) {
    const int64_t i = idx0 + k;
    const uint32_t cb = ld_one<EB>(cd.cand, i), rb = ld_one<EB>(cd.ref, i);
    L.cacc |= cb ^ (L.cpat & Tr<DT>::kElemMask);
    L.racc |= rb ^ (L.rpat & Tr<DT>::kElemMask);
    if constexpr (NIN != 0) {
      for (int j = 0; j < cd.n_elig; ++j) {
        const uint32_t xb = ld_one<EB>(cd.in_ptr[j], i);
        const int add = (cb == xb) & (rb != xb);
        if constexpr (NIN > 0) {
#pragma unroll
          for (int jj = 0; jj < NIN; ++jj)
            if (jj == j) L.eq[jj] += add;
        } else {
          atomicAdd(&P.sh_cls[8 + j], add);
        }
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
  slow_step<DT, NIN>(P, L, W, make_uint4(cw[0], cw[1], cw[2], cw[3]),
                     make_uint4(rw[0], rw[1], rw[2], rw[3]), idx0, n);
}

// Sweep one segment [lo, hi) with the whole warp.
template <int DT, int NIN>
__device__ __forceinline__ void sweep(const PieceSh &P, Lane<NIN> &L, WarpSt &W, int64_t lo, int64_t hi) {
  constexpr int V = Tr<DT>::V;
  constexpr int EB = Tr<DT>::EB;
  constexpr int STEP = 32 * V;
  constexpr int NX = NIN > 0 ? NIN : 1;
  const int lane = threadIdx.x & 31;
  const CaseDesc &cd = P.cd;
  const char *cp = (const char *)cd.cand;
  const char *rp = (const char *)cd.ref;
  const char *xp[NX];
#pragma unroll
  for (int j = 0; j < NX; ++j) xp[j] = (const char *)cd.in_ptr[j];
  const float lo_r = cd.lo_r, lo_a = cd.lo_a;
  const uint32_t *g_thr = P.g_thr;
  int64_t base = lo;
  if (cd.vec_ok) {
    while (base + (int64_t)STEP * kUnroll <= hi) {
      const uint32_t gA = __ldcg(&g_thr[0]);
      const uint32_t gR = __ldcg(&g_thr[1]);
      uint4 cv[kUnroll], rv[kUnroll];
      uint4 xv[NIN > 0 ? kUnroll : 1][NX];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t e = base + (int64_t)u * STEP + lane * V;
        cv[u] = ld_v4(cp + e * EB);
        rv[u] = ld_v4(rp + e * EB);
        if constexpr (NIN > 0) {
#pragma unroll
          for (int j = 0; j < NIN; ++j) xv[u][j] = ld_v4(xp[j] + e * EB);
        }
      }
      merge_thresholds(W, gA, gR);
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t e = base + (int64_t)u * STEP + lane * V;
        if constexpr (NIN > 0) {
#pragma unroll
          for (int j = 0; j < NIN; ++j) eq_vec<DT, NIN>(L, cv[u], rv[u], xv[u][j], j);
        } else if constexpr (NIN < 0) {
          for (int j = 0; j < cd.n_elig; ++j) {
            const uint4 x = ld_v4((const char *)cd.in_ptr[j] + e * EB);
            int add = 0;
#pragma unroll
            for (int k = 0; k < V; ++k) {
              const uint32_t xb = vbits<DT>(x, k);
              add += (vbits<DT>(cv[u], k) == xb) & (vbits<DT>(rv[u], k) != xb);
            }
            atomicAdd(&P.sh_cls[8 + j], add);
          }
        }
        step_vec<DT, NIN>(P, L, W, lo_r, lo_a, cv[u], rv[u], e);
      }
      sse_flush(L.sse);
      base += (int64_t)STEP * kUnroll;
    }
    while (base + STEP <= hi) {
      const int64_t e = base + lane * V;
      merge_thresholds(W, __ldcg(&g_thr[0]), __ldcg(&g_thr[1]));
      const uint4 cv = ld_v4(cp + e * EB), rv = ld_v4(rp + e * EB);
      if constexpr (NIN > 0) {
#pragma unroll
        for (int j = 0; j < NIN; ++j) eq_vec<DT, NIN>(L, cv, rv, ld_v4(xp[j] + e * EB), j);
      } else if constexpr (NIN < 0) {
        for (int j = 0; j < cd.n_elig; ++j) {
          const uint4 x = ld_v4((const char *)cd.in_ptr[j] + e * EB);
          int add = 0;
#pragma unroll
          for (int k = 0; k < V; ++k) {
            const uint32_t xb = vbits<DT>(x, k);
            add += (vbits<DT>(cv, k) == xb) & (vbits<DT>(rv, k) != xb);
          }
          atomicAdd(&P.sh_cls[8 + j], add);
        }
      }
      step_vec<DT, NIN>(P, L, W, lo_r, lo_a, cv, rv, e);
      base += STEP;
    }
  }
  while (base < hi) {
    const int64_t e = base + lane * V;
    int64_t n = hi - e;
    n = n < 0 ? 0 : (n > V ? V : n);
    merge_thresholds(W, __ldcg(&g_thr[0]), __ldcg(&g_thr[1]));
    step_tail<DT, NIN>(P, L, W, e, (int)n);
    base += STEP;
  }
  sse_flush(L.sse);
}

// ------------------------------------------------------------ the kernel
// Shared memory (dynamic, int32 words): [0, 8) class counters (NaN/+Inf/-Inf
// of c, of r, non-finite pairs), [8, 16) pass-through counts of the generic
// input path, then row profile [th], column profile [tw], histogram window.
constexpr int kShHead = 16;

template <int DT, int NIN>
__global__ void __launch_bounds__(kThreads) scan_kernel(const CaseDesc *__restrict__ cases,
                                                        const Piece *__restrict__ pieces,
                                                        const int64_t *__restrict__ block_piece,
                                                        int64_t piece_base, Partial *partials,
                                                        int32_t *seg_count, uint32_t *seg_list,
                                                        uint8_t *out, uint32_t *g_thr) {
  constexpr int V = Tr<DT>::V;
  constexpr int EB = Tr<DT>::EB;
  extern __shared__ int32_t smem[];
  __shared__ PieceSh P;
  __shared__ Partial red[kWarps];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
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
    }
    __syncthreads();
    const int64_t used = (int64_t)(P.sh_hist - smem) + (int64_t)pc.wr * pc.wc;
    for (int64_t t = threadIdx.x; t < used; t += kThreads) smem[t] = 0;
    __syncthreads();

    Lane<NIN> L;
    L.babs = {-1.0, INT64_MAX};
    L.brel = {-1.0, INT64_MAX};
    L.sse = {0.f, 0.f, 0.0};
    L.cacc = 0;
    L.racc = 0;
#pragma unroll
    for (int j = 0; j < (NIN > 0 ? NIN : 1); ++j) L.eq[j] = 0;
    {
      const uint32_t c0 = ld_one<EB>(P.cd.cand, 0), r0 = ld_one<EB>(P.cd.ref, 0);
      L.cpat = EB == 2 ? (c0 | (c0 << 16)) : c0;
      L.rpat = EB == 2 ? (r0 | (r0 << 16)) : r0;
    }
    WarpSt W;
    W.tA = W.tR = W.wA = W.wR = 0.f;
    W.pubA = W.pubR = 0;
    W.mism = 0;
    int64_t lo, hi;
    segment_range(pc.begin, pc.end, warp, V, &lo, &hi);
    const int64_t seg = (piece_base + p) * kWarps + warp;
    W.seg_list = seg_list + seg * kFirstR;
    W.seg_lo = lo;
    if (lo < hi) sweep<DT, NIN>(P, L, W, lo, hi);
    if (lane == 0) seg_count[seg] = (int32_t)W.mism;

    // ---- lanes -> warps -> the piece's partial
    const Best a = best_warp(L.babs), r = best_warp(L.brel);
    const double sse = warp_reduce(L.sse.acc, [](double x, double y) { return __dadd_rn(x, y); });
    const uint32_t cacc = warp_reduce(L.cacc, [](uint32_t x, uint32_t y) { return x | y; });
    const uint32_t racc = warp_reduce(L.racc, [](uint32_t x, uint32_t y) { return x | y; });
    int eqs[NMV_MAX_INPUTS];
#pragma unroll
    for (int j = 0; j < NMV_MAX_INPUTS; ++j)
      eqs[j] = (NIN > 0 && j < NIN) ? warp_reduce(L.eq[j < NIN ? j : 0], [](int x, int y) { return x + y; }) : 0;
    if (lane == 0) {
      Partial &w = red[warp];
      w.cnt[0] = W.mism;
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
      for (int j = 0; j < NMV_MAX_INPUTS; ++j) Q.eq[j] = NIN < 0 ? smem[8 + j] : 0;
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
                            Partial *partials, int32_t *seg_count, uint32_t *seg_list, uint8_t *out,
                            uint32_t *g_thr);
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
                                  Partial *partials, int32_t *seg_count, uint32_t *seg_list, uint8_t *out, \
                                  uint32_t *g_thr) {                                                \
    if (nin == 0)                                                                                   \
      scan_kernel<DT, 0><<<grid, kThreads, smem, st>>>(cases, pieces, block_piece, piece_base, partials, \
                                                       seg_count, seg_list, out, g_thr);            \
    else if (nin == 1)                                                                              \
      scan_kernel<DT, 1><<<grid, kThreads, smem, st>>>(cases, pieces, block_piece, piece_base, partials, \
                                                       seg_count, seg_list, out, g_thr);            \
    else                                                                                            \
      scan_kernel<DT, -1><<<grid, kThreads, smem, st>>>(cases, pieces, block_piece, piece_base, partials, \
                                                        seg_count, seg_list, out, g_thr);           \
    return cudaGetLastError();                                                                      \
  }

}  // namespace nmv
