// nmv_stats.cu -- diagnostic tensor statistics (nmv_stats): the engine's
// diagnostic instrumentation of Section 4.2 ("multi-level tensor statistics
// at pipeline boundaries"), on GB300.
//
// Levels: the whole tensor and every tile of the [M, N] view (the tile grid
// of the localisation maps).  Work is cut into units: a unit is a block of
// at most kUnitElems elements of one tile, at most kUnitCols columns wide
// (a tile is split into row and column chunks, a small tile is one unit).
// stats_kernel hands the units to warps from a counter; a warp reads its
// unit with 16-byte loads where the rows allow (scalar loads otherwise),
// each lane walking its rows with a fixed stride and accumulating class
// counts, min/max and the sums, then reduces the lanes in a fixed butterfly
// and stores the unit's partial.  stats_fin_kernel merges each tile's units
// in unit order into the tile's statistics (written straight into the
// mapped host result), and the tiles of each case in a fixed tree into the
// whole-tensor statistics: nothing depends on which warp took which unit,
// so the results are bit-identical from run to run.
//
// Sums.  float elements: the lanes first take every whole vector on a fast
// path without class tests, sum(x) and sum(x^2) as float-float pairs
// (Knuth's TwoSum; x^2 split exactly as p + pe with an fma) folded into
// fp64 every kFlush vectors.  The result stands when the unit met no NaN
// or infinity and its largest magnitude lies in [2^-44, 2^57) (the pairs
// cannot overflow and the squares' remainders are exact, or round by a
// negligible amount); otherwise the unit is taken again element by
// element, classes tested and finite values added in fp64.  int32
// elements: exact 128-bit integer sums, rounded once to fp64 at the end.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <string>
#include <vector>

#include "nmv_scan.cuh"

namespace nmv {

constexpr int kStatThreads = 256;
constexpr int64_t kUnitCols = 8192;    // elements of a unit's row segment at most
constexpr int64_t kUnitElems = 16384;  // elements of a unit at most (rows x cols), unless one row is longer
constexpr int kFinBlocks = 256;        // finalize blocks per case at most
constexpr int64_t kCoopUnits = 32;     // tiles of this many units or more are merged by a whole block
constexpr int kFlush = 32;             // float-float pairs folded into fp64 every kFlush vectors

// One buffer as the kernels see it.
struct StatsDesc {
  const void *x;
  int32_t dtype, vec_ok;               // vec_ok: 16-byte loads of whole vectors are aligned
  int64_t numel, M, N, th, tw, GR, GC;
  int64_t cw, cc;                      // unit columns, column chunks per tile
  int64_t rch, ch;                     // unit rows, row chunks per tile
  int64_t unit_begin, unit_end;        // the case's units in the launch
  int64_t fin_blocks;                  // finalize blocks of this case
  int64_t bpart_off;                   // its block partials in the workspace
  int64_t res_off;                     // byte offset of the case's nmv_stats_result in the host block
  int64_t tiles_off;                   // byte offset of its nmv_stat tile array
};

// Partial statistics of a unit, a tile, a block of tiles or the tensor.
struct StatPart {
  int64_t n;                           // elements
  int64_t cnt[4];                      // NaN, +Inf, -Inf, zero
  int64_t first_nan, first_inf;        // lowest index, or INT64_MAX
  double mn, mx;                       // finite min / max (+Inf / -Inf: none)
  double s, q;                         // float: sum(x), sum(x^2)
  uint64_t is_lo, is_hi, iq_lo, iq_hi; // int32: exact sum(x) (two's complement) and sum(x^2), 128 bits
};

// ------------------------------------------------------------ combining
__device__ __forceinline__ void add128(uint64_t &lo, uint64_t &hi, uint64_t blo, uint64_t bhi) {
  asm("add.cc.u64 %0, %0, %2;\n\taddc.u64 %1, %1, %3;" : "+l"(lo), "+l"(hi) : "l"(blo), "l"(bhi));
}

__device__ __forceinline__ void part_init(StatPart &p) {
  p.n = 0;
  for (int k = 0; k < 4; ++k) p.cnt[k] = 0;
  p.first_nan = p.first_inf = INT64_MAX;
  p.mn = INFINITY;
  p.mx = -INFINITY;
  p.s = p.q = 0.0;
  p.is_lo = p.is_hi = p.iq_lo = p.iq_hi = 0;
}

// a += b, b holding elements that follow a's (the order is fixed by the
// callers; fp64 additions are commutative, so a + b == b + a bit for bit).
__device__ __forceinline__ void part_merge(StatPart &a, const StatPart &b) {
  a.n += b.n;
  for (int k = 0; k < 4; ++k) a.cnt[k] += b.cnt[k];
  a.first_nan = min(a.first_nan, b.first_nan);
  a.first_inf = min(a.first_inf, b.first_inf);
  a.mn = fmin(a.mn, b.mn);
  a.mx = fmax(a.mx, b.mx);
  a.s = __dadd_rn(a.s, b.s);
  a.q = __dadd_rn(a.q, b.q);
  add128(a.is_lo, a.is_hi, b.is_lo, b.is_hi);
  add128(a.iq_lo, a.iq_hi, b.iq_lo, b.iq_hi);
}

__device__ __forceinline__ StatPart part_shfl(const StatPart &p, int o) {
  StatPart r;
  r.n = __shfl_xor_sync(0xffffffffu, p.n, o);
  for (int k = 0; k < 4; ++k) r.cnt[k] = __shfl_xor_sync(0xffffffffu, p.cnt[k], o);
  r.first_nan = __shfl_xor_sync(0xffffffffu, p.first_nan, o);
  r.first_inf = __shfl_xor_sync(0xffffffffu, p.first_inf, o);
  r.mn = __shfl_xor_sync(0xffffffffu, p.mn, o);
  r.mx = __shfl_xor_sync(0xffffffffu, p.mx, o);
  r.s = __shfl_xor_sync(0xffffffffu, p.s, o);
  r.q = __shfl_xor_sync(0xffffffffu, p.q, o);
  r.is_lo = __shfl_xor_sync(0xffffffffu, p.is_lo, o);
  r.is_hi = __shfl_xor_sync(0xffffffffu, p.is_hi, o);
  r.iq_lo = __shfl_xor_sync(0xffffffffu, p.iq_lo, o);
  r.iq_hi = __shfl_xor_sync(0xffffffffu, p.iq_hi, o);
  return r;
}

// exact 128-bit two's-complement integer -> fp64, one rounding to nearest
// (ties to even): the top 64 significant bits, with a sticky bit for the
// rest, converted by one integer-to-double conversion.
__device__ __forceinline__ double i128_to_f64(uint64_t lo, uint64_t hi) {
  const bool neg = (int64_t)hi < 0;
  if (neg) {  // magnitude
    lo = ~lo;
    hi = ~hi;
    add128(lo, hi, 1ull, 0ull);
  }
  double v;
  if (hi == 0) {
    v = __ull2double_rn(lo);
  } else {
    // value = top * 2^sh + rest, top holding the 64 leading bits
    const int lz = __clzll((long long)hi);
    const int sh = 64 - lz;
    uint64_t top, rest;
    if (lz == 0) {
      top = hi;
      rest = lo;
    } else {
      top = (hi << lz) | (lo >> sh);
      rest = lo << lz;
    }
    top |= rest != 0 ? 1ull : 0ull;  // sticky: bit 0 lies far below fp64's 53 bits
    v = ldexp(__ull2double_rn(top), sh);
  }
  return neg ? -v : v;
}

// The statistics of a finished region into the public record: mean and std
// from the sums with one rounding per operation.
__device__ __forceinline__ void part_out(const StatPart &p, int dt, nmv_stat *o) {
  const int64_t nf = p.n - p.cnt[0] - p.cnt[1] - p.cnt[2];
  o->n_finite = nf;
  o->n_nan = p.cnt[0];
  o->n_posinf = p.cnt[1];
  o->n_neginf = p.cnt[2];
  o->n_zero = p.cnt[3];
  if (nf == 0) {
    o->min = o->max = o->sum = o->sumsq = o->mean = o->std = 0.0;
    return;
  }
  double s, q;
  if (dt == NMV_I32) {
    s = i128_to_f64(p.is_lo, p.is_hi);
    q = i128_to_f64(p.iq_lo, p.iq_hi);
  } else {
    s = p.s;
    q = p.q;
  }
  const double n = (double)nf;
  const double mean = __ddiv_rn(s, n);
  const double var = __dsub_rn(__ddiv_rn(q, n), __dmul_rn(mean, mean));
  o->min = p.mn;
  o->max = p.mx;
  o->sum = s;
  o->sumsq = q;
  o->mean = mean;
  o->std = var > 0.0 ? __dsqrt_rn(var) : 0.0;
}

// ------------------------------------------------------------ lane sums
// Every field is a scalar (no field is indexed at run time), so a lane's
// sums stay in registers.
struct LaneStat {
  int32_t n_nan, n_pinf, n_ninf, n_zero;  // a unit has at most kUnitElems elements
  int64_t first_nan, first_inf;
  float mn, mx;          // float types
  int32_t imn, imx;      // int32
  float2 sh, sl, qh, ql; // float-float sum(x), sum(x^2): even / odd elements of each vector
  double s64, q64;
  uint64_t is_lo, is_hi, iq_lo, iq_hi;
  int pending;           // vectors since the last fold
};

__device__ __forceinline__ void lane_init(LaneStat &L) {
  L.n_nan = L.n_pinf = L.n_ninf = L.n_zero = 0;
  L.first_nan = L.first_inf = INT64_MAX;
  L.mn = INFINITY;
  L.mx = -INFINITY;
  L.imn = INT32_MAX;
  L.imx = INT32_MIN;
  L.sh = L.sl = L.qh = L.ql = make_float2(0.f, 0.f);
  L.s64 = L.q64 = 0.0;
  L.is_lo = L.is_hi = L.iq_lo = L.iq_hi = 0;
  L.pending = 0;
}

// TwoSum of x into (h, l), packed.
__device__ __forceinline__ void ff_add2(float2 &h, float2 &l, float2 x) {
  const float2 m1 = make_float2(-1.f, -1.f);
  const float2 t = __fadd2_rn(h, x);
  const float2 bp = __ffma2_rn(h, m1, t);
  const float2 x1 = __ffma2_rn(bp, m1, t);
  const float2 x2 = __ffma2_rn(x1, m1, h);
  const float2 x3 = __ffma2_rn(bp, m1, x);
  l = __fadd2_rn(l, __fadd2_rn(x2, x3));
  h = t;
}

__device__ __forceinline__ void lane_fold(LaneStat &L) {
  L.s64 = __dadd_rn(L.s64, __dadd_rn(__dadd_rn((double)L.sh.x, (double)L.sl.x),
                                     __dadd_rn((double)L.sh.y, (double)L.sl.y)));
  L.q64 = __dadd_rn(L.q64, __dadd_rn(__dadd_rn((double)L.qh.x, (double)L.ql.x),
                                     __dadd_rn((double)L.qh.y, (double)L.ql.y)));
  L.sh = L.sl = L.qh = L.ql = make_float2(0.f, 0.f);
  L.pending = 0;
}

// One element outside the fast path (float types): its class, and a finite
// value's terms in fp64.
template <int DT>
__device__ __forceinline__ void lane_slow(LaneStat &L, uint32_t b, int64_t idx) {
  const float x = to_f32<DT>(b);
  if (isnan(x)) {
    ++L.n_nan;
    L.first_nan = min(L.first_nan, idx);
    return;
  }
  if (isinf(x)) {
    if (x > 0.f) ++L.n_pinf;
    else ++L.n_ninf;
    L.first_inf = min(L.first_inf, idx);
    return;
  }
  if (x == 0.f) ++L.n_zero;
  L.mn = fminf(L.mn, x);
  L.mx = fmaxf(L.mx, x);
  const double d = (double)x;
  L.s64 = __dadd_rn(L.s64, d);
  L.q64 = __dadd_rn(L.q64, __dmul_rn(d, d));
}

// -1 if x is a zero of either sign, else 0.
__device__ __forceinline__ int32_t zero_m1(float x) {
  int32_t r;
  asm("set.eq.s32.f32 %0, %1, 0f00000000;" : "=r"(r) : "f"(x));
  return r;
}

// int32 elements (exact): V elements in v, n of them valid.
template <int DT>
__device__ __forceinline__ void lane_int(LaneStat &L, const uint4 &v, int n) {
  constexpr int V = Tr<DT>::V;
#pragma unroll
  for (int k = 0; k < V; ++k) {
    if (k < n) {
      const int32_t x = (int32_t)vbits<DT>(v, k);
      L.n_zero += x == 0;
      L.imn = min(L.imn, x);
      L.imx = max(L.imx, x);
      const int64_t x64 = x;
      add128(L.is_lo, L.is_hi, (uint64_t)x64, x64 < 0 ? ~0ull : 0ull);
      add128(L.iq_lo, L.iq_hi, (uint64_t)(x64 * x64), 0ull);
    }
  }
}

// Float elements, the fast path: V valid elements of any value, no class
// test.  Zeros are counted, min/max taken, and sum(x), sum(x^2) added as
// float-float pairs (TwoSum; x^2 split exactly into fl(x^2) and an fma
// remainder).  The pairs are exact while every |x| lies below 2^57 and the
// remainders are exact for |x| >= 2^-51; a NaN or an infinity leaves a
// non-finite sum.  The unit's end test (lane_fast_ok) decides whether the
// unit's result stands.
template <int DT>
__device__ __forceinline__ void lane_fast(LaneStat &L, const uint4 &v) {
  constexpr int V = Tr<DT>::V;
  float x[V];
#pragma unroll
  for (int k = 0; k < V; ++k) x[k] = vdec<DT>(v, k);
  int32_t z = 0;
  float mn = x[0], mx = x[0];
#pragma unroll
  for (int k = 0; k < V; ++k) z += zero_m1(x[k]);
#pragma unroll
  for (int k = 1; k < V; ++k) {
    mn = fminf(mn, x[k]);
    mx = fmaxf(mx, x[k]);
  }
  L.n_zero -= z;
  L.mn = fminf(L.mn, mn);
  L.mx = fmaxf(L.mx, mx);
#pragma unroll
  for (int k = 0; k < V; k += 2) {
    const float2 p = make_float2(x[k], x[k + 1]);
    ff_add2(L.sh, L.sl, p);
    const float2 sq = __fmul2_rn(p, p);
    const float2 pe = __ffma2_rn(p, p, __fmul2_rn(sq, make_float2(-1.f, -1.f)));
    ff_add2(L.qh, L.ql, sq);
    L.ql = __fadd2_rn(L.ql, pe);
  }
  if (++L.pending == kFlush) lane_fold(L);
}

// Every element of a whole vector zero or of magnitude in [2^-50, 2^57):
// the fast path adds such vectors exactly (the unit's second pass takes the
// others element by element).
template <int DT>
__device__ __forceinline__ bool vec_in_range(const uint4 &v) {
  constexpr int V = Tr<DT>::V;
  bool ok = true;
#pragma unroll
  for (int k = 0; k < V; ++k) {
    const uint32_t m = __float_as_uint(vdec<DT>(v, k)) & 0x7fffffffu;
    ok = ok && (m == 0u || m - 0x26800000u < 0x5c000000u - 0x26800000u);
  }
  return ok;
}

// A whole vector on the unit's second pass; its first element at index e.
template <int DT>
__device__ __forceinline__ void lane_checked(LaneStat &L, const uint4 &v, int64_t e) {
  constexpr int V = Tr<DT>::V;
  if (vec_in_range<DT>(v)) {
    lane_fast<DT>(L, v);
  } else {
#pragma unroll
    for (int q = 0; q < V; ++q) lane_slow<DT>(L, vbits<DT>(v, q), e + q);
  }
}

// After the final fold: the fast path's result stands when the sums are
// finite (no NaN or infinity met) and the largest magnitude a lies in
// [2^-44, 2^57) (or every element is zero).  Below 2^-51 a square's
// remainder may round, by at most 2^-150 per element; a unit has at most
// 2^14 elements and sum(x^2) >= a^2 >= 2^-88, so the relative error stays
// below 2^-48.
__device__ __forceinline__ bool lane_fast_ok(const LaneStat &L) {
  const float a = fmaxf(-L.mn, L.mx);  // -inf for a lane without elements
  return isfinite(L.s64) && isfinite(L.q64) && a < 0x1p57f && !(a > 0.f && a < 0x1p-44f);
}

// One unit's elements into a lane's sums.  The unit is rows [r0, r1) x
// columns [c0, c0 + cols) of the [M, N] view, cols at most
// kUnitCols elements; a row holds vpr vectors.  When vpr >= 32 a row is
// swept in windows of 32 vectors, lane l taking vector l of each window in
// every row; narrower rows are stacked, S = 32 / vpr rows per step.  Each
// lane walks its rows with a fixed byte stride, the loads software-pipelined
// (the next four rows in flight while four are added up).
// MODE 0: int32 (exact); 1: float fast path (whole vectors; partial
// vectors element by element); 2: float, the unit's second pass: whole
// vectors in range on the fast path, the rest element by element.
template <int DT, int MODE>
__device__ __forceinline__ void unit_sweep(LaneStat &L, const char *base, bool vec_ok, int64_t N, int64_t r0,
                                           int64_t r1, int64_t c0, int64_t cols, int lane) {
  constexpr int V = Tr<DT>::V;
  constexpr int EB = Tr<DT>::EB;
  const int32_t vpr = (int32_t)((cols + V - 1) / V);
  const int32_t VW = vpr < 32 ? vpr : 32;  // lanes per row
  const int32_t S = 32 / VW;               // rows per step
  const int32_t rsub = lane / VW, vl = lane - rsub * VW;
  if (rsub >= S) return;
  const int32_t nw = (vpr + 31) / 32;
  const int64_t nr = (r1 - r0 - rsub + S - 1) / S;  // this lane's rows
  const int64_t stride = (int64_t)S * N;            // elements between them
  for (int32_t w = 0; w < nw; ++w) {
    const int32_t vi = w * 32 + vl;
    if (vi >= vpr) break;
    const int64_t left = cols - (int64_t)vi * V;
    const int n = left < V ? (int)left : V;
    int64_t e = (r0 + rsub) * N + c0 + (int64_t)vi * V;  // the lane's first element in this window
    if (vec_ok && n == V) {
      const char *p = base + e * EB;
      const int64_t sb = stride * EB;
      int64_t k = 0;
      if constexpr (MODE != 2) {
        // software-pipelined: the next four rows' loads go out before this
        // four rows' arithmetic (eight 16-byte loads in flight per lane)
        if (nr >= 4) {
          uint4 a0 = ld_v4(p), a1 = ld_v4(p + sb), a2 = ld_v4(p + 2 * sb), a3 = ld_v4(p + 3 * sb);
          p += 4 * sb;
          for (k = 4; k + 4 <= nr; k += 4) {
            const uint4 b0 = ld_v4(p), b1 = ld_v4(p + sb), b2 = ld_v4(p + 2 * sb), b3 = ld_v4(p + 3 * sb);
            p += 4 * sb;
            if constexpr (MODE == 0) {
              lane_int<DT>(L, a0, V);
              lane_int<DT>(L, a1, V);
              lane_int<DT>(L, a2, V);
              lane_int<DT>(L, a3, V);
            } else {
              lane_fast<DT>(L, a0);
              lane_fast<DT>(L, a1);
              lane_fast<DT>(L, a2);
              lane_fast<DT>(L, a3);
            }
            a0 = b0;
            a1 = b1;
            a2 = b2;
            a3 = b3;
          }
          if constexpr (MODE == 0) {
            lane_int<DT>(L, a0, V);
            lane_int<DT>(L, a1, V);
            lane_int<DT>(L, a2, V);
            lane_int<DT>(L, a3, V);
          } else {
            lane_fast<DT>(L, a0);
            lane_fast<DT>(L, a1);
            lane_fast<DT>(L, a2);
            lane_fast<DT>(L, a3);
          }
        }
      }
      for (; k + 4 <= nr; k += 4) {
        const uint4 v0 = ld_v4(p), v1 = ld_v4(p + sb), v2 = ld_v4(p + 2 * sb), v3 = ld_v4(p + 3 * sb);
        p += 4 * sb;
        if constexpr (MODE == 0) {
          lane_int<DT>(L, v0, V);
          lane_int<DT>(L, v1, V);
          lane_int<DT>(L, v2, V);
          lane_int<DT>(L, v3, V);
        } else if constexpr (MODE == 1) {
          lane_fast<DT>(L, v0);
          lane_fast<DT>(L, v1);
          lane_fast<DT>(L, v2);
          lane_fast<DT>(L, v3);
        } else {
          lane_checked<DT>(L, v0, e);
          lane_checked<DT>(L, v1, e + stride);
          lane_checked<DT>(L, v2, e + 2 * stride);
          lane_checked<DT>(L, v3, e + 3 * stride);
          e += 4 * stride;
        }
      }
      for (; k < nr; ++k) {
        const uint4 v0 = ld_v4(p);
        p += sb;
        if constexpr (MODE == 0) {
          lane_int<DT>(L, v0, V);
        } else if constexpr (MODE == 1) {
          lane_fast<DT>(L, v0);
        } else {
          lane_checked<DT>(L, v0, e);
          e += stride;
        }
      }
    } else {
      for (int64_t k = 0; k < nr; ++k, e += stride) {
        uint32_t wd[4] = {0, 0, 0, 0};
#pragma unroll
        for (int q = 0; q < V; ++q) {
          if (q < n) {
            const uint32_t b = ld_one<EB>(base, e + q);
            if constexpr (EB == 2) wd[q >> 1] |= b << (16 * (q & 1));
            else wd[q] = b;
          }
        }
        const uint4 v = make_uint4(wd[0], wd[1], wd[2], wd[3]);
        if constexpr (MODE == 0) {
          lane_int<DT>(L, v, n);
        } else if (MODE == 1 && n == V) {
          lane_fast<DT>(L, v);
        } else if (MODE == 2 && n == V) {
          lane_checked<DT>(L, v, e);
        } else {
#pragma unroll
          for (int q = 0; q < V; ++q)
            if (q < n) lane_slow<DT>(L, vbits<DT>(v, q), e + q);
        }
      }
    }
  }
}

// ------------------------------------------------------------ the scan
// cases: the launch's cases (all of element type DT), ascending unit
// ranges; units [unit_base, unit_base + n_units) are theirs.
template <int DT>
__global__ void __launch_bounds__(kStatThreads) stats_kernel(const StatsDesc *__restrict__ cases, int n_cases,
                                                            int64_t unit_base, int64_t n_units,
                                                            unsigned long long *unit_ctr, StatPart *parts) {
  const int lane = threadIdx.x & 31;
  for (;;) {
    int64_t u = 0;
    if (lane == 0) u = (int64_t)atomicAdd(unit_ctr, 1ull);
    u = __shfl_sync(0xffffffffu, u, 0);
    if (u >= n_units) break;
    u += unit_base;
    // the unit's case (cases of this element type, ascending unit ranges)
    int lo = 0, hi = n_cases - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (cases[mid].unit_begin <= u) lo = mid;
      else hi = mid - 1;
    }
    const StatsDesc &d = cases[lo];
    const int64_t lu = u - d.unit_begin;
    const int64_t per_tile = d.ch * d.cc;
    const int64_t t = lu / per_tile, rem = lu - t * per_tile;
    const int64_t kr = rem / d.cc, kc = rem - kr * d.cc;
    const int64_t tr = t / d.GC, tc = t - tr * d.GC;
    const int64_t tr0 = tr * d.th, tc0 = tc * d.tw;
    const int64_t r0 = tr0 + kr * d.rch;
    const int64_t r1 = min(min(r0 + d.rch, tr0 + d.th), d.M);
    const int64_t c0 = tc0 + kc * d.cw;
    const int64_t c1 = min(min(c0 + d.cw, tc0 + d.tw), d.N);
    const int64_t rows = r1 > r0 ? r1 - r0 : 0, cols = c1 > c0 ? c1 - c0 : 0;
    const char *base = (const char *)d.x;
    LaneStat L;
    lane_init(L);
    if (rows > 0 && cols > 0) {
      const bool vec_ok = d.vec_ok != 0;
      const int64_t N = d.N;
      if constexpr (Tr<DT>::kInt) {
        unit_sweep<DT, 0>(L, base, vec_ok, N, r0, r1, c0, cols, lane);
      } else {
        unit_sweep<DT, 1>(L, base, vec_ok, N, r0, r1, c0, cols, lane);
        lane_fold(L);
        if (__any_sync(0xffffffffu, !lane_fast_ok(L))) {  // the unit again, element by element
          lane_init(L);
          unit_sweep<DT, 2>(L, base, vec_ok, N, r0, r1, c0, cols, lane);
          lane_fold(L);
        }
      }
    }
    // lanes -> the unit's partial (fixed butterfly; every lane ends with it)
    StatPart p;
    part_init(p);
    p.n = lane == 0 ? rows * cols : 0;
    p.cnt[0] = L.n_nan;
    p.cnt[1] = L.n_pinf;
    p.cnt[2] = L.n_ninf;
    p.cnt[3] = L.n_zero;
    p.first_nan = L.first_nan;
    p.first_inf = L.first_inf;
    if constexpr (Tr<DT>::kInt) {
      p.mn = L.imn <= L.imx ? (double)L.imn : INFINITY;
      p.mx = L.imn <= L.imx ? (double)L.imx : -INFINITY;
      p.is_lo = L.is_lo;
      p.is_hi = L.is_hi;
      p.iq_lo = L.iq_lo;
      p.iq_hi = L.iq_hi;
    } else {
      p.mn = L.mn <= L.mx ? (double)L.mn : INFINITY;
      p.mx = L.mn <= L.mx ? (double)L.mx : -INFINITY;
      p.s = L.s64;
      p.q = L.q64;
    }
#pragma unroll 1
    for (int o = 16; o; o >>= 1) {
      const StatPart b = part_shfl(p, o);
      part_merge(p, b);
    }
    if (lane == 0) parts[u] = p;
  }
}

// ---------------------------------------------------------- the finalize
// grid (n_cases, kFinBlocks): block b of case c merges tiles b, b + B, ...
// (B = that case's fin_blocks) and their units, writes each tile's record
// to the host result, and leaves a block partial; the case's last block
// to finish merges the block partials in block order into the tensor's
// statistics.
__global__ void __launch_bounds__(kStatThreads) stats_fin_kernel(const StatsDesc *__restrict__ cases,
                                                                const StatPart *__restrict__ parts,
                                                                StatPart *bparts, unsigned int *done,
                                                                uint8_t *host) {
  const int64_t c = blockIdx.x;
  const int64_t blk = blockIdx.y;
  const StatsDesc &d = cases[c];
  const int64_t B = d.fin_blocks;
  if (blk >= B) return;
  const int64_t tiles = d.GR * d.GC, per_tile = d.ch * d.cc;
  nmv_stat *hrec = (nmv_stat *)(host + d.tiles_off);
  __shared__ StatPart sh[kStatThreads];
  StatPart acc;
  part_init(acc);
  if (per_tile < kCoopUnits) {
    // thread t of block b takes tiles b + B (t + 256 j), ascending
    for (int64_t t = blk + B * threadIdx.x; t < tiles; t += B * kStatThreads) {
      StatPart tp;
      part_init(tp);
      const StatPart *up = parts + d.unit_begin + t * per_tile;
      for (int64_t j = 0; j < per_tile; ++j) part_merge(tp, up[j]);
      nmv_stat rec;
      part_out(tp, d.dtype, &rec);
      hrec[t] = rec;
      part_merge(acc, tp);
    }
  } else {
    // tiles of many units: block b takes tiles b, b + B, ...; thread t
    // merges units t, t + 256, ... of the tile, then the threads in a fixed
    // tree
    for (int64_t t = blk; t < tiles; t += B) {
      StatPart tp;
      part_init(tp);
      const StatPart *up = parts + d.unit_begin + t * per_tile;
      for (int64_t j = threadIdx.x; j < per_tile; j += kStatThreads) part_merge(tp, up[j]);
      sh[threadIdx.x] = tp;
      __syncthreads();
      for (int o = kStatThreads / 2; o; o >>= 1) {
        if ((int)threadIdx.x < o) part_merge(sh[threadIdx.x], sh[threadIdx.x + o]);
        __syncthreads();
      }
      if (threadIdx.x == 0) {
        nmv_stat rec;
        part_out(sh[0], d.dtype, &rec);
        hrec[t] = rec;
        part_merge(acc, sh[0]);
      }
      __syncthreads();
    }
  }
  // the block's threads in a fixed tree
  sh[threadIdx.x] = acc;
  __syncthreads();
  for (int o = kStatThreads / 2; o; o >>= 1) {
    if ((int)threadIdx.x < o) part_merge(sh[threadIdx.x], sh[threadIdx.x + o]);
    __syncthreads();
  }
  __shared__ bool last;
  if (threadIdx.x == 0) {
    bparts[d.bpart_off + blk] = sh[0];
    __threadfence();
    last = atomicAdd(&done[c], 1u) == (unsigned)(B - 1);
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  if (threadIdx.x == 0) {
    StatPart all;
    part_init(all);
    const StatPart *bp = bparts + d.bpart_off;
    for (int64_t b = 0; b < B; ++b) {
      // the other blocks' partials, read from L2 (not a stale L1 line)
      StatPart q;
      const unsigned long long *src = (const unsigned long long *)&bp[b];
      unsigned long long *dst = (unsigned long long *)&q;
      for (int w = 0; w < (int)(sizeof(StatPart) / 8); ++w) dst[w] = __ldcg(src + w);
      part_merge(all, q);
    }
    nmv_stats_result *res = (nmv_stats_result *)(host + d.res_off);
    nmv_stat rec;
    part_out(all, d.dtype, &rec);
    res->all = rec;
    res->first_nan = all.first_nan == INT64_MAX ? -1 : all.first_nan;
    res->first_inf = all.first_inf == INT64_MAX ? -1 : all.first_inf;
    done[c] = 0;  // ready for the next call
  }
}


// ------------------------------------------------------------------ host
namespace {

struct StatsWorkspace {
  void *p = nullptr;
  size_t size = 0;
};
StatsWorkspace g_sws[64];

// Units of a tile: column chunks of at most kUnitCols elements, row chunks
// of at most kUnitElems / (chunk columns) rows, over the extent a tile
// actually has (a tile taller or wider than the view is cut to it).
void unit_geometry(StatsDesc &d) {
  const int64_t er = std::max<int64_t>(1, std::min(d.th, d.M)), ec = std::max<int64_t>(1, std::min(d.tw, d.N));
  d.cw = std::min<int64_t>(ec, kUnitCols);
  d.cc = (ec + d.cw - 1) / d.cw;
  d.rch = std::max<int64_t>(1, std::min<int64_t>(er, kUnitElems / d.cw));
  d.ch = (er + d.rch - 1) / d.rch;
}

template <int DT>
cudaError_t launch_stats_dt(int sms, const StatsDesc *cases, int n_cases, int64_t unit_base, int64_t n_units,
                            unsigned long long *ctr, StatPart *parts, cudaStream_t st) {
  int occ = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, stats_kernel<DT>, kStatThreads, 0);
  if (e != cudaSuccess) return e;
  int64_t grid = (int64_t)sms * std::max(occ, 1);
  grid = std::min<int64_t>(grid, (n_units + 7) / 8);
  stats_kernel<DT><<<(int)std::max<int64_t>(grid, 1), kStatThreads, 0, st>>>(cases, n_cases, unit_base, n_units,
                                                                             ctr, parts);
  return cudaGetLastError();
}

cudaError_t launch_stats(int dt, int sms, const StatsDesc *cases, int n_cases, int64_t unit_base, int64_t n_units,
                         unsigned long long *ctr, StatPart *parts, cudaStream_t st) {
  switch (dt) {
    case NMV_F32: return launch_stats_dt<NMV_F32>(sms, cases, n_cases, unit_base, n_units, ctr, parts, st);
    case NMV_F16: return launch_stats_dt<NMV_F16>(sms, cases, n_cases, unit_base, n_units, ctr, parts, st);
    case NMV_BF16: return launch_stats_dt<NMV_BF16>(sms, cases, n_cases, unit_base, n_units, ctr, parts, st);
    default: return launch_stats_dt<NMV_I32>(sms, cases, n_cases, unit_base, n_units, ctr, parts, st);
  }
}

size_t align_to(size_t x, size_t a) { return (x + a - 1) / a * a; }

constexpr int64_t kMaxStatUnits = int64_t(1) << 26;  // unit partials of one call

int run_stats(const nmv_stats_case *cases, int64_t n, void *stream, nmv_stats_result **out) {
  if (out == nullptr) return host_fail(NMV_EINVAL, "out is NULL");
  *out = nullptr;
  if (cases == nullptr && n > 0) return host_fail(NMV_EINVAL, "cases is NULL");
  if (n < 0 || n > NMV_MAX_CASES) return host_fail(NMV_EINVAL, "case count out of range");
  std::vector<StatsDesc> desc((size_t)n);
  std::vector<int64_t> order((size_t)n);
  int64_t tiles_total = 0;
  for (int64_t i = 0; i < n; ++i) {
    const nmv_stats_case &c = cases[i];
    char pre[64];
    std::snprintf(pre, sizeof pre, "case %lld: ", (long long)i);
    const nmv_tensor &x = c.x;
    if (x.dtype < NMV_F32 || x.dtype > NMV_I32) return host_fail(NMV_EINVAL, std::string(pre) + "unknown dtype");
    const int64_t numel = host_tensor_numel(x);
    if (numel < 0) return host_fail(NMV_EINVAL, std::string(pre) + "invalid rank or shape");
    if (numel > 0 && x.data == nullptr) return host_fail(NMV_EINVAL, std::string(pre) + "NULL data");
    if (c.tile_rows < 1 || c.tile_cols < 1 || c.tile_rows > NMV_MAX_TILE || c.tile_cols > NMV_MAX_TILE)
      return host_fail(NMV_EINVAL, std::string(pre) + "tile_rows and tile_cols must lie in [1, NMV_MAX_TILE]");
    StatsDesc &d = desc[(size_t)i];
    std::memset(&d, 0, sizeof(d));
    d.x = x.data;
    d.dtype = x.dtype;
    d.numel = numel;
    d.N = x.rank == 0 ? 1 : x.shape[x.rank - 1];
    d.M = 1;
    for (int k = 0; k + 1 < x.rank; ++k) d.M *= x.shape[k];
    d.th = c.tile_rows;
    d.tw = c.tile_cols;
    d.GR = numel ? (d.M + d.th - 1) / d.th : 0;
    d.GC = numel ? (d.N + d.tw - 1) / d.tw : 0;
    if (d.GC > 0 && d.GR > NMV_MAX_STAT_TILES / d.GC)
      return host_fail(NMV_EINVAL, std::string(pre) + "tile grid exceeds NMV_MAX_STAT_TILES tiles");
    unit_geometry(d);
    // 16-byte loads need every unit row segment to start 16-byte aligned:
    // row starts (N), tile columns (tw, when there are several) and unit
    // column chunks (cw)
    const int eb = elem_bytes(d.dtype);
    d.vec_ok = ((uintptr_t)x.data % 16 == 0) && (d.N * eb) % 16 == 0 && (d.GC <= 1 || (d.tw * eb) % 16 == 0) &&
               (d.cw * eb) % 16 == 0;
    tiles_total += d.GR * d.GC;
  }
  // cases grouped by element type (one scan launch each); results keep the
  // caller's order
  for (int64_t i = 0; i < n; ++i) order[(size_t)i] = i;
  std::stable_sort(order.begin(), order.end(),
                   [&](int64_t a, int64_t b) { return desc[(size_t)a].dtype < desc[(size_t)b].dtype; });
  const size_t res_bytes = align_to(sizeof(nmv_stats_result) * (size_t)std::max<int64_t>(n, 1), 256);
  std::vector<StatsDesc> dd((size_t)n);
  int64_t units = 0, bparts = 0, max_fb = 1;
  size_t tile_off = res_bytes;
  for (int64_t j = 0; j < n; ++j) {
    const int64_t i = order[(size_t)j];
    StatsDesc d = desc[(size_t)i];
    const int64_t tiles = d.GR * d.GC;
    d.unit_begin = units;
    units += tiles * d.ch * d.cc;
    d.unit_end = units;
    d.fin_blocks = d.ch * d.cc >= kCoopUnits
                       ? std::max<int64_t>(1, std::min<int64_t>(kFinBlocks, tiles))
                       : std::max<int64_t>(1, std::min<int64_t>(kFinBlocks, (tiles + kStatThreads - 1) / kStatThreads));
    d.bpart_off = bparts;
    bparts += d.fin_blocks;
    max_fb = std::max(max_fb, d.fin_blocks);
    d.res_off = (int64_t)(sizeof(nmv_stats_result) * (size_t)i);
    d.tiles_off = (int64_t)tile_off;
    tile_off += sizeof(nmv_stat) * (size_t)tiles;
    dd[(size_t)j] = d;
  }
  if (units > kMaxStatUnits) return host_fail(NMV_EINVAL, "too many tiles and tile chunks in one call");
  if (n == 0) return NMV_OK;

  std::lock_guard<std::mutex> lock(host_mutex());
  int dev = -1, sms = 0;
  size_t smem_optin = 0;
  int rc = host_probe(&dev, &sms, &smem_optin);
  if (rc) return rc;
  if (dev >= 64) return host_fail(NMV_EUNSUPPORTED, "device ordinal out of range");
  cudaStream_t st = (cudaStream_t)stream;

  // workspace: descriptors, counters (one per element type, one per case),
  // block partials, unit partials
  const size_t sz_desc = align_to(sizeof(StatsDesc) * (size_t)n, 256);
  const size_t sz_ctr = align_to(8 * 4 + 4 * (size_t)n, 256);
  const size_t sz_bp = align_to(sizeof(StatPart) * (size_t)bparts, 256);
  const size_t sz_up = align_to(sizeof(StatPart) * (size_t)std::max<int64_t>(units, 1), 256);
  const size_t need = sz_desc + sz_ctr + sz_bp + sz_up;
  StatsWorkspace &W = g_sws[dev];
  if (host_injected("alloc")) return host_fail(NMV_ENOMEM, "injected allocation failure");
  if (need > W.size) {
    const size_t want = std::max(need, W.size * 2);
    if (W.p) cudaFree(W.p);
    W.p = nullptr;
    W.size = 0;
    const cudaError_t e = cudaMalloc(&W.p, want);
    if (e != cudaSuccess) {
      cudaGetLastError();
      W.p = nullptr;
      return host_fail(NMV_ENOMEM, std::string("cudaMalloc statistics workspace: ") + cudaGetErrorString(e));
    }
    W.size = want;
  }
  uint8_t *ws = (uint8_t *)W.p;
  StatsDesc *d_desc = (StatsDesc *)ws;
  unsigned long long *d_ctr = (unsigned long long *)(ws + sz_desc);
  unsigned int *d_done = (unsigned int *)(ws + sz_desc + 32);
  StatPart *d_bp = (StatPart *)(ws + sz_desc + sz_ctr);
  StatPart *d_up = (StatPart *)(ws + sz_desc + sz_ctr + sz_bp);

  // the results: mapped pinned host memory the finalize writes into
  uint8_t *host = (uint8_t *)host_arena_get(tile_off);
  if (!host) return host_fail(NMV_ENOMEM, "cudaHostAlloc result block");
  struct ArenaGuard {
    uint8_t *p;
    ~ArenaGuard() { host_arena_put(p); }
  } guard{host};
  uint8_t *dhost = nullptr;
  {
    void *dp = nullptr;
    const cudaError_t e = cudaHostGetDevicePointer(&dp, host, 0);
    if (e != cudaSuccess) return host_cuda_fail(e, "cudaHostGetDevicePointer (result block)");
    dhost = (uint8_t *)dp;
  }
  nmv_stats_result *res = (nmv_stats_result *)host;
  for (int64_t j = 0; j < n; ++j) {
    const StatsDesc &d = dd[(size_t)j];
    const int64_t i = order[(size_t)j];
    nmv_stats_result &r = res[i];
    std::memset(&r, 0, sizeof(r));
    r.status = NMV_OK;
    r.rank = cases[i].x.rank;
    r.numel = d.numel;
    r.grid_rows = d.GR;
    r.grid_cols = d.GC;
    r.tile_rows = d.th;
    r.tile_cols = d.tw;
    r.tiles = (nmv_stat *)(host + d.tiles_off);
    r.first_nan = r.first_inf = -1;
  }

  struct DrainOnError {
    cudaStream_t st;
    bool armed = true;
    ~DrainOnError() {
      if (armed) {
        cudaStreamSynchronize(st);
        cudaGetLastError();
      }
    }
  } drain{st};
  cudaError_t e = cudaMemcpyAsync(d_desc, dd.data(), sizeof(StatsDesc) * (size_t)n, cudaMemcpyHostToDevice, st);
  if (e != cudaSuccess) return host_cuda_fail(e, "cudaMemcpyAsync (descriptors)");
  e = cudaMemsetAsync(d_ctr, 0, sz_ctr, st);
  if (e != cudaSuccess) return host_cuda_fail(e, "cudaMemsetAsync");
  for (int64_t j = 0; j < n;) {
    int64_t k = j;
    while (k < n && dd[(size_t)k].dtype == dd[(size_t)j].dtype) ++k;
    const int64_t ub = dd[(size_t)j].unit_begin, ue = dd[(size_t)k - 1].unit_end;
    if (ue > ub) {
      e = launch_stats(dd[(size_t)j].dtype, sms, d_desc + j, (int)(k - j), ub, ue - ub, d_ctr + dd[(size_t)j].dtype,
                       d_up, st);
      if (e != cudaSuccess) return host_cuda_fail(e, "statistics kernel launch");
    }
    j = k;
  }
  stats_fin_kernel<<<dim3((unsigned)n, (unsigned)max_fb), kStatThreads, 0, st>>>(d_desc, d_up, d_bp, d_done, dhost);
  e = cudaGetLastError();
  if (e != cudaSuccess) return host_cuda_fail(e, "statistics finalize launch");
  e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return host_cuda_fail(e, "cudaStreamSynchronize");
  drain.armed = false;
  guard.p = nullptr;  // handed to the caller
  *out = res;
  host_clear_error();
  return NMV_OK;
}

}  // namespace
}  // namespace nmv

extern "C" int nmv_stats(const nmv_stats_case *cases, int64_t n, void *cuda_stream, nmv_stats_result **out) {
  return nmv::run_stats(cases, n, cuda_stream, out);
}
