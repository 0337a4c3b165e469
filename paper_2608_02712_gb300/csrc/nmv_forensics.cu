// nmv_forensics.cu -- deep forensics of a candidate/reference pair
// (nmv_forensics): the evidence behind the adaptive-scheduling rules
// "near-pass and fp16-ceiling detection" (Section 4.4), the localisation of
// a divergence that compounds along a reduction axis (Section 3.2, the
// cumsum of Table 1), and mismatch counts at every index of every axis.
//
// fx_kernel streams the pair once, viewed as R rows of L elements (L the
// last axis), in units of rb rows x g column windows handed to warps from a
// counter.  A window is 32 vectors wide and lane l owns the same V columns
// in every row of it, so the last axis' mismatch marginal (and, when the
// growth axis is the last one, the growth maxima of those columns) stay in
// the lane's registers until the window ends; the leading axes' marginals
// take one warp sum per row, gathered in the warp's shared row counters
// until the unit ends.  Per element: the predicate with the scan's fp32
// pre-filter (fp64 where the filter cannot decide), the ulp distance of the
// two stored values into a lane-private shared-memory histogram (laid out
// [warp][bin][lane], so each lane's bins sit in its own bank), and for
// mismatches the largest-ulp record and the fp16-spacing test, decided
// exactly from the fp32 difference and its TwoSum remainder.  The growth
// curve max |c - r| per index of the chosen axis is kept exact as
// (|fl32(c - r)|, remainder) pairs and written as fp64 maxima with atomics
// (maxima do not depend on the order) after an fp32 screen against each
// bin's lower bound.
// fx_fin_kernel reduces the blocks' largest-ulp candidates in block order
// and writes every field into the mapped host result.
#include <cuda_runtime.h>

#include <algorithm>
#include <cfloat>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "nmv_scan.cuh"

namespace nmv {

constexpr int kFxThreads = 256;
constexpr int kFxHistBytes = (kFxThreads / 32) * NMV_ULP_BINS * 32 * 4;  // [warp][bin][lane] ulp histograms
constexpr int64_t kFxRowsMax = 256;   // rows of a unit at most
constexpr int kFxRowBytes = (kFxThreads / 32) * (int)kFxRowsMax * 4;  // [warp][row] mismatch counts
constexpr int64_t kFxGrowCap = 2048;  // growth bins privatised in shared memory
constexpr int64_t kFxMargCap = 4096;  // marginal bins privatised in shared memory
constexpr int64_t kFxUnitElems = 65536;  // elements of a unit (rows x window columns), when the rows allow

struct FxDesc {
  const void *cand, *ref;
  int32_t dtype, vec_ok;    // vec_ok: every row of the [R, L] view starts 16-byte aligned in both tensors
  int32_t rank, axis;
  int32_t grow_smem, marg_smem, j_is_row, pad;
  int64_t numel;
  int64_t L, R;             // the pair as R rows of L elements (L the last axis; 1 x 1 for rank 0)
  int64_t CWn, rb, g, WG;   // column windows of 32 vectors; a unit is rb rows x g windows
  int64_t RBn, n_units;     // row blocks; units (row block fastest)
  int64_t shape[NMV_MAX_RANK];
  Div64 sdiv[NMV_MAX_RANK];
  int64_t marg_off[NMV_MAX_RANK + 1];
  int64_t axis_len;
  Div64 dstride, dlen;      // coordinate on the axis: (i / stride) % len
  Div64 drs;                // growth axis before the last: rows per index (row rho -> (rho / rs) % len)
  float lo_r, lo_a, hi_r, hi_a;  // fp32 pre-filter of the predicate (as nmv_validate)
  double rtol, atol;
  int64_t near_ulps;
  double near_fraction, growth_factor;
  int64_t res_off, growth_off, marg_off_host;  // byte offsets in the host result block
};

// Device accumulators of one case (cleared before its launch).
struct FxAcc {
  unsigned long long hist[NMV_ULP_BINS];
  unsigned long long mismatch, n_finite, nonfin, within;
  unsigned long long unit_ctr;  // units handed out
};

struct FxBest {
  long long u, idx;  // largest ulp distance of a finite mismatch (-1: none) and its lowest index
};

// Per-lane totals.  A lane sees at most numel / 32 elements, below 2^32 for
// any pair that fits in device memory.
struct FxLane {
  uint32_t mism, nfin, nonfin, within;
  uint32_t bu;   // largest ulp distance of a finite mismatch (0: none; a finite mismatch has u >= 1)
  int64_t bi;    // its lowest index
};

// |ord(c) - ord(r)|, ord the stored sign-magnitude bits as a signed integer
// that orders like the values with both zeros at 0 (two's complement int32
// as it is); below 2^32 for every type (fp32 magnitudes of finite values are
// at most 0x7f7fffff).  Float types through the key k(b) = magnitude for a
// positive sign, -1 - magnitude for a negative one (one xor): k orders like
// ord and differs from it by -1 on negative signs, so |ord(c) - ord(r)| =
// |k(c) - k(r)| - [the signs differ] (16-bit types: the bits moved to the
// top half, where the -1 falls below the magnitudes and the shift back
// drops it).
template <int DT>
__device__ __forceinline__ uint32_t ulp_dist(uint32_t cb, uint32_t rb) {
  if constexpr (Tr<DT>::kInt) {
    const int32_t a = (int32_t)cb, b = (int32_t)rb;
    return a >= b ? (uint32_t)a - (uint32_t)b : (uint32_t)b - (uint32_t)a;
  } else {
    constexpr int kSh = Tr<DT>::EB == 2 ? 16 : 0;   // 16-bit bits moved to the top, sign in bit 31
    const int32_t c = (int32_t)(cb << kSh), r = (int32_t)(rb << kSh);
    const int32_t kc = c ^ ((c >> 31) & 0x7fffffff), kr = r ^ ((r >> 31) & 0x7fffffff);
    const uint32_t d = kc >= kr ? (uint32_t)kc - (uint32_t)kr : (uint32_t)kr - (uint32_t)kc;
    if constexpr (kSh != 0) return d >> kSh;  // the keys' -1 sits below the shifted magnitudes
    else return d - (((uint32_t)(c ^ r)) >> 31);
  }
}

// t with a - b = s + t exactly, s = fl32(a - b) finite (TwoSum; the
// intrinsics keep every step a separately rounded operation).
__device__ __forceinline__ float twosum_err(float a, float b, float s) {
  const float nb = -b;
  const float bb = __fsub_rn(s, a);
  return __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(nb, bb));
}

// A running maximum of |c - r| (the growth curve).  Float types: the exact
// value as S + T, S = |fl32(c - r)| and T the TwoSum remainder signed
// toward S.  |T| is at most half an ulp of S (a quarter below a power of
// two), so the pairs order lexicographically like the exact values, and
// fl64(S + T) is the fp64 |c - r| (one rounding of the exact value).
// int32: the exact |c - r| (below 2^32).
template <int DT, bool INT = Tr<DT>::kInt>
struct GAcc {
  float S = 0.f, T = 0.f;
};
template <int DT>
struct GAcc<DT, true> {
  uint32_t U = 0u;
};

// An element whose fp32 difference overflowed (|c - r| > FLT_MAX, c and r
// finite): its fp64 |c - r| goes straight to the growth bin of its index.
__device__ __noinline__ void grow_direct(const FxDesc &d, int64_t i, double v, unsigned long long *gmax,
                                         uint32_t *glb) {
  int64_t j = 0;
  if (d.rank > 0) {
    const uint64_t q = div_q((uint64_t)i, d.dstride.d, d.dstride.m);
    j = (int64_t)(q - div_q(q, d.dlen.d, d.dlen.m) * d.dlen.d);
  }
  atomicMax(&gmax[j], (unsigned long long)__double_as_longlong(v));
  atomicMax(&glb[j], __float_as_uint(__double2float_rd(v)));
}

// One maximum at growth index j, unless the bin's fp32 lower bound already
// exceeds it: fl32(S (1 + 2^-22)) is above S + |T| (and fl32(U) is within
// 2^-24 of U).
template <int DT>
__device__ __forceinline__ void grow_flush(const GAcc<DT> &g, int64_t j, unsigned long long *gmax, uint32_t *glb) {
  double v;
  if constexpr (Tr<DT>::kInt) {
    if (g.U == 0u || __fmul_rn(__uint2float_rn(g.U), 1.0f + 0x1p-22f) < __uint_as_float(glb[j])) return;
    v = (double)g.U;
  } else {
    if (g.S == 0.f || __fmul_rn(g.S, 1.0f + 0x1p-22f) < __uint_as_float(glb[j])) return;
    v = __dadd_rn((double)g.S, (double)g.T);
  }
  atomicMax(&gmax[j], (unsigned long long)__double_as_longlong(v));
  atomicMax(&glb[j], __float_as_uint(__double2float_rd(v)));
}

// A float pair's exact |c - r| into a running maximum (S, T).
template <typename GA>
__device__ __forceinline__ void gacc_add(GA &g, float cf, float rf, float s, float as) {
  const float t = twosum_err(cf, rf, s), tp = s > 0.f ? t : -t;
  if (as > g.S || tp > g.T) {
    g.S = as;
    g.T = tp;
  }
}

// One element: counts, ulp histogram, growth, the predicate (the scan's
// fp32 pre-filter, fp64 where it cannot decide) and, for a mismatch, the
// largest-ulp record and the fp16-spacing test.  Returns true on mismatch.
// Growth: with AXL the element's column maximum g is made exact at once
// when the element can raise it; otherwise rmax takes |fl32(c - r)| and
// the row's exact maximum is found at the row's end.
template <int DT, bool AXL, typename GA>
__device__ __forceinline__ bool fx_el(const FxDesc &d, FxLane &L, uint32_t cb, uint32_t rb, int64_t i,
                                      uint32_t hist_sa, GA &g, float &rmax, unsigned long long *gmax, uint32_t *glb) {
  if constexpr (Tr<DT>::kInt) {
    const int32_t c = (int32_t)cb, r = (int32_t)rb;
    const uint32_t u = ulp_dist<DT>(cb, rb);  // = |c - r|
    ++L.nfin;
    sh_add_at(hist_sa + 128u * (u ? 32 - __clz(u) : 0), 1);
    g.U = max(g.U, u);
    if (u == 0u) return false;
    const float as = __uint2float_rn(u), ar = fabsf(__int2float_rn(r));
    bool pass;
    if (as <= __fmaf_rz(d.lo_r, ar, d.lo_a)) pass = true;
    else if (as > __fmaf_ru(d.hi_r, ar, d.hi_a)) pass = false;
    else pass = pass64((double)c, (double)r, d.rtol, d.atol);
    if (pass) return false;
    ++L.mism;
    if (u >= L.bu && (u > L.bu || i < L.bi)) {
      L.bu = u;
      L.bi = i;
    }
    // one fp16 spacing 2^(max(floor(log2 |r|), -14) - 10) is below 1 for
    // |r| < 2^10, where no integer mismatch lies within it
    const uint32_t mr = r < 0 ? 0u - (uint32_t)r : (uint32_t)r;
    if (mr >= 1024u && u <= (1u << (21 - __clz(mr)))) ++L.within;
    return true;
  } else {
    const float cf = to_f32<DT>(cb), rf = to_f32<DT>(rb);
    const float s = __fsub_rn(cf, rf), as = fabsf(s);
    const bool fin = fabsf(cf) <= FLT_MAX && fabsf(rf) <= FLT_MAX;
    const uint32_t u = ulp_dist<DT>(cb, rb);  // meaningful for finite pairs
    L.nfin += fin ? 1u : 0u;
    sh_add_at(hist_sa + 128u * (u ? 32 - __clz(u) : 0), fin ? 1 : 0);
    if constexpr (AXL) {
      if (fin && as >= g.S) {  // a possible new maximum: make it exact
        if (as <= FLT_MAX) gacc_add(g, cf, rf, s, as);
        else grow_direct(d, i, fabs(__dsub_rn((double)cf, (double)rf)), gmax, glb);
      }
    } else {
      rmax = fmaxf(rmax, fin ? as : 0.f);
    }
    const float ar = fabsf(rf);
    bool pass = cf == rf || (fin && as <= __fmaf_rz(d.lo_r, ar, d.lo_a));
    if (!pass && fin && !(as > __fmaf_ru(d.hi_r, ar, d.hi_a))) pass = pass64((double)cf, (double)rf, d.rtol, d.atol);
    if (pass) return false;
    ++L.mism;
    if (!fin) {
      ++L.nonfin;
      return true;
    }
    if (u >= L.bu && (u > L.bu || i < L.bi)) {
      L.bu = u;
      L.bi = i;
    }
    // fl64(|c - r|) <= h, h = 2^(max(e, -14) - 10) with e the fp32 exponent
    // of r (floor(log2 |r|) for normal r; fp32 subnormals and zero lie below
    // 2^-14 and give 2^-24 alike).  |s| < h or |s| > h decides it (|s| and h
    // are fp32 numbers, the remainder is below half an ulp of s); at |s| = h
    // the exact value h + T rounds to h in fp64 iff T <= 2^-53 h.
    const uint32_t E = (__float_as_uint(rf) >> 23) & 0xffu;
    const float h = __uint_as_float((max(E, 113u) - 10u) << 23);
    bool w = as < h;
    if (as == h) {
      const float t = twosum_err(cf, rf, s), tp = s > 0.f ? t : -t;
      w = tp <= __fmul_rn(h, 0x1p-53f);
    }
    L.within += w ? 1u : 0u;
    return true;
  }
}

// The marginals of the leading axes (all but the last) for row rho of the
// [R, L] view: its coordinates, each bin + n.
__device__ __noinline__ void marg_rows(const FxDesc &d, int64_t rho, uint32_t n, uint32_t *smarg,
                                       unsigned long long *gmarg) {
  uint64_t rest = (uint64_t)rho;
  for (int a = d.rank - 2; a >= 0; --a) {
    const uint64_t q = div_q(rest, d.sdiv[a].d, d.sdiv[a].m);
    const int64_t bin = d.marg_off[a] + (int64_t)(rest - q * d.sdiv[a].d);
    rest = q;
    if (d.marg_smem) atomicAdd(&smarg[bin], n);
    else gl_add(&gmarg[bin], (unsigned long long)n);
  }
}

// The growth index of row rho for an axis before the last: (rho / rs) % len.
__device__ __forceinline__ int64_t row_gidx(const FxDesc &d, int64_t rho) {
  if (d.j_is_row) return rho;
  const uint64_t q = div_q((uint64_t)rho, d.drs.d, d.drs.m);
  return (int64_t)(q - div_q(q, d.dlen.d, d.dlen.m) * d.dlen.d);
}

// Units: rb rows x g column windows of the [R, L] view; a window is 32
// vectors wide, lane l owning columns c0 + l V .. c0 + l V + V - 1 in every
// row, so the last axis' marginal (and, with AXL, the growth maxima of the
// lane's columns) stay in registers until the window ends, and each row's
// mismatch count adds up over the unit's windows in the warp's shared row
// counters before it goes to the leading axes' marginals.  Four rows are
// loaded at a time (eight 16-byte loads in flight per lane).
template <int DT, bool AXL>
__global__ void __launch_bounds__(kFxThreads) fx_kernel(const __grid_constant__ FxDesc d, FxAcc *acc, FxBest *blk,
                                                       unsigned long long *g_growth, uint32_t *g_glb,
                                                       unsigned long long *g_marg) {
  constexpr int V = Tr<DT>::V;
  constexpr int EB = Tr<DT>::EB;
  extern __shared__ __align__(16) uint8_t fx_sm[];
  // [warp][bin][lane] ulp histograms: a lane's bins sit in its own bank
  int32_t *hist = (int32_t *)fx_sm;
  uint32_t *s_rows = (uint32_t *)(fx_sm + kFxHistBytes);  // [warp][kFxRowsMax] row mismatch counts
  const int64_t glen = d.grow_smem ? d.axis_len : 0;
  const int64_t mlen = d.marg_smem ? d.marg_off[d.rank] : 0;
  unsigned long long *s_gmax = (unsigned long long *)(fx_sm + kFxHistBytes + kFxRowBytes);
  uint32_t *s_glb = (uint32_t *)(s_gmax + glen);
  uint32_t *s_marg = s_glb + glen;
  for (int t = threadIdx.x; t < (kFxHistBytes + kFxRowBytes) / 4; t += kFxThreads) hist[t] = 0;
  for (int64_t t = threadIdx.x; t < glen; t += kFxThreads) {
    s_gmax[t] = 0ull;
    s_glb[t] = 0u;
  }
  for (int64_t t = threadIdx.x; t < mlen; t += kFxThreads) s_marg[t] = 0u;
  __syncthreads();
  unsigned long long *gmax = d.grow_smem ? s_gmax : g_growth;
  uint32_t *glb = d.grow_smem ? s_glb : g_glb;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t myhist = (uint32_t)__cvta_generic_to_shared(hist + warp * (NMV_ULP_BINS * 32) + lane);
  uint32_t *myrows = s_rows + warp * kFxRowsMax;
  FxLane L = {0u, 0u, 0u, 0u, 0u, INT64_MAX};
  const char *cb0 = (const char *)d.cand, *rb0 = (const char *)d.ref;
  const int64_t Lw = d.L, R = d.R;
  const int64_t col_bin0 = d.rank > 0 ? d.marg_off[d.rank - 1] : 0;
  for (;;) {
    unsigned long long u = 0;
    if (lane == 0) u = atomicAdd(&acc->unit_ctr, 1ull);
    u = __shfl_sync(0xffffffffu, u, 0);
    if (u >= (unsigned long long)d.n_units) break;
    // consecutive units lie in different row blocks, so the units that run
    // at once share few rows and the growth screen sees earlier maxima
    const int64_t wg = (int64_t)(u / (unsigned long long)d.RBn), rbk = (int64_t)u - wg * d.RBn;
    const int64_t r0 = rbk * d.rb, r1 = min(R, r0 + d.rb);
    const int64_t w0 = wg * d.g, w1 = min(d.CWn, w0 + d.g);
    for (int64_t w = w0; w < w1; ++w) {
      const int64_t mycol = w * (32 * V) + lane * V;
      const int ncol = Lw - mycol >= V ? V : (Lw > mycol ? (int)(Lw - mycol) : 0);
      uint32_t colm[V];
      GAcc<DT> gc[AXL ? V : 1];
#pragma unroll
      for (int k = 0; k < V; ++k) colm[k] = 0u;
      for (int64_t r = r0; r < r1; r += 4) {
        uint4 cv[4], rv[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          cv[j] = rv[j] = make_uint4(0, 0, 0, 0);
          if (r + j < r1 && ncol > 0) {
            const int64_t e = (r + j) * Lw + mycol;
            if (d.vec_ok && ncol == V) {
              cv[j] = ld_v4(cb0 + e * EB);
              rv[j] = ld_v4(rb0 + e * EB);
            } else {
              uint32_t cw[4] = {0, 0, 0, 0}, rw[4] = {0, 0, 0, 0};
#pragma unroll
              for (int k = 0; k < V; ++k) {
                if (k < ncol) {
                  const uint32_t c = ld_one<EB>(cb0, e + k), x = ld_one<EB>(rb0, e + k);
                  if constexpr (EB == 2) {
                    cw[k >> 1] |= c << (16 * (k & 1));
                    rw[k >> 1] |= x << (16 * (k & 1));
                  } else {
                    cw[k] = c;
                    rw[k] = x;
                  }
                }
              }
              cv[j] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
              rv[j] = make_uint4(rw[0], rw[1], rw[2], rw[3]);
            }
          }
        }
        // the four rows' elements, then their row ends (the warp reductions
        // of the four rows side by side)
        uint32_t m_row[4];
        float rmax[4];
        GAcc<DT> gr[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          m_row[j] = 0u;
          rmax[j] = 0.f;
        }
        if (ncol == V) {  // whole vectors (all but a row's last window): no per-element guard
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int64_t rho = r + j;
            if (rho < r1) {  // warp-uniform
              const int64_t e = rho * Lw + mycol;
#pragma unroll
              for (int k = 0; k < V; ++k) {
                const bool mm = fx_el<DT, AXL>(d, L, vbits<DT>(cv[j], k), vbits<DT>(rv[j], k), e + k, myhist,
                                               AXL ? gc[AXL ? k : 0] : gr[j], rmax[j], gmax, glb);
                colm[k] += mm ? 1u : 0u;
                m_row[j] += mm ? 1u : 0u;
              }
            }
          }
        } else {
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int64_t rho = r + j;
            if (rho < r1) {
              const int64_t e = rho * Lw + mycol;
#pragma unroll
              for (int k = 0; k < V; ++k) {
                if (k < ncol) {
                  const bool mm = fx_el<DT, AXL>(d, L, vbits<DT>(cv[j], k), vbits<DT>(rv[j], k), e + k, myhist,
                                                 AXL ? gc[AXL ? k : 0] : gr[j], rmax[j], gmax, glb);
                  colm[k] += mm ? 1u : 0u;
                  m_row[j] += mm ? 1u : 0u;
                }
              }
            }
          }
        }
        if (d.rank >= 2) {
          uint32_t tot[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) tot[j] = __reduce_add_sync(0xffffffffu, m_row[j]);
          if (lane == 0) {
#pragma unroll
            for (int j = 0; j < 4; ++j)
              if (tot[j]) myrows[r + j - r0] += tot[j];  // zero for rows past r1
          }
        }
        if constexpr (!AXL) {
          // each row's growth: the warp's largest |fl32(c - r)| screened
          // against the bin's lower bound; past the screen, the exact
          // maximum among the elements that reach it
          uint32_t wmx[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            if constexpr (Tr<DT>::kInt) wmx[j] = __reduce_max_sync(0xffffffffu, gr[j].U);
            else wmx[j] = __reduce_max_sync(0xffffffffu, __float_as_uint(rmax[j]));
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int64_t rho = r + j;
            if (rho >= r1 || wmx[j] == 0u) continue;  // warp-uniform
            const int64_t jg = row_gidx(d, rho);
            if constexpr (Tr<DT>::kInt) {  // exact integer maxima
              GAcc<DT> m;
              m.U = wmx[j];
              if (lane == 0) grow_flush<DT>(m, jg, gmax, glb);
            } else {
              const float lb = __uint_as_float(__shfl_sync(0xffffffffu, glb[jg], 0));
              const float wmf = __uint_as_float(wmx[j]);
              if (__fmul_rn(wmf, 1.0f + 0x1p-22f) >= lb) {
                const int64_t e = rho * Lw + mycol;
                GAcc<DT> m;
#pragma unroll
                for (int k = 0; k < V; ++k) {
                  if (k < ncol) {
                    const float cf = to_f32<DT>(vbits<DT>(cv[j], k)), rf = to_f32<DT>(vbits<DT>(rv[j], k));
                    const float s = __fsub_rn(cf, rf), as = fabsf(s);
                    if (as == wmf && fabsf(cf) <= FLT_MAX && fabsf(rf) <= FLT_MAX) {
                      if (as <= FLT_MAX) {
                        const float t = twosum_err(cf, rf, s), tp = s > 0.f ? t : -t;
                        if (m.S == 0.f || tp > m.T) {
                          m.S = as;
                          m.T = tp;
                        }
                      } else {
                        grow_direct(d, e + k, fabs(__dsub_rn((double)cf, (double)rf)), gmax, glb);
                      }
                    }
                  }
                }
                // (S, T) as a pair of order-preserving words, maximised word by word
                const uint32_t hi = __float_as_uint(m.S), tb = __float_as_uint(m.T);
                const uint32_t lo = (tb & 0x80000000u) ? ~tb : (tb | 0x80000000u);
                const uint32_t mhi = __reduce_max_sync(0xffffffffu, hi);
                const uint32_t mlo = __reduce_max_sync(0xffffffffu, hi == mhi ? lo : 0u);
                m.S = __uint_as_float(mhi);
                m.T = __uint_as_float((mlo & 0x80000000u) ? (mlo & 0x7fffffffu) : ~mlo);
                if (lane == 0) grow_flush<DT>(m, jg, gmax, glb);
              }
            }
          }
        }
      }
      // the window's columns: the last axis' marginal and, with AXL, growth
      if (d.rank > 0) {
#pragma unroll
        for (int k = 0; k < V; ++k) {
          if (k < ncol && colm[k] != 0u) {
            const int64_t bin = col_bin0 + mycol + k;
            if (d.marg_smem) atomicAdd(&s_marg[bin], colm[k]);
            else gl_add(&g_marg[bin], (unsigned long long)colm[k]);
          }
        }
      }
      if constexpr (AXL) {
#pragma unroll
        for (int k = 0; k < V; ++k)
          if (k < ncol) grow_flush<DT>(gc[k], mycol + k, gmax, glb);
      }
    }
    // the unit's row counts -> the leading axes' marginals, in parallel
    if (d.rank >= 2) {
      __syncwarp();
      for (int64_t t = lane; t < r1 - r0; t += 32) {
        const uint32_t c = myrows[t];
        if (c) {
          marg_rows(d, r0 + t, c, s_marg, g_marg);
          myrows[t] = 0u;
        }
      }
      __syncwarp();
    }
  }
  // ---- the block's totals
  const unsigned long long m = warp_reduce((unsigned long long)L.mism, [](unsigned long long a, unsigned long long b) { return a + b; });
  const unsigned long long f = warp_reduce((unsigned long long)L.nfin, [](unsigned long long a, unsigned long long b) { return a + b; });
  const unsigned long long nf = warp_reduce((unsigned long long)L.nonfin, [](unsigned long long a, unsigned long long b) { return a + b; });
  const unsigned long long w = warp_reduce((unsigned long long)L.within, [](unsigned long long a, unsigned long long b) { return a + b; });
  if (lane == 0) {
    if (m) atomicAdd(&acc->mismatch, m);
    if (f) atomicAdd(&acc->n_finite, f);
    if (nf) atomicAdd(&acc->nonfin, nf);
    if (w) atomicAdd(&acc->within, w);
  }
  // largest ulp distance, lowest index on ties
  long long bu = L.bu ? (long long)L.bu : -1ll, bi = L.bu ? (long long)L.bi : -1ll;
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const long long u2 = __shfl_xor_sync(0xffffffffu, bu, o), i2 = __shfl_xor_sync(0xffffffffu, bi, o);
    if (u2 > bu || (u2 == bu && u2 >= 0 && i2 < bi)) {
      bu = u2;
      bi = i2;
    }
  }
  __shared__ FxBest wb[kFxThreads / 32];
  if (lane == 0) wb[warp] = {bu, bi};
  __syncthreads();
  if (threadIdx.x == 0) {
    FxBest b = wb[0];
    for (int k = 1; k < kFxThreads / 32; ++k)
      if (wb[k].u > b.u || (wb[k].u == b.u && b.u >= 0 && wb[k].idx < b.idx)) b = wb[k];
    blk[blockIdx.x] = b;
  }
  if (threadIdx.x < NMV_ULP_BINS) {
    unsigned long long sum = 0;
    for (int t = 0; t < kFxThreads; ++t) sum += (unsigned)hist[(t >> 5) * (NMV_ULP_BINS * 32) + threadIdx.x * 32 + (t & 31)];
    if (sum) atomicAdd(&acc->hist[threadIdx.x], sum);
  }
  for (int64_t t = threadIdx.x; t < glen; t += kFxThreads)
    if (s_gmax[t]) atomicMax(&g_growth[t], s_gmax[t]);
  for (int64_t t = threadIdx.x; t < mlen; t += kFxThreads)
    if (s_marg[t]) gl_add(&g_marg[t], (unsigned long long)s_marg[t]);
}

// One block: the blocks' candidates in block order, every field of the
// result into the mapped host block, the growth means and the flags.
__global__ void __launch_bounds__(kFxThreads) fx_fin_kernel(const FxDesc *__restrict__ dp, const FxAcc *acc,
                                                           const FxBest *blk, int n_blk,
                                                           const unsigned long long *g_growth,
                                                           const unsigned long long *g_marg, uint8_t *host) {
  const FxDesc &d = *dp;
  nmv_forensics_result *res = (nmv_forensics_result *)(host + d.res_off);
  double *hg = (double *)(host + d.growth_off);
  int64_t *hm = (int64_t *)(host + d.marg_off_host);
  for (int64_t j = threadIdx.x; j < d.axis_len; j += kFxThreads) hg[j] = __longlong_as_double((long long)g_growth[j]);
  for (int64_t t = threadIdx.x; t < d.marg_off[d.rank]; t += kFxThreads) hm[t] = (int64_t)g_marg[t];
  if (threadIdx.x < NMV_ULP_BINS) res->ulp_hist[threadIdx.x] = (int64_t)acc->hist[threadIdx.x];
  if (threadIdx.x != 0) return;
  FxBest b = {-1, -1};
  for (int k = 0; k < n_blk; ++k)
    if (blk[k].u > b.u || (blk[k].u == b.u && b.u >= 0 && blk[k].idx < b.idx)) b = blk[k];
  const int64_t mism = (int64_t)acc->mismatch, nonfin = (int64_t)acc->nonfin, within = (int64_t)acc->within;
  res->mismatch = mism;
  res->n_finite_pairs = (int64_t)acc->n_finite;
  res->max_ulp_mismatch = b.u;
  res->argmax_ulp_mismatch = b.u >= 0 ? b.idx : -1;
  res->mism_nonfinite = nonfin;
  res->mism_within_f16 = within;
  const int64_t len = d.axis_len;
  int64_t q = len / 4;
  if (q < 1) q = 1;
  double lo = 0.0, hi = 0.0;
  if (len > 0) {
    for (int64_t j = 0; j < q && j < len; ++j) lo = __dadd_rn(lo, __longlong_as_double((long long)g_growth[j]));
    for (int64_t j = len - q; j < len; ++j) hi = __dadd_rn(hi, __longlong_as_double((long long)g_growth[j]));
    lo = __ddiv_rn(lo, (double)q);
    hi = __ddiv_rn(hi, (double)q);
  }
  res->growth_lo = lo;
  res->growth_hi = hi;
  uint32_t fl = 0;
  if (mism > 0 && nonfin == 0 && b.u <= d.near_ulps && (double)mism <= __dmul_rn(d.near_fraction, (double)d.numel))
    fl |= NMV_FX_NEAR_PASS;
  if (mism > 0 && nonfin == 0 && within == mism) fl |= NMV_FX_F16_CEILING;
  if (len >= 4 && hi > 0.0 && hi >= __dmul_rn(d.growth_factor, lo)) fl |= NMV_FX_AXIS_GROWTH;
  res->flags = fl;
}

// ------------------------------------------------------------------ host
namespace {

struct FxWorkspace {
  void *p = nullptr;
  size_t size = 0;
};
FxWorkspace g_fxws[64];

size_t align_to(size_t x, size_t a) { return (x + a - 1) / a * a; }

float f32_down(double x) {
  float f = (float)x;
  if ((double)f > x) f = std::nextafter(f, -INFINITY);
  return f;
}

float f32_up(double x) {
  float f = (float)x;
  if ((double)f < x) f = std::nextafter(f, INFINITY);
  return f;
}

size_t fx_smem(const FxDesc &d) {
  size_t b = (size_t)kFxHistBytes + kFxRowBytes;
  if (d.grow_smem) b += (size_t)d.axis_len * 12;
  if (d.marg_smem) b += (size_t)d.marg_off[d.rank] * 4;
  return b;
}

template <int DT, bool AXL>
cudaError_t launch_fx_dt(int sms, const FxDesc &h, const FxDesc *dd, FxAcc *acc, FxBest *blk, int *n_blk,
                         unsigned long long *gg, uint32_t *glb, unsigned long long *gm, cudaStream_t st) {
  const size_t smem = fx_smem(h);
  cudaError_t e = cudaFuncSetAttribute(fx_kernel<DT, AXL>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  int occ = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fx_kernel<DT, AXL>, kFxThreads, smem);
  if (e != cudaSuccess) return e;
  int64_t grid = (int64_t)sms * std::max(occ, 1);
  grid = std::max<int64_t>(1, std::min<int64_t>(grid, (h.n_units + kFxThreads / 32 - 1) / (kFxThreads / 32)));
  *n_blk = (int)grid;
  fx_kernel<DT, AXL><<<(int)grid, kFxThreads, smem, st>>>(h, acc, blk, gg, glb, gm);
  return cudaGetLastError();
}

template <int DT>
cudaError_t launch_fx_ax(int sms, const FxDesc &h, const FxDesc *dd, FxAcc *acc, FxBest *blk, int *n_blk,
                         unsigned long long *gg, uint32_t *glb, unsigned long long *gm, cudaStream_t st) {
  // the growth axis is the last one (or the tensor has rank 0 or 1)
  if (h.rank <= 1 || h.axis == h.rank - 1) return launch_fx_dt<DT, true>(sms, h, dd, acc, blk, n_blk, gg, glb, gm, st);
  return launch_fx_dt<DT, false>(sms, h, dd, acc, blk, n_blk, gg, glb, gm, st);
}

cudaError_t launch_fx(int sms, const FxDesc &h, const FxDesc *dd, FxAcc *acc, FxBest *blk, int *n_blk,
                      unsigned long long *gg, uint32_t *glb, unsigned long long *gm, cudaStream_t st) {
  switch (h.dtype) {
    case NMV_F32: return launch_fx_ax<NMV_F32>(sms, h, dd, acc, blk, n_blk, gg, glb, gm, st);
    case NMV_F16: return launch_fx_ax<NMV_F16>(sms, h, dd, acc, blk, n_blk, gg, glb, gm, st);
    case NMV_BF16: return launch_fx_ax<NMV_BF16>(sms, h, dd, acc, blk, n_blk, gg, glb, gm, st);
    default: return launch_fx_ax<NMV_I32>(sms, h, dd, acc, blk, n_blk, gg, glb, gm, st);
  }
}

int check_fx_case(const nmv_forensics_case &c, FxDesc &d, int64_t i) {
  char pre[64];
  std::snprintf(pre, sizeof pre, "case %lld: ", (long long)i);
  auto bad = [&](const char *m) { return host_fail(NMV_EINVAL, std::string(pre) + m); };
  const nmv_tensor &a = c.cand, &b = c.ref;
  if (a.dtype < NMV_F32 || a.dtype > NMV_I32) return bad("unknown dtype");
  if (a.dtype != b.dtype) return bad("cand and ref dtypes differ");
  const int64_t n = host_tensor_numel(a), nr = host_tensor_numel(b);
  if (n < 0 || nr < 0) return bad("invalid rank or shape");
  if (a.rank != b.rank) return bad("cand and ref ranks differ");
  for (int k = 0; k < a.rank; ++k)
    if (a.shape[k] != b.shape[k]) return bad("cand and ref shapes differ");
  if (n > 0 && (a.data == nullptr || b.data == nullptr)) return bad("NULL data");
  if (c.reserved != 0) return bad("reserved must be 0");
  if (!std::isfinite(c.rtol) || !std::isfinite(c.atol) || c.rtol < 0 || c.atol < 0)
    return bad("rtol and atol must be finite and >= 0");
  if (c.near_ulps < 0 || !std::isfinite(c.near_fraction) || c.near_fraction < 0 || !std::isfinite(c.growth_factor) ||
      c.growth_factor < 0)
    return bad("near_ulps, near_fraction and growth_factor must be finite and >= 0");
  if (a.rank > 0 && (c.axis < -a.rank || c.axis >= a.rank)) return bad("axis out of range");
  std::memset(&d, 0, sizeof(d));
  d.cand = a.data;
  d.ref = b.data;
  d.dtype = a.dtype;
  d.numel = n;
  d.rank = a.rank;
  d.axis = a.rank > 0 ? (c.axis < 0 ? c.axis + a.rank : c.axis) : 0;
  d.marg_off[0] = 0;
  for (int k = 0; k < a.rank; ++k) {
    d.shape[k] = a.shape[k];
    d.sdiv[k] = a.shape[k] > 0 ? make_div((uint64_t)a.shape[k]) : Div64{1, ~0ull};
    d.marg_off[k + 1] = d.marg_off[k] + a.shape[k];
  }
  if (d.marg_off[a.rank] > NMV_MAX_HIST_BINS) return bad("sum(shape) exceeds NMV_MAX_HIST_BINS");
  int64_t stride = 1;
  for (int k = a.rank - 1; k > d.axis; --k) stride *= a.shape[k];
  d.axis_len = a.rank > 0 ? a.shape[d.axis] : 1;
  d.dstride = make_div((uint64_t)std::max<int64_t>(stride, 1));
  d.dlen = make_div((uint64_t)std::max<int64_t>(d.axis_len, 1));
  // the [R, L] view and its units
  const int64_t V = vec_elems(a.dtype), EB = elem_bytes(a.dtype);
  d.L = a.rank > 0 ? a.shape[a.rank - 1] : 1;
  d.R = d.L > 0 ? n / d.L : 0;
  d.CWn = (d.L + 32 * V - 1) / (32 * V);
  d.rb = std::max<int64_t>(1, std::min<int64_t>(std::min<int64_t>(d.R, kFxRowsMax), kFxUnitElems / (32 * V)));
  d.g = std::max<int64_t>(1, std::min<int64_t>(d.CWn, kFxUnitElems / (d.rb * 32 * V)));
  d.WG = (d.CWn + d.g - 1) / d.g;
  d.RBn = (d.R + d.rb - 1) / d.rb;
  d.n_units = n > 0 ? d.RBn * d.WG : 0;
  // growth on an axis before the last: rows per index of the axis
  const int64_t rs = d.L > 0 ? std::max<int64_t>(stride, 1) / std::max<int64_t>(d.L, 1) : 1;
  d.drs = make_div((uint64_t)std::max<int64_t>(rs, 1));
  d.j_is_row = (rs == 1 && d.axis_len == d.R) ? 1 : 0;
  d.vec_ok = ((uintptr_t)a.data % 16 == 0) && ((uintptr_t)b.data % 16 == 0) && (d.L * EB) % 16 == 0;
  d.rtol = c.rtol;
  d.atol = c.atol;
  const bool filter = c.rtol <= 0.5 && c.atol <= 0x1p100;
  if (filter) {
    d.lo_r = f32_down(c.rtol * (1.0 - 0x1p-20));
    d.lo_a = f32_down(c.atol * (1.0 - 0x1p-20));
    d.hi_r = f32_up(c.rtol * (1.0 + 0x1p-20));
    d.hi_a = f32_up(c.atol * (1.0 + 0x1p-20));
  } else {
    d.lo_r = 0.f;
    d.lo_a = -1.f;      // never sure-pass
    d.hi_r = 0.f;
    d.hi_a = INFINITY;  // never sure-fail
  }
  d.near_ulps = c.near_ulps;
  d.near_fraction = c.near_fraction;
  d.growth_factor = c.growth_factor;
  d.grow_smem = d.axis_len <= kFxGrowCap ? 1 : 0;
  d.marg_smem = d.marg_off[a.rank] <= kFxMargCap ? 1 : 0;
  return NMV_OK;
}

int run_fx(const nmv_forensics_case *cases, int64_t n, void *stream, nmv_forensics_result **out) {
  if (out == nullptr) return host_fail(NMV_EINVAL, "out is NULL");
  *out = nullptr;
  if (cases == nullptr && n > 0) return host_fail(NMV_EINVAL, "cases is NULL");
  if (n < 0 || n > NMV_MAX_CASES) return host_fail(NMV_EINVAL, "case count out of range");
  std::vector<FxDesc> desc((size_t)n);
  size_t off = align_to(sizeof(nmv_forensics_result) * (size_t)std::max<int64_t>(n, 1), 256);
  int64_t max_len = 1, max_marg = 1;
  for (int64_t i = 0; i < n; ++i) {
    FxDesc &d = desc[(size_t)i];
    const int rc = check_fx_case(cases[i], d, i);
    if (rc) return rc;
    d.res_off = (int64_t)(sizeof(nmv_forensics_result) * (size_t)i);
    d.growth_off = (int64_t)off;
    off = align_to(off + 8 * (size_t)d.axis_len, 256);
    d.marg_off_host = (int64_t)off;
    off = align_to(off + 8 * (size_t)d.marg_off[d.rank], 256);
    max_len = std::max(max_len, d.axis_len);
    max_marg = std::max(max_marg, d.marg_off[d.rank]);
  }
  if (n == 0) return NMV_OK;

  std::lock_guard<std::mutex> lock(host_mutex());
  int dev = -1, sms = 0;
  size_t smem_optin = 0;
  int rc = host_probe(&dev, &sms, &smem_optin);
  if (rc) return rc;
  if (dev >= 64) return host_fail(NMV_EUNSUPPORTED, "device ordinal out of range");
  for (const FxDesc &d : desc)
    if (fx_smem(d) > smem_optin) return host_fail(NMV_EINVAL, "forensics maps need more shared memory than the device has");
  cudaStream_t st = (cudaStream_t)stream;
  const int64_t max_blk = (int64_t)sms * 8;
  const size_t sz_desc = align_to(sizeof(FxDesc), 256), sz_acc = align_to(sizeof(FxAcc), 256);
  const size_t sz_blk = align_to(sizeof(FxBest) * (size_t)max_blk, 256);
  const size_t sz_g = align_to(8 * (size_t)max_len, 256), sz_glb = align_to(4 * (size_t)max_len, 256);
  const size_t sz_m = align_to(8 * (size_t)max_marg, 256);
  const size_t need = sz_desc + sz_acc + sz_blk + sz_g + sz_glb + sz_m;
  FxWorkspace &W = g_fxws[dev];
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
      return host_fail(NMV_ENOMEM, std::string("cudaMalloc forensics workspace: ") + cudaGetErrorString(e));
    }
    W.size = want;
  }
  uint8_t *ws = (uint8_t *)W.p;
  FxDesc *d_desc = (FxDesc *)ws;
  FxAcc *d_acc = (FxAcc *)(ws + sz_desc);
  FxBest *d_blk = (FxBest *)(ws + sz_desc + sz_acc);
  unsigned long long *d_g = (unsigned long long *)(ws + sz_desc + sz_acc + sz_blk);
  uint32_t *d_glb = (uint32_t *)(ws + sz_desc + sz_acc + sz_blk + sz_g);
  unsigned long long *d_m = (unsigned long long *)(ws + sz_desc + sz_acc + sz_blk + sz_g + sz_glb);

  uint8_t *host = (uint8_t *)host_arena_get(off);
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
  nmv_forensics_result *res = (nmv_forensics_result *)host;
  for (int64_t i = 0; i < n; ++i) {
    const FxDesc &d = desc[(size_t)i];
    nmv_forensics_result &r = res[i];
    std::memset(&r, 0, sizeof(r));
    r.status = NMV_OK;
    r.rank = d.rank;
    r.numel = d.numel;
    r.axis = d.axis;
    r.axis_len = d.axis_len;
    r.max_ulp_mismatch = r.argmax_ulp_mismatch = -1;
    r.growth = (double *)(host + d.growth_off);
    r.marginals = (int64_t *)(host + d.marg_off_host);
    for (int k = 0; k <= NMV_MAX_RANK; ++k) r.marg_off[k] = d.marg_off[k <= d.rank ? k : d.rank];
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
  for (int64_t i = 0; i < n; ++i) {
    const FxDesc &d = desc[(size_t)i];
    cudaError_t e = cudaMemcpyAsync(d_desc, &d, sizeof(FxDesc), cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) return host_cuda_fail(e, "cudaMemcpyAsync (descriptor)");
    e = cudaMemsetAsync(d_acc, 0, sz_acc, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d_g, 0, 8 * (size_t)std::max<int64_t>(d.axis_len, 1), st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d_glb, 0, 4 * (size_t)std::max<int64_t>(d.axis_len, 1), st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d_m, 0, 8 * (size_t)std::max<int64_t>(d.marg_off[d.rank], 1), st);
    if (e != cudaSuccess) return host_cuda_fail(e, "cudaMemsetAsync");
    int n_blk = 0;
    if (d.numel > 0) {
      e = launch_fx(sms, d, d_desc, d_acc, d_blk, &n_blk, d_g, d_glb, d_m, st);
      if (e != cudaSuccess) return host_cuda_fail(e, "forensics kernel launch");
    }
    fx_fin_kernel<<<1, kFxThreads, 0, st>>>(d_desc, d_acc, d_blk, n_blk, d_g, d_m, dhost);
    e = cudaGetLastError();
    if (e != cudaSuccess) return host_cuda_fail(e, "forensics finalize launch");
    // the descriptor and accumulators are reused by the next case
    e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return host_cuda_fail(e, "cudaStreamSynchronize");
  }
  drain.armed = false;
  guard.p = nullptr;  // handed to the caller
  *out = res;
  host_clear_error();
  return NMV_OK;
}

}  // namespace
}  // namespace nmv

extern "C" int nmv_forensics(const nmv_forensics_case *cases, int64_t n, void *cuda_stream,
                             nmv_forensics_result **out) {
  return nmv::run_fx(cases, n, cuda_stream, out);
}
