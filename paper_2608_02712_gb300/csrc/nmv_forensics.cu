// nmv_forensics.cu -- deep forensics of a candidate/reference pair
// (nmv_forensics): the evidence behind the adaptive-scheduling rules
// "near-pass and fp16-ceiling detection" (Section 4.4), the localisation of
// a divergence that compounds along a reduction axis (Section 3.2, the
// cumsum of Table 1), and mismatch counts at every index of every axis.
//
// fx_kernel streams the pair once (16-byte loads, four in flight per lane).
// Per element it takes the predicate with the scan's fp32 pre-filter (fp64
// where the filter cannot decide), the ulp distance u of the two stored
// values, and for mismatches the fp16-spacing test and the coordinates.
// Lane-private ulp histograms sit in shared memory (stride 35 words, so the
// 32 lanes of a warp hit 32 banks); the growth curve max |c - r| per index
// of the chosen axis is screened in fp32 against a lower bound of the bin's
// maximum and made exact in fp64 only for candidates (maxima do not depend
// on the order, so atomics keep them exact); the marginals are privatised
// in shared memory when they fit.  fx_fin_kernel reduces the blocks'
// largest-ulp candidates in block order and writes every field into the
// mapped host result.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "nmv_scan.cuh"

namespace nmv {

constexpr int kFxThreads = 256;
constexpr int kFxHistStride = 35;     // words per lane histogram (34 bins, odd stride)
constexpr int64_t kFxGrowCap = 2048;  // growth bins privatised in shared memory
constexpr int64_t kFxMargCap = 4096;  // marginal bins privatised in shared memory

struct FxDesc {
  const void *cand, *ref;
  int32_t dtype, vec_ok;
  int32_t rank, axis;
  int32_t idx32, grow_smem, marg_smem, pad;
  int64_t numel;
  int64_t shape[NMV_MAX_RANK];
  Div64 sdiv[NMV_MAX_RANK];
  int64_t marg_off[NMV_MAX_RANK + 1];
  int64_t axis_len;
  Div64 dstride, dlen;      // coordinate on the axis: (i / stride) % len
  uint32_t m32stride, m32len;
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
};

struct FxBest {
  long long u, idx;  // largest ulp distance of a finite mismatch (-1: none) and its lowest index
};

__device__ __forceinline__ long long ord_bits(uint32_t b, int dt) {
  if (dt == NMV_I32) return (long long)(int32_t)b;
  const int width = elem_bytes(dt) * 8;
  const uint32_t sign = (b >> (width - 1)) & 1u;
  const long long mag = (long long)(b & (width == 32 ? 0x7fffffffu : 0x7fffu));
  return sign ? -mag : mag;
}

// One fp16 spacing at |r| (r finite): 2^(max(floor(log2 |r|), -14) - 10),
// 2^-24 at 0.  Values of these types are normal in fp64, so floor(log2 |r|)
// is the fp64 exponent field less the bias.
__device__ __forceinline__ double f16_spacing(double r) {
  if (r == 0.0) return 0x1p-24;
  const int e = (int)((__double_as_longlong(fabs(r)) >> 52) & 0x7ff) - 1023;
  return ldexp(1.0, max(e, -14) - 10);
}

// The predicate of nmv_validate: the fp32 pre-filter decides where it can,
// fp64 otherwise.
template <int DT>
__device__ __forceinline__ bool fx_pass(const FxDesc &d, uint32_t cb, uint32_t rb) {
  if constexpr (Tr<DT>::kInt) {
    if (cb == rb) return true;
    const long long df = (long long)(int32_t)cb - (long long)(int32_t)rb;
    const float as = fabsf(__ll2float_rn(df)), ar = fabsf(to_f32<DT>(rb));
    if (as <= __fmaf_rz(d.lo_r, ar, d.lo_a)) return true;
    if (as > __fmaf_ru(d.hi_r, ar, d.hi_a)) return false;
  } else {
    const float cf = to_f32<DT>(cb), rf = to_f32<DT>(rb);
    if (cf == rf) return true;
    if (!(isfinite(cf) && isfinite(rf))) return false;
    const float as = fabsf(__fsub_rn(cf, rf)), ar = fabsf(rf);
    if (as <= __fmaf_rz(d.lo_r, ar, d.lo_a)) return true;
    if (as > __fmaf_ru(d.hi_r, ar, d.hi_a)) return false;
  }
  return pass64(to_f64<DT>(cb), to_f64<DT>(rb), d.rtol, d.atol);
}

struct FxLane {
  uint32_t mism, nfin, nonfin, within;
  long long bu, bi;
};

// The coordinate of element i on the growth axis.
__device__ __forceinline__ int64_t axis_coord(const FxDesc &d, int64_t i) {
  if (d.rank == 0) return 0;
  if (d.idx32) {
    const uint32_t q = div_q32((uint32_t)i, (uint32_t)d.dstride.d, d.m32stride);
    return q - div_q32(q, (uint32_t)d.dlen.d, d.m32len) * (uint32_t)d.dlen.d;
  }
  const uint64_t q = div_q((uint64_t)i, d.dstride.d, d.dstride.m);
  return (int64_t)(q - div_q(q, d.dlen.d, d.dlen.m) * d.dlen.d);
}

template <int DT>
__device__ __forceinline__ void fx_elem(const FxDesc &d, FxLane &L, uint32_t cb, uint32_t rb, int64_t i,
                                        int32_t *hist, unsigned long long *gmax, uint32_t *glb, uint32_t *smarg,
                                        unsigned long long *gmarg) {
  bool fin = true;
  float as32;
  if constexpr (Tr<DT>::kInt) {
    const long long df = (long long)(int32_t)cb - (long long)(int32_t)rb;
    as32 = __ll2float_rn(df < 0 ? -df : df);
  } else {
    const float cf = to_f32<DT>(cb), rf = to_f32<DT>(rb);
    fin = isfinite(cf) && isfinite(rf);
    as32 = fabsf(__fsub_rn(cf, rf));
  }
  long long u = ord_bits(cb, DT) - ord_bits(rb, DT);
  u = u < 0 ? -u : u;
  if (fin) {
    ++L.nfin;
    const int bin = u == 0 ? 0 : min(64 - __clzll(u), NMV_ULP_BINS - 1);
    hist[bin] += 1;
    // growth: fl32 |c - r| is within 2^-24 of the exact |c - r|, so an
    // element whose as32 (1 + 2^-22) lies below the bin's lower bound is no
    // new maximum; the others are evaluated exactly in fp64
    if (as32 > 0.f) {
      const int64_t j = axis_coord(d, i);
      if (!(__fmul_rn(as32, 1.0f + 0x1p-22f) < __uint_as_float(glb[j]))) {
        const double dv = fabs(__dsub_rn(to_f64<DT>(cb), to_f64<DT>(rb)));
        atomicMax(&gmax[j], (unsigned long long)__double_as_longlong(dv));
        atomicMax(&glb[j], __float_as_uint(__double2float_rd(dv)));
      }
    }
  }
  if (!fx_pass<DT>(d, cb, rb)) {
    ++L.mism;
    if (!fin) {
      ++L.nonfin;
    } else {
      if (u > L.bu || (u == L.bu && i < L.bi)) {
        L.bu = u;
        L.bi = i;
      }
      const double r64 = to_f64<DT>(rb);
      const double dv = fabs(__dsub_rn(to_f64<DT>(cb), r64));
      L.within += dv <= f16_spacing(r64);
    }
    // the mismatch's coordinate on every axis; the lanes here that share a
    // bin add to it once (consecutive elements mostly share all but the
    // last coordinate)
    uint64_t rest = (uint64_t)i;
    const unsigned act = __activemask();
    const int lane = threadIdx.x & 31;
    for (int a = d.rank - 1; a >= 0; --a) {
      const uint64_t q = div_q(rest, d.sdiv[a].d, d.sdiv[a].m);
      const long long bin = d.marg_off[a] + (long long)(rest - q * d.sdiv[a].d);
      rest = q;
      const unsigned peers = __match_any_sync(act, bin);
      if (lane == __ffs(peers) - 1) {
        if (d.marg_smem) atomicAdd(&smarg[bin], (unsigned)__popc(peers));
        else gl_add(&gmarg[bin], (unsigned long long)__popc(peers));
      }
    }
  }
}

template <int DT>
__global__ void __launch_bounds__(kFxThreads) fx_kernel(const FxDesc *__restrict__ dp, FxAcc *acc, FxBest *blk,
                                                       unsigned long long *g_growth, uint32_t *g_glb,
                                                       unsigned long long *g_marg) {
  constexpr int V = Tr<DT>::V;
  constexpr int EB = Tr<DT>::EB;
  const FxDesc &d = *dp;
  extern __shared__ __align__(16) uint8_t fx_sm[];
  int32_t *hist = (int32_t *)fx_sm;
  const int64_t glen = d.grow_smem ? d.axis_len : 0;
  const int64_t mlen = d.marg_smem ? d.marg_off[d.rank] : 0;
  unsigned long long *s_gmax = (unsigned long long *)(fx_sm + (size_t)kFxThreads * kFxHistStride * 4 + 16);
  uint32_t *s_glb = (uint32_t *)(s_gmax + glen);
  uint32_t *s_marg = s_glb + glen;
  for (int t = threadIdx.x; t < kFxThreads * kFxHistStride; t += kFxThreads) hist[t] = 0;
  for (int64_t t = threadIdx.x; t < glen; t += kFxThreads) {
    s_gmax[t] = 0ull;
    s_glb[t] = 0u;
  }
  for (int64_t t = threadIdx.x; t < mlen; t += kFxThreads) s_marg[t] = 0u;
  __syncthreads();
  unsigned long long *gmax = d.grow_smem ? s_gmax : g_growth;
  uint32_t *glb = d.grow_smem ? s_glb : g_glb;
  int32_t *myhist = hist + threadIdx.x * kFxHistStride;
  FxLane L = {0u, 0u, 0u, 0u, -1ll, -1ll};
  const int64_t nvec = (d.numel + V - 1) / V;
  const int64_t nth = (int64_t)gridDim.x * kFxThreads;
  const char *cb0 = (const char *)d.cand, *rb0 = (const char *)d.ref;
  for (int64_t v0 = (int64_t)blockIdx.x * kFxThreads + threadIdx.x; v0 < nvec; v0 += 4 * nth) {
    uint4 cv[4], rv[4];
    int nn[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t v = v0 + j * nth;
      nn[j] = 0;
      cv[j] = rv[j] = make_uint4(0, 0, 0, 0);
      if (v < nvec) {
        const int64_t e = v * V;
        const int n = d.numel - e < V ? (int)(d.numel - e) : V;
        nn[j] = n;
        if (d.vec_ok && n == V) {
          cv[j] = ld_v4(cb0 + e * EB);
          rv[j] = ld_v4(rb0 + e * EB);
        } else {
          uint32_t cw[4] = {0, 0, 0, 0}, rw[4] = {0, 0, 0, 0};
          for (int k = 0; k < n; ++k) {
            const uint32_t c = ld_one<EB>(cb0, e + k), r = ld_one<EB>(rb0, e + k);
            if constexpr (EB == 2) {
              cw[k >> 1] |= c << (16 * (k & 1));
              rw[k >> 1] |= r << (16 * (k & 1));
            } else {
              cw[k] = c;
              rw[k] = r;
            }
          }
          cv[j] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
          rv[j] = make_uint4(rw[0], rw[1], rw[2], rw[3]);
        }
      }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t e = (v0 + j * nth) * V;
#pragma unroll
      for (int k = 0; k < V; ++k)
        if (k < nn[j])
          fx_elem<DT>(d, L, vbits<DT>(cv[j], k), vbits<DT>(rv[j], k), e + k, myhist, gmax, glb, s_marg, g_marg);
    }
  }
  // ---- the block's totals
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
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
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const long long u2 = __shfl_xor_sync(0xffffffffu, L.bu, o), i2 = __shfl_xor_sync(0xffffffffu, L.bi, o);
    if (u2 > L.bu || (u2 == L.bu && u2 >= 0 && i2 < L.bi)) {
      L.bu = u2;
      L.bi = i2;
    }
  }
  __shared__ FxBest wb[kFxThreads / 32];
  if (lane == 0) wb[warp] = {L.bu, L.bi};
  __syncthreads();
  if (threadIdx.x == 0) {
    FxBest b = wb[0];
    for (int k = 1; k < kFxThreads / 32; ++k)
      if (wb[k].u > b.u || (wb[k].u == b.u && b.u >= 0 && wb[k].idx < b.idx)) b = wb[k];
    blk[blockIdx.x] = b;
  }
  if (threadIdx.x < NMV_ULP_BINS) {
    unsigned long long s = 0;
    for (int t = 0; t < kFxThreads; ++t) s += (unsigned)hist[t * kFxHistStride + threadIdx.x];
    if (s) atomicAdd(&acc->hist[threadIdx.x], s);
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
  size_t b = (size_t)kFxThreads * kFxHistStride * 4 + 16;
  if (d.grow_smem) b += (size_t)d.axis_len * 12;
  if (d.marg_smem) b += (size_t)d.marg_off[d.rank] * 4;
  return b;
}

template <int DT>
cudaError_t launch_fx_dt(int sms, const FxDesc &h, const FxDesc *dd, FxAcc *acc, FxBest *blk, int *n_blk,
                         unsigned long long *gg, uint32_t *glb, unsigned long long *gm, cudaStream_t st) {
  const size_t smem = fx_smem(h);
  cudaError_t e = cudaFuncSetAttribute(fx_kernel<DT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  int occ = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fx_kernel<DT>, kFxThreads, smem);
  if (e != cudaSuccess) return e;
  const int64_t V = vec_elems(h.dtype);
  int64_t grid = (int64_t)sms * std::max(occ, 1);
  grid = std::max<int64_t>(1, std::min<int64_t>(grid, (h.numel / V + 4 * kFxThreads - 1) / (4 * kFxThreads)));
  *n_blk = (int)grid;
  fx_kernel<DT><<<(int)grid, kFxThreads, smem, st>>>(dd, acc, blk, gg, glb, gm);
  return cudaGetLastError();
}

cudaError_t launch_fx(int sms, const FxDesc &h, const FxDesc *dd, FxAcc *acc, FxBest *blk, int *n_blk,
                      unsigned long long *gg, uint32_t *glb, unsigned long long *gm, cudaStream_t st) {
  switch (h.dtype) {
    case NMV_F32: return launch_fx_dt<NMV_F32>(sms, h, dd, acc, blk, n_blk, gg, glb, gm, st);
    case NMV_F16: return launch_fx_dt<NMV_F16>(sms, h, dd, acc, blk, n_blk, gg, glb, gm, st);
    case NMV_BF16: return launch_fx_dt<NMV_BF16>(sms, h, dd, acc, blk, n_blk, gg, glb, gm, st);
    default: return launch_fx_dt<NMV_I32>(sms, h, dd, acc, blk, n_blk, gg, glb, gm, st);
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
  d.idx32 = n <= (int64_t)0xffffffffll ? 1 : 0;
  d.m32stride = d.idx32 ? 0xffffffffu / (uint32_t)std::max<int64_t>(stride, 1) : 0u;
  d.m32len = d.idx32 ? 0xffffffffu / (uint32_t)std::max<int64_t>(d.axis_len, 1) : 0u;
  d.vec_ok = ((uintptr_t)a.data % 16 == 0) && ((uintptr_t)b.data % 16 == 0);
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
