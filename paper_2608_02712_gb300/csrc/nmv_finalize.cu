// nmv_finalize.cu -- one block per case: reduce the piece partials of the
// scan pass (fixed order, so the result is bit-identical run to run), derive
// the degenerate-output flags, and write the first-K mismatch records, found
// by re-reading the few batches that hold them (located through the pieces'
// and then the batches' mismatch counts).  Also the fp64 SSE re-pass for
// cases whose differences are all tiny (see nmv_scan.cuh).
#include "nmv_scan.cuh"

namespace nmv {

__device__ __forceinline__ uint32_t ld_elem(const void *base, int64_t i, int dt) {
  return elem_bytes(dt) == 2 ? ld_one<2>(base, i) : ld_one<4>(base, i);
}

__device__ __forceinline__ double widen_any(uint32_t b, int dt) {
  switch (dt) {
    case NMV_F32: return to_f64<NMV_F32>(b);
    case NMV_F16: return to_f64<NMV_F16>(b);
    case NMV_BF16: return to_f64<NMV_BF16>(b);
    default: return to_f64<NMV_I32>(b);
  }
}

// What the record pass needs of one case, loaded once into registers.
struct FkView {
  const char *cand, *ref;
  int64_t *idx;          // record arrays of the packed result (device)
  double *c64, *r64;
  uint8_t *hrec;         // the host result's record arrays (laid out as idx), or null
  int64_t *coords;       // [first_k][rank] coordinates in the host result, or null
  const Div64 *sdiv;     // the candidate's extents as divisors (rank entries)
  int64_t first_k;
  int32_t rank;
  double rtol, atol;
  float lo_r, lo_a, hi_r, hi_a;  // the fp32 pre-filter of the predicate
  int32_t ks;            // warp steps per batch
  int32_t vec_ok;
};

// o: the case's device output; ho: its host result (or null).
__device__ __forceinline__ FkView fk_view(const CaseDesc &cd, uint8_t *o, uint8_t *ho, uint8_t *hbase) {
  FkView F;
  F.cand = (const char *)cd.cand;
  F.ref = (const char *)cd.ref;
  F.idx = (int64_t *)(o + cd.fk_off);
  F.c64 = (double *)(F.idx + cd.first_k);
  F.r64 = F.c64 + cd.first_k;
  F.hrec = ho ? ho + cd.fk_off : nullptr;
  F.coords = hbase ? (int64_t *)(hbase + cd.coord_off) : nullptr;
  F.sdiv = cd.sdiv;
  F.first_k = cd.first_k;
  F.rank = cd.rank;
  F.rtol = cd.rtol;
  F.atol = cd.atol;
  F.lo_r = cd.lo_r;
  F.lo_a = cd.lo_a;
  F.hi_r = cd.hi_r;
  F.hi_a = cd.hi_a;
  F.ks = batch_steps(nin_class_of(cd.n_elig));
  F.vec_ok = cd.vec_ok;
  return F;
}

// The pre-filter's sure-pass half, without branches: true only where the
// predicate holds (the scan pass takes the same decision).
template <int DT>
__device__ __forceinline__ bool sure_pass(const FkView &F, uint32_t cb, uint32_t rb) {
  if constexpr (Tr<DT>::kInt) {
    const long long d = (long long)(int32_t)cb - (long long)(int32_t)rb;
    const float as = fabsf(__ll2float_rn(d)), ar = fabsf(to_f32<DT>(rb));
    return cb == rb || as <= __fmaf_rz(F.lo_r, ar, F.lo_a);
  } else {
    const float cf = to_f32<DT>(cb), rf = to_f32<DT>(rb);
    const float as = fabsf(__fsub_rn(cf, rf)), ar = fabsf(rf);
    return cf == rf || (isfinite(cf) && isfinite(rf) && as <= __fmaf_rz(F.lo_r, ar, F.lo_a));
  }
}

// The predicate with the scan pass's fp32 pre-filter (same decision).
template <int DT>
__device__ __forceinline__ bool pass_elem(const FkView &F, uint32_t cb, uint32_t rb) {
  const float cf = to_f32<DT>(cb), rf = to_f32<DT>(rb);
  if constexpr (Tr<DT>::kInt) {
    if (cb == rb) return true;
    const long long d = (long long)(int32_t)cb - (long long)(int32_t)rb;
    const float as = fabsf(__ll2float_rn(d)), ar = fabsf(rf);
    if (as <= __fmaf_rz(F.lo_r, ar, F.lo_a)) return true;
    if (as > __fmaf_ru(F.hi_r, ar, F.hi_a)) return false;
  } else {
    if (cf == rf) return true;
    if (!(isfinite(cf) && isfinite(rf))) return false;
    const float as = fabsf(__fsub_rn(cf, rf)), ar = fabsf(rf);
    if (as <= __fmaf_rz(F.lo_r, ar, F.lo_a)) return true;
    if (as > __fmaf_ru(F.hi_r, ar, F.hi_a)) return false;
  }
  return pass64(to_f64<DT>(cb), to_f64<DT>(rb), F.rtol, F.atol);
}

// Exclusive block-wide prefix sum of a 64-bit v; *total = the block's sum.
__device__ __forceinline__ int64_t block_excl_scan64(int64_t v, int64_t *total, int64_t *sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int64_t incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int64_t t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  __syncthreads();
  if (lane == 31) sh[warp] = incl;
  __syncthreads();
  if (threadIdx.x == 0) {
    int64_t acc = 0;
    for (int w = 0; w < kFinThreads / 32; ++w) {
      const int64_t t = sh[w];
      sh[w] = acc;
      acc += t;
    }
    sh[kFinThreads / 32] = acc;
  }
  __syncthreads();
  *total = sh[kFinThreads / 32];
  return sh[warp] + incl - v;
}

// Copy records [pos0, pos0 + n), written by this warp, from the device
// arrays to the host result, with their row-major coordinates; lane t takes
// records pos0 + t, pos0 + t + 32, ... so the stores coalesce.
__device__ void publish_records(const FkView &F, int64_t pos0, int64_t n) {
  __syncwarp();  // the warp's record stores are visible to its lanes
  int64_t *hidx = (int64_t *)F.hrec;
  double *hc = (double *)(hidx + F.first_k), *hr = hc + F.first_k;
  for (int64_t t = threadIdx.x & 31; t < n; t += 32) {
    const int64_t p = pos0 + t;
    int64_t idx = F.idx[p];
    hidx[p] = idx;
    hc[p] = F.c64[p];
    hr[p] = F.r64[p];
    if (F.coords) {
      int64_t *c = F.coords + p * F.rank;
      for (int d = F.rank - 1; d >= 0; --d) {
        const Div64 sd = F.sdiv[d];
        if (sd.d == 0) {
          c[d] = 0;
          idx = 0;
        } else {
          const uint64_t q = div_q((uint64_t)idx, sd.d, sd.m);
          c[d] = idx - (int64_t)(q * sd.d);
          idx = (int64_t)q;
        }
      }
    }
  }
}

// Re-read elements [lo, hi) (one batch, lo batch-aligned) with one warp
// and write the first `needed` mismatches at record positions pos0, pos0 +
// 1, ...  Lane l takes the V elements at lo + u * 32V + lV of each warp step
// u, as the scan does; only the steps the scan marked in sbits (those
// holding mismatches) are read.  Their vectors are loaded up front and put
// through the sure-pass filter together, so a batch costs one memory
// latency and little more; only steps where some element is not surely
// passing go through the full predicate and the warp-wide ordered
// compaction that places their records.  With a host result, the records
// are then copied there with their coordinates.
template <int DT>
__device__ void reread_warp(const FkView &F, int64_t lo, int64_t hi, int64_t pos0, int64_t needed, uint32_t sbits) {
  constexpr int V = Tr<DT>::V;
  constexpr int EB = Tr<DT>::EB;
  constexpr int STEP = 32 * V;
  constexpr int G = kMaxSteps;
  const int lane = threadIdx.x & 31;
  uint4 cv[G], rv[G];
#pragma unroll
  for (int u = 0; u < G; ++u) {
    const int64_t i0 = lo + u * STEP + lane * V;
    if (!((sbits >> u) & 1u)) {
      cv[u] = rv[u] = make_uint4(0, 0, 0, 0);  // no mismatch in this step
    } else if (F.vec_ok && i0 + V <= hi) {
      cv[u] = ld_v4(F.cand + i0 * EB);
      rv[u] = ld_v4(F.ref + i0 * EB);
    } else {
      uint32_t cw[4] = {0, 0, 0, 0}, rw[4] = {0, 0, 0, 0};
#pragma unroll
      for (int k = 0; k < V; ++k) {
        if (i0 + k < hi) {
          const uint32_t c = ld_one<EB>(F.cand, i0 + k), r = ld_one<EB>(F.ref, i0 + k);
          if constexpr (EB == 2) {
            cw[k >> 1] |= c << (16 * (k & 1));
            rw[k >> 1] |= r << (16 * (k & 1));
          } else {
            cw[k] = c;
            rw[k] = r;
          }
        }
      }
      cv[u] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
      rv[u] = make_uint4(rw[0], rw[1], rw[2], rw[3]);
    }
  }
  // elements of each step that the filter does not pass outright
  uint32_t open[G];
#pragma unroll
  for (int u = 0; u < G; ++u) {
    const int64_t i0 = lo + u * STEP + lane * V;
    uint32_t m = 0;
    if ((sbits >> u) & 1u) {
#pragma unroll
      for (int k = 0; k < V; ++k)
        if (i0 + k < hi && !sure_pass<DT>(F, vbits<DT>(cv[u], k), vbits<DT>(rv[u], k))) m |= 1u << k;
    }
    open[u] = m;
  }
  int64_t found = 0;
#pragma unroll
  for (int u = 0; u < G; ++u) {
    if (!__any_sync(0xffffffffu, open[u] != 0)) continue;
    const int64_t i0 = lo + u * STEP + lane * V;
    uint32_t mask = 0;
#pragma unroll
    for (int k = 0; k < V; ++k)
      if (((open[u] >> k) & 1u) && !pass_elem<DT>(F, vbits<DT>(cv[u], k), vbits<DT>(rv[u], k))) mask |= 1u << k;
    const int cnt = __popc(mask);
    int incl = cnt;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= d) incl += t;
    }
    int64_t pos = found + incl - cnt;
#pragma unroll
    for (int k = 0; k < V; ++k) {
      if (((mask >> k) & 1u) && pos < needed) {
        F.idx[pos0 + pos] = i0 + k;
        F.c64[pos0 + pos] = to_f64<DT>(vbits<DT>(cv[u], k));
        F.r64[pos0 + pos] = to_f64<DT>(vbits<DT>(rv[u], k));
      }
      pos += (mask >> k) & 1u;
    }
    found += __shfl_sync(0xffffffffu, incl, 31);
    if (found >= needed) break;
  }
  if (F.hrec) publish_records(F, pos0, found < needed ? found : needed);
}

// One round of the record pass over a run of at most kFinChunk consecutive
// counts (pieces' or batches'): thread t takes the kFinPer counts at
// t * kFinPer, ...; a block scan gives each count its first record position
// (from `pos`) and each nonzero count its slot among the nonzero ones, so
// every block derives the same ordered work list.
constexpr int kFinPer = 4;
constexpr int kFinChunk = kFinThreads * kFinPer;

struct FkItem {
  int64_t pos;     // first record position
  int32_t id;      // piece (within the launch) or batch (within the piece)
  uint32_t sbits;  // a batch's warp steps that hold mismatches
};

// One round of the batch level of the record pass: the counts of the
// case's batches b0, b0 + 1, ... (global indices; at most kFinChunk, up to
// the case's last batch), the first of which starts at record position pos
// (< K).  A block scan gives each batch its first record position, and
// every batch holding records below K is re-read by one warp of the nw
// warps of the case's record blocks (this warp is number gw of them).  The
// case's pieces are contiguous and cut at batch boundaries, so batch b
// starts at element (b - batch_begin) * batch_elems.  Returns the position
// after the round's batches.  Called by the whole block with uniform
// arguments.
__device__ int64_t first_k_batches(const FkView &F, const CaseDesc &cd, int dt, int nin,
                                   const int32_t *batch_count, int64_t b0, int64_t pos, int64_t K, int gw, int nw,
                                   int64_t *sh_scan, FkItem *sh_item, int *sh_cnt) {
  const int64_t be = batch_elems(dt, nin);
  const int64_t bt = b0 + (int64_t)threadIdx.x * kFinPer;
  int32_t n[kFinPer];
  uint32_t sb[kFinPer];
  // records in the low 32 bits (a round holds at most kFinChunk * be),
  // nonzero counts in the high ones
  int64_t packed = 0;
#pragma unroll
  for (int t = 0; t < kFinPer; ++t) {
    const uint32_t w = bt + t < cd.batch_end ? (uint32_t)batch_count[bt + t] : 0u;
    n[t] = (int32_t)(w & kBatchCountMask);
    sb[t] = w >> kStepBitsShift;
    packed += (int64_t)n[t] + (n[t] > 0 ? (int64_t(1) << 32) : 0);
  }
  int64_t total;
  const int64_t ex = block_excl_scan64(packed, &total, sh_scan);
  const int64_t end_pos = pos + (total & 0xffffffffll);
  const int n_nz = (int)(total >> 32);
  int64_t pre = pos + (ex & 0xffffffffll);
  int slot = (int)(ex >> 32);
#pragma unroll
  for (int t = 0; t < kFinPer; ++t) {
    if (n[t] > 0) {
      sh_item[slot] = {pre, (int32_t)(threadIdx.x * kFinPer + t), sb[t]};
      // the last batch starting below K ends at or beyond it
      if (pre < K && pre + n[t] >= K) *sh_cnt = slot + 1;
      ++slot;
    }
    pre += n[t];
  }
  __syncthreads();
  const int items = end_pos < K ? n_nz : *sh_cnt;
  for (int j = gw; j < items; j += nw) {
    const int64_t pre_j = sh_item[j].pos;
    const int64_t lo = (b0 + sh_item[j].id - cd.batch_begin) * be;
    const int64_t hi = lo + be < cd.numel ? lo + be : cd.numel;
    const int64_t nxt = j + 1 < n_nz ? sh_item[j + 1].pos : end_pos;
    const int64_t need = nxt < K ? nxt - pre_j : K - pre_j;
    const uint32_t sbits = sh_item[j].sbits;
    switch (dt) {
      case NMV_F32: reread_warp<NMV_F32>(F, lo, hi, pre_j, need, sbits); break;
      case NMV_F16: reread_warp<NMV_F16>(F, lo, hi, pre_j, need, sbits); break;
      case NMV_BF16: reread_warp<NMV_BF16>(F, lo, hi, pre_j, need, sbits); break;
      default: reread_warp<NMV_I32>(F, lo, hi, pre_j, need, sbits); break;
    }
  }
  __syncthreads();
  return end_pos;
}

// Move n 8-byte words (n even or not; src and dst 16-byte aligned) from the
// device to the host result and leave zeros behind, block `part` of
// `parts`: each thread moves 16-byte pairs four at a time, loads first.
__device__ void move_words(uint8_t *src, uint8_t *dst, int64_t n, int part, int parts) {
  uint4 *s = (uint4 *)src, *d = (uint4 *)dst;
  const int64_t n2 = n / 2;
  const int64_t stride = (int64_t)parts * kFinThreads;
  for (int64_t t0 = (int64_t)part * kFinThreads + threadIdx.x; t0 < n2; t0 += 4 * stride) {
    uint4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) v[u] = t0 + u * stride < n2 ? s[t0 + u * stride] : make_uint4(0, 0, 0, 0);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (t0 + u * stride < n2) {
        d[t0 + u * stride] = v[u];
        if (v[u].x | v[u].y | v[u].z | v[u].w) s[t0 + u * stride] = make_uint4(0, 0, 0, 0);
      }
    }
  }
  if ((n & 1) && part == 0 && threadIdx.x == 0) {
    unsigned long long *s1 = (unsigned long long *)src + (n - 1);
    const unsigned long long v = *s1;
    ((unsigned long long *)dst)[n - 1] = v;
    if (v) *s1 = 0ull;
  }
}

// What the first block reduces of the partials (the pass-through counts
// are summed separately, only for cases with inputs).
struct Red {
  int64_t cnt[8];
  Best ba, br;
  double sse;
  uint32_t cacc, racc;
};

__device__ __forceinline__ void red_clear(Red &a) {
  for (int k = 0; k < 8; ++k) a.cnt[k] = 0;
  a.ba = {-1.0, INT64_MAX};
  a.br = {-1.0, INT64_MAX};
  a.sse = 0.0;
  a.cacc = a.racc = 0;
}

__device__ __forceinline__ void red_load(Red &a, const Partial &Q) {
  for (int k = 0; k < 8; ++k) a.cnt[k] = Q.cnt[k];
  a.ba = {Q.best_abs, Q.arg_abs};
  a.br = {Q.best_rel, Q.arg_rel};
  a.sse = Q.sse;
  a.cacc = Q.cacc;
  a.racc = Q.racc;
}

__device__ __forceinline__ void red_add(Red &a, const Red &b) {
  for (int k = 0; k < 8; ++k) a.cnt[k] += b.cnt[k];
  best_offer(a.ba, b.ba.v, b.ba.i);
  best_offer(a.br, b.br.v, b.br.i);
  a.sse = __dadd_rn(a.sse, b.sse);
  a.cacc |= b.cacc;
  a.racc |= b.racc;
}

__global__ void __launch_bounds__(kFinThreads, 2) finalize_kernel(const CaseDesc *__restrict__ cases,
                                                               const Piece *__restrict__ pieces,
                                                               const Partial *__restrict__ partials,
                                                               const int32_t *__restrict__ batch_count,
                                                               uint8_t *out, uint8_t *hout, uint8_t *zthr,
                                                               size_t zthr_bytes) {
  const CaseDesc &cd = cases[blockIdx.x];
  // block 0 of the case reduces; with helpers, blocks 1 .. helpers write the
  // records meanwhile, else block 0 writes them afterwards (the descriptors
  // were uploaded before the scan started)
  const int helpers = cd.fin_help;
  const int y = blockIdx.y;
  if (y > helpers) return;
  // the inputs' first elements (for the degenerate-output flags) do not
  // depend on the scan: read before waiting for it
  uint32_t c0 = 0, r0 = 0;
  if (y == 0 && threadIdx.x == 0 && cd.numel >= 1) {
    c0 = ld_elem(cd.cand, 0, cd.dtype);
    r0 = ld_elem(cd.ref, 0, cd.dtype);
  }
  // launched as the scan's programmatic dependent: wait until the scan grid
  // has completed and its writes are visible (a no-op otherwise)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // o: the case's part of the device output (the scan's accumulators); ho:
  // where the packed result goes (the host result block when hout is set)
  uint8_t *o = out + cd.out_off;
  uint8_t *ho = hout ? hout + cd.out_off : o;
  OutHeader *H = (OutHeader *)ho;
  if (hout) {
    // The maps go to the host block and their accumulators back to zero for
    // the next call, shared over the case's blocks; block (0, 0) does the
    // same for the call's counters and error word and clears the published
    // maxima and piece counters.
    const int nb = helpers + 1;
    move_words(o + cd.hist_off, ho + cd.hist_off, cd.hist_n, y, nb);
    move_words(o + cd.rowp_off, ho + cd.rowp_off, cd.rowp_n, y, nb);
    move_words(o + cd.colp_off, ho + cd.colp_off, cd.colp_n, y, nb);
    if (blockIdx.x == 0 && y == 0) {
      // the call header to the host block; its words back to zero except the
      // scan's error word, which every block reads below (a failed call's
      // accumulators are cleared by the host before the next call)
      unsigned long long *src = (unsigned long long *)out, *dst = (unsigned long long *)hout;
      for (int t = threadIdx.x; t < (int)(kCallHeader / 8); t += kFinThreads) {
        const unsigned long long v = src[t];
        dst[t] = v;
        if (v && t != (int)(kCallErrOff / 8)) src[t] = 0ull;
      }
      for (size_t t = threadIdx.x; t < zthr_bytes / 8; t += kFinThreads) ((unsigned long long *)zthr)[t] = 0ull;
    }
  }
  // A scan that gave up waiting for its copies left batch counts and
  // partials incomplete (the call is void and reports NMV_ETIMEOUT): nothing
  // more is read.
  if (*(volatile const uint32_t *)(out + kCallErrOff) != 0) return;
  __shared__ int64_t sh_scan[kFinThreads / 32 + 1];
  __shared__ int64_t sh_mism;
  __shared__ FkItem sh_need[kFinChunk], sh_item[kFinChunk];
  __shared__ int sh_cnt;
  __shared__ Red sh_red[kFinThreads / 32];
  __shared__ int64_t sh_eq[NMV_MAX_INPUTS];

  if (y == 0) {
    // ---- 1. reduce the partials: thread t takes pieces t, t + kFinThreads,
    // ... in order, then a fixed butterfly within each warp and the warps in
    // order (the same tree on every run).
    {
      Red a;
      red_clear(a);
      // partials two at a time per thread, both loads before the adds (the
      // order of the adds is the thread's pieces in ascending order)
      for (int64_t p0 = cd.piece_begin + threadIdx.x; p0 < cd.piece_end; p0 += 2 * kFinThreads) {
        const int64_t p1 = p0 + kFinThreads;
        Red b0, b1;
        red_load(b0, partials[p0]);
        if (p1 < cd.piece_end) red_load(b1, partials[p1]);
        red_add(a, b0);
        if (p1 < cd.piece_end) red_add(a, b1);
      }
  #pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        Red b;
  #pragma unroll
        for (int k = 0; k < 8; ++k) b.cnt[k] = __shfl_xor_sync(0xffffffffu, a.cnt[k], off);
        b.ba.v = __shfl_xor_sync(0xffffffffu, a.ba.v, off);
        b.ba.i = __shfl_xor_sync(0xffffffffu, a.ba.i, off);
        b.br.v = __shfl_xor_sync(0xffffffffu, a.br.v, off);
        b.br.i = __shfl_xor_sync(0xffffffffu, a.br.i, off);
        b.sse = __shfl_xor_sync(0xffffffffu, a.sse, off);
        b.cacc = __shfl_xor_sync(0xffffffffu, a.cacc, off);
        b.racc = __shfl_xor_sync(0xffffffffu, a.racc, off);
        // lanes below the partner add the partner's value second, lanes above
        // first, so both hold the same bits
        if ((threadIdx.x & off) == 0) {
          red_add(a, b);
        } else {
          red_add(b, a);
          a = b;
        }
      }
      if ((threadIdx.x & 31) == 0) sh_red[threadIdx.x >> 5] = a;
      // the pass-through counts (integers: any order)
      if (threadIdx.x < NMV_MAX_INPUTS) sh_eq[threadIdx.x] = 0;
      __syncthreads();
      if (cd.n_elig > 0) {
        int64_t e[NMV_MAX_INPUTS];
  #pragma unroll
        for (int j = 0; j < NMV_MAX_INPUTS; ++j) e[j] = 0;
        for (int64_t p = cd.piece_begin + threadIdx.x; p < cd.piece_end; p += kFinThreads) {
  #pragma unroll
          for (int j = 0; j < NMV_MAX_INPUTS; ++j)
            if (j < cd.n_elig) e[j] += partials[p].eq[j];
        }
  #pragma unroll
        for (int j = 0; j < NMV_MAX_INPUTS; ++j) {
          if (j < cd.n_elig) {
            const int64_t t = warp_reduce(e[j], [](int64_t x, int64_t y) { return x + y; });
            if ((threadIdx.x & 31) == 0) atomicAdd((unsigned long long *)&sh_eq[j], (unsigned long long)t);
          }
        }
      }
      if (threadIdx.x == 0) {
        for (int w = 1; w < kFinThreads / 32; ++w) red_add(sh_red[0], sh_red[w]);
      }
      __syncthreads();
    }
    if (threadIdx.x == 0) {
      const Red &a = sh_red[0];
      for (int k = 0; k < 7; ++k) H->cnt[k] = a.cnt[k];
      H->cnt[7] = cd.numel - a.cnt[7];  // n_finite_pairs
      H->max_abs = a.ba.v < 0.0 ? 0.0 : a.ba.v;
      H->argmax_abs = a.ba.v < 0.0 ? -1 : a.ba.i;
      H->max_rel = a.br.v < 0.0 ? 0.0 : a.br.v;
      H->argmax_rel = a.br.v < 0.0 ? -1 : a.br.i;
      H->sse = a.sse;
      H->k_out = a.cnt[0] < cd.first_k ? a.cnt[0] : cd.first_k;
      // degenerate-output flags
      uint32_t flags = 0;
      int32_t pt = -1;
      for (int j = 0; j < NMV_MAX_INPUTS; ++j) H->input_eq[j] = -1;
      for (int j = 0; j < cd.n_elig; ++j) H->input_eq[cd.in_slot[j]] = sh_eq[j];
      const int64_t thr = cd.numel >= 100 ? (cd.numel + 99) / 100 : 1;
      for (int j = 0; j < cd.n_inputs; ++j) {
        if (H->input_eq[j] >= thr) {
          flags |= NMV_FLAG_CAND_EQ_INPUT;
          if (pt < 0) pt = j;
        }
      }
      if (cd.numel >= 1) {
        const bool two = elem_bytes(cd.dtype) == 2;
          const uint32_t mag = cd.dtype == NMV_I32 ? 0xffffffffu : (two ? 0x7fffu : 0x7fffffffu);
        const uint32_t cfold = two ? ((a.cacc | (a.cacc >> 16)) & 0xffffu) : a.cacc;
        const uint32_t rfold = two ? ((a.racc | (a.racc >> 16)) & 0xffffu) : a.racc;
        if ((c0 & mag) == 0 && (cfold & mag) == 0) flags |= NMV_FLAG_CAND_ALL_ZERO;
        if ((r0 & mag) == 0 && (rfold & mag) == 0) flags |= NMV_FLAG_REF_ALL_ZERO;
        if (cd.numel >= 2 && cfold == 0) flags |= NMV_FLAG_CAND_CONSTANT;
        if (cd.numel >= 2 && rfold == 0) flags |= NMV_FLAG_REF_CONSTANT;
      }
      H->flags = flags;
      H->passthrough = pt;
      H->status = 0;
      sh_mism = a.cnt[0];
    }
    __syncthreads();
    if (helpers > 0 || cd.first_k == 0 || sh_mism == 0) return;
  }

  // ---- 2. first-K records, in two levels.  The pieces' mismatch counts
  // are taken kFinChunk at a time: block scans of them and of their nonzero
  // flags give each piece its first record position and each nonzero piece
  // its slot, in order.  From the first piece holding records below K, the
  // batch counts are then scanned kFinChunk batches at a time across piece
  // boundaries (first_k_batches), jumping over runs of pieces without
  // records, until K records are placed.
  const int64_t K = cd.first_k;
  if (K == 0) return;
  const FkView F = fk_view(cd, o, hout ? ho : nullptr, hout);
  const int dt = cd.dtype, nin = nin_class_of(cd.n_elig);
  // items go round the blocks first, so a few items land on different SMs
  const int gw = helpers > 0 ? (y - 1) + helpers * (threadIdx.x >> 5) : (threadIdx.x >> 5);
  const int nw = (helpers > 0 ? helpers : 1) * (kFinThreads / 32);
  int64_t base = 0;               // records in the pieces before this round
  int64_t cur = cd.batch_begin;   // first batch not scanned yet
  int64_t pos = 0;                // records before batch cur
  for (int64_t q0 = cd.piece_begin; q0 < cd.piece_end && base < K && pos < K; q0 += kFinChunk) {
    const int64_t qt = q0 + (int64_t)threadIdx.x * kFinPer;
    int64_t n[kFinPer], s = 0, nz = 0;
#pragma unroll
    for (int t = 0; t < kFinPer; ++t) {
      n[t] = qt + t < cd.piece_end ? partials[qt + t].cnt[0] : 0;
      s += n[t];
      nz += n[t] > 0;
    }
    int64_t total, n_nz;
    int64_t pre = base + block_excl_scan64(s, &total, sh_scan);
    int64_t slot = block_excl_scan64(nz, &n_nz, sh_scan);
#pragma unroll
    for (int t = 0; t < kFinPer; ++t) {
      if (n[t] > 0) sh_need[slot++] = {pre, (int32_t)(qt + t), 0u};
      pre += n[t];
    }
    __syncthreads();
    for (int64_t j = 0; j < n_nz && pos < K; ++j) {
      const int64_t pos0 = sh_need[j].pos;
      if (pos0 >= K) break;
      const Piece &pc = pieces[sh_need[j].id];
      const int64_t pend = pc.batch_base + piece_batches(pc.begin, pc.end, dt, nin);
      if (pend <= cur) continue;  // scanned with an earlier piece
      if (pc.batch_base > cur) {
        cur = pc.batch_base;      // the batches before hold no records
        pos = pos0;
      }
      while (cur < pend && pos < K) {
        pos = first_k_batches(F, cd, dt, nin, batch_count, cur, pos, K, gw, nw, sh_scan, sh_item, &sh_cnt);
        cur = cur + kFinChunk < cd.batch_end ? cur + kFinChunk : cd.batch_end;
      }
    }
    base += total;
    __syncthreads();
  }
}

// ---- fp64 SSE re-pass: block b sums its contiguous range in index order per
// thread, then a fixed tree; sse64_final adds the block sums in order.
constexpr int kSseBlocks = 1024;

__global__ void __launch_bounds__(kFinThreads) sse64_kernel(const CaseDesc *__restrict__ cd_p, double *part) {
  const CaseDesc &cd = *cd_p;
  __shared__ double sh[kFinThreads];
  const int64_t per_block = (cd.numel + gridDim.x - 1) / gridDim.x;
  const int64_t b0 = (int64_t)blockIdx.x * per_block;
  const int64_t b1 = b0 + per_block < cd.numel ? b0 + per_block : cd.numel;
  const int64_t per_thr = (per_block + kFinThreads - 1) / kFinThreads;
  const int64_t t0 = b0 + (int64_t)threadIdx.x * per_thr;
  const int64_t t1 = t0 + per_thr < b1 ? t0 + per_thr : b1;
  double acc = 0.0;
  for (int64_t i = t0; i < t1; ++i) {
    const double c = widen_any(ld_elem(cd.cand, i, cd.dtype), cd.dtype);
    const double r = widen_any(ld_elem(cd.ref, i, cd.dtype), cd.dtype);
    if (isfinite(c) && isfinite(r)) {
      const double d = __dsub_rn(c, r);
      acc = __dadd_rn(acc, __dmul_rn(d, d));
    }
  }
  sh[threadIdx.x] = acc;
  __syncthreads();
  for (int half = kFinThreads / 2; half > 0; half >>= 1) {
    if (threadIdx.x < half) sh[threadIdx.x] = __dadd_rn(sh[threadIdx.x], sh[threadIdx.x + half]);
    __syncthreads();
  }
  if (threadIdx.x == 0) part[blockIdx.x] = sh[0];
}

__global__ void sse64_final(const double *part, int n, double *dst) {
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    double acc = 0.0;
    for (int b = 0; b < n; ++b) acc = __dadd_rn(acc, part[b]);
    *dst = acc;
  }
}

// Grid: one column of 1 + max_helpers blocks per case (CaseDesc::fin_help).
// With hout set (a device pointer to mapped host memory laid out like
// out), the packed results go there directly, the accumulators in out are
// left zero, and so are the zthr_bytes (a multiple of 8) at zthr.
// Launched with programmatic stream serialization: its blocks may start
// while the scan kernel before it on the stream drains, and wait for it
// inside (griddepcontrol.wait).
cudaError_t launch_finalize(const CaseDesc *cases, const Piece *pieces, const Partial *partials,
                            const int32_t *batch_count, uint8_t *out, uint8_t *hout, uint8_t *zthr,
                            size_t zthr_bytes, int n_cases, int max_helpers, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_cases, 1 + max_helpers);
  cfg.blockDim = dim3(kFinThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, finalize_kernel, cases, pieces, partials, batch_count, out, hout,
                                           zthr, zthr_bytes);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// Recompute one case's SSE in fp64 into *dst (device).  `part` holds
// kSseBlocks doubles of scratch.
cudaError_t launch_sse64(const CaseDesc *cd, double *part, double *dst, cudaStream_t st) {
  sse64_kernel<<<kSseBlocks, kFinThreads, 0, st>>>(cd, part);
  sse64_final<<<1, 32, 0, st>>>(part, kSseBlocks, dst);
  return cudaGetLastError();
}

}  // namespace nmv
