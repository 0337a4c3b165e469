// nmv_finalize.cu -- one block per case: reduce the piece partials of the
// scan pass in piece order (deterministic), derive the degenerate-output
// flags, and write the first-K mismatch records: copied from the per-segment
// offset lists, or found by re-reading a segment whose list overflowed.
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

// Exclusive block-wide prefix sum of v; *total = the block's sum.
__device__ __forceinline__ int block_excl_scan(int v, int *total, int *sh /*[kFinThreads/32 + 1]*/) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  __syncthreads();
  if (lane == 31) sh[warp] = incl;
  __syncthreads();
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int w = 0; w < kFinThreads / 32; ++w) {
      const int t = sh[w];
      sh[w] = acc;
      acc += t;
    }
    sh[kFinThreads / 32] = acc;
  }
  __syncthreads();
  *total = sh[kFinThreads / 32];
  return sh[warp] + incl - v;
}

__device__ void write_record(const CaseDesc &cd, uint8_t *o, int64_t pos, int64_t idx) {
  int64_t *fk_index = (int64_t *)(o + cd.fk_off);
  double *fk_c = (double *)(fk_index + cd.first_k);
  double *fk_r = fk_c + cd.first_k;
  fk_index[pos] = idx;
  fk_c[pos] = widen_any(ld_elem(cd.cand, idx, cd.dtype), cd.dtype);
  fk_r[pos] = widen_any(ld_elem(cd.ref, idx, cd.dtype), cd.dtype);
}

// Re-read segment [lo, hi) and write its first `needed` mismatches at
// record positions pos0, pos0 + 1, ...  (the whole block, E elements per
// thread, block-wide ordered compaction).
__device__ void reread_segment(const CaseDesc &cd, uint8_t *o, int64_t lo, int64_t hi, int64_t pos0,
                               int64_t needed, int *sh) {
  constexpr int E = 8;
  int64_t found = 0;
  for (int64_t base = lo; base < hi && found < needed; base += (int64_t)kFinThreads * E) {
    const int64_t i0 = base + (int64_t)threadIdx.x * E;
    uint32_t mask = 0;
    for (int k = 0; k < E; ++k) {
      const int64_t i = i0 + k;
      if (i < hi) {
        const double c = widen_any(ld_elem(cd.cand, i, cd.dtype), cd.dtype);
        const double r = widen_any(ld_elem(cd.ref, i, cd.dtype), cd.dtype);
        if (!pass64(c, r, cd.rtol, cd.atol)) mask |= 1u << k;
      }
    }
    int total;
    const int excl = block_excl_scan(__popc(mask), &total, sh);
    int64_t pos = found + excl;
    while (mask) {
      const int k = __ffs(mask) - 1;
      mask &= mask - 1;
      if (pos < needed) write_record(cd, o, pos0 + pos, i0 + k);
      ++pos;
    }
    found += total;
  }
}

__global__ void __launch_bounds__(kFinThreads) finalize_kernel(const CaseDesc *__restrict__ cases,
                                                               const Piece *__restrict__ pieces,
                                                               const Partial *__restrict__ partials,
                                                               const int32_t *__restrict__ seg_count,
                                                               const uint32_t *__restrict__ seg_list,
                                                               uint8_t *out) {
  const CaseDesc &cd = cases[blockIdx.x];
  uint8_t *o = out + cd.out_off;
  OutHeader *H = (OutHeader *)o;
  __shared__ int sh_scan[kFinThreads / 32 + 1];
  __shared__ int64_t sh_mism;
  __shared__ int64_t sh_re[kFinThreads][3];
  __shared__ int sh_nre;

  // ---- 1. reduce the partials of this case in piece order
  if (threadIdx.x == 0) {
    int64_t cnt[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    Best ba = {-1.0, INT64_MAX}, br = {-1.0, INT64_MAX};
    double sse = 0.0;
    uint32_t cacc = 0, racc = 0;
    int64_t eq[NMV_MAX_INPUTS] = {0, 0, 0, 0, 0, 0, 0, 0};
    for (int64_t p = cd.piece_begin; p < cd.piece_end; ++p) {
      const Partial &Q = partials[p];
      for (int k = 0; k < 8; ++k) cnt[k] += Q.cnt[k];
      best_offer(ba, Q.best_abs, Q.arg_abs);
      best_offer(br, Q.best_rel, Q.arg_rel);
      sse = __dadd_rn(sse, Q.sse);
      cacc |= Q.cacc;
      racc |= Q.racc;
      for (int j = 0; j < NMV_MAX_INPUTS; ++j) eq[j] += Q.eq[j];
    }
    for (int k = 0; k < 7; ++k) H->cnt[k] = cnt[k];
    H->cnt[7] = cd.numel - cnt[7];  // n_finite_pairs
    H->max_abs = ba.v < 0.0 ? 0.0 : ba.v;
    H->argmax_abs = ba.v < 0.0 ? -1 : ba.i;
    H->max_rel = br.v < 0.0 ? 0.0 : br.v;
    H->argmax_rel = br.v < 0.0 ? -1 : br.i;
    H->sse = sse;
    H->k_out = cnt[0] < cd.first_k ? cnt[0] : cd.first_k;
    // degenerate-output flags
    uint32_t flags = 0;
    int32_t pt = -1;
    for (int j = 0; j < NMV_MAX_INPUTS; ++j) H->input_eq[j] = -1;
    for (int j = 0; j < cd.n_elig; ++j) H->input_eq[cd.in_slot[j]] = eq[j];
    const int64_t thr = cd.numel >= 100 ? (cd.numel + 99) / 100 : 1;
    for (int j = 0; j < cd.n_inputs; ++j) {
      if (H->input_eq[j] >= thr) {
        flags |= NMV_FLAG_CAND_EQ_INPUT;
        if (pt < 0) pt = j;
      }
    }
    if (cd.numel >= 1) {
      const bool two = elem_bytes(cd.dtype) == 2;
      const uint32_t c0 = ld_elem(cd.cand, 0, cd.dtype), r0 = ld_elem(cd.ref, 0, cd.dtype);
      const uint32_t mag = cd.dtype == NMV_I32 ? 0xffffffffu : (two ? 0x7fffu : 0x7fffffffu);
      const uint32_t cfold = two ? ((cacc | (cacc >> 16)) & 0xffffu) : cacc;
      const uint32_t rfold = two ? ((racc | (racc >> 16)) & 0xffffu) : racc;
      if ((c0 & mag) == 0 && (cfold & mag) == 0) flags |= NMV_FLAG_CAND_ALL_ZERO;
      if ((r0 & mag) == 0 && (rfold & mag) == 0) flags |= NMV_FLAG_REF_ALL_ZERO;
      if (cd.numel >= 2 && cfold == 0) flags |= NMV_FLAG_CAND_CONSTANT;
      if (cd.numel >= 2 && rfold == 0) flags |= NMV_FLAG_REF_CONSTANT;
    }
    H->flags = flags;
    H->passthrough = pt;
    H->status = 0;
    sh_mism = cnt[0];
  }
  __syncthreads();

  // ---- 2. first-K records, segment by segment in index order
  const int64_t K = cd.first_k;
  if (K == 0 || sh_mism == 0) return;
  const int vec = vec_elems(cd.dtype);
  const int64_t s0 = cd.piece_begin * kWarps, s1 = cd.piece_end * kWarps;
  int64_t carry = 0;
  for (int64_t sb = s0; sb < s1 && carry < K; sb += kFinThreads) {
    const int64_t s = sb + threadIdx.x;
    const int cnt = s < s1 ? seg_count[s] : 0;
    int total;
    const int excl = block_excl_scan(cnt, &total, sh_scan);
    if (threadIdx.x == 0) sh_nre = 0;
    __syncthreads();
    const int64_t prefix = carry + excl;
    if (cnt > 0 && prefix < K) {
      const int64_t needed = (K - prefix) < cnt ? (K - prefix) : cnt;
      const Piece &pc = pieces[s / kWarps];
      int64_t lo, hi;
      segment_range(pc.begin, pc.end, (int)(s % kWarps), vec, &lo, &hi);
      if (needed <= kFirstR) {
        for (int64_t j = 0; j < needed; ++j) write_record(cd, o, prefix + j, lo + seg_list[s * kFirstR + j]);
      } else {
        const int slot = atomicAdd(&sh_nre, 1);
        sh_re[slot][0] = s;
        sh_re[slot][1] = prefix;
        sh_re[slot][2] = needed;
      }
    }
    __syncthreads();
    const int nre = sh_nre;
    for (int t = 0; t < nre; ++t) {
      const int64_t s2 = sh_re[t][0];
      const Piece &pc = pieces[s2 / kWarps];
      int64_t lo, hi;
      segment_range(pc.begin, pc.end, (int)(s2 % kWarps), vec, &lo, &hi);
      reread_segment(cd, o, lo, hi, sh_re[t][1], sh_re[t][2], sh_scan);
    }
    carry += total;
    __syncthreads();
  }
}

cudaError_t launch_finalize(const CaseDesc *cases, const Piece *pieces, const Partial *partials,
                            const int32_t *seg_count, const uint32_t *seg_list, uint8_t *out,
                            int n_cases, cudaStream_t st) {
  finalize_kernel<<<n_cases, kFinThreads, 0, st>>>(cases, pieces, partials, seg_count, seg_list, out);
  return cudaGetLastError();
}

}  // namespace nmv
