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

// The predicate with the scan pass's fp32 pre-filter (same decision).
template <int DT>
__device__ __forceinline__ bool pass_elem(const CaseDesc &cd, uint32_t cb, uint32_t rb) {
  const float cf = to_f32<DT>(cb), rf = to_f32<DT>(rb);
  if constexpr (Tr<DT>::kInt) {
    if (cb == rb) return true;
    const long long d = (long long)(int32_t)cb - (long long)(int32_t)rb;
    const float as = fabsf(__ll2float_rn(d)), ar = fabsf(rf);
    if (as <= __fmaf_rz(cd.lo_r, ar, cd.lo_a)) return true;
    if (as > __fmaf_ru(cd.hi_r, ar, cd.hi_a)) return false;
  } else {
    if (cf == rf) return true;
    if (!(isfinite(cf) && isfinite(rf))) return false;
    const float as = fabsf(__fsub_rn(cf, rf)), ar = fabsf(rf);
    if (as <= __fmaf_rz(cd.lo_r, ar, cd.lo_a)) return true;
    if (as > __fmaf_ru(cd.hi_r, ar, cd.hi_a)) return false;
  }
  return pass64(to_f64<DT>(cb), to_f64<DT>(rb), cd.rtol, cd.atol);
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

__device__ __forceinline__ void write_record(const CaseDesc &cd, uint8_t *o, int64_t pos, int64_t idx,
                                             uint32_t cb, uint32_t rb) {
  int64_t *fk_index = (int64_t *)(o + cd.fk_off);
  double *fk_c = (double *)(fk_index + cd.first_k);
  double *fk_r = fk_c + cd.first_k;
  fk_index[pos] = idx;
  fk_c[pos] = widen_any(cb, cd.dtype);
  fk_r[pos] = widen_any(rb, cd.dtype);
}

// Re-read elements [lo, hi) (one batch, lo batch-aligned) with one warp
// and write the first `needed` mismatches at record positions pos0, pos0 +
// 1, ...  Lane l takes the V elements at lo + u * 32V + lV of each warp step
// u, as the scan does; a 16-byte aligned case loads all of the batch's
// vectors up front, so the batch costs one memory latency.  Records are
// placed by a warp-wide ordered compaction, step by step.
template <int DT>
__device__ void reread_warp(const CaseDesc &cd, uint8_t *o, int64_t lo, int64_t hi, int64_t pos0,
                            int64_t needed) {
  constexpr int V = Tr<DT>::V;
  constexpr int EB = Tr<DT>::EB;
  constexpr int STEP = 32 * V;
  const int lane = threadIdx.x & 31;
  const int ks = batch_steps(nin_class_of(cd.n_elig));
  uint4 cv[kMaxSteps], rv[kMaxSteps];
#pragma unroll
  for (int u = 0; u < kMaxSteps; ++u) {
    const int64_t i0 = lo + u * STEP + lane * V;
    if (u >= ks) {
      cv[u] = rv[u] = make_uint4(0, 0, 0, 0);
      continue;
    }
    if (cd.vec_ok && i0 + V <= hi) {
      cv[u] = ld_v4((const char *)cd.cand + i0 * EB);
      rv[u] = ld_v4((const char *)cd.ref + i0 * EB);
    } else {
      uint32_t cw[4] = {0, 0, 0, 0}, rw[4] = {0, 0, 0, 0};
      for (int k = 0; k < V; ++k) {
        if (i0 + k >= hi) break;
        const uint32_t c = ld_one<EB>(cd.cand, i0 + k), r = ld_one<EB>(cd.ref, i0 + k);
        if constexpr (EB == 2) {
          cw[k >> 1] |= c << (16 * (k & 1));
          rw[k >> 1] |= r << (16 * (k & 1));
        } else {
          cw[k] = c;
          rw[k] = r;
        }
      }
      cv[u] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
      rv[u] = make_uint4(rw[0], rw[1], rw[2], rw[3]);
    }
  }
  int64_t found = 0;
#pragma unroll
  for (int u = 0; u < kMaxSteps; ++u) {
    if (u >= ks) break;
    const int64_t i0 = lo + u * STEP + lane * V;
    uint32_t mask = 0;
#pragma unroll
    for (int k = 0; k < V; ++k)
      if (i0 + k < hi && !pass_elem<DT>(cd, vbits<DT>(cv[u], k), vbits<DT>(rv[u], k))) mask |= 1u << k;
    const int cnt = __popc(mask);
    int incl = cnt;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= d) incl += t;
    }
    const int64_t pos = found + incl - cnt;
    for (int k = 0, j = 0; k < V; ++k) {
      if ((mask >> k) & 1u) {
        if (pos + j < needed)
          write_record(cd, o, pos0 + pos + j, i0 + k, vbits<DT>(cv[u], k), vbits<DT>(rv[u], k));
        ++j;
      }
    }
    found += __shfl_sync(0xffffffffu, incl, 31);
    if (found >= needed) break;
  }
}

// Records of one piece whose first record has position pos0 (< K): its
// batches are taken kFinThreads at a time, a block scan of their mismatch
// counts places them, and each batch holding records below K is re-read by
// one warp.  Called by the whole block with uniform arguments.
__device__ void first_k_piece(const CaseDesc &cd, uint8_t *o, const Piece &pc, const int32_t *batch_count,
                              int64_t pos0, int64_t K, int64_t *sh_scan, int64_t (*sh_item)[3], int *sh_nitems) {
  const int nin = nin_class_of(cd.n_elig);
  const int64_t be = batch_elems(cd.dtype, nin);
  const int64_t nb = piece_batches(pc.begin, pc.end, cd.dtype, nin);
  const int warp = threadIdx.x >> 5;
  int64_t pos = pos0;
  for (int64_t b0 = 0; b0 < nb && pos < K; b0 += kFinThreads) {
    const int64_t b = b0 + threadIdx.x;
    const int64_t n = b < nb ? batch_count[pc.batch_base + b] : 0;
    int64_t total;
    const int64_t pre = pos + block_excl_scan64(n, &total, sh_scan);
    if (threadIdx.x == 0) *sh_nitems = 0;
    __syncthreads();
    if (n > 0 && pre < K) {
      const int it = atomicAdd(sh_nitems, 1);
      sh_item[it][0] = b;
      sh_item[it][1] = pre;
      sh_item[it][2] = n < K - pre ? n : K - pre;
    }
    __syncthreads();
    for (int j = warp; j < *sh_nitems; j += kFinThreads / 32) {
      const int64_t lo = pc.begin + sh_item[j][0] * be;
      const int64_t hi = lo + be < pc.end ? lo + be : pc.end;
      switch (cd.dtype) {
        case NMV_F32: reread_warp<NMV_F32>(cd, o, lo, hi, sh_item[j][1], sh_item[j][2]); break;
        case NMV_F16: reread_warp<NMV_F16>(cd, o, lo, hi, sh_item[j][1], sh_item[j][2]); break;
        case NMV_BF16: reread_warp<NMV_BF16>(cd, o, lo, hi, sh_item[j][1], sh_item[j][2]); break;
        default: reread_warp<NMV_I32>(cd, o, lo, hi, sh_item[j][1], sh_item[j][2]); break;
      }
    }
    __syncthreads();
    pos += total;
  }
}

struct Red {
  int64_t cnt[8];
  Best ba, br;
  double sse;
  uint32_t cacc, racc;
  int64_t eq[NMV_MAX_INPUTS];
};

__device__ __forceinline__ void red_add(Red &a, const Red &b) {
  for (int k = 0; k < 8; ++k) a.cnt[k] += b.cnt[k];
  best_offer(a.ba, b.ba.v, b.ba.i);
  best_offer(a.br, b.br.v, b.br.i);
  a.sse = __dadd_rn(a.sse, b.sse);
  a.cacc |= b.cacc;
  a.racc |= b.racc;
  for (int j = 0; j < NMV_MAX_INPUTS; ++j) a.eq[j] += b.eq[j];
}

__global__ void __launch_bounds__(kFinThreads) finalize_kernel(const CaseDesc *__restrict__ cases,
                                                               const Piece *__restrict__ pieces,
                                                               const Partial *__restrict__ partials,
                                                               const int32_t *__restrict__ batch_count,
                                                               uint8_t *out) {
  const CaseDesc &cd = cases[blockIdx.x];
  uint8_t *o = out + cd.out_off;
  OutHeader *H = (OutHeader *)o;
  __shared__ int64_t sh_scan[kFinThreads / 32 + 1];
  __shared__ int64_t sh_mism;
  __shared__ int64_t sh_need[kFinThreads], sh_need_p[kFinThreads];
  __shared__ int64_t sh_item[kFinThreads][3];
  __shared__ int sh_nitems;
  __shared__ Red sh_red[kFinThreads / 32];

  // ---- 1. reduce the partials: thread t takes pieces t, t + kFinThreads,
  // ... in order, then a fixed butterfly within each warp and the warps in
  // order (the same tree on every run).
  {
    Red a;
    for (int k = 0; k < 8; ++k) a.cnt[k] = 0;
    a.ba = {-1.0, INT64_MAX};
    a.br = {-1.0, INT64_MAX};
    a.sse = 0.0;
    a.cacc = a.racc = 0;
    for (int j = 0; j < NMV_MAX_INPUTS; ++j) a.eq[j] = 0;
    for (int64_t p = cd.piece_begin + threadIdx.x; p < cd.piece_end; p += kFinThreads) {
      const Partial &Q = partials[p];
      Red b;
      for (int k = 0; k < 8; ++k) b.cnt[k] = Q.cnt[k];
      b.ba = {Q.best_abs, Q.arg_abs};
      b.br = {Q.best_rel, Q.arg_rel};
      b.sse = Q.sse;
      b.cacc = Q.cacc;
      b.racc = Q.racc;
      for (int j = 0; j < NMV_MAX_INPUTS; ++j) b.eq[j] = Q.eq[j];
      red_add(a, b);
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
#pragma unroll
      for (int j = 0; j < NMV_MAX_INPUTS; ++j) b.eq[j] = __shfl_xor_sync(0xffffffffu, a.eq[j], off);
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
    __syncthreads();
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
    for (int j = 0; j < cd.n_elig; ++j) H->input_eq[cd.in_slot[j]] = a.eq[j];
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

  // ---- 2. first-K records.  Pieces are taken kFinThreads at a time, one
  // per thread; a block scan of their mismatch counts gives each piece its
  // first record position.  Each piece holding records below K is then
  // scanned the same way over its batch counts, and every batch holding
  // records below K is re-read by one warp.
  const int64_t K = cd.first_k;
  if (K == 0 || sh_mism == 0) return;
  int64_t base = 0;  // records in the pieces before this round
  for (int64_t q0 = cd.piece_begin; q0 < cd.piece_end && base < K; q0 += kFinThreads) {
    const int64_t p = q0 + threadIdx.x;
    const int64_t n = p < cd.piece_end ? partials[p].cnt[0] : 0;
    int64_t total;
    const int64_t pre = base + block_excl_scan64(n, &total, sh_scan);
    // compact the pieces holding records below K, in order
    const bool need = n > 0 && pre < K;
    int64_t n_need;
    const int64_t slot = block_excl_scan64(need ? 1 : 0, &n_need, sh_scan);
    if (need) {
      sh_need[slot] = pre;
      sh_need_p[slot] = p;
    }
    __syncthreads();
    for (int64_t j = 0; j < n_need; ++j) {
      const int64_t pos0 = sh_need[j], pj = sh_need_p[j];
      first_k_piece(cd, o, pieces[pj], batch_count, pos0, K, sh_scan, sh_item, &sh_nitems);
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

cudaError_t launch_finalize(const CaseDesc *cases, const Piece *pieces, const Partial *partials,
                            const int32_t *batch_count, uint8_t *out, int n_cases, cudaStream_t st) {
  finalize_kernel<<<n_cases, kFinThreads, 0, st>>>(cases, pieces, partials, batch_count, out);
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
