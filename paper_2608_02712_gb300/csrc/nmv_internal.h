// nmv_internal.h -- descriptors shared by the host planner (nmv_api.cu) and
// the kernels (nmv_scan.cuh, nmv_finalize.cu).  Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>
#include <mutex>
#include <string>

#include "../../include/nmv.h"

#ifdef __CUDACC__
#define NMV_HD __host__ __device__ __forceinline__
#else
#define NMV_HD inline
#endif

namespace nmv {

// ---- launch geometry ----------------------------------------------------
constexpr int kWarps = 8;                 // warps per block of the scan kernel
constexpr int kThreads = kWarps * 32;
constexpr int kFinThreads = 256;          // threads per block of the finalize kernel
constexpr int64_t kHistCap = 8192;        // smem tile-histogram window (bins)
constexpr int64_t kProfCap = 4096;        // smem row / column profile (bins each)
// Elements per piece at most: a multiple of every batch size (so piece
// boundaries stay on batch boundaries), small enough for int32 shared-memory
// counters and 32-bit byte offsets within a piece.
constexpr int kPiecesPerBlock = 2;       // pieces per scan block of the no-allocation entry point
constexpr int64_t kMaxPiece = int64_t(3) << 27;

// Element size in bytes and elements per 16-byte vector.
NMV_HD int elem_bytes(int dt) { return (dt == NMV_F16 || dt == NMV_BF16) ? 2 : 4; }
NMV_HD int vec_elems(int dt) { return 16 / elem_bytes(dt); }

// Division of a 64-bit unsigned value by an invariant d >= 1:
// m = floor((2^64 - 1) / d) gives q0 = mulhi(n, m) in {q - 1, q} for
// n < 2^63, and one compare fixes it.
struct Div64 {
  uint64_t d;
  uint64_t m;
};

inline Div64 make_div(uint64_t d) {
  Div64 r;
  r.d = d;
  r.m = ~uint64_t(0) / d;
  return r;
}

// One validation case as the kernels see it.
struct CaseDesc {
  const void *cand;
  const void *ref;
  const void *in_ptr[NMV_MAX_INPUTS];  // eligible inputs only (same dtype, numel)
  int32_t in_slot[NMV_MAX_INPUTS];     // their index in the caller's input list
  int32_t n_elig;
  int32_t n_inputs;                    // caller's input count
  int32_t dtype;
  int32_t vec_ok;                      // all buffers 16-byte aligned
  int32_t filter_ok;                   // the fp32 pre-filter of the predicate is valid
  int32_t fin_help;                    // finalize helper blocks of this case (fin_helpers)
  int64_t numel, M, N, th, tw, GR, GC;
  Div64 dN, dth, dtw;
  // 32-bit reciprocals floor((2^32 - 1) / d) of N, th, tw, used when every
  // element index fits in 32 bits (idx32 != 0)
  uint32_t m32N, m32th, m32tw, idx32;
  double rtol, atol;
  // fp32 pre-filter of the predicate: sure-pass if |s| <= fma_rz(lo_r, |r|, lo_a),
  // sure-fail if |s| > fma_ru(hi_r, |r|, hi_a) (see nmv_scan.cuh).
  float lo_r, lo_a, hi_r, hi_a;
  int64_t first_k;
  int64_t piece_begin, piece_end;      // this case's pieces
  int64_t batch_begin, batch_end;      // this case's batches (global batch indices)
  int64_t out_off;                     // byte offset of this case's packed result
  int64_t hist_off, rowp_off, colp_off, fk_off;  // byte offsets inside the packed result
  int64_t hist_n, rowp_n, colp_n;      // entries of the histogram and the profiles
  // Aligned localisation (amode != 0): indices fit in 32 bits, N is a
  // multiple of the warp step (32 vec_elems elements), and the tile width
  // divides the warp step and is a multiple of vec_elems.  A warp step then
  // lies in one row, and lane l's elements lie in one tile column at column
  // offsets (l mod 2^a_shift) * vec_elems + k, with 2^a_shift = tw /
  // vec_elems lanes per tile.
  int32_t amode, a_shift;
  // the candidate's shape as divisors, for the records' coordinates
  // (written at byte coord_off of the host result when the finalize writes
  // there; a zero extent has d = 0)
  int32_t rank;
  int32_t test_stall;                  // test hook of the scan's wait limit (NMV_FAULT_INJECT=stall)
  Div64 sdiv[NMV_MAX_RANK];
  int64_t coord_off;
};

// The packed results start with a call header holding the scan pass's
// exact-path counters (filled when profiling is on) and, at byte
// kCallErrOff, the scan kernel's error word (nonzero: a bulk copy into
// shared memory did not complete within the kernel's wait limit).
constexpr size_t kCallHeader = 256;
constexpr size_t kCallErrOff = 128;

// A contiguous element range of one case processed by one block.  It is
// cut into batches of batch_elems(dtype) elements (the last one may be
// shorter); warp w of the block takes batches w, w + kWarps, ... in order.
struct Piece {
  int64_t begin, end;
  int64_t batch_base;   // global index of the piece's first batch
  int64_t tr0, tc0;     // smem tile-histogram window origin (tile coordinates)
  int32_t wr, wc;       // window extent; wr == 0 -> histogram via global atomics
  int32_t case_id;
  int32_t prof_smem;    // 1 -> row / column profiles privatised in smem
};

// Per-piece partial result, reduced by the finalize kernel.
struct Partial {
  int64_t cnt[8];       // mismatch, cnan, cpinf, cninf, rnan, rpinf, rninf, nonfinite pairs
  double best_abs;
  double best_rel;
  double sse;
  int64_t arg_abs;
  int64_t arg_rel;
  uint32_t cacc, racc;  // OR of (bits ^ bits of element 0)
  int64_t eq[NMV_MAX_INPUTS];
};

// Header of one case's packed result (followed by the arrays).
struct OutHeader {
  int64_t cnt[8];       // as Partial::cnt, but [7] = n_finite_pairs
  double max_abs, max_rel, sse;
  int64_t argmax_abs, argmax_rel, k_out;
  uint32_t flags;
  int32_t passthrough;
  int64_t input_eq[NMV_MAX_INPUTS];
  int64_t status;
  int64_t pad[3];
};

#ifdef __CUDACC__
#define NMV_CHD __host__ __device__ constexpr
#else
#define NMV_CHD constexpr
#endif

// Warp steps (32 lanes x 16 bytes of each tensor) per batch, and per ring
// stage, by input class (0, 1 or -1 = several inputs read from global
// memory), and elements per batch.  A batch is the unit of the first-K
// counts and of the scan's bookkeeping; it streams through a warp's
// two-stage shared-memory ring as batch_steps / stage_steps stages: two of
// four steps, or, with one staged input (three tensors in each stage), four
// of two steps, so the ring's shared memory stays the same.
constexpr int kMaxSteps = 8;
NMV_CHD int batch_steps(int) { return 8; }
NMV_CHD int stage_steps(int nin) { return nin == 1 ? 2 : 4; }
// A batch's entry in the batch-count array: its mismatch count (below 2^24)
// in the low bits, and from bit kStepBitsShift the warp steps that hold them.
constexpr int kStepBitsShift = 24;
constexpr uint32_t kBatchCountMask = (1u << kStepBitsShift) - 1;
NMV_CHD int stage_bytes(int nin) { return 32 * 16 * stage_steps(nin); }  // one tensor's bytes per stage
NMV_CHD int nin_class_of(int n_elig) { return n_elig == 0 ? 0 : (n_elig == 1 ? 1 : -1); }
NMV_HD int64_t batch_elems(int dt, int nin) { return (int64_t)32 * vec_elems(dt) * batch_steps(nin); }
NMV_HD int64_t piece_batches(int64_t begin, int64_t end, int dt, int nin) {
  const int64_t be = batch_elems(dt, nin);
  return (end - begin + be - 1) / be;
}

// Finalize blocks of one case beyond the first.  A case with records to
// write gets one helper block per kFinHelperBatches batches; in a call of at
// most kFinFewCases cases (whose finalize grid is otherwise small) also one
// per kFinHelperItems batches that may hold records (min(first_k,
// batches)), so that sparse mismatches, one or two per batch, are re-read by
// many warps at once.  At most kFinMaxHelpers; the helpers then write the
// records while the first block reduces the partials.
constexpr int kFinMaxHelpers = 16;
constexpr int64_t kFinHelperBatches = 4096;
constexpr int64_t kFinHelperItems = 16;
constexpr int64_t kFinFewCases = 16;
NMV_HD int fin_helpers(int64_t first_k, int64_t n_batches, int64_t n_cases) {
  if (first_k <= 0) return 0;
  int64_t h = n_batches / kFinHelperBatches;
  if (n_cases <= kFinFewCases) {
    const int64_t items = first_k < n_batches ? first_k : n_batches;
    if (items / kFinHelperItems > h) h = items / kFinHelperItems;
  }
  return h < kFinMaxHelpers ? (int)h : kFinMaxHelpers;
}

// Ring of each scan warp, by input class: stages, tensors staged per batch,
// and the dynamic shared memory of all rings of a block (stage data, then
// one 8-byte mbarrier per stage).
NMV_CHD int ring_stages(int) { return 2; }
NMV_CHD int ring_streams(int nin) { return nin == 1 ? 3 : 2; }
NMV_CHD size_t ring_bytes(int nin) {
  return (size_t)kWarps * ring_stages(nin) * ((size_t)ring_streams(nin) * stage_bytes(nin) + 8);
}

// Host services of nmv_api.cu used by the library's other entry points: the
// thread-local error text (nmv_last_error), the library lock, the device
// probe (sm_103 only), and the pool of mapped pinned result blocks.
int host_fail(int code, const std::string &msg);
int host_cuda_fail(cudaError_t e, const char *what);
void host_clear_error();
std::mutex &host_mutex();
int host_probe(int *dev, int *sms, size_t *smem_optin);  // call with host_mutex() held
int64_t host_tensor_numel(const nmv_tensor &t);          // -1 for an invalid shape
void *host_arena_get(size_t bytes);                      // mapped pinned block, or NULL
void host_arena_put(void *p);
bool host_injected(const char *step);                    // NMV_FAULT_INJECT test hook

}  // namespace nmv
