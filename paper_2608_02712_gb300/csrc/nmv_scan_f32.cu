// Streaming validation pass for NMV_F32 tensors (see nmv_scan.cuh).
#include "nmv_scan.cuh"

namespace nmv {
NMV_DEFINE_SCAN_OPS(NMV_F32)
template struct ScanOps<NMV_F32>;
}  // namespace nmv
