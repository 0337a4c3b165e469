// Streaming validation pass for NMV_I32 tensors (see nmv_scan.cuh).
#include "nmv_scan.cuh"

namespace nmv {
NMV_DEFINE_SCAN_OPS(NMV_I32)
template struct ScanOps<NMV_I32>;
}  // namespace nmv
