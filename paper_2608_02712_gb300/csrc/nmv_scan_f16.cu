// Streaming validation pass for NMV_F16 tensors (see nmv_scan.cuh).
#include "nmv_scan.cuh"

namespace nmv {
NMV_DEFINE_SCAN_OPS(NMV_F16)
template struct ScanOps<NMV_F16>;
}  // namespace nmv
