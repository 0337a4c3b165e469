// Streaming validation pass for NMV_BF16 tensors (see nmv_scan.cuh).
#include "nmv_scan.cuh"

namespace nmv {
NMV_DEFINE_SCAN_OPS(NMV_BF16)
template struct ScanOps<NMV_BF16>;
}  // namespace nmv
