// Instantiations of the tcgen05 GEMM for the forward (A and B K-major) operand layout.
#include "gemm_tc.cuh"

namespace fl_gemm {
FL_GEMM_INSTANTIATE(false, false)
}  // namespace fl_gemm
