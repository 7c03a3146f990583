// Instantiations of the tcgen05 GEMM for the weight-gradient (A and B MN-major) operand layout.
#include "gemm_tc.cuh"

namespace fl_gemm {
FL_GEMM_INSTANTIATE(true, true)
}  // namespace fl_gemm
