// Instantiations of the tcgen05 GEMM for the data-gradient (A K-major, B MN-major) operand layout.
#include "gemm_tc.cuh"

namespace fl_gemm {
FL_GEMM_INSTANTIATE(false, true)
}  // namespace fl_gemm
