// k_gemm_tc.cu -- tcgen05 / TMEM / TMA GEMM (placeholder until the kernel lands).
#include "kernels.h"

namespace ra {
bool tc_available() { return false; }
cudaError_t gemm_tc(const GemmArgs&, cudaStream_t) { return cudaErrorNotSupported; }
}  // namespace ra
