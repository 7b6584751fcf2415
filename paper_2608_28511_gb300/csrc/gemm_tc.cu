// Tensor-core grouped GEMM engine (placeholder until the tcgen05 path lands).
#include "launch.h"

namespace moe {

bool gemm_tc_supports(const GemmDesc&) { return false; }

cudaError_t launch_gemm_tc(const Ctx&, const GemmDesc&, const char*) { return cudaErrorNotSupported; }

}  // namespace moe
