// tcgen05 GEMMs (placeholder: every layer takes the SIMT path until the
// tensor-core kernels are in).
#include "vfl_tc.cuh"

namespace vfl {

bool tc_supported_fwd(int, int, bool, int, bool) { return false; }
bool tc_supported_dx(int, int, int, bool) { return false; }
bool tc_supported_dw(int, int, bool, int) { return false; }
cudaError_t launch_tc_gemm(const TcGemm&, cudaStream_t) { return cudaErrorNotSupported; }

}  // namespace vfl
