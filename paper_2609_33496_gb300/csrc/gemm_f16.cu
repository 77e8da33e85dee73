// gemm_f16.cu -- the fp16-output instantiations of the GEMM kernel (gemm_kernel.cuh).
#include "gemm_kernel.cuh"

namespace cham {

template cudaError_t launch_gemm_yt<CHAM_Y_F16>(const CUtensorMap&, const GemmArgs&, int, int, cudaStream_t);

}  // namespace cham
