// gemm_bf16.cu -- the bf16-output instantiations of the GEMM kernel (gemm_kernel.cuh).
#include "gemm_kernel.cuh"

namespace cham {

template cudaError_t launch_gemm_yt<CHAM_Y_BF16>(const CUtensorMap&, const GemmArgs&, int, int, cudaStream_t);

}  // namespace cham
