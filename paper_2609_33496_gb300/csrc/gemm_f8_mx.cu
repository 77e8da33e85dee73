// gemm_f8_mx.cu -- instantiations of the FP8 kernel (gemm_f8_kernel.cuh) for MXFP8 activations,
// whose block exponents are the MMA's B scale factors (no per-tensor scale): every output type, and
// the split-K partial sums.
#include "gemm_f8_kernel.cuh"

namespace cham {

template <int YT, bool MXA>
cudaError_t launch_gemm_f8_yt(const CUtensorMap& map8, const CUtensorMap& map16, const GemmArgs& a, int num_sms, int bn,
                              cudaStream_t st) {
  return launch_f8_epi<2 * YT, MXA>(map8, map16, a, num_sms, bn, st);
}

template cudaError_t launch_gemm_f8_yt<CHAM_Y_F32, true>(CHAM_F8_LAUNCH_ARGS);
template cudaError_t launch_gemm_f8_yt<CHAM_Y_F16, true>(CHAM_F8_LAUNCH_ARGS);
template cudaError_t launch_gemm_f8_yt<CHAM_Y_BF16, true>(CHAM_F8_LAUNCH_ARGS);
template cudaError_t launch_gemm_f8_yt<kPartialYT, true>(CHAM_F8_LAUNCH_ARGS);

}  // namespace cham
