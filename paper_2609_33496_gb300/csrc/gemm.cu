// gemm.cu -- the GEMM's host side (token-tile choice, dispatch by output type) and the fp32-output
// instantiations of the kernel in gemm_kernel.cuh.
#include "gemm_kernel.cuh"

namespace cham {

template cudaError_t launch_gemm_yt<CHAM_Y_F32>(const CUtensorMap&, const GemmArgs&, int, int, cudaStream_t);

int gemm_pick_bn(int M, int n_tiles, int num_sms) {
  (void)n_tiles;
  (void)num_sms;
  if (M <= 16) return 16;
  if (M <= 32) return 32;
  if (M <= 64) return 64;
  if (M <= 128) return 128;
  return 192;
}

cudaError_t launch_gemm_f16(const CUtensorMap& map, const GemmArgs& a, int num_sms, int bn, cudaStream_t st) {
  switch (a.y_type) {
    case CHAM_Y_F16: return launch_gemm_yt<CHAM_Y_F16>(map, a, num_sms, bn, st);
    case CHAM_Y_BF16: return launch_gemm_yt<CHAM_Y_BF16>(map, a, num_sms, bn, st);
    default: return launch_gemm_yt<CHAM_Y_F32>(map, a, num_sms, bn, st);
  }
}

}  // namespace cham
