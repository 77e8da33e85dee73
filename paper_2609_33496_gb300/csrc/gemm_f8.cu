// gemm_f8.cu -- instantiations of the FP8 kernel (gemm_f8_kernel.cuh) for activation codes with a
// per-tensor or per-sample scale (E4M3, E5M2): every output type, and the split-K partial sums.
#include "gemm_f8_kernel.cuh"

namespace cham {

template <int YT, bool MXA>
cudaError_t launch_gemm_f8_yt(const CUtensorMap& map8, const CUtensorMap& map16, const GemmArgs& a, int num_sms, int bn,
                              cudaStream_t st) {
  const bool per_sample = a.act_scale != nullptr && a.rows_per_group < a.M;
  if constexpr (YT == kPartialYT || MXA) {
    return launch_f8_epi<2 * YT, MXA>(map8, map16, a, num_sms, bn, st);  // scales are applied by the reduction / are 1
  } else {
    return per_sample ? launch_f8_epi<2 * YT + 1, MXA>(map8, map16, a, num_sms, bn, st)
                      : launch_f8_epi<2 * YT, MXA>(map8, map16, a, num_sms, bn, st);
  }
}

template cudaError_t launch_gemm_f8_yt<CHAM_Y_F32, false>(CHAM_F8_LAUNCH_ARGS);
template cudaError_t launch_gemm_f8_yt<CHAM_Y_F16, false>(CHAM_F8_LAUNCH_ARGS);
template cudaError_t launch_gemm_f8_yt<CHAM_Y_BF16, false>(CHAM_F8_LAUNCH_ARGS);
template cudaError_t launch_gemm_f8_yt<kPartialYT, false>(CHAM_F8_LAUNCH_ARGS);

}  // namespace cham
