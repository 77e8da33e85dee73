// gemm.cu -- the GEMM's host side (token-tile choice, dispatch by output type) and the fp32-output
// instantiations of the kernel in gemm_kernel.cuh.
#include "gemm_kernel.cuh"

namespace cham {

template cudaError_t launch_gemm_yt<CHAM_Y_F32>(const CUtensorMap&, const GemmArgs&, int, int, cudaStream_t);

// Split-K units: raw partial sums (EPI 6); the reduction applies scales, bias and output type.
static cudaError_t launch_gemm_partial(const CUtensorMap& map, const GemmArgs& a, int num_sms, int bn,
                                       cudaStream_t st) {
  if (a.bits == 8) return launch_gw<8, 2 * kPartialOut>(map, a, num_sms, bn, st);
  return launch_gw<4, 2 * kPartialOut>(map, a, num_sms, bn, st);
}

// Split-K reduction: Y[tok, perm[p]] = (sum_j partial[j][tok][p]) * (s_a(tok) * s_w[p]) + bias,
// the K ranges added in order (deterministic), rounded to the output type like the fused epilogue.
// Only the launch's channel tiles [tile0, tile0 + n_ch_tiles) are reduced: the other MMA class of
// the same layer may be written by a launch of its own.
__global__ void __launch_bounds__(256) k_splitk_reduce(const GemmArgs a) {
  griddep_wait();  // the partial sums of the GEMM just before
  griddep_launch_dependents();
  const int64_t width = static_cast<int64_t>(a.n_ch_tiles) * 128;
  const int64_t total = static_cast<int64_t>(a.M) * width;
  const int64_t plane = static_cast<int64_t>(a.M) * a.Np;
  const bool per_sample = a.act_scale != nullptr && a.rows_per_group < a.M;
  const float sa0 = a.act_scale != nullptr ? *a.act_scale : 1.f;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int tok = static_cast<int>(i / width);
    const int p = a.tile0 * 128 + static_cast<int>(i % width);
    const int orig = a.perm[p];
    if (orig < 0) continue;
    const int64_t o0 = static_cast<int64_t>(tok) * a.Np + p;
    float acc = a.partial[o0];
    for (int j = 1; j < a.k_split; ++j) acc = __fadd_rn(acc, a.partial[j * plane + o0]);
    const float sa = per_sample ? a.act_scale[tok / a.rows_per_group] : sa0;
    const float y = fmaf(acc, __fmul_rn(sa, a.wscale[p]), a.bias != nullptr ? a.bias[orig] : 0.f);
    const size_t o = static_cast<size_t>(tok) * a.N + orig;
    if (a.y_type == CHAM_Y_F16) static_cast<__half*>(a.Y)[o] = __float2half_rn(y);
    else if (a.y_type == CHAM_Y_BF16) static_cast<__nv_bfloat16*>(a.Y)[o] = __float2bfloat16_rn(y);
    else static_cast<float*>(a.Y)[o] = y;
  }
}

cudaError_t launch_splitk_reduce(const GemmArgs& a, int num_sms, cudaStream_t st) {
  const int64_t total = static_cast<int64_t>(a.M) * a.n_ch_tiles * 128;
  int64_t g = (total + 255) / 256;
  if (g > static_cast<int64_t>(num_sms) * 8) g = static_cast<int64_t>(num_sms) * 8;
  return launch_pdl(k_splitk_reduce, dim3(static_cast<int>(g)), dim3(256), 0, st, a);
}

int gemm_pick_split(int tiles, int n_chunks, int num_sms) {
  // a short K (under 8 chunks) gains less from the split than the reduction launch costs
  if (tiles * 2 > num_sms || n_chunks < 8) return 1;
  int ks = num_sms / tiles;
  if (ks > n_chunks / 2) ks = n_chunks / 2;  // at least one full commit group per unit
  return ks < 1 ? 1 : ks;
}

int gemm_pick_bn_f8(int M, bool mx) {
  if (M <= 32) return 32;
  if (M <= 64) return 64;
  if (M <= 128) return 128;
  return mx ? kF8TokenTileMx : kF8TokenTile;
}

cudaError_t launch_gemm_f8(const CUtensorMap& map8, const CUtensorMap& map16, const GemmArgs& a, int num_sms, int bn,
                           cudaStream_t st) {
  const bool mxa = a.act_e8 != nullptr;
  if (a.k_split > 1) {
    const cudaError_t e = mxa ? launch_gemm_f8_yt<kPartialYT, true>(map8, map16, a, num_sms, bn, st)
                              : launch_gemm_f8_yt<kPartialYT, false>(map8, map16, a, num_sms, bn, st);
    if (e != cudaSuccess) return e;
    return launch_splitk_reduce(a, num_sms, st);
  }
  switch (a.y_type) {
    case CHAM_Y_F16:
      return mxa ? launch_gemm_f8_yt<CHAM_Y_F16, true>(map8, map16, a, num_sms, bn, st)
                 : launch_gemm_f8_yt<CHAM_Y_F16, false>(map8, map16, a, num_sms, bn, st);
    case CHAM_Y_BF16:
      return mxa ? launch_gemm_f8_yt<CHAM_Y_BF16, true>(map8, map16, a, num_sms, bn, st)
                 : launch_gemm_f8_yt<CHAM_Y_BF16, false>(map8, map16, a, num_sms, bn, st);
    default:
      return mxa ? launch_gemm_f8_yt<CHAM_Y_F32, true>(map8, map16, a, num_sms, bn, st)
                 : launch_gemm_f8_yt<CHAM_Y_F32, false>(map8, map16, a, num_sms, bn, st);
  }
}

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
  if (a.k_split > 1) {
    const cudaError_t e = launch_gemm_partial(map, a, num_sms, bn, st);
    if (e != cudaSuccess) return e;
    return launch_splitk_reduce(a, num_sms, st);
  }
  switch (a.y_type) {
    case CHAM_Y_F16: return launch_gemm_yt<CHAM_Y_F16>(map, a, num_sms, bn, st);
    case CHAM_Y_BF16: return launch_gemm_yt<CHAM_Y_BF16>(map, a, num_sms, bn, st);
    default: return launch_gemm_yt<CHAM_Y_F32>(map, a, num_sms, bn, st);
  }
}

}  // namespace cham
