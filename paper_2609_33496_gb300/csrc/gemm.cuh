// gemm.cuh -- mixed-format quantized linear on tcgen05 (steps a7, a8): declarations.
#pragma once

#include <cuda_runtime.h>

#include "weights.cuh"

namespace cham {

struct GemmArgs {
  const uint8_t* codes;      // blob code region (tiled, include/chameleon.h)
  const float* wscale;       // [Np] per packed channel
  const uint8_t* wzero;      // [Np]
  const uint8_t* we8m0;      // [tiles][chunks][128][2] (group-wise blobs: the blocks' zero points)
  const uint32_t* wgscale;   // group-wise blobs: [tiles][chunks][128] two fp16 block scales, else null
  const uint8_t* wfmt;       // [Np]
  const int32_t* perm;       // [Np]
  const float* bias;         // [N] in original order, or null
  const float* act_scale;    // device s_a per row group (per-tensor formats: one group), or null for 1
  void* Y;                   // [M][N] of y_type
  int y_type;                // CHAM_Y_F32, CHAM_Y_F16 or CHAM_Y_BF16
  int rows_per_group;        // rows sharing one act_scale entry (per-sample scales); >= M: one
  int k_split;               // split-K: each tile's K-chunks in k_split contiguous ranges (1: off)
  float* partial;            // split-K: raw fp32 sums [k_split][M][Np], reduced by a second kernel
  int Np;                    // packed channels (128 per channel tile)
  int M, N, n_chunks;        // n_chunks = Kp / 64
  int tile0;                 // first 128-channel tile of this launch
  int n_ch_tiles;            // 128-channel tiles of this launch
  int bits;                  // 4 or 8
  int stall_chunk;           // test hook: CTA 0's producer withholds this K-chunk's copies (-1: off)
  int* dev_status;
  uint32_t nf4_lo[4];        // NF4 levels as fp16: low bytes of levels 4r..4r+3 in word r
  uint32_t nf4_hi[4];        // high bytes, same layout
  // FP8 kernel only (n_chunks then counts chunks of 128 elements)
  const uint8_t* act_e8;     // MXFP8 activations: E8M0 [n_chunks][act_mp][4] (chunk-major), else null
  int64_t act_e8_plane;      // bytes per chunk of act_e8 (act_mp * 4)
  int act_mp;                // rows per chunk of act_e8: M rounded up to 4
  int kblocks;               // K / 32
  int nk64;                  // 64-element chunks of the blob (Kp / 64)
  int b_fmt;                 // activation element type of the MMA: 0 E4M3, 1 E5M2
  int f8_tiles;              // the first f8_tiles channel tiles of the launch run on FP8 MMAs, the rest
                             // (NF4) on fp16 MMAs
};

// Token tile of the FP8 kernel for M > 128: 160 leaves room in tensor memory for the scale factors
// next to two accumulators and four decoded-weight slots.
constexpr int kF8TokenTile = 192;    // per-tensor / per-sample activation scales
constexpr int kF8TokenTileMx = 160;  // MXFP8 activations (their scale factors need tensor memory per slot)
// Up to this many tokens the linear runs on the weight-streaming kernel (gemm_small.cu).
constexpr int kSmallM = 16;

// Token-tile (MMA N) size for M tokens: 16, 32, 64, 128 or 192.
int gemm_pick_bn(int M, int n_tiles, int num_sms);
// Split-K factor: 1 when the tiles fill the GPU, else enough K ranges (of at least two chunks)
// to give every SM work.
int gemm_pick_split(int tiles, int n_chunks, int num_sms);
// Token tile of the FP8 kernel: 32, 64, 128, or kF8TokenTile (kF8TokenTileMx for MXFP8 activations).
int gemm_pick_bn_f8(int M, bool mx);
// Persistent launch: min(tiles, num_sms) CTAs walk the (channel tile, token tile) grid.
cudaError_t launch_gemm_f16(const CUtensorMap& act_map, const GemmArgs& a, int num_sms, int bn, cudaStream_t st);
// The FP8 kernel (gemm_f8_kernel.cuh) over a 4-bit layout: its first f8_tiles channel tiles on
// FP8 MMAs with the activation codes (map8, uint8), the rest (NF4) on fp16 MMAs with the fp16
// operand (map16).
cudaError_t launch_gemm_f8(const CUtensorMap& map8, const CUtensorMap& map16, const GemmArgs& a, int num_sms, int bn,
                           cudaStream_t st);
template <int YT, bool MXA>
cudaError_t launch_gemm_f8_yt(const CUtensorMap& map8, const CUtensorMap& map16, const GemmArgs& a, int num_sms,
                              int bn, cudaStream_t st);
// The weight-streaming kernel for M <= kSmallM: ks K ranges per 64-channel CTA group (a cluster).
int gemm_small_split(int n_ch_tiles, int n_chunks, int num_sms);
cudaError_t launch_gemm_small(const __half* X, const GemmArgs& a, int ks, cudaStream_t st);
// Split-K units' raw sums (EPI 6) and the reduction over the launch's tiles.
cudaError_t launch_splitk_reduce(const GemmArgs& a, int num_sms, cudaStream_t st);
// The launches of one output type (instantiated in gemm.cu, gemm_f16.cu, gemm_bf16.cu).
template <int YT>
cudaError_t launch_gemm_yt(const CUtensorMap& act_map, const GemmArgs& a, int num_sms, int bn, cudaStream_t st);
extern template cudaError_t launch_gemm_yt<CHAM_Y_F32>(const CUtensorMap&, const GemmArgs&, int, int, cudaStream_t);
extern template cudaError_t launch_gemm_yt<CHAM_Y_F16>(const CUtensorMap&, const GemmArgs&, int, int, cudaStream_t);
extern template cudaError_t launch_gemm_yt<CHAM_Y_BF16>(const CUtensorMap&, const GemmArgs&, int, int, cudaStream_t);
constexpr int kPartialYT = 3;  // "output type" of split-K units: raw fp32 partial sums
// the FP8 launcher's signature, instantiated per output type and activation kind
#define CHAM_F8_LAUNCH_ARGS const CUtensorMap&, const CUtensorMap&, const GemmArgs&, int, int, cudaStream_t
extern template cudaError_t launch_gemm_f8_yt<CHAM_Y_F32, false>(CHAM_F8_LAUNCH_ARGS);
extern template cudaError_t launch_gemm_f8_yt<CHAM_Y_F16, false>(CHAM_F8_LAUNCH_ARGS);
extern template cudaError_t launch_gemm_f8_yt<CHAM_Y_BF16, false>(CHAM_F8_LAUNCH_ARGS);
extern template cudaError_t launch_gemm_f8_yt<kPartialYT, false>(CHAM_F8_LAUNCH_ARGS);
extern template cudaError_t launch_gemm_f8_yt<CHAM_Y_F32, true>(CHAM_F8_LAUNCH_ARGS);
extern template cudaError_t launch_gemm_f8_yt<CHAM_Y_F16, true>(CHAM_F8_LAUNCH_ARGS);
extern template cudaError_t launch_gemm_f8_yt<CHAM_Y_BF16, true>(CHAM_F8_LAUNCH_ARGS);
extern template cudaError_t launch_gemm_f8_yt<kPartialYT, true>(CHAM_F8_LAUNCH_ARGS);

}  // namespace cham
