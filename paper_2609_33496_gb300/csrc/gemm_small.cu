// gemm_small.cu -- the quantized linear for a handful of tokens (M <= kSmallM): step a7/a8 when the
// layer is bound by streaming its packed weights and by launch latency, not by the tensor cores
// (the time-embedding projections, batch-1..16 rows of the few-step fork).  The tcgen05 kernels pay
// a fixed cost per launch (tensor-memory allocation, barrier rings, a 128-channel x 16-token tile
// per CTA) that dwarfs such a GEMM; here the work is spread over the GPU by channels and by K, with
// enough independent warps per SM to hide the load and shared-memory latencies:
//
//   * a CTA owns 32 packed channels (one per lane) and a contiguous range of the K-chunks; its four
//     warps take the range's chunks in turn (warp w: chunks kc0 + w, kc0 + w + 4, ...).  The CTAs
//     that share the 32 channels form one thread-block cluster (up to 8, one per K range);
//   * per 64-element chunk a warp stages the MB activation rows of the chunk in its own shared
//     memory as fp32 (rows M..MB-1 zero; MB = M rounded up to a power of two, a template argument,
//     so the FMA loop has no per-row predicates), every lane loads its channel's codes with 16-byte
//     loads (the tiled blob layout makes the 32 lanes' loads one contiguous 512-byte run), decodes
//     them with the GEMM's decoders to the exact fp16 operand values and accumulates the MB dot
//     products in fp32 (each product of two fp16 values is exact in fp32);
//   * the four warps' sums are added in warp order in shared memory; after a cluster barrier CTA 0
//     adds the cluster's sums in rank order through distributed shared memory (a fixed order:
//     deterministic), applies s_a * s_w[p] and the bias as the GEMM epilogue does and stores Y; a
//     second barrier keeps the other CTAs' shared memory alive until it has been read.
// One launch, no workspace beyond the operand, no counters.
#include <cuda_bf16.h>

#include "gemm_kernel.cuh"

namespace cham {

constexpr int kSmallWarps = 4;   // warps per CTA, splitting the CTA's K-chunks
constexpr int kSmallMaxCluster = 8;

CHAM_DEV void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
CHAM_DEV uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
CHAM_DEV float ld_dsmem_f32(const float* local_addr, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local_addr)), "r"(rank));
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(remote) : "memory");
  return v;
}

// grid: (ks, 4 * n_ch_tiles); cluster (ks, 1, 1): blockIdx.x is the K range (= cluster rank),
// blockIdx.y the 32-channel quarter tile.  X: the fp16 operand (M x K row-major).  MB >= M.
template <int BITS, bool GW, int MB>
__global__ void __launch_bounds__(32 * kSmallWarps) k_gemm_small(const __half* __restrict__ X, const GemmArgs a) {
  __shared__ __align__(16) float xs[kSmallWarps][MB][64];
  __shared__ float part[kSmallWarps][MB][32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ks = gridDim.x;
  const uint32_t rank = cluster_rank();
  const int tile = a.tile0 + blockIdx.y / 4;
  const int r = (blockIdx.y & 3) * 32 + lane;   // channel within the 128-channel tile
  const int p = tile * 128 + r;
  const int nk = a.n_chunks, M = a.M;
  const int kc0 = static_cast<int>(rank) * nk / ks, kc1 = (static_cast<int>(rank) + 1) * nk / ks;
  constexpr int CB = BITS == 8 ? 64 : 32;  // code bytes per channel and chunk
  const int f = a.wfmt[p];
  const ChanDecode cd = chan_decode(f, a.wzero[p]);
  float acc[MB];
#pragma unroll
  for (int m = 0; m < MB; ++m) acc[m] = 0.f;
  griddep_wait();  // the operand is the previous kernel's output
  griddep_launch_dependents();
  const int kreal = a.kblocks * 32;  // K (elements beyond it are zero codes; their x is staged as 0)
  float(*xw)[64] = xs[warp];
  for (int kc = kc0 + warp; kc < kc1; kc += kSmallWarps) {
    // this warp's chunk: its MB x 64 activations as fp32 (zeros beyond K and beyond M)
    __syncwarp();
#pragma unroll
    for (int i = lane; i < MB * 8; i += 32) {
      const int m = i >> 3, v = i & 7, k = kc * 64 + v * 8;
      uint4 q = make_uint4(0, 0, 0, 0);
      if (m < M && k < kreal) q = *reinterpret_cast<const uint4*>(X + static_cast<size_t>(m) * kreal + k);
      const float2 t0 = __half22float2(u32_as_h2(q.x)), t1 = __half22float2(u32_as_h2(q.y));
      const float2 t2 = __half22float2(u32_as_h2(q.z)), t3 = __half22float2(u32_as_h2(q.w));
      *reinterpret_cast<float4*>(&xw[m][v * 8]) = make_float4(t0.x, t0.y, t1.x, t1.y);
      *reinterpret_cast<float4*>(&xw[m][v * 8 + 4]) = make_float4(t2.x, t2.y, t3.x, t3.y);
    }
    const size_t chunk = static_cast<size_t>(tile) * nk + kc;
    const uint8_t* cp = a.codes + chunk * 128 * CB;
    const uint32_t e8 = reinterpret_cast<const uint16_t*>(a.we8m0 + chunk * 256)[r];
    ChanDecode cdk = cd;
    uint32_t gs = 0;
    if constexpr (GW) {
      gs = a.wgscale[chunk * 128 + r];
      if (cd.f == CHAM_W_INT8_ASYM || cd.f == CHAM_W_INT4_ASYM) {
        cdk.off0 = static_cast<int>(e8 & 0xFFu);
        cdk.off1 = static_cast<int>((e8 >> 8) & 0xFFu);
      }
    }
    uint32_t raw[BITS * 2];
#pragma unroll
    for (int j = 0; j < BITS / 2; ++j) {
      const uint4 u = *reinterpret_cast<const uint4*>(cp + j * 2048 + r * 16);
      raw[4 * j] = u.x;
      raw[4 * j + 1] = u.y;
      raw[4 * j + 2] = u.z;
      raw[4 * j + 3] = u.w;
    }
    uint32_t out[32];
    if constexpr (BITS == 8) decode_w8(raw, cdk, e8, out);
    else decode_w4(raw, cdk, e8, a.nf4_lo, a.nf4_hi, out);
    if constexpr (GW) {
      const uint32_t g0 = dup16(gs & 0xFFFFu), g1 = dup16(gs >> 16);
#pragma unroll
      for (int i = 0; i < 32; ++i) out[i] = hmul2u(out[i], i < 16 ? g0 : g1);
    }
    __syncwarp();  // the staged activations are visible to the whole warp
#pragma unroll
    for (int c = 0; c < 16; ++c) {   // out[2c], out[2c+1] = elements 4c .. 4c+3 of the chunk
      const float2 w01 = __half22float2(u32_as_h2(out[2 * c]));
      const float2 w23 = __half22float2(u32_as_h2(out[2 * c + 1]));
#pragma unroll
      for (int m = 0; m < MB; ++m) {
        const float4 xv = *reinterpret_cast<const float4*>(&xw[m][4 * c]);
        acc[m] = fmaf(w23.y, xv.w, fmaf(w23.x, xv.z, fmaf(w01.y, xv.y, fmaf(w01.x, xv.x, acc[m]))));
      }
    }
  }
#pragma unroll
  for (int m = 0; m < MB; ++m) part[warp][m][lane] = acc[m];
  __syncthreads();
  // the CTA's sums, warps added in order, into warp 0's slots
  for (int i = threadIdx.x; i < MB * 32; i += blockDim.x) {
    const int m = i >> 5, l = i & 31;
    float y = part[0][m][l];
#pragma unroll
    for (int w = 1; w < kSmallWarps; ++w) y = __fadd_rn(y, part[w][m][l]);
    part[0][m][l] = y;
  }
  cluster_sync();  // every CTA's sums are in its shared memory
  if (rank == 0) {
    const int orig = a.perm[p];
    if (orig >= 0) {
      const float ws = a.wscale[p];
      const float bv = a.bias != nullptr ? a.bias[orig] : 0.f;
      const float sa0 = a.act_scale != nullptr ? *a.act_scale : 1.f;
      const bool per_sample = a.act_scale != nullptr && a.rows_per_group < M;
      for (int m = warp; m < M; m += kSmallWarps) {
        float y = part[0][m][lane];
        for (int q = 1; q < ks; ++q) y = __fadd_rn(y, ld_dsmem_f32(&part[0][m][lane], q));
        const float sa = per_sample ? a.act_scale[m / a.rows_per_group] : sa0;
        const float o = fmaf(y, __fmul_rn(sa, ws), bv);
        const size_t idx = static_cast<size_t>(m) * a.N + orig;
        if (a.y_type == CHAM_Y_F16) static_cast<__half*>(a.Y)[idx] = __float2half_rn(o);
        else if (a.y_type == CHAM_Y_BF16) static_cast<__nv_bfloat16*>(a.Y)[idx] = __float2bfloat16_rn(o);
        else static_cast<float*>(a.Y)[idx] = o;
      }
    }
  }
  cluster_sync();  // the other CTAs' shared memory stays alive until CTA 0 has read it
}

int gemm_small_split(int n_ch_tiles, int n_chunks, int num_sms) {
  // about four CTAs (16 warps) per SM, and every warp with at least one chunk where K allows
  const int groups = 4 * n_ch_tiles;
  int ks = (4 * num_sms + groups - 1) / groups;
  const int by_k = (n_chunks + kSmallWarps - 1) / kSmallWarps;
  if (ks > by_k) ks = by_k;
  if (ks > kSmallMaxCluster) ks = kSmallMaxCluster;
  return ks < 1 ? 1 : ks;
}

template <int BITS, bool GW, int MB>
static cudaError_t launch_small(const __half* X, const GemmArgs& a, int ks, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(ks, 4 * a.n_ch_tiles);
  cfg.blockDim = dim3(32 * kSmallWarps);
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = ks;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, k_gemm_small<BITS, GW, MB>, X, a);
}

template <int BITS, bool GW>
static cudaError_t launch_small_m(const __half* X, const GemmArgs& a, int ks, cudaStream_t st) {
  if (a.M <= 1) return launch_small<BITS, GW, 1>(X, a, ks, st);
  if (a.M <= 2) return launch_small<BITS, GW, 2>(X, a, ks, st);
  if (a.M <= 4) return launch_small<BITS, GW, 4>(X, a, ks, st);
  if (a.M <= 8) return launch_small<BITS, GW, 8>(X, a, ks, st);
  return launch_small<BITS, GW, 16>(X, a, ks, st);
}

cudaError_t launch_gemm_small(const __half* X, const GemmArgs& a, int ks, cudaStream_t st) {
  static_assert(kSmallM == 16, "the row buckets above end at 16");
  if (a.bits == 8) return a.wgscale != nullptr ? launch_small_m<8, true>(X, a, ks, st) : launch_small_m<8, false>(X, a, ks, st);
  return a.wgscale != nullptr ? launch_small_m<4, true>(X, a, ks, st) : launch_small_m<4, false>(X, a, ks, st);
}

}  // namespace cham
