// probe.cu -- tensor-core throughput probe (libchameleon_probe.so, used by the benchmark only).
//
// Measures what one SM's tcgen05 pipe sustains for the instruction forms the GEMM uses, to give
// the roofline its dense fp16 and 8-bit-float denominators on this GPU: one CTA per SM issues
// `iters` groups of four back-to-back MMAs (M = 128, N, K = 16 for kind::f16 or 32 for
// kind::f8f6f4) into one accumulator, then waits for their commit.  The operands are filled with
// a seeded pattern of finite values (power draw, and so the clock, depends on the data).  Every
// wait is bounded; a timeout is reported through *status.
#include <cuda_runtime.h>

#include "common.cuh"

namespace cham {

constexpr int kProbeOperand = 128 * 128;  // A tile: 128 rows x 128 bytes

// kind: 0 = kind::f16, A from shared memory; 1 = kind::f16, A from tensor memory;
//       2 = kind::f8f6f4 (E4M3 x E4M3), A from shared memory; 3 = the same, A from tensor memory;
//       4 = kind::mxf8f6f4.block_scale (E4M3 x E4M3, UE8M0 scale factors in tensor memory), A from
//       tensor memory -- the 4-bit GEMM's FP8 form; 5 = the same, A from shared memory; 6 = kind 4
//       with the GEMM's per-chunk bookkeeping after every four MMAs: a commit to an mbarrier, an
//       arrive-and-wait on another (a phase that is complete when tested) and the fence after it;
//       7 = kind 6 issued by two threads (warps 0 and 1) into two accumulators, half the
//       iterations each: whether a second issuer fills the pipe during the other's bookkeeping.
template <int KIND, int N>
__global__ void __launch_bounds__(128, 1) k_mma_probe(int iters, unsigned long long* cycles, int* status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kProbeOperand;
  // per issuing thread w (0, and 1 for kind 7): bar[w] final commit, bar[2 + w] per-iteration
  // commits (kinds 6, 7), bar[4 + w] per-iteration arrive + wait
  uint64_t* bar = reinterpret_cast<uint64_t*>(sB + N * 128);
  uint32_t* slot = reinterpret_cast<uint32_t*>(bar + 6);
  __shared__ int abort_flag;
  // finite operands: bytes 0x30..0x3F are small positive E4M3 values, and as fp16 pairs they are
  // small positive normals
  for (int i = threadIdx.x; i < (kProbeOperand + N * 128) / 4; i += blockDim.x)
    reinterpret_cast<uint32_t*>(smem)[i] = 0x30303030u + ((i * 2654435761u) >> 28) * 0x01010101u;
  if (threadIdx.x == 0) {
    for (int i = 0; i < 6; ++i) mbar_init(&bar[i], 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // operands visible to the tensor core
  if (threadIdx.x < 32) tmem_alloc(slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *slot;
  const uint32_t lane_off = static_cast<uint32_t>((threadIdx.x >> 5) * 32) << 16;
  // A operand and scale factors in tensor memory: columns 256.. (kind 7: 384.., after the second
  // accumulator at N)
  constexpr uint32_t kACol = KIND == 7 ? 384 : 256, kSfa = kACol + 64, kSfb = kSfa + 8;
  if (KIND == 1 || KIND == 3 || KIND == 4 || KIND >= 6) {
    uint32_t z[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) z[i] = 0x30303030u + i;
    tmem_st_32x32b_x32(tmem + kACol + lane_off, z);
    tmem_wait_st();
  }
  if (KIND >= 4) {  // scale factors 2^0 in every byte (A at kSfa, B at kSfb)
    uint32_t one[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) one[i] = 0x7F7F7F7Fu;
    tmem_st_32x32b_x8(tmem + kSfa + lane_off, one);
    tmem_st_32x32b_x8(tmem + kSfb + lane_off, one);
    tmem_wait_st();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (threadIdx.x == 0 || (KIND == 7 && threadIdx.x == 32)) {
    const int w = threadIdx.x >> 5;                       // issuing thread 0 or 1
    const uint32_t d = tmem + (KIND == 7 ? w * N : 0);    // its accumulator
    const int n_it = KIND == 7 ? iters / 2 : iters;
    const uint32_t a0 = smem_u32(sA), b0 = smem_u32(sB);
    uint32_t idesc = idesc_f16(128, N);
    if (KIND == 2 || KIND == 3) idesc &= ~((7u << 7) | (7u << 10));  // E4M3 x E4M3 (format code 0), F32 D
    // kind::mxf8f6f4: E4M3 x E4M3, N, UE8M0 scale factors (bit 23), M; scale-factor ids added per MMA
    const uint32_t idesc_mx = (static_cast<uint32_t>(N >> 3) << 17) | (1u << 23) | (128u >> 4 << 24);
    const unsigned long long t0 = clock64();
    for (int it = 0; it < n_it; ++it) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const uint64_t bd = smem_desc_sw128(b0 + kk * 32);
        const uint64_t ad = smem_desc_sw128(a0 + kk * 32);
        if (KIND == 0) {
          asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                       "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d),
                       "l"(ad), "l"(bd), "r"(idesc), "r"(1u)
                       : "memory");
        } else if (KIND == 1) {
          mma_f16_ts(d, tmem + kACol + kk * 8, bd, idesc, 1u);
        } else if (KIND == 3) {
          asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                       "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d),
                       "r"(tmem + kACol + kk * 8), "l"(bd), "r"(idesc), "r"(1u)
                       : "memory");
        } else if (KIND == 4 || KIND >= 6) {
          const uint32_t id = idesc_mx | (static_cast<uint32_t>(kk) << 4) | (static_cast<uint32_t>(kk) << 29);
          asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %6, 0;\n\t"
                       "tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], [%1], %2, %3, [%4], "
                       "[%5], p;\n\t}\n" ::"r"(d),
                       "r"(tmem + kACol + kk * 8), "l"(bd), "r"(id), "r"(tmem + kSfa), "r"(tmem + kSfb), "r"(1u)
                       : "memory");
        } else if (KIND == 5) {
          const uint32_t id = idesc_mx | (static_cast<uint32_t>(kk) << 4) | (static_cast<uint32_t>(kk) << 29);
          asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %6, 0;\n\t"
                       "tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], %1, %2, %3, [%4], "
                       "[%5], p;\n\t}\n" ::"r"(d),
                       "l"(ad), "l"(bd), "r"(id), "r"(tmem + kSfa), "r"(tmem + kSfb), "r"(1u)
                       : "memory");
        } else {
          asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                       "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d),
                       "l"(ad), "l"(bd), "r"(idesc), "r"(1u)
                       : "memory");
        }
      }
      if (KIND >= 6) {
        mma_commit(&bar[2 + w]);
        mbar_arrive(&bar[4 + w]);
        if (!mbar_wait(&bar[4 + w], it & 1, reinterpret_cast<volatile int*>(&abort_flag), status)) break;
        tc_fence_after();
      }
    }
    mma_commit(&bar[w]);
    mbar_wait(&bar[w], 0, reinterpret_cast<volatile int*>(&abort_flag), status);
    const unsigned long long t1 = clock64();
    if (blockIdx.x == 0 && w == 0) *cycles = t1 - t0;
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x < 32) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int KIND, int N>
static int launch_probe(int ctas, int iters, unsigned long long* cycles, int* status, cudaStream_t st) {
  const int smem = 1024 + kProbeOperand + N * 128 + 64;
  const int req = smem > 120 * 1024 ? smem : 120 * 1024;  // one CTA per SM
  cudaFuncSetAttribute(k_mma_probe<KIND, N>, cudaFuncAttributeMaxDynamicSharedMemorySize, req);
  k_mma_probe<KIND, N><<<ctas, 128, req, st>>>(iters, cycles, status);
  return static_cast<int>(cudaGetLastError());
}

}  // namespace cham

// kind 0..7 as above, n in {128, 160, 192, 256}; ctas CTAs of 128 threads, one per SM; *cycles gets
// CTA 0's clock cycles.  Returns a cudaError_t value (-1 for an unsupported kind / n).
extern "C" int chameleon_probe_mma(int kind, int n, int ctas, int iters, unsigned long long* cycles, int* status,
                                   void* stream) {
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  using namespace cham;
#define PROBE_CASE(K, NN) \
  if (kind == K && n == NN) return launch_probe<K, NN>(ctas, iters, cycles, status, st);
  PROBE_CASE(0, 128) PROBE_CASE(0, 192) PROBE_CASE(0, 256)
  PROBE_CASE(1, 128) PROBE_CASE(1, 192) PROBE_CASE(1, 256)
  PROBE_CASE(2, 128) PROBE_CASE(2, 192) PROBE_CASE(2, 256)
  PROBE_CASE(3, 160) PROBE_CASE(3, 192)
  PROBE_CASE(4, 160) PROBE_CASE(4, 192)
  PROBE_CASE(5, 160) PROBE_CASE(5, 192)
  PROBE_CASE(6, 160) PROBE_CASE(6, 192)
  PROBE_CASE(7, 192)
#undef PROBE_CASE
  return -1;
}
