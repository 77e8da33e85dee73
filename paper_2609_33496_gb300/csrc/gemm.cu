// gemm.cu -- mixed-format quantized linear on tcgen05 tensor cores (steps a7, a8).
//
// Y[m, perm[p]] = s_a * s_w[p] * sum_k A^[m, k] * W^[p, k] + bias[perm[p]]   (Sec. 3.6, Alg. 2/3)
//
// Operand roles are swapped relative to the textbook layout so that the weight side -- the
// operand that needs per-channel decoding -- never touches shared memory:
//   * MMA "A" (M = 128 rows) = one tile of 128 packed weight channels.  Four decode warps own one
//     channel per thread, read its codes with coalesced 16-byte loads, decode them in registers to
//     exact fp16 operand values (the MX block exponent folded in, the per-channel scale kept for
//     the epilogue) and write them straight into tensor memory with tcgen05.st.
//   * MMA "B" (N = BN tokens) = a tile of activation operand rows, brought into shared memory by
//     TMA with 128-byte swizzling, K-major.
//   * D (128 channels x BN tokens, fp32) accumulates in tensor memory; the same four warps read
//     it back with tcgen05.ld, apply s_a * s_w and the bias, and store Y in original channel order.
// A 4-stage ring over K-chunks of 64 couples them: TMA and decode fill stage s, one thread issues
// four kind::f16 MMAs (K = 16 each) on it, and the MMA commit frees the stage for both producers.
// Every wait is bounded (common.cuh); on a timeout the kernel records CHAM_ERR_TIMEOUT, drains
// its own copies and MMAs, releases tensor memory and returns.
#include "gemm.cuh"

namespace cham {

constexpr int kStages = 4;
constexpr int kBK = 64;  // K elements per stage: 128 bytes of fp16 per activation row
constexpr int kGemmThreads = 256;

template <int BN>
struct GemmCfg {
  static constexpr int kBStage = BN * 128;
  static constexpr int kData = kStages * kBStage;
  static constexpr int kTmemCols = (BN + kStages * 32) <= 256 ? 256 : 512;
  static constexpr int kACol = kTmemCols - kStages * 32;  // first TMEM column of the A stages
  static constexpr int kMisc = 1024 /*NF4 pair table*/ + 8 * (3 * kStages + 1) + 16;
  static constexpr int kNeed = 1024 /*alignment slack*/ + kData + kMisc;
  // Shared-memory request: at most two CTAs per SM when each holds 256 TMEM columns, one when it
  // holds 512, so tensor-memory allocations never have to wait for each other.
  static constexpr int kFloor = kTmemCols == 512 ? 120 * 1024 : 80 * 1024;
  static constexpr int kSmem = kNeed > kFloor ? kNeed : kFloor;
  static_assert(BN % 16 == 0 && BN >= 16 && BN <= 256, "MMA N for M = 128");
};

CHAM_DEV float exp2i_clamped(int e) { return exp2i_f32(e < -126 ? -126 : e); }

CHAM_DEV bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* st) {
  const bool ok = mbar_wait(bar, parity, abort_flag, st);
  return __all_sync(0xffffffffu, ok);
}

// Drain wait used only on the way out: ignores the abort flag, still bounded.
CHAM_DEV void drain_wait(uint64_t* bar, uint32_t parity) {
  for (uint32_t i = 0; i < kWaitPolls; ++i) {
    if (mbar_test(bar, parity)) return;
    if (i > 64) __nanosleep(128);
  }
}

// 8-bit codes of one channel's 64-element chunk -> 32 fp16 pairs (element 2c, 2c+1 in column c).
CHAM_DEV void decode_w8(const uint32_t (&w)[16], int f, int z, uint32_t e8, uint32_t (&out)[32]) {
  if (f == CHAM_W_MXINT8) {
    const float sc0 = exp2i_clamped(static_cast<int>(e8 & 0xFFu) - 127 - 6);
    const float sc1 = exp2i_clamped(static_cast<int>((e8 >> 8) & 0xFFu) - 127 - 6);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const float sc = i < 8 ? sc0 : sc1;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int b0 = static_cast<int>(static_cast<int8_t>((w[i] >> (16 * h)) & 0xFFu));
        const int b1 = static_cast<int>(static_cast<int8_t>((w[i] >> (16 * h + 8)) & 0xFFu));
        out[2 * i + h] = h2_as_u32(__floats2half2_rn(__fmul_rn(static_cast<float>(b0), sc),
                                                     __fmul_rn(static_cast<float>(b1), sc)));
      }
    }
  } else {
    // 0x64XX as fp16 is 1024 + XX: subtract 1024 + 128 (sym, codes biased by the xor) or 1024 + z
    const uint32_t flip = f == CHAM_W_INT8_SYM ? 0x80808080u : 0u;
    const __half2 sub = __float2half2_rn(f == CHAM_W_INT8_SYM ? 1152.f : 1024.f + static_cast<float>(z));
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const uint32_t v = w[i] ^ flip;
      out[2 * i] = h2_as_u32(__hsub2(u32_as_h2(__byte_perm(v, 0x64646464u, 0x4140)), sub));
      out[2 * i + 1] = h2_as_u32(__hsub2(u32_as_h2(__byte_perm(v, 0x64646464u, 0x4342)), sub));
    }
  }
}

// 4-bit codes of one channel's chunk -> 32 fp16 pairs.  Word i holds elements 8i..8i+7 with
// nibble j = element 2j and nibble 4+j = element 2j+1, so (x >> 4j) & 0x000F000F isolates a pair.
CHAM_DEV void decode_w4(const uint32_t (&w)[8], int f, int z, uint32_t e8, const uint32_t* lut,
                        uint32_t (&out)[32]) {
  if (f == CHAM_W_NF4) {
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) out[4 * i + j] = lut[((w[i] >> (4 * j)) & 0xFu) | ((w[i] >> (4 * j + 12)) & 0xF0u)];
    return;
  }
  if (f == CHAM_W_E2M1 || f == CHAM_W_MXFP4) {
    // E2M1 s.e1e0.m placed at fp16 bits 15 and 11..9 is value * 2^-14: multiply back by 2^14
    const __half2 k = __float2half2_rn(16384.f);
    const float up0 = exp2i_clamped(static_cast<int>(e8 & 0xFFu) - 127);
    const float up1 = exp2i_clamped(static_cast<int>((e8 >> 8) & 0xFFu) - 127);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t x = w[i] >> (4 * j);
        const uint32_t bits = ((x & 0x00070007u) << 9) | ((x & 0x00080008u) << 12);
        const __half2 h = __hmul2(u32_as_h2(bits), k);
        if (f == CHAM_W_E2M1) {
          out[4 * i + j] = h2_as_u32(h);
        } else {
          const float up = i < 4 ? up0 : up1;
          const float2 v = __half22float2(h);
          out[4 * i + j] = h2_as_u32(__floats2half2_rn(__fmul_rn(v.x, up), __fmul_rn(v.y, up)));
        }
      }
    }
    return;
  }
  // INT4-sym, INT4-asym, MXINT4: 0x640N as fp16 is 1024 + N
  const bool sym = f != CHAM_W_INT4_ASYM;
  const uint32_t flip = sym ? 0x88888888u : 0u;
  const __half2 sub = __float2half2_rn(sym ? 1032.f : 1024.f + static_cast<float>(z));
  const float up0 = exp2i_clamped(static_cast<int>(e8 & 0xFFu) - 127 - 2);
  const float up1 = exp2i_clamped(static_cast<int>((e8 >> 8) & 0xFFu) - 127 - 2);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t v = w[i] ^ flip;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const __half2 h = __hsub2(u32_as_h2(((v >> (4 * j)) & 0x000F000Fu) | 0x64006400u), sub);
      if (f != CHAM_W_MXINT4) {
        out[4 * i + j] = h2_as_u32(h);
      } else {
        const float up = i < 4 ? up0 : up1;
        const float2 q = __half22float2(h);
        out[4 * i + j] = h2_as_u32(__floats2half2_rn(__fmul_rn(q.x, up), __fmul_rn(q.y, up)));
      }
    }
  }
}

CHAM_DEV void tmem_ld_32x32b_x16(uint32_t taddr, uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%16];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
        "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
      : "r"(taddr)
      : "memory");
}

template <int BITS>
CHAM_DEV void load_raw(const uint8_t* chunk_base, uint32_t (&raw)[16]) {
  // slab j of a chunk holds bytes [16j, 16j+16) of all 128 channels, 2048 bytes apart
#pragma unroll
  for (int j = 0; j < BITS / 2; ++j) {
    const uint4 u = __ldg(reinterpret_cast<const uint4*>(chunk_base + j * 2048));
    raw[4 * j] = u.x;
    raw[4 * j + 1] = u.y;
    raw[4 * j + 2] = u.z;
    raw[4 * j + 3] = u.w;
  }
}

template <int BN, int BITS>
__global__ void __launch_bounds__(kGemmThreads, 1)
    k_gemm_ts_f16(const __grid_constant__ CUtensorMap act_map, const GemmArgs a) {
  using C = GemmCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sB = smem;
  uint32_t* lut = reinterpret_cast<uint32_t*>(smem + C::kData);
  uint64_t* full_b = reinterpret_cast<uint64_t*>(lut + 256);
  uint64_t* full_a = full_b + kStages;
  uint64_t* empty = full_a + kStages;
  uint64_t* accum = empty + kStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tile = a.tile0 + blockIdx.x;
  const int tok0 = blockIdx.y * BN;
  const int nk = a.n_chunks;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full_b[s], 1);
      mbar_init(&full_a[s], 128);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accum, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  for (int i = threadIdx.x; i < 256; i += kGemmThreads)  // NF4 pair table (low half = even element)
    lut[i] = static_cast<uint32_t>(a.nf4_level[i & 15]) | (static_cast<uint32_t>(a.nf4_level[i >> 4]) << 16);
  if (warp == 0 && lane == 0) tma_prefetch_desc(&act_map);
  if (warp == 2) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t d_tmem = tmem;               // columns [0, BN)
  const uint32_t a_tmem = tmem + C::kACol;    // stage s at columns kACol + 32 s

  if (warp == 0) {
    // ---------------- TMA producer: activation tiles
    if (lane == 0) {
      int issued = 0;
      for (int kc = 0; kc < nk; ++kc) {
        const int s = kc % kStages;
        const uint32_t ph = (kc / kStages) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, a.dev_status)) break;
        mbar_arrive_expect_tx(&full_b[s], C::kBStage);
        tma_load_2d(smem_u32(sB + s * C::kBStage), &act_map, &full_b[s], kc * kBK, tok0);
        issued = kc + 1;
      }
      for (int kc = issued > kStages ? issued - kStages : 0; kc < issued; ++kc)
        drain_wait(&full_b[kc % kStages], (kc / kStages) & 1);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f16(128, BN);
      for (int kc = 0; kc < nk; ++kc) {
        const int s = kc % kStages;
        const uint32_t ph = (kc / kStages) & 1;
        if (!mbar_wait(&full_b[s], ph, abort_flag, a.dev_status)) break;
        if (!mbar_wait(&full_a[s], ph, abort_flag, a.dev_status)) break;
        tc_fence_after();
        const uint32_t b0 = smem_u32(sB + s * C::kBStage);
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk)
          mma_f16_ts(d_tmem, a_tmem + s * 32 + kk * 8, smem_desc_sw128(b0 + kk * 32), idesc, (kc | kk) != 0);
        mma_commit(&empty[s]);
      }
      mma_commit(accum);
      drain_wait(accum, 0);  // all issued MMAs have finished before tensor memory is released
    }
  } else if (warp >= 4) {
    // ---------------- weight decode (one channel per thread), then the epilogue
    const int q = warp - 4;  // tensor-memory lane quadrant of this warp
    const int r = q * 32 + lane;
    const int p = tile * 128 + r;
    const int f = a.wfmt[p];
    const int z = a.wzero[p];
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    constexpr int kChunkBytes = BITS == 8 ? 8192 : 4096;
    const uint8_t* cbase = a.codes + static_cast<size_t>(tile) * nk * kChunkBytes + r * 16;
    const uint16_t* e8base = reinterpret_cast<const uint16_t*>(a.we8m0) + static_cast<size_t>(tile) * nk * 128 + r;
    uint32_t raw[16];
    load_raw<BITS>(cbase, raw);
    uint32_t e8 = e8base[0];
    bool ok = true;
    for (int kc = 0; kc < nk; ++kc) {
      const int s = kc % kStages;
      const uint32_t ph = (kc / kStages) & 1;
      uint32_t out[32];
      if constexpr (BITS == 8) {
        decode_w8(raw, f, z, e8, out);
      } else {
        const uint32_t (&r8)[8] = *reinterpret_cast<const uint32_t(*)[8]>(&raw[0]);
        decode_w4(r8, f, z, e8, lut, out);
      }
      if (kc + 1 < nk) {
        load_raw<BITS>(cbase + static_cast<size_t>(kc + 1) * kChunkBytes, raw);
        e8 = e8base[static_cast<size_t>(kc + 1) * 128];
      }
      if (!warp_wait(&empty[s], ph ^ 1, abort_flag, a.dev_status)) {
        ok = false;
        break;
      }
      tc_fence_after();
      tmem_st_32x32b_x32(a_tmem + lane_off + s * 32, out);
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(&full_a[s]);
    }
    if (ok && warp_wait(accum, 0, abort_flag, a.dev_status)) {
      tc_fence_after();
      const int orig = a.perm[p];
      const float sa = a.act_scale != nullptr ? *a.act_scale : 1.f;
      const float scale = __fmul_rn(sa, a.wscale[p]);
      const float b = (a.bias != nullptr && orig >= 0) ? a.bias[orig] : 0.f;
      float* yc = a.Y + (orig >= 0 ? orig : 0);
#pragma unroll 1
      for (int j = 0; j < BN / 16; ++j) {
        uint32_t v[16];
        tmem_ld_32x32b_x16(d_tmem + lane_off + j * 16, v);
        tmem_wait_ld();
        if (orig >= 0) {
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int tok = tok0 + j * 16 + i;
            if (tok < a.M) yc[static_cast<size_t>(tok) * a.N] = fmaf(__uint_as_float(v[i]), scale, b);
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

int gemm_pick_bn(int M, int n_tiles, int num_sms) {
  if (M <= 16) return 16;
  if (M <= 32) return 32;
  if (M <= 64) return 64;
  if (M <= 128) return 128;
  const long ctas256 = static_cast<long>(n_tiles) * ((M + 255) / 256);
  return ctas256 >= num_sms ? 256 : 128;
}

template <int BN, int BITS>
static cudaError_t launch_bn(const CUtensorMap& map, const GemmArgs& a, int n_tiles, cudaStream_t st) {
  using C = GemmCfg<BN>;
  static int configured_device = -1;  // attribute is per device; re-set when the device changes
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured_device != dev) {
    const cudaError_t e =
        cudaFuncSetAttribute(k_gemm_ts_f16<BN, BITS>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
    if (e != cudaSuccess) return e;
    configured_device = dev;
  }
  const dim3 grid(n_tiles, (a.M + BN - 1) / BN);
  k_gemm_ts_f16<BN, BITS><<<grid, kGemmThreads, C::kSmem, st>>>(map, a);
  return cudaGetLastError();
}

cudaError_t launch_gemm_f16(const CUtensorMap& map, const GemmArgs& a, int n_tiles, int bn, cudaStream_t st) {
  if (a.bits == 8) {
    switch (bn) {
      case 16: return launch_bn<16, 8>(map, a, n_tiles, st);
      case 32: return launch_bn<32, 8>(map, a, n_tiles, st);
      case 64: return launch_bn<64, 8>(map, a, n_tiles, st);
      case 128: return launch_bn<128, 8>(map, a, n_tiles, st);
      default: return launch_bn<256, 8>(map, a, n_tiles, st);
    }
  }
  switch (bn) {
    case 16: return launch_bn<16, 4>(map, a, n_tiles, st);
    case 32: return launch_bn<32, 4>(map, a, n_tiles, st);
    case 64: return launch_bn<64, 4>(map, a, n_tiles, st);
    case 128: return launch_bn<128, 4>(map, a, n_tiles, st);
    default: return launch_bn<256, 4>(map, a, n_tiles, st);
  }
}

}  // namespace cham
