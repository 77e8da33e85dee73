// gemm_f8_kernel.cuh -- the 4-bit mixed-format linear on 8-bit tensor cores (steps a7, Sec. 3.6):
// the kernel template for the 4-bit per-channel layouts whose class-0 channels (every decoded value
// an exact E4M3 number) meet FP8 activation codes (E4M3 or E5M2 with a per-tensor scale, or MXFP8
// blocks).  Instantiated in gemm_f8.cu (per-tensor activations) and gemm_f8_mx.cu (MXFP8).
//
// Y[m, perm[p]] = s_a * s_w[p] * sum_b 2^(e_w[p, b] + e_a[m, b]) sum_{k in block b} A^[m, k] W^[p, k] + bias
//
// Which weights qualify (MMA class 0 of the packed layout): INT4-sym and INT4-asym (q - z in
// [-15, 15]), E2M1, and the element values of MXINT4 (code / 4) and MXFP4 -- all are E4M3 values, so
// the FP8 operand is exact, and the per-32 block exponents of the MX formats ride in the MMA's block
// scale factors.  The activation codes are the quantizer's own bytes: E4M3 / E5M2 bit patterns with
// the per-tensor scale s_a applied in the epilogue, or MXFP8 E4M3 elements whose E8M0 exponents are
// the activation-side scale factors.  The product is the same sum the fp16 path forms from the
// dequantized operands; only the accumulation order inside the tensor core differs.
//
// One launch covers every tile of the layer: the class-1 tiles of a 4-bit layout (NF4, whose levels
// are not 8-bit floats) take a second mainloop in the same kernel -- kind::f16 MMAs on the exact
// fp16 activation operand, NF4 levels decoded to fp16 -- so that the two classes' output columns,
// which interleave in Y, are written at the same time (two launches would each leave fp32 output
// sectors half written, and the second one's writes would miss in L2), and neither class waits for
// the other's last wave.
//
// Structure (as the fp16 kernel in gemm_kernel.cuh, whose epilogue role it shares):
//   * MMA "A" (M = 128) = 128 packed weight channels decoded into tensor memory, one thread per
//     channel.  FP8 tiles: every 4-bit code indexes that channel's own 16-entry table of E4M3 bytes
//     (built once per tile from the format and zero point), so channels of different formats in
//     one tile take the same instructions; the channel's four block exponents of the chunk go to
//     the A scale-factor columns.  NF4 tiles: the levels as fp16 pairs from byte tables.
//   * MMA "B" (N = BN tokens) = 128 bytes per activation row, loaded by TMA with 128-byte
//     swizzling: 128 FP8 codes (MXFP8 also brings its chunk's exponents, 4 bytes per token) or 64
//     fp16 operand values.
//   * K-chunks of 128 (FP8: 4 MMAs kind::mxf8f6f4, K = 32 each, scale vector 1X -- one E8M0 per row
//     per MMA, selected by the instruction's scale-factor ids -- the last chunk issuing only the
//     MMAs of the 32-element blocks inside K) or of 64 (NF4: 4 MMAs kind::f16, K = 16).
// Tensor-memory columns: two accumulators, four decoded-weight slots of 32 columns, the A scale
// factors of each slot (8 columns apart, lane m reads column base + m / 32), and the B scale
// factors (every lane quadrant holds all BN tokens: lane 32q + n % 32, column base + n / 32) --
// one constant copy for per-tensor activations, one per slot for MXFP8.
#pragma once

#include "gemm_kernel.cuh"

namespace cham {

constexpr int kBK8 = 128;  // K elements per FP8 chunk: 128 bytes per activation row

template <int BN, bool MXA>
struct F8Cfg {
  static constexpr int kBBytes = BN * 128;       // activation codes
  static constexpr int kWBytes = 2 * 128 * 32;   // two 64-element blob chunks of 4-bit codes
  static constexpr int kEBytes = 2 * 256;        // their E8M0 pairs
  static constexpr int kSBytes = MXA ? 1024 : 0; // MXFP8: 4 exponent bytes per token, up to 256 tokens
  static constexpr int kStage = (kBBytes + kWBytes + kEBytes + kSBytes + 1023) / 1024 * 1024;
  static constexpr int kStages = (200 * 1024) / kStage > 8 ? 8 : (200 * 1024) / kStage;
  static constexpr int kData = kStages * kStage;
  static constexpr int kAccCols = BN < 32 ? 32 : BN;
  static constexpr int kACol = 2 * kAccCols;
  // decoded-weight slots (32 columns each) with their A scale factors (8 columns each; MXFP8: and
  // their B scale factors, 8 more), as many as fit next to the accumulators, at most 8.  Every
  // chunk is its own commit group: a slot goes back to the decoders as soon as its MMAs have
  // completed (pairs of chunks per commit measured 4-5 % slower on 8192 x 1152 x 4608)
  static constexpr int kPerSlot = 32 + 8 + (MXA ? 8 : 0);
  static constexpr int kAFit = (512 - kACol - (MXA ? 0 : 8)) / kPerSlot;
  static constexpr int kAStages = kAFit > 8 ? 8 : kAFit;
  static constexpr int kGroup = 1, kDone = 16;
  static constexpr int kSFA = kACol + kAStages * 32;          // slot s: columns kSFA + 8 s .. + 3
  static constexpr int kSFB = kSFA + kAStages * 8;            // per-tensor: one copy; MXFP8: slot s at + 8 s
  static constexpr int kSFBCols = (BN + 31) / 32;
  static constexpr int kNeedCols = kSFB + (MXA ? kAStages * 8 : 8);
  static constexpr int kTmemCols = kNeedCols <= 256 ? 256 : 512;
  static constexpr int kMisc = 8 * (kStages + kDone + kAStages / kGroup + 4) + 16;
  static constexpr int kNeed = 1024 + kData + kMisc;
  static constexpr int kSmem = kNeed > 116 * 1024 ? kNeed : 116 * 1024;  // one CTA per SM
  static_assert(BN % 32 == 0 && BN >= 32 && BN <= 256, "token tile: a multiple of 32 (accumulator columns)");
  static_assert(kStages >= 4, "ring depth");
  static_assert(kSmem <= 227 * 1024, "within the opt-in shared-memory limit");
  static_assert(kNeedCols <= 512, "tensor memory budget");
  static_assert(kSFBCols <= 8, "B scale factors: 8 columns per copy");
  static_assert(kAStages >= 3, "decoded-weight slots in flight");
  static_assert(kDone * kGroup > kStages + kGroup, "group barrier rotation");
};

// D[tmem] (+)= A[tmem] * B[smem]^T with per-32 block scale factors, kind::mxf8f6f4.
CHAM_DEV void mma_mxf8_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc, uint32_t sfa,
                          uint32_t sfb, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %6, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], [%1], %2, %3, [%4], [%5], p;\n\t}\n" ::"r"(
          d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(sfa), "r"(sfb), "r"(accumulate)
      : "memory");
}

// The same MMA issued by the warp's elected lane: the whole warp executes the instruction with
// warp-uniform operands, one lane (the lowest active one, so always the same lane of a converged
// warp) issues it.
CHAM_DEV void mma_mxf8_ts_elect(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc, uint32_t sfa,
                                uint32_t sfb, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred e, p;\n\t"
      "elect.sync _|e, 0xffffffff;\n\t"
      "setp.ne.b32 p, %6, 0;\n\t"
      "@e tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], [%1], %2, %3, [%4], [%5], p;\n\t}\n" ::
          "r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(sfa), "r"(sfb), "r"(accumulate)
      : "memory");
}

// Instruction descriptor of kind::mxf8f6f4: A E4M3 (weights), B E4M3 or E5M2 (btype 0 / 1), both
// K-major, M x N, UE8M0 scale factors (bit 23); the A / B scale-factor ids (bits 29-30 / 4-5) pick
// the byte of the scale-factor column each MMA uses.
__host__ __device__ constexpr uint32_t idesc_mxf8(int M, int N, int btype) {
  return (0u << 7) | (static_cast<uint32_t>(btype) << 10) | (static_cast<uint32_t>(N >> 3) << 17) | (1u << 23) |
         (static_cast<uint32_t>(M >> 4) << 24);
}
__host__ __device__ constexpr uint32_t idesc_sf_ids(uint32_t idesc, int i) {
  return idesc | (static_cast<uint32_t>(i) << 4) | (static_cast<uint32_t>(i) << 29);
}


// Value of 4-bit code n of a class-0 channel in format f (zero point z for INT4-asym): INT4-sym and
// MXINT4 store q + 8 (MXINT4 elements are q / 4, the block exponent apart), INT4-asym stores q with
// value q - z, E2M1 and MXFP4 store the sign-exponent-mantissa bits.  Other formats (padding): 0.
CHAM_DEV float f8_level(int f, int z, int n) {
  switch (f) {
    case CHAM_W_INT4_SYM: return static_cast<float>(n - 8);
    case CHAM_W_MXINT4: return 0.25f * static_cast<float>(n - 8);
    case CHAM_W_INT4_ASYM: return static_cast<float>(n - z);
    case CHAM_W_E2M1:
    case CHAM_W_MXFP4: {
      const int e = (n >> 1) & 3, m = n & 1;
      const float mag = e == 0 ? 0.5f * m : exp2i_f32(e - 1) * (1.f + 0.5f * m);
      return (n & 8) ? -mag : mag;
    }
    default: return 0.f;
  }
}

// The channel's 16-entry E4M3 table: byte n % 4 of word n / 4 holds the code of f8_level(n)
// (every level is an E4M3 value, so the conversion is exact).
CHAM_DEV void f8_table(int f, int z, uint32_t (&T)[4]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) T[i] = 0;
#pragma unroll
  for (int n = 0; n < 16; n += 2) {
    const uint32_t e = cvt_e4m3x2(f8_level(f, z, n + 1), f8_level(f, z, n));
    T[n >> 2] |= e << (8 * (n & 2));
  }
}

// Sign-magnitude formats (E2M1, MXFP4: bit 3 of the code is the sign, bits 0-2 the magnitude).
CHAM_DEV bool f8_sign_magnitude(int f) { return f == CHAM_W_E2M1 || f == CHAM_W_MXFP4; }

// Four codes (the selector nibbles of sel; bit 3 of each code in the byte mask m) -> four table bytes.
CHAM_DEV uint32_t f8_lookup4(uint32_t sel, uint32_t m, const uint32_t (&T)[4]) {
  const uint32_t lo = prmt(T[0], T[1], sel), hi = prmt(T[2], T[3], sel);
  return (lo & ~m) | (hi & m);
}

// 128 codes of one channel (16 words, word i = elements 8i..8i+7 with nibble j = element 2j for
// j < 4 and element 2(j - 4) + 1 for j >= 4, the blob's 4-bit order) -> 32 columns of E4M3 bytes in
// the same group order: column 2i holds elements 8i, 8i+2, 8i+4, 8i+6 and column 2i+1 holds 8i+1,
// 8i+3, 8i+5, 8i+7 (the activation codes of the FP8 operand are stored in that order too, so the
// MMA still pairs element k with element k).  SM: every lane's table is sign-magnitude (entries
// 8..15 are 0..7 with the sign bit), so one permute of the magnitudes and the sign bit suffice.
template <bool SM>
CHAM_DEV void decode_f8(const uint32_t (&w)[16], const uint32_t (&T)[4], uint32_t (&out)[32]) {
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const uint32_t x = w[i];
    const uint32_t s = x & 0x77777777u, x4 = x << 4;
    // byte mask of each code's bit 3: PRMT with the sign-replicate selector bit copies bit 7 of the
    // byte that holds that bit (x << 4 for the low nibble of a byte, x for the high one)
    const uint32_t mlo = prmt(x4, x, 0xD9C8u), mhi = prmt(x4, x, 0xFBEAu);
    if constexpr (SM) {
      out[2 * i] = prmt(T[0], T[1], s) | (mlo & 0x80808080u);
      out[2 * i + 1] = prmt(T[0], T[1], s >> 16) | (mhi & 0x80808080u);
    } else {
      out[2 * i] = f8_lookup4(s, mlo, T);
      out[2 * i + 1] = f8_lookup4(s >> 16, mhi, T);
    }
  }
}

// MXA: the activations are MXFP8 (their exponents come with every FP8 stage); otherwise E4M3 /
// E5M2 codes with a per-tensor (or per-sample) scale and constant unit B scale factors.  Channel
// tiles tile0 .. tile0 + f8_tiles - 1 take the FP8 mainloop (map8: the codes), the rest of the
// launch's tiles the NF4 / fp16 one (map16: the fp16 operand).
template <int BN, int EPI, bool MXA>
__global__ void __launch_bounds__(kGemmThreads, 1)
    k_gemm_ts_f8(const __grid_constant__ CUtensorMap map8, const __grid_constant__ CUtensorMap map16,
                 const GemmArgs a) {
  using C = F8Cfg<BN, MXA>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint32_t* misc = reinterpret_cast<uint32_t*>(smem + C::kData);
  constexpr int S = C::kStages;
  constexpr int kAStages = C::kAStages, kGroup = C::kGroup, kAGroups = kAStages / kGroup;
  constexpr int kDone = C::kDone;
  constexpr int kDec = Roles<4>::kDec, kEpi = Roles<4>::kEpi;
  uint64_t* full = reinterpret_cast<uint64_t*>(misc);       // [S] producer -> decoders (tx bytes)
  uint64_t* done = full + S;                                 // [kDone] MMA group commit -> producer, decoders
  uint64_t* afull = done + kDone;                            // [kAGroups] decode warps -> MMA
  uint64_t* accfull = afull + kAGroups;                      // [2] MMA commit -> epilogue
  uint64_t* accempty = accfull + 2;                          // [2] epilogue warps -> MMA
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nk8 = (a.nk64 + 1) / 2;  // chunks of 128 (FP8 tiles); NF4 tiles walk the nk64 chunks of 64
  const int n_ch = a.n_ch_tiles;
  const int n_tiles = n_ch * ((a.M + BN - 1) / BN);
  const int ks = a.k_split;
  const int n_units = n_tiles * ks;
  auto is_f8 = [&](int u) { return (u / ks) % n_ch < a.f8_tiles; };
  auto kc_begin = [&](int u) { return ks == 1 ? 0 : (u % ks) * (is_f8(u) ? nk8 : a.nk64) / ks; };
  auto kc_end = [&](int u) { const int nk = is_f8(u) ? nk8 : a.nk64; return ks == 1 ? nk : (u % ks + 1) * nk / ks; };
  uint32_t total = 0;
  for (int u = blockIdx.x; u < n_units; u += gridDim.x) total += static_cast<uint32_t>(kc_end(u) - kc_begin(u));
  auto wait_done = [&](uint32_t j) {
    const uint32_t g = j / kGroup;
    return mbar_wait(&done[g % kDone], (g / kDone) & 1, abort_flag, a.dev_status);
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) mbar_init(&full[s], 2);  // the two producer threads
    for (int g = 0; g < kDone; ++g) mbar_init(&done[g], 1);
    for (int g = 0; g < kAGroups; ++g) mbar_init(&afull[g], 4 * kGroup);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accfull[b], 1);
      mbar_init(&accempty[b], 4 * kEpi);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&map8);
    if (a.f8_tiles < n_ch) tma_prefetch_desc(&map16);
  }
  if (warp == 2) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();
  griddep_launch_dependents();

  if (warp == 0 || warp == 3) {
    // ---------------- producers: one chunk sequence, two threads.  Warp 0 loads the activation
    // operand (TMA: FP8 codes, or the fp16 operand of an NF4 chunk) and, MXFP8, the chunk's
    // activation exponents of the tile's tokens (bulk); warp 3 the weight codes (two blob chunks
    // of 64, one for an NF4 chunk or the last FP8 chunk of an odd K) and their E8M0 bytes (bulk).
    // Each arrives on the stage's barrier with its own byte count (the barrier counts two): issuing
    // the copies is most of a producer's time per chunk, and one thread alone came close to the
    // MMA thread's chunk period
    if (lane == 0) {
      const bool act = warp == 0;
      uint32_t it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        const int t = u / ks;
        const int ch = a.tile0 + t % n_ch, tok0 = (t / n_ch) * BN;
        const bool f8 = is_f8(u);
        const int kc1 = kc_end(u);
        const uint32_t sf_bytes = MXA ? static_cast<uint32_t>(min(BN, a.act_mp - tok0)) * 4u : 0u;
        for (int kc = kc_begin(u); kc < kc1; ++kc, ++it) {
          const int s = it % S;
          if (it >= static_cast<uint32_t>(S) && !wait_done(it - S)) {
            ok = false;
            break;
          }
          uint8_t* st = smem + s * C::kStage;
          const bool stall = blockIdx.x == 0 && static_cast<int>(it) == a.stall_chunk;  // test hook (see the fp16 kernel)
          if (act) {
            mbar_arrive_expect_tx(&full[s], C::kBBytes + (f8 ? sf_bytes : 0u));
            if (stall) continue;
            if (f8) tma_load_2d(smem_u32(st), &map8, &full[s], kc * kBK8, tok0);
            else tma_load_2d(smem_u32(st), &map16, &full[s], kc * kBK, tok0);
            if constexpr (MXA)
              if (f8)
                bulk_load(smem_u32(st + C::kBBytes + C::kWBytes + C::kEBytes),
                          a.act_e8 + static_cast<size_t>(kc) * a.act_e8_plane + static_cast<size_t>(tok0) * 4,
                          sf_bytes, &full[s]);
          } else {
            const int nh = f8 ? (2 * kc + 1 < a.nk64 ? 2 : 1) : 1;
            const size_t chunk64 = static_cast<size_t>(ch) * a.nk64 + (f8 ? 2 * kc : kc);
            const uint32_t e_bytes = f8 ? nh * (C::kEBytes / 2) : 0u;
            mbar_arrive_expect_tx(&full[s], nh * (C::kWBytes / 2) + e_bytes);
            if (stall) continue;
            bulk_load(smem_u32(st + C::kBBytes), a.codes + chunk64 * (C::kWBytes / 2), nh * (C::kWBytes / 2), &full[s]);
            if (f8)
              bulk_load(smem_u32(st + C::kBBytes + C::kWBytes), a.we8m0 + chunk64 * (C::kEBytes / 2), e_bytes,
                        &full[s]);
          }
        }
      }
      // every issued copy must have landed before the CTA may exit
      const uint32_t first = it > S ? it - S : 0;
      for (uint32_t j = first; j < it; ++j) drain_wait(&full[j % S], (j / S) & 1);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer.  The whole warp runs the loop, so the descriptors and counters
    // are warp-uniform values; the MMAs and commits are issued by the elected lane (the lowest,
    // the same one every time, so each commit covers every MMA issued before it)
    const uint32_t idesc8 = idesc_mxf8(128, BN, a.b_fmt);
    constexpr uint32_t idesc16 = idesc_f16(128, BN);
    const uint64_t desc0 = smem_desc_sw128(smem_u32(smem));
    constexpr uint32_t kStageDesc = C::kStage >> 4;
    uint32_t it = 0, acc_it = 0, s = 0, sa = 0, gi = 0;
    bool ok = true;
    bool ready = false;  // the chunk's decoded operands are known to be in place (tested a chunk ahead)
    for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x, ++acc_it) {
      const int b = acc_it & 1;
      const int kc0 = kc_begin(u), kc1 = kc_end(u);
      const bool f8 = is_f8(u);
      if (!warp_wait(&accempty[b], ((acc_it >> 1) & 1) ^ 1, abort_flag, a.dev_status)) break;
      tc_fence_after();
      const uint32_t d_tmem = tmem + b * C::kAccCols;
      for (int kc = kc0; kc < kc1; ++kc, ++it) {
        if (gi == 0) {
          if (!ready && !warp_wait(&afull[(it / kGroup) % kAGroups], (it / kAStages) & 1, abort_flag, a.dev_status)) {
            ok = false;
            break;
          }
          tc_fence_after();
        }
        // test the next chunk's barrier now (its previous phases were all waited for here, in
        // order): the result is used after this chunk's MMAs and commit, so the test's latency,
        // a fifth of the chunk period when it sat in front of the MMAs, hides behind them
        const uint32_t nx = it + 1;
        const bool nready = static_cast<int>(nx % kGroup) == 0 && nx < total &&
                            mbar_ready(&afull[(nx / kGroup) % kAGroups], (nx / kAStages) & 1);
        const uint64_t bd = desc0 + s * kStageDesc;
        const uint32_t ad = tmem + C::kACol + sa * 32;
        if (f8) {
          const uint32_t sfa = tmem + C::kSFA + sa * 8;
          const uint32_t sfb = tmem + C::kSFB + (MXA ? sa * 8 : 0);
          const int nmma = min(4, a.kblocks - 4 * kc);  // 32-element blocks of this chunk inside K
#pragma unroll
          for (int i = 0; i < 4; ++i)
            if (i < nmma)
              mma_mxf8_ts_elect(d_tmem, ad + 8 * i, bd + 2 * i, idesc_sf_ids(idesc8, i), sfa, sfb, kc != kc0 || i > 0);
        } else {
#pragma unroll
          for (int i = 0; i < 4; ++i) mma_f16_ts_elect(d_tmem, ad + 8 * i, bd + 2 * i, idesc16, kc != kc0 || i > 0);
        }
        if (++gi == kGroup || it + 1 == total) {
          mma_commit_elect(&done[(it / kGroup) % kDone]);
          gi = gi == kGroup ? 0 : gi;
        }
        s = s + 1 == static_cast<uint32_t>(S) ? 0 : s + 1;
        sa = sa + 1 == static_cast<uint32_t>(kAStages) ? 0 : sa + 1;
        ready = __all_sync(0xffffffffu, nready);
      }
      mma_commit_elect(&accfull[b]);  // after an abort inside the tile this still covers every MMA issued
    }
    // all issued MMAs have finished before tensor memory is released
    if (lane == 0 && acc_it > 0) drain_wait(&accfull[(acc_it - 1) & 1], ((acc_it - 1) >> 1) & 1);
  } else if (warp >= 4 && warp < 4 + 4 * kDec) {
    // ---------------- weight decode: one channel per thread; group g takes chunks it % kDec == g
    const int q = warp & 3;
    const int grp = (warp - 4) >> 2;
    const int r = q * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    if constexpr (!MXA) {
      // unit B scale factors for the whole launch, before this group's first arrival
      if (grp == 0) {
        uint32_t one[8];
#pragma unroll
        for (int c = 0; c < 8; ++c) one[c] = 0x7F7F7F7Fu;
        tmem_st_32x32b_x8(tmem + lane_off + C::kSFB, one);
      }
    }
    uint32_t it = 0;
    bool ok = true;
    int nf = 0, nz = 0;
    if (static_cast<int>(blockIdx.x) < n_units) {
      const int p0 = (a.tile0 + (static_cast<int>(blockIdx.x) / ks) % n_ch) * 128 + r;
      nf = a.wfmt[p0];
      nz = a.wzero[p0];
    }
    for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
      const bool f8 = is_f8(u);
      uint32_t T[4];
      f8_table(nf, nz, T);
      const bool sm = __all_sync(0xffffffffu, f8_sign_magnitude(nf));  // the warp's channels
      if (u + static_cast<int>(gridDim.x) < n_units) {
        const int pn = (a.tile0 + ((u + static_cast<int>(gridDim.x)) / ks) % n_ch) * 128 + r;
        nf = a.wfmt[pn];
        nz = a.wzero[pn];
      }
      const int kc1 = kc_end(u);
      for (int kc = kc_begin(u); kc < kc1; ++kc, ++it) {
        if (static_cast<int>(it % kDec) != grp) continue;
        const int s = it % S, sa = it % kAStages;
        const uint32_t ph = (it / S) & 1;
        // when S is not a multiple of the decode groups, the stage's previous chunk (it - S) is
        // another group's, and testing this chunk's parity while that chunk's phase is still open
        // would pass on the opposite parity.  That chunk's commit closes its phase (its MMAs
        // follow its decode) and costs no extra wait: the producer waits for the same commit
        // before it loads this chunk
        if constexpr (S % kDec != 0) {
          if (it >= static_cast<uint32_t>(S) && !__all_sync(0xffffffffu, wait_done(it - S))) {
            ok = false;
            break;
          }
        }
        if (!warp_wait(&full[s], ph, abort_flag, a.dev_status)) {
          ok = false;
          break;
        }
        const uint8_t* st = smem + s * C::kStage;
        uint32_t out[32];
        uint32_t sfa = 0;
        uint32_t sfb[8];
        if (f8) {
          const int nh = 2 * kc + 1 < a.nk64 ? 2 : 1;
          const uint16_t* e8 = reinterpret_cast<const uint16_t*>(st + C::kBBytes + C::kWBytes);
          // block exponents of the chunk's four 32-element blocks (a missing second half is never read)
          sfa = static_cast<uint32_t>(e8[r]) | (nh == 2 ? static_cast<uint32_t>(e8[128 + r]) << 16 : 0x7F7F0000u);
          uint32_t raw[16];
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int j = 0; j < 2; ++j) {
              uint4 v = make_uint4(0, 0, 0, 0);
              if (h < nh) v = *reinterpret_cast<const uint4*>(st + C::kBBytes + h * 4096 + j * 2048 + r * 16);
              raw[8 * h + 4 * j] = v.x;
              raw[8 * h + 4 * j + 1] = v.y;
              raw[8 * h + 4 * j + 2] = v.z;
              raw[8 * h + 4 * j + 3] = v.w;
            }
          if (sm) decode_f8<true>(raw, T, out);
          else decode_f8<false>(raw, T, out);
          if constexpr (MXA) {
            // this lane's tokens n = 32 c + lane of the tile, in every lane quadrant
            const uint32_t* se = reinterpret_cast<const uint32_t*>(st + C::kBBytes + C::kWBytes + C::kEBytes);
#pragma unroll
            for (int c = 0; c < 8; ++c) sfb[c] = c < C::kSFBCols ? se[32 * c + lane] : 0x7F7F7F7Fu;
          }
        } else {
          // NF4 (element order in the codes): levels as fp16 pairs; the scale stays in the epilogue
          uint32_t raw[8];
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            const uint4 v = *reinterpret_cast<const uint4*>(st + C::kBBytes + j * 2048 + r * 16);
            raw[4 * j] = v.x;
            raw[4 * j + 1] = v.y;
            raw[4 * j + 2] = v.z;
            raw[4 * j + 3] = v.w;
          }
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            nf4_lookup4(raw[i] & 0xFFFFu, a.nf4_lo, a.nf4_hi, out[4 * i], out[4 * i + 1]);
            nf4_lookup4(raw[i] >> 16, a.nf4_lo, a.nf4_hi, out[4 * i + 2], out[4 * i + 3]);
          }
        }
        const bool free_ok = it < static_cast<uint32_t>(kAStages) || wait_done(it - kAStages);
        if (!__all_sync(0xffffffffu, free_ok)) {
          ok = false;
          break;
        }
        __syncwarp();
        tc_fence_after();
        tmem_st_32x32b_x32(tmem + C::kACol + lane_off + sa * 32, out);
        if (f8) {
          tmem_st_32x32b_x1(tmem + C::kSFA + lane_off + sa * 8 + q, sfa);
          if constexpr (MXA) tmem_st_32x32b_x8(tmem + C::kSFB + lane_off + sa * 8, sfb);
        }
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          const int missing = it + 1 == total ? kGroup - 1 - static_cast<int>(it % kGroup) : 0;
          for (int m = 0; m <= missing; ++m) mbar_arrive(&afull[(it / kGroup) % kAGroups]);
        }
      }
    }
  } else if (warp >= 4 + 4 * kDec) {
    epilogue_role<BN, EPI, kEpi, C::kAccCols>(a, tmem, accfull, accempty, abort_flag, warp, 4 + 4 * kDec, n_units,
                                              ks, n_ch);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

template <int BN, int EPI, bool MXA>
static cudaError_t launch_f8_bn(const CUtensorMap& map8, const CUtensorMap& map16, const GemmArgs& a, int num_sms,
                                cudaStream_t st) {
  using C = F8Cfg<BN, MXA>;
  static int configured_device = -1;
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured_device != dev) {
    const cudaError_t e =
        cudaFuncSetAttribute(k_gemm_ts_f8<BN, EPI, MXA>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
    if (e != cudaSuccess) return e;
    configured_device = dev;
  }
  const long units = static_cast<long>(a.n_ch_tiles) * ((a.M + BN - 1) / BN) * a.k_split;
  const int grid = static_cast<int>(units < num_sms ? units : num_sms);
  return launch_pdl(k_gemm_ts_f8<BN, EPI, MXA>, dim3(grid), dim3(kGemmThreads), C::kSmem, st, map8, map16, a);
}

template <int EPI, bool MXA>
static cudaError_t launch_f8_epi(const CUtensorMap& map8, const CUtensorMap& map16, const GemmArgs& a, int num_sms,
                                 int bn, cudaStream_t st) {
  switch (bn) {
    case 32: return launch_f8_bn<32, EPI, MXA>(map8, map16, a, num_sms, st);
    case 64: return launch_f8_bn<64, EPI, MXA>(map8, map16, a, num_sms, st);
    case 128: return launch_f8_bn<128, EPI, MXA>(map8, map16, a, num_sms, st);
    default:
      // the widest tile: kF8TokenTileMx for MXFP8 activations, kF8TokenTile otherwise
      if constexpr (MXA) return launch_f8_bn<kF8TokenTileMx, EPI, MXA>(map8, map16, a, num_sms, st);
      else return launch_f8_bn<kF8TokenTile, EPI, MXA>(map8, map16, a, num_sms, st);
  }
}

}  // namespace cham
