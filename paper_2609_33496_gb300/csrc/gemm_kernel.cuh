// gemm_kernel.cuh -- mixed-format quantized linear on tcgen05 tensor cores (steps a7, a8): the
// kernel template, included by gemm.cu (fp32 outputs), gemm_f16.cu and gemm_bf16.cu, each of which
// instantiates it for one output type so that the three compile in parallel.
//
// Y[m, perm[p]] = s_a * s_w[p] * sum_k A^[m, k] * W^[p, k] + bias[perm[p]]   (Sec. 3.6, Alg. 2/3)
//
// Operand roles are swapped relative to the textbook layout so that the weight side -- the
// operand that needs per-channel decoding -- never has to be written to shared memory:
//   * MMA "A" (M = 128 rows) = one tile of 128 packed weight channels.  Four decode warps own one
//     channel per thread, read its codes from a shared-memory stage that a bulk copy filled,
//     decode them in registers to the exact fp16 operand values (MX block exponent folded in, the
//     per-channel scale kept for the epilogue) and write them into tensor memory (tcgen05.st).
//   * MMA "B" (N = BN tokens) = a tile of activation operand rows, brought into shared memory by
//     TMA with 128-byte swizzling, K-major.
//   * D (128 channels x BN tokens, fp32) accumulates in tensor memory, double buffered: eight
//     epilogue warps (two per lane quadrant, alternate 16-column slices) drain one buffer (tcgen05.ld, s_a * s_w, bias, coalesced stores of Y in
//     original channel order) while the MMA fills the other with the next tile.
// The kernel is persistent: each CTA walks tiles t = blockIdx.x, blockIdx.x + gridDim.x, ... of
// the (channel tile, token tile) grid.  Two rings over K-chunks of 64 couple the roles: a 6-8
// stage shared-memory ring (activation tile + raw weight codes + their E8M0 bytes, filled by TMA
// and bulk copies, deep enough to cover the load round trip) and a 4-8 slot tensor-memory ring of
// decoded weight operands in two commit groups; one thread issues four kind::f16 MMAs (K = 16
// each) per chunk and one commit per group, which frees the group's slots in both rings.  Every wait is bounded (common.cuh); on a timeout
// the kernel records CHAM_ERR_TIMEOUT, drains its own copies and MMAs, releases tensor memory and
// returns.
#pragma once

#include <cuda_bf16.h>

#include <type_traits>

#include "gemm.cuh"

namespace cham {

constexpr int kBK = 64;  // K elements per stage: 128 bytes of fp16 per activation row
// decode warpgroups (taking K-chunks in turn) and epilogue warpgroups (taking alternate 16-column
// slices): the 4-bit decode (NF4 tables) is about three times the 8-bit one per chunk
template <int BITS> struct Roles {
  static constexpr int kDec = BITS == 4 ? 3 : 2, kEpi = BITS == 4 ? 1 : 2;
};
constexpr int kDecodeGroups = 2, kEpiGroups = 2;  // the 8-bit split; the thread count is the same
constexpr int kPartialOut = kPartialYT;  // epilogue "output type" of split-K units: raw fp32 partial sums
constexpr int kGemmThreads = 128 * (1 + kDecodeGroups + kEpiGroups);

template <int BN, int BITS>
struct GemmCfg {
  static constexpr int kBBytes = BN * 128;                        // activation tile
  static constexpr int kWBytes = 128 * (BITS == 8 ? 64 : 32);     // raw codes of 128 channels
  static constexpr int kEBytes = 256;                             // their E8M0 pairs (or zero points)
  static constexpr int kGBytes = 512;                             // group-wise blobs: fp16 block scales
  static constexpr int kStage = (kBBytes + kWBytes + kEBytes + kGBytes + 1023) / 1024 * 1024;
  // shared-memory ring: as deep as fits in ~200 KiB, to cover the TMA round trip (~1000 cycles)
  // plus decode and MMA time of the stages in flight
  static constexpr int kStages = (200 * 1024) / kStage > 8 ? 8 : (200 * 1024) / kStage;
  static constexpr int kData = kStages * kStage;
  static constexpr int kAccCols = (BN + 31) / 32 * 32;
  static constexpr int kACol = 2 * kAccCols;                      // first column of the A stages
  // Tensor-memory ring of decoded weight operands (32 columns per K-chunk), as deep as the 512
  // columns allow next to the two accumulators, split into commit groups of kGroup chunks.
  // The MMA thread commits once per group, and that one barrier frees both the group's
  // shared-memory stages and its tensor-memory stages.  One chunk per group: a slot returns to
  // the decoders as soon as its own MMAs are done (two chunks per commit measured 2-6 % slower
  // on 2048 x 1280 x 10240 and 8192 x 1152 x 4608).
  static constexpr int kAFit = (512 - kACol) / 32;
  static constexpr int kAStages = kAFit > 8 ? 8 : kAFit;
  static constexpr int kGroup = 1;   // chunks per commit group: kAStages groups in flight
  static constexpr int kDone = 16;                                // group-completion barriers
  static constexpr int kNeedCols = kACol + kAStages * 32;
  static constexpr int kTmemCols = kNeedCols <= 256 ? 256 : 512;
  // the mbarriers (full[S], done[kDone], afull[kAStages / kGroup], accfull[2], accempty[2]),
  // the TMEM address slot and the abort flag
  static constexpr int kMisc = 8 * (kStages + kDone + kAStages / kGroup + 4) + 16;
  static constexpr int kNeed = 1024 /*alignment slack*/ + kData + kMisc;
  // at least 116 KiB so that two CTAs (and two tensor-memory allocations) never share an SM
  static constexpr int kSmem = kNeed > 116 * 1024 ? kNeed : 116 * 1024;
  static_assert(kStages >= 4, "ring depth");
  static_assert(kSmem <= 227 * 1024, "within the opt-in shared-memory limit");
  static_assert(BN % 16 == 0 && BN >= 16 && BN <= 256, "MMA N for M = 128");
  static_assert(kNeedCols <= 512 && kAStages >= 4, "tensor memory budget");
  // a shared-memory stage is refilled only after the group holding its previous chunk completed;
  // kDone barriers in rotation keep a waiter from missing a phase
  static_assert(kDone * kGroup > kStages + kGroup, "group barrier rotation");
};

CHAM_DEV bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* st) {
  const bool ok = mbar_wait(bar, parity, abort_flag, st);
  return __all_sync(0xffffffffu, ok);
}

// Drain wait used only on the way out: ignores the abort flag, gives up after about a second of
// SM clock (non-suspending tests, so the bound does not depend on how long a suspended wait lasts).
constexpr long long kDrainCycles = 2000000000LL;
CHAM_DEV void drain_wait(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!mbar_ready(bar, parity)) {
    if (clock64() - t0 > kDrainCycles) return;
    __nanosleep(128);
  }
}

CHAM_DEV void bulk_load(uint32_t smem_dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(smem_dst),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// 2^e as an fp16 bit pattern for e in [-24, 15] (0 below).
CHAM_DEV uint32_t exp2_h(int e) {
  if (e >= -14) return static_cast<uint32_t>(e + 15) << 10;
  if (e >= -24) return 1u << (e + 24);
  return 0u;
}

// Two fp16 factors (as half2 bit patterns) whose product is 2^e, each applied exactly: the first
// keeps an integer or E2M1 code in the normal range, the second carries what is left (the
// product is an exact fp16 value, which the packer checks for MX weights).
CHAM_DEV void pow2_factors(int e, uint32_t& f1, uint32_t& f2) {
  const int a = min(max(e, -14), 15);
  const uint32_t h1 = exp2_h(a), h2 = exp2_h(e - a);
  f1 = h1 | (h1 << 16);
  f2 = h2 | (h2 << 16);
}

CHAM_DEV uint32_t hsub2u(uint32_t a, uint32_t b) { return h2_as_u32(__hsub2(u32_as_h2(a), u32_as_h2(b))); }
CHAM_DEV uint32_t hmul2u(uint32_t a, uint32_t b) { return h2_as_u32(__hmul2(u32_as_h2(a), u32_as_h2(b))); }

// Per-channel decode constants.
struct ChanDecode {
  int f;          // weight format
  int off;        // stored code of the value 0: zero point (asym) or the offset-binary bias
  int off0, off1; // the same for the chunk's two 32-element blocks (group-wise asym: their own)
  int e_off;      // MX: block exponent offset of the element scale (MXINT8 -6, MXINT4 -2, MXFP4 0)
  bool mx;
};

CHAM_DEV ChanDecode chan_decode(int f, int z) {
  ChanDecode c;
  c.f = f;
  const bool asym = f == CHAM_W_INT8_ASYM || f == CHAM_W_INT4_ASYM;
  c.off = asym ? z : (wbits(f) == 8 ? 128 : 8);
  c.off0 = c.off1 = c.off;
  c.e_off = f == CHAM_W_MXINT8 ? -6 : (f == CHAM_W_MXINT4 ? -2 : 0);
  c.mx = w_is_mx(f);
  return c;
}

// Element-scale exponent of block b (0 or 1) of a chunk: 0 for per-channel formats.
CHAM_DEV int block_exp(const ChanDecode& c, uint32_t e8, int b) {
  return c.mx ? static_cast<int>((e8 >> (8 * b)) & 0xFFu) - 127 + c.e_off : 0;
}

// Magic-number decode of integer codes.  An fp16 whose exponent field is E and whose low
// mantissa bits hold the code u (shifted left by t bits) has the value 2^(E-25) * (1024 + u * 2^t);
// subtracting the same construction with u = off leaves (u - off) * 2^(E-25+t) exactly (both
// operands lie in one binade).  Choosing E = e + 25 - t puts the block's power-of-two element
// scale 2^e into the same two instructions (PRMT or LOP3, then HSUB2), for every e that keeps E
// in [1, 30].
CHAM_DEV uint32_t dup16(uint32_t h) { return h | (h << 16); }

// 8-bit codes of one channel's 64-element chunk -> 32 fp16 pairs (element 2c, 2c+1 in column c).
// Called by whole warps (the vote below needs every lane).
CHAM_DEV void decode_w8(const uint32_t (&w)[16], const ChanDecode& c, uint32_t e8, uint32_t (&out)[32]) {
  const int e0 = block_exp(c, e8, 0), e1 = block_exp(c, e8, 1);
  // a block decodes on the fast path when its exponent fits; an all-zero MX block (E8M0 byte 0)
  // decodes to zeros whatever exponent is used
  const bool z0 = c.mx && (e8 & 0xFFu) == 0, z1 = c.mx && ((e8 >> 8) & 0xFFu) == 0;
  const bool fast = (z0 || (e0 >= -24 && e0 <= 5)) && (z1 || (e1 >= -24 && e1 <= 5));
  if (__all_sync(0xffffffffu, fast)) {
    const int E0 = min(max(e0, -24), 5) + 25, E1 = min(max(e1, -24), 5) + 25;
    const uint32_t hi[2] = {static_cast<uint32_t>(E0) << 2, static_cast<uint32_t>(E1) << 2};
    const uint32_t sub[2] = {dup16((static_cast<uint32_t>(E0) << 10) | static_cast<uint32_t>(c.off0)),
                             dup16((static_cast<uint32_t>(E1) << 10) | static_cast<uint32_t>(c.off1))};
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int b = i >> 3;
      out[2 * i] = hsub2u(__byte_perm(w[i], hi[b], 0x4140), sub[b]);
      out[2 * i + 1] = hsub2u(__byte_perm(w[i], hi[b], 0x4342), sub[b]);
    }
  } else {
    // general path: unscaled integers, then the block scale as two exact power-of-two factors
    uint32_t f1[2], f2[2];
    pow2_factors(e0, f1[0], f2[0]);
    pow2_factors(e1, f1[1], f2[1]);
    const uint32_t sub[2] = {dup16((25u << 10) | static_cast<uint32_t>(c.off0)),
                             dup16((25u << 10) | static_cast<uint32_t>(c.off1))};
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int b = i >> 3;
      out[2 * i] = hmul2u(hmul2u(hsub2u(__byte_perm(w[i], 0x64u, 0x4140), sub[b]), f1[b]), f2[b]);
      out[2 * i + 1] = hmul2u(hmul2u(hsub2u(__byte_perm(w[i], 0x64u, 0x4342), sub[b]), f1[b]), f2[b]);
    }
  }
}

// 4-bit codes -> 32 fp16 pairs.  Word i holds elements 8i..8i+7 with nibble j = element 2j and
// nibble 4+j = element 2j+1, so a mask of 0x000F000F << 4j isolates a pair.  The lanes of a warp
// hold channels of different formats: every warp vote is taken before the per-format branches.
CHAM_DEV uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));  // selector bit 3: sign replicate
  return d;
}

// Four NF4 level indices (nibbles of the low 16 bits of h, element order) -> two fp16 pairs, from
// byte tables in registers: PRMT picks the low and the high byte of each level among entries
// 0..7 and 8..15, and a per-byte mask built from each index's bit 3 chooses between the two.
CHAM_DEV void nf4_lookup4(uint32_t h, const uint32_t (&lo)[4], const uint32_t (&hi)[4], uint32_t& p01, uint32_t& p23) {
  const uint32_t sel = h & 0x7777u;
  const uint32_t m = prmt(h << 4, h, 0xD9C8u);  // byte k = 0xFF where index k >= 8
  const uint32_t l = (prmt(lo[0], lo[1], sel) & ~m) | (prmt(lo[2], lo[3], sel) & m);
  const uint32_t u = (prmt(hi[0], hi[1], sel) & ~m) | (prmt(hi[2], hi[3], sel) & m);
  p01 = prmt(l, u, 0x5140u);
  p23 = prmt(l, u, 0x7362u);
}

CHAM_DEV void decode_w4(const uint32_t (&w)[8], const ChanDecode& c, uint32_t e8, const uint32_t (&nlo)[4],
                        const uint32_t (&nhi)[4], uint32_t (&out)[32]) {
  const int e0 = block_exp(c, e8, 0), e1 = block_exp(c, e8, 1);
  const bool is_nf4 = c.f == CHAM_W_NF4;
  const bool is_fp4 = c.f == CHAM_W_E2M1 || c.f == CHAM_W_MXFP4;
  // E2M1 s.e1e0.m placed at fp16 bits 15 and 11..9 is value * 2^-14: multiply back by 2^(14 + e);
  // integer codes use the unscaled magic-number construction on the general path
  uint32_t f1[2], f2[2];
  pow2_factors(is_fp4 ? e0 + 14 : e0, f1[0], f2[0]);
  pow2_factors(is_fp4 ? e1 + 14 : e1, f1[1], f2[1]);
  // INT4-sym, INT4-asym, MXINT4 fast path: nibble at bit 0 of a half uses E = e + 25, nibble at
  // bit 4 uses E = e + 21, so both pairs of a byte need no shift; all-zero MX blocks decode to 0
  const bool z0 = c.mx && (e8 & 0xFFu) == 0, z1 = c.mx && ((e8 >> 8) & 0xFFu) == 0;
  const bool int_fast = (z0 || (e0 >= -20 && e0 <= 5)) && (z1 || (e1 >= -20 && e1 <= 5));
  const bool fp4_fast = f2[0] == 0x3C003C00u && f2[1] == 0x3C003C00u;
  const bool all_int_fast = __all_sync(0xffffffffu, is_nf4 || is_fp4 || int_fast);
  const bool all_fp4_fast = __all_sync(0xffffffffu, !is_fp4 || fp4_fast);
  if (is_nf4) {
    // NF4 codes are stored in element order (nibble j of word i = element 8i + j); levels from
    // the register tables (per-channel scale in the epilogue)
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      nf4_lookup4(w[i] & 0xFFFFu, nlo, nhi, out[4 * i], out[4 * i + 1]);
      nf4_lookup4(w[i] >> 16, nlo, nhi, out[4 * i + 2], out[4 * i + 3]);
    }
  } else if (is_fp4) {
    if (all_fp4_fast) {
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t x = w[i] >> (4 * j);
          out[4 * i + j] = hmul2u(((x & 0x00070007u) << 9) | ((x & 0x00080008u) << 12), f1[i >> 2]);
        }
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t x = w[i] >> (4 * j);
          out[4 * i + j] =
              hmul2u(hmul2u(((x & 0x00070007u) << 9) | ((x & 0x00080008u) << 12), f1[i >> 2]), f2[i >> 2]);
        }
    }
  } else if (all_int_fast) {
    const int c0 = min(max(e0, -20), 5), c1 = min(max(e1, -20), 5);
    const uint32_t m0[2] = {dup16(static_cast<uint32_t>(c0 + 25) << 10), dup16(static_cast<uint32_t>(c1 + 25) << 10)};
    const uint32_t m1[2] = {dup16(static_cast<uint32_t>(c0 + 21) << 10), dup16(static_cast<uint32_t>(c1 + 21) << 10)};
    const uint32_t o0 = static_cast<uint32_t>(c.off0), o1 = static_cast<uint32_t>(c.off1);
    const uint32_t s0[2] = {m0[0] | dup16(o0), m0[1] | dup16(o1)};
    const uint32_t s1[2] = {m1[0] | dup16(o0 << 4), m1[1] | dup16(o1 << 4)};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int b = i >> 2;
      const uint32_t v = w[i], t = w[i] >> 8;
      out[4 * i + 0] = hsub2u((v & 0x000F000Fu) | m0[b], s0[b]);
      out[4 * i + 1] = hsub2u((v & 0x00F000F0u) | m1[b], s1[b]);
      out[4 * i + 2] = hsub2u((t & 0x000F000Fu) | m0[b], s0[b]);
      out[4 * i + 3] = hsub2u((t & 0x00F000F0u) | m1[b], s1[b]);
    }
  } else {
    const uint32_t sub[2] = {dup16((25u << 10) | static_cast<uint32_t>(c.off0)),
                             dup16((25u << 10) | static_cast<uint32_t>(c.off1))};
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j)
        out[4 * i + j] = hmul2u(
            hmul2u(hsub2u(((w[i] >> (4 * j)) & 0x000F000Fu) | 0x64006400u, sub[i >> 2]), f1[i >> 2]), f2[i >> 2]);
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

// Epilogue role, shared by the fp16 and FP8 kernels: the warps first_warp .. first_warp + 4 * kEpiGrp - 1
// drain one accumulator buffer per tile (buffer b at column b * kAccCols); warpgroup h takes the
// 16-column slices j = h, h + kEpiGrp, ...
template <int BN, int EPI, int kEpiGrp, int kAccCols>
CHAM_DEV void epilogue_role(const GemmArgs& a, uint32_t tmem, uint64_t* accfull, uint64_t* accempty,
                            volatile int* abort_flag, int warp, int first_warp, int n_units, int ks, int n_ch) {
  const int lane = threadIdx.x & 31;
  const int q = warp & 3;
  const int h = (warp - first_warp) >> 2;
  const int r = q * 32 + lane;
  const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
  const float sa = a.act_scale != nullptr ? *a.act_scale : 1.f;
  uint32_t acc_it = 0;
  for (int u = blockIdx.x; u < n_units; u += gridDim.x, ++acc_it) {
    const int b = acc_it & 1;
    const int t = u / ks;
    // per-channel constants first: their (dependent) loads overlap the wait for the accumulator
    const int p = (a.tile0 + t % n_ch) * 128 + r;
    const int tok0 = (t / n_ch) * BN;
    const int orig = a.perm[p];
    const float ws = a.wscale[p];
    const float scale = __fmul_rn(sa, ws);
    const float bv = (a.bias != nullptr && orig >= 0) ? a.bias[orig] : 0.f;
    if (!warp_wait(&accfull[b], (acc_it >> 1) & 1, abort_flag, a.dev_status)) break;
    tc_fence_after();
    const uint32_t d_tmem = tmem + b * kAccCols + lane_off;
    // y = acc * (s_a * s_w) + bias, rounded once to fp32, then (f16 / bf16 outputs) to the output
    // type; one instantiation per output type and scale granularity keeps each variant as lean
    // as the fp32 per-tensor one
    // YT = kPartialOut (EPI = 6, split-K): the raw fp32 sums go to a.partial[u % ks][tok][p]
    // and the reduction kernel applies scales, bias and the output type
    auto drain = [&](auto yt, auto grouped_tag) {
      constexpr int YT = decltype(yt)::value;
      constexpr bool GROUPED = decltype(grouped_tag)::value;
      using OutT = std::conditional_t<YT == CHAM_Y_F32 || YT == kPartialOut, float,
                                      std::conditional_t<YT == CHAM_Y_F16, __half, __nv_bfloat16>>;
      OutT* yc = static_cast<OutT*>(a.Y) + (orig >= 0 ? orig : 0);
      float* pc = a.partial + static_cast<size_t>(u % ks) * a.M * a.Np + p;
      // 16 token columns per tcgen05.ld; the load of the warp's next slice is in flight while
      // the current one is scaled and stored (a wait per load would serialise its latency)
      auto store16 = [&](const uint32_t (&v)[16], int j) {
        if (orig < 0) return;
        const int t0 = tok0 + j * 16;
        if constexpr (YT == kPartialOut) {
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int tok = t0 + i;
            if (tok >= a.M) break;
            pc[static_cast<size_t>(tok) * a.Np] = __uint_as_float(v[i]);
          }
          return;
        }
        if (t0 + 16 <= a.M) {
          // a full slice inside one row group (always, for a per-tensor scale): no bounds or
          // group checks, one running pointer
          float s16 = scale;
          bool one = true;
          if constexpr (GROUPED) {
            const int g0 = t0 / a.rows_per_group;
            one = (t0 + 15) / a.rows_per_group == g0;
            if (one) s16 = __fmul_rn(a.act_scale[g0], ws);
          }
          if (one) {
            OutT* yp = yc + static_cast<size_t>(t0) * a.N;
            const size_t stride = static_cast<size_t>(a.N);
#pragma unroll
            for (int i = 0; i < 16; ++i, yp += stride) {
              const float y = fmaf(__uint_as_float(v[i]), s16, bv);
              if constexpr (YT == CHAM_Y_F32) *yp = y;
              else if constexpr (YT == CHAM_Y_F16) *yp = __float2half_rn(y);
              else *yp = __float2bfloat16_rn(y);
            }
            return;
          }
        }
        float sc = scale;
        int grp = 0, next = 0;
        if constexpr (GROUPED) {  // per-sample scales: the group advances at most a few times
          grp = t0 / a.rows_per_group;
          next = (grp + 1) * a.rows_per_group;
          sc = __fmul_rn(a.act_scale[grp], ws);
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int tok = t0 + i;
          if (tok >= a.M) break;
          if constexpr (GROUPED) {
            if (tok >= next) {
              ++grp;
              next += a.rows_per_group;
              sc = __fmul_rn(a.act_scale[grp], ws);
            }
          }
          const float y = fmaf(__uint_as_float(v[i]), sc, bv);
          if constexpr (YT == CHAM_Y_F32) yc[static_cast<size_t>(tok) * a.N] = y;
          else if constexpr (YT == CHAM_Y_F16) yc[static_cast<size_t>(tok) * a.N] = __float2half_rn(y);
          else yc[static_cast<size_t>(tok) * a.N] = __float2bfloat16_rn(y);
        }
      };
      constexpr int kLoads = BN / 16, kE = kEpiGrp;
      uint32_t va[16], vb[16];
      if (h < kLoads) {
        tmem_ld_32x32b_x16(d_tmem + h * 16, va);
        tmem_wait_ld();
      }
#pragma unroll 1
      for (int j = h; j < kLoads; j += 2 * kE) {
        if (j + kE < kLoads) tmem_ld_32x32b_x16(d_tmem + (j + kE) * 16, vb);
        store16(va, j);
        tmem_wait_ld();
        if (j + 2 * kE < kLoads) tmem_ld_32x32b_x16(d_tmem + (j + 2 * kE) * 16, va);
        if (j + kE < kLoads) store16(vb, j + kE);
        tmem_wait_ld();
      }
    };
    drain(std::integral_constant<int, EPI / 2>{}, std::bool_constant<(EPI % 2) == 1>{});
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&accempty[b]);
  }
}

// EPI = 2 * output type (CHAM_Y_*) + per-sample scales: one epilogue variant per instantiation
// (several inlined into one kernel raise its register count past what the split allows); GW =
// group-wise weights (per-block fp16 scales and zero points staged with every chunk)
template <int BN, int BITS, int EPI, bool GW>
__global__ void __launch_bounds__(kGemmThreads, 1)
    k_gemm_ts_f16(const __grid_constant__ CUtensorMap act_map, const GemmArgs a) {
  using C = GemmCfg<BN, BITS>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint32_t* misc = reinterpret_cast<uint32_t*>(smem + C::kData);
  constexpr int S = C::kStages;
  constexpr int kAStages = C::kAStages, kGroup = C::kGroup, kAGroups = kAStages / kGroup;
  constexpr int kDone = C::kDone;
  uint64_t* full = reinterpret_cast<uint64_t*>(misc);       // [S] producer -> decoders, MMA (tx bytes)
  uint64_t* done = full + S;                                 // [kDone] MMA group commit -> producer, decoders
  uint64_t* afull = done + kDone;                            // [kAGroups] decode warps -> MMA
  uint64_t* accfull = afull + kAGroups;                      // [2] MMA commit -> epilogue
  uint64_t* accempty = accfull + 2;                          // [2] epilogue warps (8) -> MMA
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nk = a.n_chunks;
  constexpr bool grouped = GW;  // group-wise blob: per-block fp16 scales
  const int n_ch = a.n_ch_tiles;
  const int n_tiles = n_ch * ((a.M + BN - 1) / BN);
  // Work units: tile t = u / ks over its K-chunk range j = u % ks (ks = 1: whole tiles).  Units
  // u = blockIdx.x, blockIdx.x + gridDim.x, ... belong to this CTA.
  const int ks = a.k_split;
  const int n_units = n_tiles * ks;
  auto kc_begin = [&](int u) { return ks == 1 ? 0 : (u % ks) * nk / ks; };
  auto kc_end = [&](int u) { return ks == 1 ? nk : (u % ks + 1) * nk / ks; };
  // K-chunks this CTA processes; the last commit group may be partial
  uint32_t total = 0;
  for (int u = blockIdx.x; u < n_units; u += gridDim.x) total += static_cast<uint32_t>(kc_end(u) - kc_begin(u));
  // wait until the MMAs of chunk j have completed (the commit of its group)
  auto wait_done = [&](uint32_t j) {
    const uint32_t g = j / kGroup;
    return mbar_wait(&done[g % kDone], (g / kDone) & 1, abort_flag, a.dev_status);
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) mbar_init(&full[s], 1);
    for (int g = 0; g < kDone; ++g) mbar_init(&done[g], 1);
    for (int g = 0; g < kAGroups; ++g) mbar_init(&afull[g], 4 * kGroup);  // one elected lane per warp and chunk
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accfull[b], 1);
      mbar_init(&accempty[b], 4 * Roles<BITS>::kEpi);  // one elected lane per epilogue warp
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) tma_prefetch_desc(&act_map);
  if (warp == 2) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // the set-up above overlaps the previous kernel's tail; everything below may read its results
  griddep_wait();
  griddep_launch_dependents();

  if (warp == 0) {
    // ---------------- producer: activation tile (TMA), raw weight codes and E8M0 bytes (bulk)
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        const int t = u / ks;
        const int ch = a.tile0 + t % n_ch, tok0 = (t / n_ch) * BN;
        const int kc1 = kc_end(u);
        for (int kc = kc_begin(u); kc < kc1; ++kc, ++it) {
          const int s = it % S;
          if (it >= static_cast<uint32_t>(S) && !wait_done(it - S)) {  // the stage's previous chunk is consumed
            ok = false;
            break;
          }
          uint8_t* st = smem + s * C::kStage;
          const size_t chunk = static_cast<size_t>(ch) * nk + kc;
          mbar_arrive_expect_tx(&full[s], C::kBBytes + C::kWBytes + C::kEBytes + (grouped ? C::kGBytes : 0));
          // test hook: the stage's transaction bytes never arrive, so every wait on it runs out
          if (blockIdx.x == 0 && static_cast<int>(it) == a.stall_chunk) continue;
          tma_load_2d(smem_u32(st), &act_map, &full[s], kc * kBK, tok0);
          bulk_load(smem_u32(st + C::kBBytes), a.codes + chunk * C::kWBytes, C::kWBytes, &full[s]);
          bulk_load(smem_u32(st + C::kBBytes + C::kWBytes), a.we8m0 + chunk * C::kEBytes, C::kEBytes, &full[s]);
          if constexpr (grouped)
            bulk_load(smem_u32(st + C::kBBytes + C::kWBytes + C::kEBytes), a.wgscale + chunk * 128, C::kGBytes,
                      &full[s]);
        }
      }
      // every issued copy must have landed before the CTA may exit
      const uint32_t first = it > S ? it - S : 0;
      for (uint32_t j = first; j < it; ++j) drain_wait(&full[j % S], (j / S) & 1);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f16(128, BN);
      // operand addresses advance incrementally: the activation stage's descriptor (start address
      // in 16-byte units in the low bits) and the decoded-weight stage's tensor-memory column
      const uint64_t desc0 = smem_desc_sw128(smem_u32(smem));
      constexpr uint32_t kStageDesc = C::kStage >> 4;
      uint32_t it = 0, acc_it = 0, s = 0, sa = 0, gi = 0;  // s = it % S, sa = it % kAStages, gi = it % kGroup
      bool ok = true;
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x, ++acc_it) {
        const int b = acc_it & 1;
        const int kc0 = kc_begin(u), kc1 = kc_end(u);
        if (!mbar_wait(&accempty[b], ((acc_it >> 1) & 1) ^ 1, abort_flag, a.dev_status)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem + b * C::kAccCols;
        // One wait per group of kGroup consecutive K-chunks, on the decoded-operand barrier only:
        // the decoders arrive on it after they have themselves observed the stage's TMA barrier,
        // so the activation tile has landed too.  A group may straddle two tiles.
        for (int kc = kc0; kc < kc1; ++kc, ++it) {
          if (gi == 0) {
            if (!mbar_wait(&afull[(it / kGroup) % kAGroups], (it / kAStages) & 1, abort_flag, a.dev_status)) {
              ok = false;
              break;
            }
            tc_fence_after();
          }
          const uint64_t bd = desc0 + s * kStageDesc;
          const uint32_t ad = tmem + C::kACol + sa * 32;
          mma_f16_ts(d_tmem, ad, bd, idesc, kc != kc0);
          mma_f16_ts(d_tmem, ad + 8, bd + 2, idesc, 1u);
          mma_f16_ts(d_tmem, ad + 16, bd + 4, idesc, 1u);
          mma_f16_ts(d_tmem, ad + 24, bd + 6, idesc, 1u);
          if (++gi == kGroup || it + 1 == total) {
            mma_commit(&done[(it / kGroup) % kDone]);
            gi = gi == kGroup ? 0 : gi;
          }
          s = s + 1 == static_cast<uint32_t>(S) ? 0 : s + 1;
          sa = sa + 1 == static_cast<uint32_t>(kAStages) ? 0 : sa + 1;
        }
        mma_commit(&accfull[b]);  // after an abort inside the tile this still covers every MMA issued
      }
      // all issued MMAs have finished before tensor memory is released
      if (acc_it > 0) drain_wait(&accfull[(acc_it - 1) & 1], ((acc_it - 1) >> 1) & 1);
    }
  } else if (warp >= 4 && warp < 4 + 4 * Roles<BITS>::kDec) {
    // ---------------- weight decode: one channel per thread; group g takes chunks it % G == g
    const int q = warp & 3;  // tensor-memory lane quadrant of this warp (warp % 4)
    const int grp = (warp - 4) >> 2;
    const int r = q * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    uint32_t it = 0;
    bool ok = true;
    // the last chunk of this CTA also arrives for the missing chunks of its group
    // the channel's format and zero point for the next tile are loaded one tile ahead
    int nf = 0, nz = 0;
    if (static_cast<int>(blockIdx.x) < n_units) {
      const int p0 = (a.tile0 + (static_cast<int>(blockIdx.x) / ks) % n_ch) * 128 + r;
      nf = a.wfmt[p0];
      nz = a.wzero[p0];
    }
    for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
      const ChanDecode cd = chan_decode(nf, nz);
      if (u + static_cast<int>(gridDim.x) < n_units) {
        const int pn = (a.tile0 + ((u + static_cast<int>(gridDim.x)) / ks) % n_ch) * 128 + r;
        nf = a.wfmt[pn];
        nz = a.wzero[pn];
      }
      const int kc1 = kc_end(u);
      for (int kc = kc_begin(u); kc < kc1; ++kc, ++it) {
        if (static_cast<int>(it % Roles<BITS>::kDec) != grp) continue;
        const int s = it % S, sa = it % kAStages;
        const uint32_t ph = (it / S) & 1;
        // decode as soon as the codes have landed; the tensor-memory slot (its previous chunk,
        // it - kAStages, must be consumed by the MMAs) is waited for only before the store, so
        // the decode stays off the MMA-completion -> store -> MMA-issue loop
        // when S is not a multiple of the decode groups, the stage's previous chunk (it - S) is
        // another group's, and testing this chunk's parity while that chunk's phase is still open
        // would pass on the opposite parity.  That chunk's commit closes its phase (its MMAs
        // follow its decode) and costs no extra wait: the producer waits for the same commit
        // before it loads this chunk
        if constexpr (S % Roles<BITS>::kDec != 0) {
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
        const uint32_t e8 = reinterpret_cast<const uint16_t*>(st + C::kBBytes + C::kWBytes)[r];
        ChanDecode cdk = cd;
        uint32_t gs = 0;
        if constexpr (grouped) {  // group-wise blob: the E8M0 slot holds the blocks' zero points (asym)
          gs = reinterpret_cast<const uint32_t*>(st + C::kBBytes + C::kWBytes + C::kEBytes)[r];
          if (cd.f == CHAM_W_INT8_ASYM || cd.f == CHAM_W_INT4_ASYM) {
            cdk.off0 = static_cast<int>(e8 & 0xFFu);
            cdk.off1 = static_cast<int>((e8 >> 8) & 0xFFu);
          }
        }
        uint32_t raw[16];
#pragma unroll
        for (int j = 0; j < BITS / 2; ++j) {  // slab j: bytes [16j, 16j+16) of every channel
          const uint4 u = *reinterpret_cast<const uint4*>(st + C::kBBytes + j * 2048 + r * 16);
          raw[4 * j] = u.x;
          raw[4 * j + 1] = u.y;
          raw[4 * j + 2] = u.z;
          raw[4 * j + 3] = u.w;
        }
        uint32_t out[32];
        if constexpr (BITS == 8) {
          decode_w8(raw, cdk, e8, out);
        } else {
          const uint32_t (&r8)[8] = *reinterpret_cast<const uint32_t(*)[8]>(&raw[0]);
          decode_w4(r8, cdk, e8, a.nf4_lo, a.nf4_hi, out);
        }
        if constexpr (grouped) {  // each block's group scale: one fp16 product, rounded once
          const uint32_t g0 = dup16(gs & 0xFFFFu), g1 = dup16(gs >> 16);
#pragma unroll
          for (int i = 0; i < 32; ++i) out[i] = hmul2u(out[i], i < 16 ? g0 : g1);
        }
        const bool free_ok = it < static_cast<uint32_t>(kAStages) || wait_done(it - kAStages);
        if (!__all_sync(0xffffffffu, free_ok)) {
          ok = false;
          break;
        }
        __syncwarp();  // the per-format decode branches reconverge before the warp-wide store
        tc_fence_after();
        tmem_st_32x32b_x32(tmem + C::kACol + lane_off + sa * 32, out);
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();  // 128 separate arrivals on one barrier word serialise: one per warp
        if (lane == 0) {
          const int missing = it + 1 == total ? kGroup - 1 - static_cast<int>(it % kGroup) : 0;
          for (int m = 0; m <= missing; ++m) mbar_arrive(&afull[(it / kGroup) % kAGroups]);
        }
      }
    }
  } else if (warp >= 4 + 4 * Roles<BITS>::kDec) {
    epilogue_role<BN, EPI, Roles<BITS>::kEpi, C::kAccCols>(a, tmem, accfull, accempty, abort_flag, warp,
                                                          4 + 4 * Roles<BITS>::kDec, n_units, ks, n_ch);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

template <int BN, int BITS, int EPI, bool GW>
static cudaError_t launch_bn(const CUtensorMap& map, const GemmArgs& a, int num_sms, cudaStream_t st) {
  using C = GemmCfg<BN, BITS>;
  static int configured_device = -1;  // the attribute is per device; set again when it changes
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured_device != dev) {
    const cudaError_t e =
        cudaFuncSetAttribute(k_gemm_ts_f16<BN, BITS, EPI, GW>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
    if (e != cudaSuccess) return e;
    configured_device = dev;
  }
  const long units = static_cast<long>(a.n_ch_tiles) * ((a.M + BN - 1) / BN) * a.k_split;
  const int grid = static_cast<int>(units < num_sms ? units : num_sms);
  return launch_pdl(k_gemm_ts_f16<BN, BITS, EPI, GW>, dim3(grid), dim3(kGemmThreads), C::kSmem, st, map, a);
}

template <int BITS, int EPI, bool GW>
static cudaError_t launch_bits(const CUtensorMap& map, const GemmArgs& a, int num_sms, int bn, cudaStream_t st) {
  switch (bn) {
    case 16: return launch_bn<16, BITS, EPI, GW>(map, a, num_sms, st);
    case 32: return launch_bn<32, BITS, EPI, GW>(map, a, num_sms, st);
    case 64: return launch_bn<64, BITS, EPI, GW>(map, a, num_sms, st);
    case 128: return launch_bn<128, BITS, EPI, GW>(map, a, num_sms, st);
    default: return launch_bn<192, BITS, EPI, GW>(map, a, num_sms, st);
  }
}

template <int BITS, int EPI>
static cudaError_t launch_gw(const CUtensorMap& map, const GemmArgs& a, int num_sms, int bn, cudaStream_t st) {
  return a.wgscale != nullptr ? launch_bits<BITS, EPI, true>(map, a, num_sms, bn, st)
                              : launch_bits<BITS, EPI, false>(map, a, num_sms, bn, st);
}

// The launches of one output type YT: both weight widths, every token-tile size, per-tensor or
// per-sample activation scales, per-channel or group-wise weights.

template <int YT>
cudaError_t launch_gemm_yt(const CUtensorMap& map, const GemmArgs& a, int num_sms, int bn, cudaStream_t st) {
  const bool per_sample = a.act_scale != nullptr && a.rows_per_group < a.M;
  if (a.bits == 8)
    return per_sample ? launch_gw<8, 2 * YT + 1>(map, a, num_sms, bn, st) : launch_gw<8, 2 * YT>(map, a, num_sms, bn, st);
  return per_sample ? launch_gw<4, 2 * YT + 1>(map, a, num_sms, bn, st) : launch_gw<4, 2 * YT>(map, a, num_sms, bn, st);
}

}  // namespace cham
