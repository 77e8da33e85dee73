// act_quant.cu -- activation quantizer kernels (steps a2-a4) and calibration power sums.
//
// The dynamic path of Alg. 3: lo, hi = min x, max x over the tensor; ScaleZP (App. A.7); every
// element encoded in the format the LUT picked.  Per-tensor formats need the range before any
// element can be encoded, so they take two launches: range partials, then encode (the second
// read of X mostly hits L2).  A single cooperative launch that stages X in shared memory across
// a grid barrier was measured slower: the barrier costs as much as the load.
// MX formats (32-element blocks along K, E8M0 exponent, Sec. 3.6 / App. A.11) need only the
// block's own amax and run in one launch, four lanes per block.  Every kernel keeps several
// 16-byte loads in flight per thread (HBM latency x bandwidth needs ~7 MB in flight).
//
// All scale arithmetic is IEEE fp32 with explicit round-to-nearest intrinsics (no contraction),
// in the order of readings R4-R8: inv by one correctly rounded division, the product x * inv
// rounded to fp32, then the format rounding.  The same arithmetic gives the codes (public
// chameleon_act_quant) and the exact fp16 operand values the GEMM consumes (R13).
#include <cooperative_groups.h>

#include "act_quant.cuh"

namespace cham {

constexpr int kUnroll = 4;       // independent 16-byte loads in flight per thread (encoders)
constexpr int kRangeUnroll = 8;  // the range pass: a grid of range_grid CTAs reads the tensor in one round

// Running min / max of eight fp16 values packed in a uint4.  The NaN-propagating forms keep a NaN
// lane in both results, and an infinity lands in one of them, so the non-finite test runs once
// on the results (nonfinite_h2) instead of once per element.
CHAM_DEV void range8(const uint4& v, __half2& lo2, __half2& hi2) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const __half2 h = u32_as_h2(w[j]);
    lo2 = __hmin2_nan(lo2, h);
    hi2 = __hmax2_nan(hi2, h);
  }
}

// 1 when either half is Inf or NaN (exponent field all ones).
CHAM_DEV uint32_t nonfinite_h2(__half2 h) {
  const uint32_t w = h2_as_u32(h);
  return ((w & 0x7C00u) == 0x7C00u) | ((w & 0x7C000000u) == 0x7C000000u);
}

// CTA-wide reduction of (lo, hi, nonfinite); the result is valid in every thread.
CHAM_DEV void block_range(float& lo, float& hi, uint32_t& nf) {
  __shared__ float s_lo[32], s_hi[32];
  __shared__ uint32_t s_nf[32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    nf |= __shfl_xor_sync(0xffffffffu, nf, o);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) {
    s_lo[warp] = lo;
    s_hi[warp] = hi;
    s_nf[warp] = nf;
  }
  __syncthreads();
  lo = s_lo[0];
  hi = s_hi[0];
  nf = s_nf[0];
  for (int k = 1; k < static_cast<int>(blockDim.x >> 5); ++k) {
    lo = fminf(lo, s_lo[k]);
    hi = fmaxf(hi, s_hi[k]);
    nf |= s_nf[k];
  }
}

// ScaleZP (App. A.7) of a per-tensor format from the tensor's range (readings R4-R8, R11).
CHAM_DEV TensorParams scale_zp(int fmt, float lo, float hi) {
  TensorParams p;
  if (fmt == CHAM_A_INT8_ASYM) {
    // s = (hi - lo)/255, z = round(-lo/s), zero-inclusive range (R4), degenerate range (R7)
    const float lo_ = fminf(lo, 0.f), hi_ = fmaxf(hi, 0.f);
    const float d = __fsub_rn(hi_, lo_);
    if (d == 0.f) {
      p.s = 1.f;
      p.inv = 1.f;
      p.z = 0;
    } else {
      p.s = __fdiv_rn(d, 255.f);
      p.inv = __fdiv_rn(255.f, d);
      p.z = min(max(__float2int_rn(__fmul_rn(-lo_, p.inv)), 0), 255);
    }
  } else {
    // FP8: s = amax / Fmax, inv = Fmax / amax
    const float fmax = (fmt == CHAM_A_E4M3) ? 448.f : 57344.f;
    const float amax = fmaxf(fabsf(lo), fabsf(hi));
    if (amax == 0.f) {
      p.s = 1.f;
      p.inv = 1.f;
    } else {
      p.s = __fdiv_rn(amax, fmax);
      p.inv = __fdiv_rn(fmax, amax);
    }
    p.z = 0;
  }
  return p;
}

// Reduce `nparts` range partials (identically in every CTA: min/max are exact and order-free).
CHAM_DEV void reduce_partials(const RangePartial* parts, int nparts, float& lo, float& hi, uint32_t& nf) {
  lo = INFINITY;
  hi = -INFINITY;
  nf = 0;
  for (int i = threadIdx.x; i < nparts; i += blockDim.x) {
    const RangePartial p = parts[i];
    lo = fminf(lo, p.lo);
    hi = fmaxf(hi, p.hi);
    nf |= static_cast<uint32_t>(p.nonfinite);
  }
  block_range(lo, hi, nf);
}

// Eight elements of a per-tensor format: code bytes (element 0 in the low byte) and the exact
// fp16 operand values (q - z for INT8-asym, value(code) for FP8; the scale s stays outside).
template <int FMT, bool DEQ>
CHAM_DEV void encode8_tensor(const uint4& v, const TensorParams& p, uint2& code, uint4& deq) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  uint32_t c[2] = {0, 0};
  uint32_t d[4] = {0, 0, 0, 0};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 f = __half22float2(u32_as_h2(w[j]));
    const float a = __fmul_rn(f.x, p.inv), b = __fmul_rn(f.y, p.inv);
    uint32_t pair;
    if constexpr (FMT == CHAM_A_INT8_ASYM) {
      const int qa = min(max(__float2int_rn(a) + p.z, 0), 255);
      const int qb = min(max(__float2int_rn(b) + p.z, 0), 255);
      pair = static_cast<uint32_t>(qa) | (static_cast<uint32_t>(qb) << 8);
      if constexpr (DEQ) d[j] = h2_as_u32(__halves2half2(__int2half_rn(qa - p.z), __int2half_rn(qb - p.z)));
    } else if constexpr (FMT == CHAM_A_E4M3) {
      const uint16_t e = cvt_e4m3x2(b, a);
      pair = e;
      if constexpr (DEQ) d[j] = cvt_e4m3x2_to_f16x2(e);
    } else {
      const uint16_t e = cvt_e5m2x2(b, a);
      pair = e;
      if constexpr (DEQ) d[j] = cvt_e5m2x2_to_f16x2(e);
    }
    c[j >> 1] |= pair << (16 * (j & 1));
  }
  code = make_uint2(c[0], c[1]);
  deq = make_uint4(d[0], d[1], d[2], d[3]);
}

// Eight code bytes (element 0 in the low byte) -> the group order 0, 2, 4, 6, 1, 3, 5, 7.
CHAM_DEV uint2 kperm8(const uint2& c) {
  uint32_t lo, hi;
  asm("prmt.b32 %0, %1, %2, 0x6420;" : "=r"(lo) : "r"(c.x), "r"(c.y));
  asm("prmt.b32 %0, %1, %2, 0x7531;" : "=r"(hi) : "r"(c.x), "r"(c.y));
  return make_uint2(lo, hi);
}

// ------------------------------------------------------------------ L2 eviction priority
// The dynamic path reads X twice (range, then encode).  The range pass marks the lines it loads
// as the last to evict, so that a tensor smaller than the L2 is still there for the encode pass;
// the encode pass, their last use, marks them as the first.
CHAM_DEV uint64_t l2_policy_keep() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
CHAM_DEV uint64_t l2_policy_drop() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
CHAM_DEV uint4 ldg_hint(const uint4* p, uint64_t pol) {
  uint4 v;
  asm volatile("ld.global.nc.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p), "l"(pol));
  return v;
}

// ------------------------------------------------------------------ a2: range partials
// Group blockIdx.y (rows split into gridDim.y equal groups, nvec vectors each; one group for a
// per-tensor range) writes its gridDim.x partials at parts[blockIdx.y * gridDim.x ...].
__global__ void __launch_bounds__(256) k_act_range(const uint4* __restrict__ X, int64_t nvec,
                                                  RangePartial* __restrict__ parts) {
  // X may be the previous kernel's output (a linear's fp16 Y fed to the next linear), and that
  // kernel lets its dependents start early: wait for it before the first read
  griddep_wait();
  griddep_launch_dependents();
  X += static_cast<int64_t>(blockIdx.y) * nvec;
  parts += static_cast<int64_t>(blockIdx.y) * gridDim.x;
  __half2 lo2 = __float2half2_rn(65504.f), hi2 = __float2half2_rn(-65504.f);
  const uint64_t keep = l2_policy_keep();
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i0 < nvec;
       i0 += stride * kRangeUnroll) {
    uint4 v[kRangeUnroll];
#pragma unroll
    for (int u = 0; u < kRangeUnroll; ++u) {
      const int64_t i = i0 + u * stride;
      v[u] = i < nvec ? ldg_hint(X + i, keep) : make_uint4(0x3C003C00u, 0x3C003C00u, 0x3C003C00u, 0x3C003C00u);
    }
#pragma unroll
    for (int u = 0; u < kRangeUnroll; ++u)
      if (i0 + u * stride < nvec) range8(v[u], lo2, hi2);
  }
  uint32_t nonfinite = nonfinite_h2(lo2) | nonfinite_h2(hi2);
  float lo = fminf(__low2float(lo2), __high2float(lo2));
  float hi = fmaxf(__low2float(hi2), __high2float(hi2));
  block_range(lo, hi, nonfinite);
  if (threadIdx.x == 0) parts[blockIdx.x] = RangePartial{lo, hi, static_cast<int>(nonfinite), 0};
}

// ------------------------------------------------------------------ a3: per-tensor encode
// Non-finite fp16 lanes of one 16-byte vector (exponent field all ones), as a 0/1 flag.
CHAM_DEV uint32_t nonfinite8(const uint4& v) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  uint32_t nf = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) nf |= ((w[j] & 0x7C00u) == 0x7C00u) | ((w[j] & 0x7C000000u) == 0x7C000000u);
  return nf;
}

// Grid-stride encode of the whole tensor with parameters p; CHECK also returns whether any input
// lane was non-finite (the static path has no range pass to find out).
// CHECK is the static path (one pass); otherwise X's lines are read for the last time here.
template <int FMT, bool CODES, bool DEQ, bool CHECK>
CHAM_DEV uint32_t encode_tensor_body(const uint4* __restrict__ X, int64_t nvec, const TensorParams& p,
                                     uint2* __restrict__ codes, uint4* __restrict__ deq, bool kperm) {
  uint32_t nf = 0;
  const uint64_t drop = l2_policy_drop();
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i0 < nvec; i0 += stride * kUnroll) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t i = i0 + u * stride;
      if constexpr (CHECK) v[u] = i < nvec ? __ldg(X + i) : make_uint4(0, 0, 0, 0);
      else v[u] = i < nvec ? ldg_hint(X + i, drop) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t i = i0 + u * stride;
      if (i < nvec) {
        if constexpr (CHECK) nf |= nonfinite8(v[u]);
        uint2 c;
        uint4 d;
        encode8_tensor<FMT, DEQ>(v[u], p, c, d);
        if constexpr (CODES) codes[i] = kperm ? kperm8(c) : c;
        if constexpr (DEQ) deq[i] = d;
      }
    }
  }
  return nf;
}

// Dynamic path (Alg. 3): ScaleZP of the tensor's own range, reduced from the range partials.
// Per-sample scales: group blockIdx.y (nvec vectors) uses the range of its own nparts partials
// and stores its scale at scale_out[blockIdx.y] (params, of the public call, has one slot).
template <int FMT, bool CODES, bool DEQ>
__global__ void __launch_bounds__(256)
    k_act_encode_tensor(const uint4* __restrict__ X, int64_t nvec, const RangePartial* __restrict__ parts,
                        int nparts, uint2* __restrict__ codes, uint4* __restrict__ deq,
                        cham_qparams* __restrict__ params, float* __restrict__ scale_out, int* dev_status, bool kperm) {
  griddep_wait();  // the range partials
  griddep_launch_dependents();
  const int64_t g = blockIdx.y;
  float lo, hi;
  uint32_t nf;
  reduce_partials(parts + g * nparts, nparts, lo, hi, nf);
  const TensorParams p = scale_zp(FMT, lo, hi);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    if (params != nullptr && g == 0) *params = cham_qparams{p.s, p.z, p.inv, FMT};
    if (scale_out != nullptr) scale_out[g] = p.s;
    if (nf) set_status(dev_status, CHAM_ERR_NONFINITE);
  }
  encode_tensor_body<FMT, CODES, DEQ, false>(X + g * nvec, nvec, p, codes == nullptr ? nullptr : codes + g * nvec,
                                             deq == nullptr ? nullptr : deq + g * nvec, kperm);
}

// Dynamic path (Alg. 3) in one launch, for a tensor whose vectors fit in the registers of one
// co-resident grid (a cooperative launch): every thread loads its kCoopVec vectors once, each CTA
// writes its range partial, the grid meets at one barrier, every CTA reduces its group's
// partials to the same ScaleZP and encodes the vectors it still holds.  X is read from DRAM once
// and one launch replaces the range and encode launches.  Same grid shape as the range pass
// (gridDim.x CTAs per group, 256 x kCoopVec vectors each), same results as the two-launch path.
constexpr int kCoopVec = kRangeUnroll;
template <int FMT, bool CODES, bool DEQ>
__global__ void __launch_bounds__(256, 4)
    k_act_quant_coop(const uint4* __restrict__ X, int64_t nvec, RangePartial* __restrict__ parts,
                     uint2* __restrict__ codes, uint4* __restrict__ deq, cham_qparams* __restrict__ params,
                     float* __restrict__ scale_out, int* dev_status, bool kperm) {
  griddep_wait();  // X may be the previous kernel's output
  const int64_t g = blockIdx.y;
  const int P = gridDim.x;
  X += g * nvec;
  const int64_t i0 = static_cast<int64_t>(blockIdx.x) * (256 * kCoopVec) + threadIdx.x;
  uint4 v[kCoopVec];
  __half2 lo2 = __float2half2_rn(65504.f), hi2 = __float2half2_rn(-65504.f);
#pragma unroll
  for (int u = 0; u < kCoopVec; ++u) {
    const int64_t i = i0 + u * 256;
    v[u] = i < nvec ? __ldg(X + i) : make_uint4(0, 0, 0, 0);
  }
#pragma unroll
  for (int u = 0; u < kCoopVec; ++u)
    if (i0 + u * 256 < nvec) range8(v[u], lo2, hi2);
  uint32_t nf = nonfinite_h2(lo2) | nonfinite_h2(hi2);
  float lo = fminf(__low2float(lo2), __high2float(lo2));
  float hi = fmaxf(__low2float(hi2), __high2float(hi2));
  block_range(lo, hi, nf);
  if (threadIdx.x == 0) {
    parts[g * P + blockIdx.x] = RangePartial{lo, hi, static_cast<int>(nf), 0};
    __threadfence();
  }
  cooperative_groups::this_grid().sync();
  griddep_launch_dependents();
  reduce_partials(parts + g * P, P, lo, hi, nf);
  const TensorParams p = scale_zp(FMT, lo, hi);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    if (params != nullptr && g == 0) *params = cham_qparams{p.s, p.z, p.inv, FMT};
    if (scale_out != nullptr) scale_out[g] = p.s;
    if (nf) set_status(dev_status, CHAM_ERR_NONFINITE);
  }
#pragma unroll
  for (int u = 0; u < kCoopVec; ++u) {
    const int64_t i = i0 + u * 256;
    if (i < nvec) {
      uint2 c;
      uint4 d;
      encode8_tensor<FMT, DEQ>(v[u], p, c, d);
      if constexpr (CODES) codes[g * nvec + i] = kperm ? kperm8(c) : c;
      if constexpr (DEQ) deq[g * nvec + i] = d;
    }
  }
}

// Static path (Alg. 2): (s, z) fixed beforehand -- ScaleZP of the calibration range that Alg. 1
// stored for this layer and bucket -- so one pass encodes; values outside that range clamp to the
// extreme codes (INT8) or saturate (FP8).  Non-finite inputs are flagged on the fly.
template <int FMT, bool CODES, bool DEQ>
__global__ void __launch_bounds__(256)
    k_act_encode_static(const uint4* __restrict__ X, int64_t nvec, TensorParams p, uint2* __restrict__ codes,
                        uint4* __restrict__ deq, cham_qparams* __restrict__ params, float* __restrict__ scale_out,
                        int* dev_status, bool kperm) {
  griddep_wait();  // X may be the previous kernel's output; the outputs may still be read by it
  griddep_launch_dependents();
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    if (params != nullptr) *params = cham_qparams{p.s, p.z, p.inv, FMT};
    if (scale_out != nullptr) *scale_out = p.s;
  }
  const uint32_t nf = encode_tensor_body<FMT, CODES, DEQ, true>(X, nvec, p, codes, deq, kperm);
  if (__any_sync(0xffffffffu, nf != 0) && (threadIdx.x & 31) == 0) set_status(dev_status, CHAM_ERR_NONFINITE);
}

// ------------------------------------------------------------------ a4: MX encode
// Four consecutive lanes own one 32-element block (8 elements each).  Shared exponent
// X = floor(log2 amax) - emax_elem (R1; 8 for the E4M3 body, 0 for the int8 body), element
// v = x * 2^-X (exact), body code; all-zero block -> E8M0 byte 0 (R2).
template <int FMT, bool DEQ>
CHAM_DEV void encode8_mx(const uint4& v, int lane, uint2& code, uint4& deq, int& byte_out, uint32_t& nonfinite) {
  constexpr int kOff = (FMT == CHAM_A_MXFP8) ? 8 : 0;
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  float f[8];
  float amax = 0.f;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    nonfinite |= (((w[j] & 0x7C00u) == 0x7C00u) | ((w[j] & 0x7C000000u) == 0x7C000000u));
    const float2 t = __half22float2(u32_as_h2(w[j]));
    f[2 * j] = t.x;
    f[2 * j + 1] = t.y;
    amax = fmaxf(amax, fmaxf(fabsf(t.x), fabsf(t.y)));
  }
  amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 1));  // 4 lanes = one 32-element block
  amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 2));
  int Xe, byte;
  if (amax == 0.f) {
    Xe = -127;
    byte = 0;
  } else {
    Xe = floor_log2_f32(amax) - kOff;
    byte = min(max(Xe + 127, 0), 254);
    Xe = byte - 127;
  }
  const float down = exp2i_f32(-Xe);  // 2^-X, exact scaling
  uint32_t c[2] = {0, 0};
  uint32_t d[4] = {0, 0, 0, 0};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float a = __fmul_rn(f[2 * j], down), b = __fmul_rn(f[2 * j + 1], down);
    uint32_t pair;
    if constexpr (FMT == CHAM_A_MXFP8) {
      const uint16_t e = cvt_e4m3x2(b, a);
      pair = e;
      if constexpr (DEQ) {
        const float2 val = __half22float2(u32_as_h2(cvt_e4m3x2_to_f16x2(e)));
        const float up = exp2i_f32(Xe);
        d[j] = h2_as_u32(__floats2half2_rn(__fmul_rn(val.x, up), __fmul_rn(val.y, up)));
      }
    } else {
      const int qa = min(max(__float2int_rn(__fmul_rn(a, 64.f)), -127), 127);
      const int qb = min(max(__float2int_rn(__fmul_rn(b, 64.f)), -127), 127);
      pair = (static_cast<uint32_t>(qa) & 0xFFu) | ((static_cast<uint32_t>(qb) & 0xFFu) << 8);
      if constexpr (DEQ) {
        const float up = exp2i_f32(max(Xe - 6, -126));  // zero block (Xe = -127): codes are 0
        d[j] = h2_as_u32(__floats2half2_rn(__fmul_rn(static_cast<float>(qa), up),
                                           __fmul_rn(static_cast<float>(qb), up)));
      }
    }
    c[j >> 1] |= pair << (16 * (j & 1));
  }
  code = make_uint2(c[0], c[1]);
  deq = make_uint4(d[0], d[1], d[2], d[3]);
  byte_out = byte;
  (void)lane;
}

template <int FMT, bool CODES, bool DEQ>
__global__ void __launch_bounds__(256)
    k_act_encode_mx(const uint4* __restrict__ X, int64_t nvec, uint2* __restrict__ codes, uint4* __restrict__ deq,
                    uint8_t* __restrict__ e8m0, uint8_t* __restrict__ e8cm, int kblocks, int64_t cm_plane,
                    cham_qparams* __restrict__ params, int* dev_status, bool kperm) {
  griddep_wait();  // its outputs may still be read by the previous kernel
  griddep_launch_dependents();
  if (blockIdx.x == 0 && threadIdx.x == 0 && params != nullptr) *params = cham_qparams{1.f, 0, 1.f, FMT};
  const int lane = threadIdx.x & 31;
  const int64_t warp_global = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t span = (static_cast<int64_t>(gridDim.x) * blockDim.x);  // vectors per unrolled step
  uint32_t nonfinite = 0;
  // lanes of a warp cover 32 consecutive vectors (8 blocks); every lane runs the same trip count
  for (int64_t base = warp_global * 32; base < nvec; base += span * kUnroll) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t i = base + u * span + lane;
      v[u] = i < nvec ? __ldg(X + i) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t i = base + u * span + lane;  // nvec is a multiple of 4: a block's lanes agree
      uint2 c;
      uint4 d;
      int byte;
      encode8_mx<FMT, DEQ>(v[u], lane, c, d, byte, nonfinite);
      if (i < nvec) {
        if constexpr (CODES) codes[i] = kperm ? kperm8(c) : c;
        if constexpr (DEQ) deq[i] = d;
        if (e8m0 != nullptr && (lane & 3) == 0) e8m0[i >> 2] = static_cast<uint8_t>(byte);
        if (e8cm != nullptr && (lane & 3) == 0) {  // chunk-major copy for the FP8 GEMM
          const int64_t blk = i >> 2, m = blk / kblocks;
          const int kb = static_cast<int>(blk - m * kblocks);
          e8cm[(kb >> 2) * cm_plane + m * 4 + (kb & 3)] = static_cast<uint8_t>(byte);
        }
      }
    }
  }
  if (nonfinite) set_status(dev_status, CHAM_ERR_NONFINITE);
}

// ------------------------------------------------------------------ activation-format argmin (Eq. format-argmin)
// Sum over 8 elements of (x - s * deq)^2: the error of each element rounded once (fma), squared
// and summed in fp32 (a fixed order).  s = 1 for the MX formats, whose deq is the full value.
CHAM_DEV float sq_err8(const float (&x)[8], const uint4& deq, float s) {
  const uint32_t d[4] = {deq.x, deq.y, deq.z, deq.w};
  float acc = 0.f;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 q = __half22float2(u32_as_h2(d[j]));
    const float ea = fmaf(-q.x, s, x[2 * j]), eb = fmaf(-q.y, s, x[2 * j + 1]);
    acc = __fadd_rn(acc, __fadd_rn(__fmul_rn(ea, ea), __fmul_rn(eb, eb)));
  }
  return acc;
}

// Per CTA: SSE_f for the five activation formats over its vectors, f = 0..4 (Sec. 3.1): the
// per-tensor formats with ScaleZP of the tensor's range (reduced from the range partials), the
// MX formats per 32-element block (four consecutive lanes per block, as in the MX encoder).
__global__ void __launch_bounds__(256)
    k_act_format_sse(const uint4* __restrict__ X, int64_t nvec, const RangePartial* __restrict__ parts, int nparts,
                     double* __restrict__ sse_parts, int* dev_status) {
  griddep_wait();  // the range partials
  griddep_launch_dependents();
  float lo, hi;
  uint32_t nf;
  reduce_partials(parts, nparts, lo, hi, nf);
  const TensorParams p0 = scale_zp(CHAM_A_INT8_ASYM, lo, hi);
  const TensorParams p1 = scale_zp(CHAM_A_E4M3, lo, hi);
  const TensorParams p2 = scale_zp(CHAM_A_E5M2, lo, hi);
  if (blockIdx.x == 0 && threadIdx.x == 0 && nf) set_status(dev_status, CHAM_ERR_NONFINITE);
  double acc[5] = {0, 0, 0, 0, 0};
  const int lane = threadIdx.x & 31;
  const int64_t warp_global = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t span = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t base = warp_global * 32; base < nvec; base += span) {
    const int64_t i = base + lane;  // nvec is a multiple of 4: the lanes of one block agree
    const uint4 v = i < nvec ? __ldg(X + i) : make_uint4(0, 0, 0, 0);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    float x[8];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 t = __half22float2(u32_as_h2(w[j]));
      x[2 * j] = t.x;
      x[2 * j + 1] = t.y;
    }
    uint2 c;
    uint4 d;
    int byte;
    uint32_t nfx = 0;
    float e[5];
    encode8_tensor<CHAM_A_INT8_ASYM, true>(v, p0, c, d);
    e[0] = sq_err8(x, d, p0.s);
    encode8_tensor<CHAM_A_E4M3, true>(v, p1, c, d);
    e[1] = sq_err8(x, d, p1.s);
    encode8_tensor<CHAM_A_E5M2, true>(v, p2, c, d);
    e[2] = sq_err8(x, d, p2.s);
    encode8_mx<CHAM_A_MXFP8, true>(v, lane, c, d, byte, nfx);
    e[3] = sq_err8(x, d, 1.f);
    encode8_mx<CHAM_A_MXINT8, true>(v, lane, c, d, byte, nfx);
    e[4] = sq_err8(x, d, 1.f);
    if (i < nvec) {
#pragma unroll
      for (int f = 0; f < 5; ++f) acc[f] += static_cast<double>(e[f]);
    }
  }
  __shared__ double sh[5][8];
#pragma unroll
  for (int f = 0; f < 5; ++f) {
    double a = acc[f];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
    if (lane == 0) sh[f][threadIdx.x >> 5] = a;
  }
  __syncthreads();
  if (threadIdx.x < 5) {
    double a = 0;
    for (int k = 0; k < static_cast<int>(blockDim.x >> 5); ++k) a += sh[threadIdx.x][k];
    sse_parts[static_cast<int64_t>(blockIdx.x) * 5 + threadIdx.x] = a;
  }
}

// Adds the CTAs' sums, in CTA order, to out[0..4] (so that calls accumulate over the
// calibration tensors of one layer and bucket).
__global__ void __launch_bounds__(32) k_act_format_sse_finish(const double* __restrict__ sse_parts, int nparts,
                                                             double* __restrict__ out) {
  griddep_wait();
  if (threadIdx.x < 5) {
    double a = 0;
    for (int k = 0; k < nparts; ++k) a += sse_parts[static_cast<int64_t>(k) * 5 + threadIdx.x];
    out[threadIdx.x] += a;
  }
}

// ------------------------------------------------------------------ calibration power sums (Alg. 1)
__global__ void __launch_bounds__(256) k_act_moments(const uint4* __restrict__ X, int64_t nvec,
                                                    MomentPartial* __restrict__ parts) {
  double s1 = 0, s2 = 0, s3 = 0, s4 = 0;
  float lo = INFINITY, hi = -INFINITY;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec; i += stride) {
    const uint4 v = __ldg(X + i);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = __half22float2(u32_as_h2(w[j]));
      lo = fminf(lo, fminf(f.x, f.y));
      hi = fmaxf(hi, fmaxf(f.x, f.y));
      const double a = f.x, b = f.y;
      const double a2 = a * a, b2 = b * b;  // exact: 22-bit products of fp16 values
      s1 += a + b;
      s2 += a2 + b2;
      s3 += a2 * a + b2 * b;
      s4 += a2 * a2 + b2 * b2;
    }
  }
  __shared__ double sh[4][256];
  __shared__ float sl[256], shh[256];
  sh[0][threadIdx.x] = s1;
  sh[1][threadIdx.x] = s2;
  sh[2][threadIdx.x] = s3;
  sh[3][threadIdx.x] = s4;
  sl[threadIdx.x] = lo;
  shh[threadIdx.x] = hi;
  __syncthreads();
  for (int o = blockDim.x / 2; o > 0; o >>= 1) {  // fixed-order tree: deterministic
    if (threadIdx.x < o) {
      for (int k = 0; k < 4; ++k) sh[k][threadIdx.x] += sh[k][threadIdx.x + o];
      sl[threadIdx.x] = fminf(sl[threadIdx.x], sl[threadIdx.x + o]);
      shh[threadIdx.x] = fmaxf(shh[threadIdx.x], shh[threadIdx.x + o]);
    }
    __syncthreads();
  }
  if (threadIdx.x == 0)
    parts[blockIdx.x] = MomentPartial{{sh[0][0], sh[1][0], sh[2][0], sh[3][0]}, sl[0], shh[0]};
}

// Sum the partials in a fixed order: 256 threads each add a strided subset, then a fixed tree.
__global__ void __launch_bounds__(256) k_act_moments_finish(const MomentPartial* __restrict__ parts, int nparts,
                                                           int64_t count, double* __restrict__ out) {
  __shared__ double sh[4][256];
  __shared__ float sl[256], shh[256];
  double s[4] = {0, 0, 0, 0};
  float lo = INFINITY, hi = -INFINITY;
  for (int i = threadIdx.x; i < nparts; i += blockDim.x) {
    for (int k = 0; k < 4; ++k) s[k] += parts[i].s[k];
    lo = fminf(lo, parts[i].lo);
    hi = fmaxf(hi, parts[i].hi);
  }
  for (int k = 0; k < 4; ++k) sh[k][threadIdx.x] = s[k];
  sl[threadIdx.x] = lo;
  shh[threadIdx.x] = hi;
  __syncthreads();
  for (int o = blockDim.x / 2; o > 0; o >>= 1) {
    if (threadIdx.x < o) {
      for (int k = 0; k < 4; ++k) sh[k][threadIdx.x] += sh[k][threadIdx.x + o];
      sl[threadIdx.x] = fminf(sl[threadIdx.x], sl[threadIdx.x + o]);
      shh[threadIdx.x] = fmaxf(shh[threadIdx.x], shh[threadIdx.x + o]);
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    out[0] += static_cast<double>(count);
    for (int k = 0; k < 4; ++k) out[1 + k] += sh[k][0];
    out[5] = fmin(out[5], static_cast<double>(sl[0]));
    out[6] = fmax(out[6], static_cast<double>(shh[0]));
  }
}

// ------------------------------------------------------------------ host-side launchers
// Enough CTAs that each thread's kRangeUnroll loads cover the tensor in one round (the DRAM latency
// is paid once), up to 8 resident CTAs of 256 threads per SM.
int range_grid(int64_t nvec, int num_sms) {
  const int64_t want = (nvec + 256 * kRangeUnroll - 1) / (256 * kRangeUnroll);
  const int64_t cap = static_cast<int64_t>(num_sms) * 8;
  return static_cast<int>(want < 1 ? 1 : (want < cap ? want : cap));
}

int group_grid(int64_t nvec, int n_groups, int num_sms) {
  const int g = range_grid(nvec, num_sms) / (n_groups > 1 ? n_groups : 1);
  return g < 1 ? 1 : g;
}

// CTAs of k_act_quant_coop that can be resident at once on this device (0 if unknown).
template <int FMT, bool CODES, bool DEQ>
static int64_t coop_capacity(int num_sms) {
  static int cached_device = -1;
  static int per_sm = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (dev != cached_device) {
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_act_quant_coop<FMT, CODES, DEQ>, 256, 0) != cudaSuccess) {
      (void)cudaGetLastError();
      n = 0;
    }
    per_sm = n;
    cached_device = dev;
  }
  return static_cast<int64_t>(per_sm) * num_sms;
}

template <int FMT, bool CODES, bool DEQ>
static void launch_tensor(const ActQuantArgs& a, cudaStream_t st) {
  if (a.use_static) {
    // one pass: enough CTAs that every thread's kUnroll loads cover the tensor (up to 8 resident
    // CTAs per SM), so no thread needs a second DRAM round trip for a tail
    const int64_t want = (a.nvec + 256 * kUnroll - 1) / (256 * kUnroll);
    const int64_t cap = static_cast<int64_t>(a.num_sms) * 8;
    const int g = static_cast<int>(want < 1 ? 1 : (want < cap ? want : cap));
    launch_pdl(k_act_encode_static<FMT, CODES, DEQ>, dim3(g), dim3(256), 0, st, a.X, a.nvec, a.stat, a.codes,
               a.deq, a.params, a.scale_out, a.dev_status, a.kperm);
    return;
  }
  // per-sample groups: each group's range and encode grids are the per-tensor ones split evenly
  const int G = a.n_groups > 1 ? a.n_groups : 1;
  const int64_t nvg = a.nvec / G;
  // one cooperative launch when the range pass's grid fits on the GPU at once and the partials'
  // slots hold it
  const int64_t P = (nvg + 256 * kCoopVec - 1) / (256 * kCoopVec);
  if (P <= a.nparts && P * G <= coop_capacity<FMT, CODES, DEQ>(a.num_sms)) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(P), G);
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, k_act_quant_coop<FMT, CODES, DEQ>, a.X, nvg, a.parts, a.codes, a.deq, a.params,
                           a.scale_out, a.dev_status, a.kperm) == cudaSuccess)
      return;
    (void)cudaGetLastError();  // not launched: the two-launch path below
  }
  launch_pdl(k_act_range, dim3(a.nparts, G), dim3(256), 0, st, a.X, nvg, a.parts);
  // the encode grid covers each group in one pass of kUnroll loads per thread (8 CTAs per SM at most)
  const int64_t want = (nvg + 256 * kUnroll - 1) / (256 * kUnroll);
  const int64_t cap = static_cast<int64_t>(a.num_sms) * 8 / G;
  const int eg = static_cast<int>(want < 1 ? 1 : (want < cap ? want : (cap < 1 ? 1 : cap)));
  launch_pdl(k_act_encode_tensor<FMT, CODES, DEQ>, dim3(eg, G), dim3(256), 0, st, a.X, nvg,
             static_cast<const RangePartial*>(a.parts), a.nparts, a.codes, a.deq, a.params, a.scale_out,
             a.dev_status, a.kperm);
}

template <int FMT, bool CODES, bool DEQ>
static void launch_mx(const ActQuantArgs& a, cudaStream_t st) {
  const int64_t warps = (a.nvec + 31) / 32;
  int64_t g = (warps + 7) / 8;
  const int64_t cap = static_cast<int64_t>(a.num_sms) * 8;
  if (g > cap) g = cap;
  if (g < 1) g = 1;
  launch_pdl(k_act_encode_mx<FMT, CODES, DEQ>, dim3(static_cast<int>(g)), dim3(256), 0, st, a.X, a.nvec, a.codes,
             a.deq, a.e8m0, a.e8cm, a.kblocks, a.cm_plane, a.params, a.dev_status, a.kperm);
}

template <bool CODES, bool DEQ>
static void dispatch(int fmt, const ActQuantArgs& a, cudaStream_t st) {
  switch (fmt) {
    case CHAM_A_INT8_ASYM: launch_tensor<CHAM_A_INT8_ASYM, CODES, DEQ>(a, st); break;
    case CHAM_A_E4M3: launch_tensor<CHAM_A_E4M3, CODES, DEQ>(a, st); break;
    case CHAM_A_E5M2: launch_tensor<CHAM_A_E5M2, CODES, DEQ>(a, st); break;
    case CHAM_A_MXFP8: launch_mx<CHAM_A_MXFP8, CODES, DEQ>(a, st); break;
    case CHAM_A_MXINT8: launch_mx<CHAM_A_MXINT8, CODES, DEQ>(a, st); break;
    default: break;
  }
}

void launch_act_quant(int fmt, const ActQuantArgs& a, bool codes, bool deq, cudaStream_t st) {
  if (codes && deq) dispatch<true, true>(fmt, a, st);
  else if (codes) dispatch<true, false>(fmt, a, st);
  else dispatch<false, true>(fmt, a, st);
}

void launch_act_format_sse(const uint4* X, int64_t nvec, RangePartial* parts, int nparts, double* sse_parts,
                           double* out, int* dev_status, cudaStream_t st) {
  launch_pdl(k_act_range, dim3(nparts), dim3(256), 0, st, X, nvec, parts);
  launch_pdl(k_act_format_sse, dim3(nparts), dim3(256), 0, st, X, nvec, static_cast<const RangePartial*>(parts),
             nparts, sse_parts, dev_status);
  launch_pdl(k_act_format_sse_finish, dim3(1), dim3(32), 0, st, static_cast<const double*>(sse_parts), nparts, out);
}

void launch_act_moments(const uint4* X, int64_t nvec, int64_t count, MomentPartial* parts, int nparts,
                        double* out, cudaStream_t st) {
  k_act_moments<<<nparts, 256, 0, st>>>(X, nvec, parts);
  k_act_moments_finish<<<1, 256, 0, st>>>(parts, nparts, count, out);
}

}  // namespace cham
