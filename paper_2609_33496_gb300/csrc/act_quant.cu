// act_quant.cu -- activation quantizer kernels (steps a2-a4) and calibration power sums.
//
// The dynamic path of Alg. 3: lo, hi = min x, max x over the tensor; ScaleZP (App. A.7); every
// element encoded in the format the LUT picked.  Per-tensor formats need the range before any
// element can be encoded, so they take two launches (range partials, then encode; the second
// read of X mostly hits L2).  MX formats (32-element blocks along K, E8M0 exponent, Sec. 3.6 /
// App. A.11) need only the block's own amax and run in one launch, four lanes per block.
//
// All scale arithmetic is IEEE fp32 with explicit round-to-nearest intrinsics (no contraction),
// in the order of readings R4-R8: inv by one correctly rounded division, the product x * inv
// rounded to fp32, then the format rounding.  The same arithmetic gives the codes (public
// chameleon_act_quant) and the exact fp16 operand values the GEMM consumes (R13).
#include "act_quant.cuh"

namespace cham {

// ------------------------------------------------------------------ a2: range partials
__global__ void __launch_bounds__(256) k_act_range(const uint4* __restrict__ X, int64_t nvec,
                                                  RangePartial* __restrict__ parts) {
  __half2 lo2 = __float2half2_rn(65504.f), hi2 = __float2half2_rn(-65504.f);
  uint32_t nonfinite = 0;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec; i += stride) {
    const uint4 v = __ldg(X + i);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      // exponent field all ones in either half: Inf or NaN
      nonfinite |= (((w[j] & 0x7C00u) == 0x7C00u) | ((w[j] & 0x7C000000u) == 0x7C000000u));
      const __half2 h = *reinterpret_cast<const __half2*>(&w[j]);
      lo2 = __hmin2(lo2, h);
      hi2 = __hmax2(hi2, h);
    }
  }
  float lo = fminf(__low2float(lo2), __high2float(lo2));
  float hi = fmaxf(__low2float(hi2), __high2float(hi2));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    nonfinite |= __shfl_xor_sync(0xffffffffu, nonfinite, o);
  }
  __shared__ float s_lo[8], s_hi[8];
  __shared__ uint32_t s_nf[8];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    s_lo[warp] = lo;
    s_hi[warp] = hi;
    s_nf[warp] = nonfinite;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int k = 1; k < static_cast<int>(blockDim.x >> 5); ++k) {
      lo = fminf(lo, s_lo[k]);
      hi = fmaxf(hi, s_hi[k]);
      nonfinite |= s_nf[k];
    }
    parts[blockIdx.x] = RangePartial{lo, hi, static_cast<int>(nonfinite), 0};
  }
}

// Reduce the range partials (identically in every CTA: min/max are exact and order-free) and
// derive the per-tensor quantizer parameters.  Returns false for a non-finite tensor.
__device__ bool tensor_params(const RangePartial* parts, int nparts, int fmt, TensorParams* out) {
  __shared__ float s_lo[32], s_hi[32];
  __shared__ int s_nf[32];
  float lo = INFINITY, hi = -INFINITY;
  int nf = 0;
  for (int i = threadIdx.x; i < nparts; i += blockDim.x) {
    const RangePartial p = parts[i];
    lo = fminf(lo, p.lo);
    hi = fmaxf(hi, p.hi);
    nf |= p.nonfinite;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    nf |= __shfl_xor_sync(0xffffffffu, nf, o);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    s_lo[warp] = lo;
    s_hi[warp] = hi;
    s_nf[warp] = nf;
  }
  __syncthreads();
  lo = INFINITY;
  hi = -INFINITY;
  nf = 0;
  for (int k = 0; k < static_cast<int>(blockDim.x >> 5); ++k) {
    lo = fminf(lo, s_lo[k]);
    hi = fmaxf(hi, s_hi[k]);
    nf |= s_nf[k];
  }
  TensorParams p;
  if (fmt == CHAM_A_INT8_ASYM) {
    // ScaleZP: s = (hi - lo)/255, z = round(-lo/s), zero-inclusive range (R4), degenerate (R7)
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
    // FP8: s = amax / Fmax, inv = Fmax / amax (App. A.7, R11)
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
  *out = p;
  return nf == 0;
}

// ------------------------------------------------------------------ a3: per-tensor encode
// Eight elements per thread per iteration (one 16-byte load): eight code bytes and/or eight exact
// fp16 operand values (q - z for INT8-asym, value(code) for FP8; the scale s stays outside).
template <int FMT, bool CODES, bool DEQ>
__global__ void __launch_bounds__(256)
    k_act_encode_tensor(const uint4* __restrict__ X, int64_t nvec, const RangePartial* __restrict__ parts,
                        int nparts, uint2* __restrict__ codes, uint4* __restrict__ deq,
                        cham_qparams* __restrict__ params, float* __restrict__ scale_out, int* dev_status) {
  TensorParams p;
  const bool finite = tensor_params(parts, nparts, FMT, &p);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    if (params != nullptr) *params = cham_qparams{p.s, p.z, p.inv, FMT};
    if (scale_out != nullptr) *scale_out = p.s;
    if (!finite) set_status(dev_status, CHAM_ERR_NONFINITE);
  }
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec; i += stride) {
    const uint4 v = __ldg(X + i);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    uint32_t c[2] = {0, 0};
    uint32_t d[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[j]));
      const float a = __fmul_rn(f.x, p.inv), b = __fmul_rn(f.y, p.inv);
      uint32_t pair;  // two code bytes, element 2j in the low byte
      if constexpr (FMT == CHAM_A_INT8_ASYM) {
        const int qa = min(max(__float2int_rn(a) + p.z, 0), 255);
        const int qb = min(max(__float2int_rn(b) + p.z, 0), 255);
        pair = static_cast<uint32_t>(qa) | (static_cast<uint32_t>(qb) << 8);
        if constexpr (DEQ) {
          const __half2 h = __halves2half2(__int2half_rn(qa - p.z), __int2half_rn(qb - p.z));
          d[j] = *reinterpret_cast<const uint32_t*>(&h);
        }
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
    if constexpr (CODES) codes[i] = make_uint2(c[0], c[1]);
    if constexpr (DEQ) deq[i] = make_uint4(d[0], d[1], d[2], d[3]);
  }
}

// ------------------------------------------------------------------ a4: MX encode
// Four consecutive lanes own one 32-element block (8 elements each).  Shared exponent
// X = floor(log2 amax) - emax_elem (R1; 8 for the E4M3 body, 0 for the int8 body), element
// v = x * 2^-X (exact), body code; all-zero block -> E8M0 byte 0 (R2).
template <int FMT, bool CODES, bool DEQ>
__global__ void __launch_bounds__(256)
    k_act_encode_mx(const uint4* __restrict__ X, int64_t nvec, uint2* __restrict__ codes, uint4* __restrict__ deq,
                    uint8_t* __restrict__ e8m0, cham_qparams* __restrict__ params, int* dev_status) {
  constexpr int kOff = (FMT == CHAM_A_MXFP8) ? 8 : 0;
  if (blockIdx.x == 0 && threadIdx.x == 0 && params != nullptr) *params = cham_qparams{1.f, 0, 1.f, FMT};
  const int lane = threadIdx.x & 31;
  const int64_t warp_global = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t warps_total = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  uint32_t nonfinite = 0;
  for (int64_t base = warp_global * 32; base < nvec; base += warps_total * 32) {
    const int64_t i = base + lane;
    const bool active = i < nvec;  // nvec is a multiple of 4: a block's lanes agree
    const uint4 v = active ? __ldg(X + i) : make_uint4(0, 0, 0, 0);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    float f[8];
    float amax = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      nonfinite |= (((w[j] & 0x7C00u) == 0x7C00u) | ((w[j] & 0x7C000000u) == 0x7C000000u));
      const float2 t = __half22float2(*reinterpret_cast<const __half2*>(&w[j]));
      f[2 * j] = t.x;
      f[2 * j + 1] = t.y;
      amax = fmaxf(amax, fmaxf(fabsf(t.x), fabsf(t.y)));
    }
    amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 1));
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
    uint32_t d[4];
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
          const __half2 h = __floats2half2_rn(__fmul_rn(val.x, up), __fmul_rn(val.y, up));
          d[j] = *reinterpret_cast<const uint32_t*>(&h);
        }
      } else {
        const int qa = min(max(__float2int_rn(__fmul_rn(a, 64.f)), -127), 127);
        const int qb = min(max(__float2int_rn(__fmul_rn(b, 64.f)), -127), 127);
        pair = (static_cast<uint32_t>(qa) & 0xFFu) | ((static_cast<uint32_t>(qb) & 0xFFu) << 8);
        if constexpr (DEQ) {
          const float up = exp2i_f32(max(Xe - 6, -126));  // zero block (Xe = -127): codes are 0
          const __half2 h = __floats2half2_rn(__fmul_rn(static_cast<float>(qa), up),
                                              __fmul_rn(static_cast<float>(qb), up));
          d[j] = *reinterpret_cast<const uint32_t*>(&h);
        }
      }
      c[j >> 1] |= pair << (16 * (j & 1));
    }
    if (active) {
      if constexpr (CODES) codes[i] = make_uint2(c[0], c[1]);
      if constexpr (DEQ) deq[i] = make_uint4(d[0], d[1], d[2], d[3]);
      if (e8m0 != nullptr && (lane & 3) == 0) e8m0[i >> 2] = static_cast<uint8_t>(byte);
    }
  }
  if (nonfinite) set_status(dev_status, CHAM_ERR_NONFINITE);
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
      const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[j]));
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

__global__ void k_act_moments_finish(const MomentPartial* __restrict__ parts, int nparts, int64_t count,
                                     double* __restrict__ out) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  double s[4] = {0, 0, 0, 0};
  float lo = INFINITY, hi = -INFINITY;
  for (int i = 0; i < nparts; ++i) {
    for (int k = 0; k < 4; ++k) s[k] += parts[i].s[k];
    lo = fminf(lo, parts[i].lo);
    hi = fmaxf(hi, parts[i].hi);
  }
  out[0] += static_cast<double>(count);
  for (int k = 0; k < 4; ++k) out[1 + k] += s[k];
  out[5] = fmin(out[5], static_cast<double>(lo));
  out[6] = fmax(out[6], static_cast<double>(hi));
}

// ------------------------------------------------------------------ host-side launchers
int range_grid(int64_t nvec, int num_sms) {
  const int64_t want = (nvec + 255) / 256;
  const int64_t cap = static_cast<int64_t>(num_sms) * 4;
  return static_cast<int>(want < 1 ? 1 : (want < cap ? want : cap));
}

template <int FMT, bool CODES, bool DEQ>
static void launch_tensor(const ActQuantArgs& a, cudaStream_t st) {
  const int g = range_grid(a.nvec, a.num_sms);
  k_act_encode_tensor<FMT, CODES, DEQ><<<g, 256, 0, st>>>(a.X, a.nvec, a.parts, a.nparts, a.codes, a.deq,
                                                          a.params, a.scale_out, a.dev_status);
}
template <int FMT, bool CODES, bool DEQ>
static void launch_mx(const ActQuantArgs& a, cudaStream_t st) {
  const int64_t warps = (a.nvec + 31) / 32;
  int64_t g = (warps + 7) / 8;
  const int64_t cap = static_cast<int64_t>(a.num_sms) * 8;
  if (g > cap) g = cap;
  if (g < 1) g = 1;
  k_act_encode_mx<FMT, CODES, DEQ><<<static_cast<int>(g), 256, 0, st>>>(a.X, a.nvec, a.codes, a.deq, a.e8m0,
                                                                         a.params, a.dev_status);
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
  const bool per_tensor = fmt <= CHAM_A_E5M2;
  if (per_tensor) k_act_range<<<a.nparts, 256, 0, st>>>(a.X, a.nvec, a.parts);
  if (codes && deq) dispatch<true, true>(fmt, a, st);
  else if (codes) dispatch<true, false>(fmt, a, st);
  else dispatch<false, true>(fmt, a, st);
}

void launch_act_moments(const uint4* X, int64_t nvec, int64_t count, MomentPartial* parts, int nparts,
                        double* out, cudaStream_t st) {
  k_act_moments<<<nparts, 256, 0, st>>>(X, nvec, parts);
  k_act_moments_finish<<<1, 32, 0, st>>>(parts, nparts, count, out);
}

}  // namespace cham
