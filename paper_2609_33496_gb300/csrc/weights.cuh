// weights.cuh -- per-channel weight codecs shared by the selection and pack kernels (steps a5, a6).
//
// One definition per weight format of Sec. 3.2, at the granularity of reading R10: per output
// channel (INT8/INT4 sym/asym, NF4, E2M1) or per 32-element block along K with an E8M0 exponent
// (MXINT8, MXINT4, MXFP4).  Arithmetic follows readings R4-R9: fp32 scales from one correctly
// rounded division, the product rounded to fp32, then round-to-nearest-even onto the code grid.
#pragma once

#include <cuda_runtime.h>

#include "common.cuh"

namespace cham {

// NF4 levels (fp16 bit patterns, ascending) and the fp32 midpoints between neighbours.
struct NF4Table {
  uint16_t level[16];
  float mid[15];
};

// Channel statistics every format derives its scale from.
struct ChanStats {
  float amax, lo, hi;
};

struct ChanScale {  // per-channel scale, reciprocal, zero point
  float s, inv;
  int z;
};

__host__ __device__ constexpr int wbits(int fmt) { return fmt <= CHAM_W_MXINT8 ? 8 : 4; }
__host__ __device__ constexpr bool w_is_mx(int fmt) {
  return fmt == CHAM_W_MXINT8 || fmt == CHAM_W_MXINT4 || fmt == CHAM_W_MXFP4;
}
// MMA class: 0 = a 4-bit format whose values are exact 8-bit floats (tensor-core FP8 path),
// 1 = needs fp16 operands (NF4 levels, 8-bit integers).
__host__ __device__ constexpr int w_class(int fmt) {
  return (fmt == CHAM_W_INT4_SYM || fmt == CHAM_W_INT4_ASYM || fmt == CHAM_W_E2M1 || fmt == CHAM_W_MXINT4 ||
          fmt == CHAM_W_MXFP4)
             ? 0
             : 1;
}

// Per-channel scale of a non-MX format from the channel statistics.
CHAM_DEV ChanScale chan_scale(int fmt, const ChanStats& st) {
  ChanScale c{1.f, 1.f, 0};
  switch (fmt) {
    case CHAM_W_INT8_SYM:
    case CHAM_W_INT4_SYM:
    case CHAM_W_E2M1: {
      const float qmax = fmt == CHAM_W_INT8_SYM ? 127.f : (fmt == CHAM_W_INT4_SYM ? 7.f : 6.f);
      if (st.amax != 0.f) {
        c.s = __fdiv_rn(st.amax, qmax);
        c.inv = __fdiv_rn(qmax, st.amax);
      }
      break;
    }
    case CHAM_W_INT8_ASYM:
    case CHAM_W_INT4_ASYM: {
      const float lv = fmt == CHAM_W_INT8_ASYM ? 255.f : 15.f;
      const float lo = fminf(st.lo, 0.f), hi = fmaxf(st.hi, 0.f);
      const float d = __fsub_rn(hi, lo);
      if (d != 0.f) {
        c.s = __fdiv_rn(d, lv);
        c.inv = __fdiv_rn(lv, d);
        c.z = min(max(__float2int_rn(__fmul_rn(-lo, c.inv)), 0), static_cast<int>(lv));
      }
      break;
    }
    case CHAM_W_NF4:
      if (st.amax != 0.f) c.s = st.amax;  // v = w / amax (R9)
      break;
    default:
      break;
  }
  return c;
}

// E2M1 value of a 4-bit pattern (exact in fp32).
CHAM_DEV float e2m1_value(uint32_t n) {
  const uint32_t e = (n >> 1) & 3u, m = n & 1u;
  const float mag = e == 0 ? 0.5f * static_cast<float>(m) : exp2i_f32(static_cast<int>(e) - 1) * (1.f + 0.5f * m);
  return (n & 8u) ? -mag : mag;
}

// Encode one element of a non-MX format; returns the stored code (int for INT formats, level
// index for NF4, bit pattern for E2M1) and writes the exact reconstruction error w - DQ rounded
// once to fp32 (FMA of the exact product).
CHAM_DEV int encode_chan(int fmt, float w, const ChanScale& c, const NF4Table& nf4, float* err) {
  switch (fmt) {
    case CHAM_W_INT8_SYM:
    case CHAM_W_INT4_SYM: {
      const int qmax = fmt == CHAM_W_INT8_SYM ? 127 : 7;
      const int q = min(max(__float2int_rn(__fmul_rn(w, c.inv)), -qmax), qmax);
      *err = __fmaf_rn(-static_cast<float>(q), c.s, w);
      return q;
    }
    case CHAM_W_INT8_ASYM:
    case CHAM_W_INT4_ASYM: {
      const int lv = fmt == CHAM_W_INT8_ASYM ? 255 : 15;
      const int q = min(max(__float2int_rn(__fmul_rn(w, c.inv)) + c.z, 0), lv);
      *err = __fmaf_rn(-static_cast<float>(q - c.z), c.s, w);
      return q;
    }
    case CHAM_W_E2M1: {
      const uint32_t n = cvt_e2m1x2(0.f, __fmul_rn(w, c.inv)) & 0xFu;
      *err = __fmaf_rn(-e2m1_value(n), c.s, w);
      return static_cast<int>(n);
    }
    case CHAM_W_NF4: {
      const float v = __fdiv_rn(w, c.s);
      int code = 0;
#pragma unroll
      for (int i = 0; i < 15; ++i) code += (nf4.mid[i] < v) ? 1 : 0;  // ties go to the lower level
      const float L = __half2float(__ushort_as_half(nf4.level[code]));
      *err = __fmaf_rn(-L, c.s, w);
      return code;
    }
    default:
      *err = 0.f;
      return 0;
  }
}

// MX block exponent from the block's amax: X = floor(log2 amax) - emax_elem (R1); all-zero
// block -> -127 (E8M0 byte 0, R2).
CHAM_DEV int mx_exponent(int fmt, float amax) {
  if (amax == 0.f) return -127;
  const int off = fmt == CHAM_W_MXFP4 ? 2 : 0;
  return max(min(floor_log2_f32(amax) - off + 127, 254), 0) - 127;
}

// Encode one MX element given its block exponent; returns the code (two's complement byte /
// nibble or E2M1 pattern) and the exact DQ value in fp32.
CHAM_DEV int encode_mx(int fmt, float w, int X, float* dq) {
  // an all-zero block has X = -127: its codes are 0 and its decode scale only needs to be finite
  const float v = __fmul_rn(w, exp2i_f32(-X));
  if (fmt == CHAM_W_MXINT8) {
    const int q = min(max(__float2int_rn(__fmul_rn(v, 64.f)), -127), 127);
    *dq = __fmul_rn(static_cast<float>(q), exp2i_f32(max(X - 6, -126)));
    return q & 0xFF;
  }
  if (fmt == CHAM_W_MXINT4) {
    const int q = min(max(__float2int_rn(__fmul_rn(v, 4.f)), -7), 7);
    *dq = __fmul_rn(static_cast<float>(q), exp2i_f32(max(X - 2, -126)));
    return q & 0xF;
  }
  const uint32_t n = cvt_e2m1x2(0.f, v) & 0xFu;
  *dq = __fmul_rn(e2m1_value(n), exp2i_f32(max(X, -126)));
  return static_cast<int>(n);
}

constexpr int kMaxRowGroups = 256;  // groups per row of a group-wise blob (K <= 8192 at g = 32)
constexpr int kMaxCands = 48;       // (g, f) candidates of one search

struct GroupCand {
  int g, f;
};

struct GroupSearchArgs {
  const __half* W;
  int N, K;
  const double* energy;   // [K] or null (e_k = 1)
  float* energy32;        // [K] scratch: energy as fp32
  double* parts;          // [N][n_cand] per-channel weighted errors
  double* scores;         // [n_cand] output
  int n_cand;
  GroupCand cand[kMaxCands];
};

constexpr int kMaxPackGroups = 12;  // 9 formats + 2 class tails (layout 1), or the 2 classes

struct PackArgs {
  const __half* W;
  const uint8_t* fmt_dev;   // selected format of each original channel
  uint8_t* fmt_out;         // fused selection + pack: where the selected formats go
  int N, K, Kp, bits, n_chunks;
  int n_packed;             // Np
  int cls_base[2];          // first packed slot of each MMA class
  int cls_count[2];         // channels of each class (from the host plan)
  // the packed groups (layout 0: one per class; layout 1: per format and class tails), in slot
  // order: group of each format, first slot and channel count of each group
  int n_groups;
  int8_t group_of_fmt[CHAM_W_NFORMATS];
  int group_base[kMaxPackGroups];
  int group_count[kMaxPackGroups];
  int one_class;            // the class of every channel when the plan has one (slot = channel), else -1
  cham_wpack_desc desc;     // copied to desc_out (the blob header) by the pack kernel
  cham_wpack_desc* desc_out;
  uint8_t* codes;
  float* scale;
  uint8_t* zero;
  uint8_t* e8m0;
  uint8_t* fmtp;
  int32_t* perm;
  int group;                // group-wise blob: g input channels per scale (0: per channel)
  uint32_t* gscale;         // group-wise blob: [tiles][chunks][128] two fp16 block scales
  int* dev_status;
};

void launch_select(const __half* W, int N, int K, uint32_t mask, uint8_t* fmt_out, double* sse_out,
                   const NF4Table& nf4, cudaStream_t st);
void launch_pack(const PackArgs& a, const NF4Table& nf4, cudaStream_t st);
// Fused selection + pack of a one-class plan (every palette member in one MMA class).
void launch_select_pack(const PackArgs& a, uint32_t mask, const NF4Table& nf4, cudaStream_t st);
void launch_select_groups(const GroupSearchArgs& a, const NF4Table& nf4, cudaStream_t st);
void launch_channel_energy(const __half* X, int M, int K, double* energy, cudaStream_t st);

}  // namespace cham
