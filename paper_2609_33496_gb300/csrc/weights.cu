// weights.cu -- weight-format selection (step a5) and weight pack (step a6).
//
// Selection (Sec. 3.4, Eq. weight-argmax): every output channel is round-tripped through every
// palette format; the squared reconstruction error SSE_f(c) is accumulated from per-element
// errors that are exact up to one fp32 rounding (fp32 sums of eight squares, added exactly as
// fp32 pairs; relative error below 2.4e-7); the smallest error wins, the earlier palette member on ties
// (strict '<').  One warp per channel: the row (at most 10 KB for K = 5120) stays in L1 across
// the format passes, and every reduction is a warp shuffle tree.
//
// Pack: channels are reordered (Sec. 5 proposes grouping the channels of one format by a
// permutation so that each group runs as its own GEMM) into the two MMA classes, each kept in original channel order and padded to 128-channel tiles, and
// encoded in the tiled layout the GEMM reads with bulk copies (include/chameleon.h).
#include "weights.cuh"

namespace cham {

// One warp per channel (shuffle reductions only, no block barriers), kWWarps channels per CTA.
constexpr int kWWarps = 8;
constexpr int kWThreads = 32 * kWWarps;

// Warp-wide reduction in a fixed xor-tree order; the result is valid in every lane.
template <typename T, typename Op>
CHAM_DEV T warp_reduce(T v, Op op) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

struct FMin {
  CHAM_DEV float operator()(float a, float b) const { return fminf(a, b); }
};
struct FMax {
  CHAM_DEV float operator()(float a, float b) const { return fmaxf(a, b); }
};
struct DAdd {
  CHAM_DEV double operator()(double a, double b) const { return a + b; }
};

// Eight consecutive elements of a row as fp32.
CHAM_DEV void load8(const __half* row, int v, float (&x)[8]) {
  const uint4 u = __ldg(reinterpret_cast<const uint4*>(row) + v);
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 f = __half22float2(u32_as_h2(w[j]));
    x[2 * j] = f.x;
    x[2 * j + 1] = f.y;
  }
}

// Channel statistics (amax, lo, hi) of one row, reduced over the warp.
CHAM_DEV ChanStats row_stats(const __half* row, int nvec, int lane) {
  float amax = 0.f, lo = INFINITY, hi = -INFINITY;
  for (int v = lane; v < nvec; v += 32) {
    float x[8];
    load8(row, v, x);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      amax = fmaxf(amax, fabsf(x[i]));
      lo = fminf(lo, x[i]);
      hi = fmaxf(hi, x[i]);
    }
  }
  ChanStats s;
  s.amax = warp_reduce(amax, FMax());
  s.lo = warp_reduce(lo, FMin());
  s.hi = warp_reduce(hi, FMax());
  return s;
}

// ------------------------------------------------------------------ a5: selection
// Pairwise fp32 sum of eight non-negative squared errors.  Each square and each of the three
// levels of additions rounds once, so the group sum is within 4 * 2^-24 relative of the exact
// sum; the groups are then added exactly (Sum2 below).  Every term being non-negative, the
// channel's SSE keeps that relative bound (about 2.4e-7).
CHAM_DEV float sum8(const float (&e2)[8]) {
  const float a = __fadd_rn(e2[0], e2[1]), b = __fadd_rn(e2[2], e2[3]);
  const float c = __fadd_rn(e2[4], e2[5]), d = __fadd_rn(e2[6], e2[7]);
  return __fadd_rn(__fadd_rn(a, b), __fadd_rn(c, d));
}

// A sum kept as an unevaluated pair hi + lo of fp32 values: each addition splits the rounding
// error of hi + x off exactly (Knuth's TwoSum; this file is compiled without FMA contraction) and
// carries it in lo.  The pair tracks the exact sum of its fp32 inputs to about 2^-24 relative of
// lo, far below the 4 * 2^-24 of each eight-element group sum, without the fp64 pipe (a small
// fraction of the fp32 rate on this GPU) inside the loops.
struct Sum2 {
  float hi, lo;
};

CHAM_DEV Sum2 two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  const float err = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return Sum2{s, err};
}

CHAM_DEV void sum2_add(Sum2& acc, float x) {
  const Sum2 t = two_sum(acc.hi, x);
  acc.hi = t.hi;
  acc.lo = __fadd_rn(acc.lo, t.lo);
}

// Warp-wide total of the lanes' pairs (fixed xor-tree order), as fp64, in every lane.
CHAM_DEV double warp_sum2(Sum2 v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float h = __shfl_xor_sync(0xffffffffu, v.hi, o), l = __shfl_xor_sync(0xffffffffu, v.lo, o);
    const Sum2 t = two_sum(v.hi, h);
    v.hi = t.hi;
    v.lo = __fadd_rn(__fadd_rn(v.lo, l), t.lo);
  }
  return static_cast<double>(v.hi) + static_cast<double>(v.lo);
}

// The selection of one channel (one warp): the first format of the palette with the least
// SSE; sse_row (9 slots, +inf for non-members) may be null.  Every lane returns the result.
CHAM_DEV int select_row(const __half* row, int K, uint32_t mask, int lane, const NF4Table& nf4, double* sse_row,
                        ChanStats* st_out = nullptr) {
  const int nvec = K / 8;
  const ChanStats st = row_stats(row, nvec, lane);
  if (st_out != nullptr) *st_out = st;
  const int iters = (nvec + 31) / 32;  // same trip count in every lane (shuffles)
  const bool any_mx = (mask & ((1u << CHAM_W_MXINT8) | (1u << CHAM_W_MXINT4) | (1u << CHAM_W_MXFP4))) != 0u;
  // one pass over the row for every palette member: each vector is loaded once and the members'
  // round trips are independent work for the scheduler
  ChanScale cs[CHAM_W_NFORMATS];
  Sum2 acc[CHAM_W_NFORMATS];
#pragma unroll
  for (int f = 0; f < CHAM_W_NFORMATS; ++f) {
    cs[f] = (((mask >> f) & 1u) && !w_is_mx(f)) ? chan_scale(f, st) : ChanScale{1.f, 1.f, 0};
    acc[f] = Sum2{0.f, 0.f};
  }
  for (int it = 0; it < iters; ++it) {
    const int v = it * 32 + lane;
    float x[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    if (v < nvec) load8(row, v, x);
    float am = 0.f;
    if (any_mx) {  // the palette is the same in every lane: all of them take the shuffles
#pragma unroll
      for (int i = 0; i < 8; ++i) am = fmaxf(am, fabsf(x[i]));
      am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, 1));  // 4 lanes = one 32-element block
      am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, 2));
    }
    if (v < nvec) {
#pragma unroll
      for (int f = 0; f < CHAM_W_NFORMATS; ++f) {
        if (!((mask >> f) & 1u)) continue;
        float e2[8];
        if (w_is_mx(f)) {
          const int X = mx_exponent(f, am);
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            float dq;
            encode_mx(f, x[i], X, &dq);
            const float e = __fsub_rn(x[i], dq);
            e2[i] = __fmul_rn(e, e);
          }
        } else {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            float err;
            encode_chan(f, x[i], cs[f], nf4, &err);
            e2[i] = __fmul_rn(err, err);
          }
        }
        sum2_add(acc[f], sum8(e2));
      }
    }
  }
  int best = -1;
  double best_e = 0.0;
#pragma unroll
  for (int f = 0; f < CHAM_W_NFORMATS; ++f) {
    if (!((mask >> f) & 1u)) {
      if (lane == 0 && sse_row != nullptr) sse_row[f] = INFINITY;
      continue;
    }
    const double tot = warp_sum2(acc[f]);
    if (best < 0 || tot < best_e) {  // palette order: the earlier member wins a tie
      best = f;
      best_e = tot;
    }
    if (lane == 0 && sse_row != nullptr) sse_row[f] = tot;
  }
  return best;
}

__global__ void __launch_bounds__(kWThreads) k_w_select(const __half* __restrict__ W, int N, int K, uint32_t mask,
                                                       uint8_t* __restrict__ fmt_out, double* __restrict__ sse_out,
                                                       NF4Table nf4) {
  const int lane = threadIdx.x & 31;
  const int c = blockIdx.x * kWWarps + (threadIdx.x >> 5);
  if (c >= N) return;  // whole warps: no block-wide barrier follows
  const int best = select_row(W + static_cast<size_t>(c) * K, K, mask, lane, nf4,
                              sse_out != nullptr ? sse_out + static_cast<size_t>(c) * CHAM_W_NFORMATS : nullptr);
  if (lane == 0) fmt_out[c] = static_cast<uint8_t>(best);
}

void launch_select(const __half* W, int N, int K, uint32_t mask, uint8_t* fmt_out, double* sse_out,
                   const NF4Table& nf4, cudaStream_t st) {
  k_w_select<<<(N + kWWarps - 1) / kWWarps, kWThreads, 0, st>>>(W, N, K, mask, fmt_out, sse_out, nf4);
}

// ------------------------------------------------------------------ a6: slot assignment
// Packed slot of every channel: the first slot of its group (its MMA class, or in the format-group
// layout its format's group or its class's tail) plus the number of earlier channels of the same
// group, so each group keeps the original channel order.  One CTA walks the channels in chunks of
// 1024 with warp ballots.
__global__ void __launch_bounds__(1024) k_w_slots(PackArgs a) {
  __shared__ int warp_cnt[32][kMaxPackGroups];
  __shared__ int running[kMaxPackGroups];
  for (int p = threadIdx.x; p < a.n_packed; p += blockDim.x) {
    a.perm[p] = -1;
    a.fmtp[p] = 0xFF;
  }
  if (threadIdx.x < kMaxPackGroups) running[threadIdx.x] = 0;
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int c0 = 0; c0 < a.N; c0 += blockDim.x) {
    const int c = c0 + threadIdx.x;
    const int f = c < a.N ? a.fmt_dev[c] : -1;
    const bool valid = f >= 0 && f < CHAM_W_NFORMATS && a.group_of_fmt[f] >= 0;
    const int grp = valid ? a.group_of_fmt[f] : -1;
    int my_rank_in_warp = 0;
    for (int g = 0; g < a.n_groups; ++g) {
      const uint32_t m = __ballot_sync(0xffffffffu, grp == g);
      if (grp == g) my_rank_in_warp = __popc(m & ((1u << lane) - 1u));
      if (lane == 0) warp_cnt[warp][g] = __popc(m);
    }
    __syncthreads();
    if (c < a.N) {
      if (!valid) {
        set_status(a.dev_status, CHAM_ERR_INVALID_ARG);
      } else {
        int rank = running[grp] + my_rank_in_warp;
        for (int w = 0; w < warp; ++w) rank += warp_cnt[w][grp];
        if (rank < a.group_count[grp]) {  // device formats must match the host plan
          const int slot = a.group_base[grp] + rank;
          a.perm[slot] = c;
          a.fmtp[slot] = static_cast<uint8_t>(f);
        } else {
          set_status(a.dev_status, CHAM_ERR_INVALID_ARG);
        }
      }
    }
    __syncthreads();
    if (threadIdx.x < a.n_groups) {
      int t = 0;
      for (int w = 0; w < 32; ++w) t += warp_cnt[w][threadIdx.x];
      running[threadIdx.x] += t;
    }
    __syncthreads();
  }
}

// ------------------------------------------------------------------ a6: encode one packed slot
// Byte offset of the 8 codes of elements [k0, k0+8) of packed slot p in the tiled code layout.
CHAM_DEV size_t code_offset(int p, int k0, int n_chunks, int bits) {
  const int tile = p >> 7, r = p & 127;
  const int chunk = k0 >> 6, kk = k0 & 63;
  const size_t chunk_base = (static_cast<size_t>(tile) * n_chunks + chunk) * (bits == 8 ? 8192u : 4096u);
  if (bits == 8) return chunk_base + static_cast<size_t>(kk >> 4) * 2048 + r * 16 + (kk & 15);
  return chunk_base + static_cast<size_t>(kk >> 5) * 2048 + r * 16 + ((kk & 31) >> 3) * 4;
}

// Stores the 8 codes of elements [8v, 8v+8) of packed slot p in the tiled layout: symmetric
// integer codes in offset binary (q + 128, q + 8); 4-bit words with nibble j (j < 4) = element 2j
// and nibble 4 + j = element 2j + 1 (the integer and E2M1 decodes isolate a pair with one mask),
// NF4 with nibble j = element j (the register-table decode).
CHAM_DEV void store_codes(const PackArgs& a, int p, int v, int f, int (&code)[8]) {
  const int bias = (f == CHAM_W_INT8_SYM || f == CHAM_W_MXINT8) ? 0x80
                   : ((f == CHAM_W_INT4_SYM || f == CHAM_W_MXINT4) ? 0x8 : 0);
#pragma unroll
  for (int i = 0; i < 8; ++i) code[i] = (code[i] & (a.bits == 8 ? 0xFF : 0xF)) ^ bias;
  const size_t off = code_offset(p, v * 8, a.n_chunks, a.bits);
  if (a.bits == 8) {
    uint32_t lo = 0, hi = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      lo |= (static_cast<uint32_t>(code[i]) & 0xFFu) << (8 * i);
      hi |= (static_cast<uint32_t>(code[4 + i]) & 0xFFu) << (8 * i);
    }
    *reinterpret_cast<uint2*>(a.codes + off) = make_uint2(lo, hi);
  } else {
    uint32_t w = 0;
    if (f == CHAM_W_NF4) {
#pragma unroll
      for (int j = 0; j < 8; ++j) w |= (static_cast<uint32_t>(code[j]) & 0xFu) << (4 * j);
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        w |= (static_cast<uint32_t>(code[2 * j]) & 0xFu) << (4 * j);
        w |= (static_cast<uint32_t>(code[2 * j + 1]) & 0xFu) << (4 * (j + 4));
      }
    }
    *reinterpret_cast<uint32_t*>(a.codes + off) = w;
  }
}

// ------------------------------------------------------------------ group-wise formats (Sec. 3.5 forks)
struct GroupParam {  // scale, reciprocal and zero point of one group of one row
  float s, inv;
  int z;
};

// Statistics of elements [k0, k1) of a row, by one lane (k0, k1 multiples of 8).
CHAM_DEV ChanStats range_stats(const __half* row, int k0, int k1) {
  float amax = 0.f, lo = INFINITY, hi = -INFINITY;
  for (int v = k0 / 8; v < k1 / 8; ++v) {
    float x[8];
    load8(row, v, x);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      amax = fmaxf(amax, fabsf(x[i]));
      lo = fminf(lo, x[i]);
      hi = fmaxf(hi, x[i]);
    }
  }
  return ChanStats{amax, lo, hi};
}

// The scale rule of format f on every group of g elements of a row (lane j takes groups j, j + 32,
// ...), into this warp's shared-memory table.
CHAM_DEV void group_params(const __half* row, int K, int g, int f, int lane, GroupParam* gp) {
  const int ng = (K + g - 1) / g;
  for (int j = lane; j < ng; j += 32) {
    const ChanScale cs = chan_scale(f, range_stats(row, j * g, min((j + 1) * g, K)));
    gp[j] = GroupParam{cs.s, cs.inv, cs.z};
  }
  __syncwarp();
}

// The value a non-MX code stands for, before its scale: q (sym), q - z (asym), the NF4 level,
// the E2M1 value.
CHAM_DEV float code_value(int f, int code, int z, const NF4Table& nf4) {
  switch (f) {
    case CHAM_W_INT8_ASYM:
    case CHAM_W_INT4_ASYM: return static_cast<float>(code - z);
    case CHAM_W_NF4: return __half2float(__ushort_as_half(nf4.level[code]));
    case CHAM_W_E2M1: return e2m1_value(static_cast<uint32_t>(code));
    default: return static_cast<float>(code);
  }
}

// Encodes packed slot p holding original channel c (-1: padding) in format f (one warp).
CHAM_DEV void pack_slot(const PackArgs& a, int p, int c, int f, int lane, const NF4Table& nf4, GroupParam* s_gp_warp,
                        const ChanStats* pre = nullptr) {
  const int nvec_p = a.Kp / 8;
  const int tile = p >> 7, r = p & 127;
  if (c < 0) {  // padding slot: zero codes, unit scale
    for (int v = lane; v < nvec_p; v += 32) {
      const size_t off = code_offset(p, v * 8, a.n_chunks, a.bits);
      if (a.bits == 8) *reinterpret_cast<uint2*>(a.codes + off) = make_uint2(0, 0);
      else *reinterpret_cast<uint32_t*>(a.codes + off) = 0u;
    }
    for (int ch = lane; ch < a.n_chunks; ch += 32) {
      const size_t e = ((static_cast<size_t>(tile) * a.n_chunks + ch) * 128 + r) * 2;
      a.e8m0[e] = 127;
      a.e8m0[e + 1] = 127;
      if (a.gscale != nullptr) a.gscale[e / 2] = 0u;
    }
    if (lane == 0) {
      a.scale[p] = 1.f;
      a.zero[p] = 0;
    }
    return;
  }
  const __half* row = a.W + static_cast<size_t>(c) * a.K;
  const int nvec = a.K / 8;
  if (a.group > 0) {
    // group-wise: codes with their group's parameters; per 32-element block its zero point (in
    // the E8M0 slot) and its group's scale as fp16; the per-channel scale is 1
    if (lane == 0 && a.desc.n_fmt[f] != a.N) set_status(a.dev_status, CHAM_ERR_INVALID_ARG);  // one format per plan
    GroupParam* gp = s_gp_warp;
    group_params(row, a.K, a.group, f, lane, gp);
    const bool asym = f == CHAM_W_INT8_ASYM || f == CHAM_W_INT4_ASYM;
    for (int v = lane; v < nvec_p; v += 32) {
      int code[8] = {0, 0, 0, 0, 0, 0, 0, 0};
      GroupParam q{0.f, 1.f, 0};  // beyond K: code 0, zero point 0, scale 0 -> the value 0
      if (v < nvec) {
        q = gp[(v * 8) / a.group];
        float x[8];
        load8(row, v, x);
        const ChanScale cs{q.s, q.inv, q.z};
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          float err;
          code[i] = encode_chan(f, x[i], cs, nf4, &err);
        }
      }
      store_codes(a, p, v, f, code);
      if ((v & 3) == 0) {
        const int k0 = v * 8;
        const size_t e = ((static_cast<size_t>(tile) * a.n_chunks + (k0 >> 6)) * 128 + r) * 2 + ((k0 & 63) >> 5);
        a.e8m0[e] = asym ? static_cast<uint8_t>(q.z) : 0;
        reinterpret_cast<__half*>(a.gscale)[e] = __float2half_rn(v < nvec ? q.s : 0.f);
      }
    }
    if (lane == 0) {
      a.scale[p] = 1.f;
      a.zero[p] = 0;
    }
    return;
  }
  const ChanStats st = pre != nullptr ? *pre : row_stats(row, nvec, lane);  // the selection's, when fused
  const ChanScale cs = chan_scale(f, st);
  const bool mx = w_is_mx(f);
  const int iters = (nvec_p + 31) / 32;
  bool range_ok = true;
  for (int it = 0; it < iters; ++it) {
    const int v = it * 32 + lane;
    float x[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    if (v < nvec) load8(row, v, x);
    int code[8];
    int X = 0;
    if (mx) {
      float am = 0.f;
#pragma unroll
      for (int i = 0; i < 8; ++i) am = fmaxf(am, fabsf(x[i]));
      am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, 1));
      am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, 2));
      X = mx_exponent(f, am);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        float dq;
        code[i] = encode_mx(f, x[i], X, &dq);
        // the GEMM's fp16 operand must equal DQ exactly (R13)
        range_ok &= (__half2float(__float2half_rn(dq)) == dq);
      }
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        float err;
        code[i] = encode_chan(f, x[i], cs, nf4, &err);
      }
    }
    if (v >= nvec_p) continue;
    if (v >= nvec) {  // K padding up to a multiple of 64: the value 0
#pragma unroll
      for (int i = 0; i < 8; ++i) code[i] = f == CHAM_W_INT8_ASYM || f == CHAM_W_INT4_ASYM ? cs.z : 0;
    }
    store_codes(a, p, v, f, code);
    if ((lane & 3) == 0) {  // one E8M0 byte per 32-element block
      const int k0 = v * 8;
      const size_t e = ((static_cast<size_t>(tile) * a.n_chunks + (k0 >> 6)) * 128 + r) * 2 + ((k0 & 63) >> 5);
      a.e8m0[e] = mx ? static_cast<uint8_t>(X + 127) : 127;
    }
  }
  if (mx && !range_ok) set_status(a.dev_status, CHAM_ERR_RANGE);
  if (lane == 0) {
    a.scale[p] = mx ? 1.f : cs.s;
    a.zero[p] = static_cast<uint8_t>(cs.z);
  }
}

__global__ void __launch_bounds__(kWThreads) k_w_pack(PackArgs a, NF4Table nf4) {
  __shared__ GroupParam s_gp[kWWarps][kMaxRowGroups];
  if (blockIdx.x == 0 && threadIdx.x < 64)  // the blob's header: a copy of the descriptor
    reinterpret_cast<uint32_t*>(a.desc_out)[threadIdx.x] = reinterpret_cast<const uint32_t*>(&a.desc)[threadIdx.x];
  const int lane = threadIdx.x & 31;
  const int p = blockIdx.x * kWWarps + (threadIdx.x >> 5);  // one warp per packed slot
  if (p >= a.n_packed) return;
  int c;
  if (a.one_class >= 0) {
    // one MMA class: slot p holds channel p - base in original order, the rest is padding
    const int rank = p - a.cls_base[a.one_class];
    c = (rank >= 0 && rank < a.cls_count[a.one_class]) ? rank : -1;
    if (lane == 0) {
      const int f = c >= 0 ? a.fmt_dev[c] : -1;
      const bool valid = f >= 0 && f < CHAM_W_NFORMATS && w_class(f) == a.one_class;
      if (c >= 0 && !valid) set_status(a.dev_status, CHAM_ERR_INVALID_ARG);  // formats must match the plan
      a.perm[p] = c;
      a.fmtp[p] = c >= 0 ? static_cast<uint8_t>(valid ? f : 0xFF) : static_cast<uint8_t>(0xFF);
    }
    __syncwarp();
    if (c >= 0 && (a.fmtp[p] == 0xFF)) return;  // invalid format: nothing to encode
  } else {
    c = a.perm[p];
  }
  pack_slot(a, p, c, c >= 0 ? a.fmtp[p] : -1, lane, nf4, s_gp[threadIdx.x >> 5]);
}

// Selection and pack in one pass for a one-class plan (slot = channel): the warp that selects
// channel c's format (Sec. 3.4) encodes the channel right away, so the row is read from DRAM once
// and one launch serves both steps.
__global__ void __launch_bounds__(kWThreads) k_w_select_pack(PackArgs a, uint32_t mask, NF4Table nf4) {
  if (blockIdx.x == 0 && threadIdx.x < 64)  // the blob's header: a copy of the descriptor
    reinterpret_cast<uint32_t*>(a.desc_out)[threadIdx.x] = reinterpret_cast<const uint32_t*>(&a.desc)[threadIdx.x];
  const int lane = threadIdx.x & 31;
  const int p = blockIdx.x * kWWarps + (threadIdx.x >> 5);
  if (p >= a.n_packed) return;
  const int rank = p - a.cls_base[a.one_class];
  const int c = (rank >= 0 && rank < a.cls_count[a.one_class]) ? rank : -1;
  int f = -1;
  ChanStats st{0.f, 0.f, 0.f};
  if (c >= 0) f = select_row(a.W + static_cast<size_t>(c) * a.K, a.K, mask, lane, nf4, nullptr, &st);
  if (lane == 0) {
    if (c >= 0) a.fmt_out[c] = static_cast<uint8_t>(f);
    a.perm[p] = c;
    a.fmtp[p] = c >= 0 ? static_cast<uint8_t>(f) : static_cast<uint8_t>(0xFF);
  }
  pack_slot(a, p, c, f, lane, nf4, nullptr, &st);
}

void launch_select_pack(const PackArgs& a, uint32_t mask, const NF4Table& nf4, cudaStream_t st) {
  k_w_select_pack<<<(a.n_packed + kWWarps - 1) / kWWarps, kWThreads, 0, st>>>(a, mask, nf4);
}

// ------------------------------------------------------------------ (g, f) search (Sec. 3.5 forks)
__global__ void __launch_bounds__(256) k_energy_f32(const double* __restrict__ energy, int K, float* __restrict__ out) {
  for (int k = blockIdx.x * blockDim.x + threadIdx.x; k < K; k += gridDim.x * blockDim.x)
    out[k] = energy != nullptr ? static_cast<float>(energy[k]) : 1.f;
}

// Per channel (one warp) and candidate: sum_k e_k (w - DQ(w))^2, with the element error rounded
// once to fp32, weighted and squared in fp32, summed in fp32 over 8 elements, then in fp64.
__global__ void __launch_bounds__(kWThreads) k_w_select_groups(GroupSearchArgs a, NF4Table nf4) {
  __shared__ GroupParam s_gp[kWWarps][kMaxRowGroups];
  const int lane = threadIdx.x & 31;
  const int c = blockIdx.x * kWWarps + (threadIdx.x >> 5);
  if (c >= a.N) return;  // whole warps: no block-wide barrier follows
  GroupParam* gp = s_gp[threadIdx.x >> 5];
  const __half* row = a.W + static_cast<size_t>(c) * a.K;
  const int nvec = a.K / 8;
  const int iters = (nvec + 31) / 32;  // same trip count in every lane (shuffles)
  for (int ci = 0; ci < a.n_cand; ++ci) {
    const int g = a.cand[ci].g, f = a.cand[ci].f;
    Sum2 acc{0.f, 0.f};
    if (w_is_mx(f)) {
      for (int it = 0; it < iters; ++it) {
        const int v = it * 32 + lane;
        float x[8] = {0, 0, 0, 0, 0, 0, 0, 0};
        if (v < nvec) load8(row, v, x);
        float am = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) am = fmaxf(am, fabsf(x[i]));
        am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, 1));  // 4 lanes = one 32-element block
        am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, 2));
        const int X = mx_exponent(f, am);
        if (v < nvec) {
          float e2[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            float dq;
            encode_mx(f, x[i], X, &dq);
            const float e = __fsub_rn(x[i], dq);
            e2[i] = __fmul_rn(__fmul_rn(e, e), a.energy32[v * 8 + i]);
          }
          sum2_add(acc, sum8(e2));
        }
      }
    } else {
      __syncwarp();  // the previous candidate's table is no longer read
      group_params(row, a.K, g, f, lane, gp);
      for (int v = lane; v < nvec; v += 32) {
        const GroupParam q = gp[(v * 8) / g];
        const ChanScale cs{q.s, q.inv, q.z};
        const float s16 = __half2float(__float2half_rn(q.s));
        float x[8], e2[8];
        load8(row, v, x);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          float err;
          const int code = encode_chan(f, x[i], cs, nf4, &err);
          // DQ = fp16(value * fp16(s)): the product of two fp16 values is exact in fp32
          const float dq = __half2float(__float2half_rn(__fmul_rn(code_value(f, code, q.z, nf4), s16)));
          const float e = __fsub_rn(x[i], dq);
          e2[i] = __fmul_rn(__fmul_rn(e, e), a.energy32[v * 8 + i]);
        }
        sum2_add(acc, sum8(e2));
      }
    }
    const double tot = warp_sum2(acc);
    if (lane == 0) a.parts[static_cast<size_t>(c) * a.n_cand + ci] = tot;
  }
}

// scores[i] = sum over channels, in channel order, of the per-channel errors of candidate i.
__global__ void __launch_bounds__(64) k_w_select_groups_finish(GroupSearchArgs a) {
  for (int ci = threadIdx.x; ci < a.n_cand; ci += blockDim.x) {
    double t = 0.0;
    for (int c = 0; c < a.N; ++c) t += a.parts[static_cast<size_t>(c) * a.n_cand + ci];
    a.scores[ci] = t;
  }
}

void launch_select_groups(const GroupSearchArgs& a, const NF4Table& nf4, cudaStream_t st) {
  k_energy_f32<<<(a.K + 255) / 256, 256, 0, st>>>(a.energy, a.K, a.energy32);
  k_w_select_groups<<<(a.N + kWWarps - 1) / kWWarps, kWThreads, 0, st>>>(a, nf4);
  k_w_select_groups_finish<<<1, 64, 0, st>>>(a);
}

// energy[k] += sum_m x[m, k]^2.  A CTA of 32 x 32 threads owns 32 column vectors (lane = vector,
// warp = one of 32 row strides); each thread sums its rows' squares in fp32 over runs of 8 rows
// and in fp64 across runs; the 32 row strides are then added in warp order (deterministic).
__global__ void __launch_bounds__(1024) k_channel_energy(const __half* __restrict__ X, int M, int K,
                                                        double* __restrict__ energy) {
  __shared__ double sh[32][33];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nv = K / 8;
  const int v = blockIdx.x * 32 + lane;
  double acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  if (v < nv) {
    for (int m0 = warp * 8; m0 < M; m0 += 32 * 8) {
      float part[8] = {0, 0, 0, 0, 0, 0, 0, 0};
      for (int m = m0; m < min(m0 + 8, M); ++m) {
        float x[8];
        load8(X + static_cast<size_t>(m) * K, v, x);
#pragma unroll
        for (int i = 0; i < 8; ++i) part[i] = __fadd_rn(part[i], __fmul_rn(x[i], x[i]));
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] += static_cast<double>(part[i]);
    }
  }
#pragma unroll 1
  for (int i = 0; i < 8; ++i) {
    sh[warp][lane] = acc[i];
    __syncthreads();
    if (warp == 0 && v < nv) {
      double t = 0.0;
      for (int w = 0; w < 32; ++w) t += sh[w][lane];
      energy[v * 8 + i] += t;
    }
    __syncthreads();
  }
}

void launch_channel_energy(const __half* X, int M, int K, double* energy, cudaStream_t st) {
  k_channel_energy<<<(K / 8 + 31) / 32, 1024, 0, st>>>(X, M, K, energy);
}

void launch_pack(const PackArgs& a, const NF4Table& nf4, cudaStream_t st) {
  if (a.one_class < 0) k_w_slots<<<1, 1024, 0, st>>>(a);  // two classes: rank the channels of each
  k_w_pack<<<(a.n_packed + kWWarps - 1) / kWWarps, kWThreads, 0, st>>>(a, nf4);
}

}  // namespace cham
