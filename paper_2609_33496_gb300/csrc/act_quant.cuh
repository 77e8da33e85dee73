// act_quant.cuh -- declarations shared by the activation-quantizer kernels and the host API.
#pragma once

#include <cuda_runtime.h>

#include "common.cuh"

namespace cham {

struct RangePartial {  // one CTA's min / max / non-finite flag of an activation tensor
  float lo, hi;
  int nonfinite, pad;
};

struct TensorParams {  // ScaleZP result of a per-tensor format
  float s, inv;
  int z;
};

struct MomentPartial {  // one CTA's power sums (Alg. 1 accumulator)
  double s[4];
  float lo, hi;
};

struct ActQuantArgs {
  const uint4* X;          // fp16 tensor, 8 elements per vector
  int64_t nvec;            // M*K/8
  RangePartial* parts;     // per-tensor formats: range partials (scratch), nparts per group
  int nparts;              // range CTAs per group: range_grid (one group) or group_grid
  int n_groups;            // per-sample scales: rows in n_groups equal groups (0 or 1: per tensor)
  uint2* codes;            // 8 code bytes per vector, or null
  uint4* deq;              // 8 exact fp16 operand values per vector, or null
  uint8_t* e8m0;           // MX formats: one byte per 4 vectors, or null
  uint8_t* e8cm;           // MX formats, FP8 GEMM operand: the same bytes chunk-major, or null:
                           // block kb of row m at e8cm[(kb / 4) * cm_plane + 4 m + kb % 4]
  int kblocks;             // K / 32 (blocks per row), with e8cm
  int64_t cm_plane;        // bytes per chunk of 4 blocks in e8cm
  bool kperm;              // codes of each 8-element group stored in the order 0, 2, 4, 6, 1, 3, 5, 7
                           // (the FP8 GEMM operand: the order in which the 4-bit weight codes
                           // decode; both operands permuted alike leave the dot product unchanged)
  cham_qparams* params;    // per-tensor parameters, or null
  float* scale_out;        // the per-tensor (per-group) scale s as bare floats (GEMM epilogue), or null
  int* dev_status;
  int num_sms;
  bool use_static;         // per-tensor formats: encode with `stat` (Alg. 2), no range pass
  TensorParams stat;
};

int range_grid(int64_t nvec, int num_sms);
// CTAs per group when nvec vectors are split into n_groups groups (at least 1)
int group_grid(int64_t nvec, int n_groups, int num_sms);
constexpr int kMaxGroups = 64;  // per-sample groups: the scale slots of the linear workspace
void launch_act_quant(int fmt, const ActQuantArgs& a, bool codes, bool deq, cudaStream_t st);
// Eq. format-argmin: range pass, per-CTA SSE of the five activation formats (nparts CTAs, 5
// doubles each in sse_parts), then a one-CTA sum added to out[0..4].
void launch_act_format_sse(const uint4* X, int64_t nvec, RangePartial* parts, int nparts, double* sse_parts,
                           double* out, int* dev_status, cudaStream_t st);
void launch_act_moments(const uint4* X, int64_t nvec, int64_t count, MomentPartial* parts, int nparts,
                        double* out, cudaStream_t st);

}  // namespace cham
