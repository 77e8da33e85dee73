/*
 * chameleon.h -- C ABI of the Chameleon format-adaptive quantized linear layer on GB300 (sm_103a).
 *
 * Method: arXiv 2609.33496 ("Chameleon: Dynamic Format Adapter for Efficient Diffusion").
 * Activations are quantized per tensor in the format a per-(layer, timestep-bucket) table picks
 * (Sec. 3.2-3.3, Alg. 2/3); every weight output channel carries its own format, chosen offline by
 * reconstruction error (Sec. 3.4); the layer multiplies the two on tcgen05 tensor cores.
 *
 * Conventions (all entry points):
 *   - every call returns a cham_status; CHAM_OK is 0.  chameleon_last_error_detail() gives a
 *     one-line message for the last failure on the calling host thread.
 *   - pointers marked (device) are CUDA device pointers owned by the caller; (host) are host
 *     pointers.  The library never allocates device memory: size queries come first and the caller
 *     passes buffers of at least the returned size.
 *   - calls are asynchronous on `stream` (a cudaStream_t passed as void*; NULL = legacy stream) and
 *     never synchronise, except where a host value is computed.  Errors detected by the kernels
 *     (non-finite input, a wait that timed out, an MX weight outside fp16) are written to the
 *     caller's device status word `dev_status` (int32, device): the kernels only ever store a
 *     non-zero cham_status there; the caller zeroes it and reads it after synchronising.
 *   - X is fp16, M x K, row-major (K contiguous); W is fp16, N x K (nn.Linear layout); Y is fp32
 *     M x N row-major; bias is fp32 [N].  Row pitches are exactly K (resp. N) elements.
 *   - all device pointers must be 16-byte aligned; K must be a multiple of 32.
 */
#ifndef CHAMELEON_H
#define CHAMELEON_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int cham_status;
#define CHAM_OK 0
#define CHAM_ERR_INVALID_ARG 1  /* bad size, pointer, alignment or format code (host check) */
#define CHAM_ERR_UNSUPPORTED 2  /* a valid request this build does not handle */
#define CHAM_ERR_WORKSPACE 3    /* a buffer is smaller than its size query returned */
#define CHAM_ERR_NONFINITE 4    /* device: the activation tensor holds Inf or NaN */
#define CHAM_ERR_TIMEOUT 5      /* device: a bounded wait inside a kernel gave up */
#define CHAM_ERR_CUDA 6         /* a CUDA runtime/driver call failed */
#define CHAM_ERR_RANGE 7        /* device: an MX weight block does not decode exactly in fp16 */

/* Activation formats: the runtime LUT codes 0..4 of Sec. 3.2 (F_a), plus 5 = fp16 operands for the
 * weight-only few-step fork of Sec. 3.5. */
#define CHAM_A_INT8_ASYM 0
#define CHAM_A_E4M3 1
#define CHAM_A_E5M2 2
#define CHAM_A_MXFP8 3
#define CHAM_A_MXINT8 4
#define CHAM_A_FP16 5

/* Weight formats (Sec. 3.2: F_w^(8) and F_w^(4), in palette order = tie-break order). */
#define CHAM_W_INT8_SYM 0
#define CHAM_W_INT8_ASYM 1
#define CHAM_W_MXINT8 2
#define CHAM_W_INT4_SYM 3
#define CHAM_W_INT4_ASYM 4
#define CHAM_W_NF4 5
#define CHAM_W_E2M1 6
#define CHAM_W_MXINT4 7
#define CHAM_W_MXFP4 8
#define CHAM_W_NFORMATS 9
#define CHAM_PALETTE_W8 0x007u   /* INT8-sym, INT8-asym, MXINT8 */
#define CHAM_PALETTE_W4 0x1F8u   /* INT4-sym, INT4-asym, NF4, E2M1, MXINT4, MXFP4 */

/* Output element types of chameleon_linear_gemm_ex. */
#define CHAM_Y_F32 0
#define CHAM_Y_F16 1
#define CHAM_Y_BF16 2
/* Most row groups (samples) of chameleon_linear_prepare_groups. */
#define CHAM_MAX_GROUPS 64

/* Noise schedules for chameleon_snr (App. A.1, A.11): scaled-linear (SDXL, beta 0.00085 -> 0.012)
 * and linear (PixArt-alpha, beta 1e-4 -> 0.02). */
#define CHAM_SCHEDULE_SCALED_LINEAR 0
#define CHAM_SCHEDULE_LINEAR 1

/* Static name of a status code ("ok", "invalid argument", ...); "unknown status" for other values. */
const char* chameleon_status_string(cham_status s);
/* One-line description of the last failed call on the calling host thread (a thread-local
 * buffer, empty before any failure; its contents change at that thread's next failing call). */
const char* chameleon_last_error_detail(void);

/* Waits for the work queued on `stream` (a cudaStream_t; NULL = the legacy default stream) and
 * returns the device status word dev_status (device int, written by the kernels of the calls
 * that were given it: 0 = CHAM_OK, else the first device-detected error, e.g.
 * CHAM_ERR_NONFINITE or CHAM_ERR_TIMEOUT).  The word is left as it is.  CHAM_ERR_CUDA when the
 * synchronisation or the copy fails; CHAM_ERR_INVALID_ARG when dev_status is NULL. */
cham_status chameleon_check(const int* dev_status, void* stream);
/* ABI version of this library: 3 (packed-weight descriptors with group-wise weights and the MMA
 * path switch; the linear prepare calls take the descriptor). */
int chameleon_version(void);

/* ------------------------------------------------------------------ host helpers (a1, L2) */

/* Bucket of timestep t: b = min(floor(t / (T/B)), B-1) (Alg. 2 and Alg. 3).  Returns -1 when
 * T <= 0, B <= 0 or t < 0. */
int chameleon_bucket(int t, int T, int B);

/* SNR(t) = abar_t / (1 - abar_t), abar_t = prod_{s<=t} (1 - beta_s), t = 0..T-1 (Sec. 2.1,
 * Eq. snr).  snr_out (host) receives T doubles. */
cham_status chameleon_snr(int schedule, int T, double* snr_out);

/* Kurtosis kappa = m4 / m2^2 from the power sums {n, S1, S2, S3, S4} (App. A.2 Eq. kurt, Alg. 1);
 * 0 when the variance is 0. */
double chameleon_kurtosis(const double sums[5]);

/* Routing rule of Sec. 3.3 at SNR(t_b): shortcut -> MXFP8; kappa > 5 or snr < 0.2 -> E5M2;
 * kappa <= 3 and snr > 2 -> INT8-asym; else E4M3.  Returns an activation format code. */
int chameleon_route(double kappa, double snr_b, int is_shortcut);

/* ------------------------------------------------------------------ calibration statistics */

/* Power sums of one activation tensor, the accumulator of Alg. 1 (Sec. 3.5):
 * out (device, 7 doubles) = {n, sum x, sum x^2, sum x^3, sum x^4, min, max}, ADDED to what `out`
 * holds for n and the sums, min/max merged (so calls accumulate across steps like Alg. 1; zero
 * the first five and set min = +inf, max = -inf before the first call).  X fp16 (device), count
 * elements.  ws (device) >= chameleon_act_moments_workspace_size bytes. */
cham_status chameleon_act_moments_workspace_size(int64_t count, size_t* ws_bytes);
cham_status chameleon_act_moments(const void* X, int64_t count, double* out, void* ws,
                                  size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------ a2-a4: activation quantizer */

/* Quantized-activation buffer layout (qact, device), for fmt in 0..4:
 *   [0, M*K)                codes, uint8 row-major: INT8-asym q; E4M3 / E5M2 / MXFP8 bit pattern;
 *                           MXINT8 two's-complement int8
 *   [P, P+16), P = round_up(M*K, 256): cham_qparams {float s; int32 z; float inv; int32 fmt}
 *                           (per-tensor formats; MX formats store s = 1, z = 0, inv = 1)
 *   [P+256, P+256+M*K/32)   E8M0 block exponents, uint8 M x (K/32) row-major (MX formats only)
 * Dequantized value: INT8-asym (q - z) * s; E4M3/E5M2 value(code) * s; MXFP8 value(code) * 2^(e-127);
 * MXINT8 code * 2^-6 * 2^(e-127)  (App. A.7 ScaleZP, App. A.11).  MX shared exponent floor(log2 amax) - emax
 * of the element body (8 for E4M3, 0 for the int8 body); an all-zero block has E8M0 byte 0. */
typedef struct {
  float s;
  int32_t z;
  float inv;
  int32_t fmt;
} cham_qparams;

/* Size query for chameleon_act_quant: *qact_bytes of the layout above and *ws_bytes of scratch
 * (0 for the MX formats; either pointer may be NULL).  Host only.  CHAM_ERR_INVALID_ARG for
 * M, K <= 0, K not a multiple of 32 or fmt outside 0..4. */
cham_status chameleon_act_quant_size(int M, int K, int fmt, size_t* qact_bytes, size_t* ws_bytes);

/* Quantize X (device, fp16 M x K) in activation format fmt with its own dynamic range (Alg. 3:
 * lo, hi = min x, max x; ScaleZP; fq_f).  Writes qact (device, qact_bytes); ws (device) is
 * scratch of ws_bytes.  Non-finite input sets *dev_status = CHAM_ERR_NONFINITE (codes then
 * unspecified). */
cham_status chameleon_act_quant(const void* X, int M, int K, int fmt, void* qact, size_t qact_bytes,
                                void* ws, size_t ws_bytes, int* dev_status, void* stream);

/* ScaleZP of a per-tensor format (0..2) from a range [lo, hi] (App. A.7; the helper Alg. 1 uses
 * when it stores the scale of each layer and bucket from the calibration range, and the one the
 * quantizer applies to a tensor's own range in Alg. 3).  INT8-asym: s = (hi' - lo')/255,
 * inv = 255/(hi' - lo'), z = round_half_even(-lo' * inv) clamped to [0, 255], where lo' = min(lo, 0),
 * hi' = max(hi, 0); E4M3 / E5M2: s = amax/Fmax, inv = Fmax/amax, z = 0 (amax = max(|lo|, |hi|),
 * Fmax 448 / 57344); a degenerate range gives s = inv = 1, z = 0.  Each step is one fp32 operation
 * rounded to nearest, as the device quantizer computes it, so the same range gives the same bits.
 * Host only (out is host memory).  CHAM_ERR_INVALID_ARG for another format, a non-finite or
 * reversed range (lo > hi), or a range whose width overflows fp32. */
cham_status chameleon_scale_zp(int fmt, float lo, float hi, cham_qparams* out);

/* The static path of Alg. 2: quantize X (device, fp16 M x K) with the per-tensor parameters
 * *params (host; made by chameleon_scale_zp from the calibration range of this layer and bucket)
 * instead of X's own range: one pass, no workspace.  Values outside that range clamp to codes 0 /
 * 255 (INT8-asym) or saturate to +-Fmax (FP8).  The qact layout and the stored cham_qparams are
 * those of chameleon_act_quant.  MX formats (3, 4) have no per-tensor parameters: params is
 * ignored (may be NULL) and the result equals chameleon_act_quant's.  CHAM_ERR_INVALID_ARG when
 * params is NULL for fmt 0..2, its fmt field differs, s or inv is not finite and positive, or z is
 * outside the format's range (0..255 for INT8-asym, 0 for FP8).  Non-finite input sets
 * *dev_status = CHAM_ERR_NONFINITE (codes then unspecified). */
cham_status chameleon_act_quant_static(const void* X, int M, int K, int fmt, const cham_qparams* params,
                                       void* qact, size_t qact_bytes, int* dev_status, void* stream);

/* ------------------------------------------------------------------ Eq. format-argmin */

/* The exhaustive activation-format choice of Eq. format-argmin (Sec. 3.1), the objective that the
 * kappa / SNR route approximates: for one activation tensor X (device, fp16 M x K, K a multiple of
 * 32), SSE_f = sum over the elements of (x - DQ_f(Q_f(x)))^2 for the five activation formats f =
 * 0..4 at their native granularity -- INT8-asym, E4M3, E5M2 with ScaleZP of X's own range (as
 * chameleon_act_quant), MXFP8 and MXINT8 per 32-element block -- ADDED to sse (device, 5 doubles),
 * so that calls accumulate over the calibration tensors of one (layer, bucket).  Each element's
 * error is one fp32 fused multiply-add, squared and summed in fp32 over 8 elements, then in fp64
 * in a fixed order (deterministic).  ws (device) >= the size query.  Non-finite input sets
 * *dev_status = CHAM_ERR_NONFINITE (sums then unspecified). */
cham_status chameleon_act_format_sse_workspace_size(int M, int K, size_t* ws_bytes);
cham_status chameleon_act_format_sse(const void* X, int M, int K, double* sse, void* ws, size_t ws_bytes,
                                     int* dev_status, void* stream);
/* f* = the first format with the least accumulated error (host, sse = 5 doubles; ties go to the
 * earlier format in palette order); -1 when sse is NULL. */
int chameleon_act_format_argmin(const double* sse);

/* ------------------------------------------------------------------ a5: weight-format selection */

/* Per output channel c of W (device, fp16 N x K): SSE_f(c) = sum_k (w - DQ_f(Q_f(w)))^2 for every
 * format f in palette_mask (bits = weight format codes; all members of one bit width), and
 * fmt_out[c] (device, uint8 [N]) = argmin, first in palette order on ties (Sec. 3.4, Eq.
 * weight-argmax: the SQNR argmax is the SSE argmin).  sse_out (device, double N x 9, row c holds
 * the 9 format slots, +inf for non-members) may be NULL. */
cham_status chameleon_select_weight_formats(const void* W, int N, int K, uint32_t palette_mask,
                                            uint8_t* fmt_out, double* sse_out, void* stream);

/* The per-linear (g, f) search of the DiT and few-step forks (Sec. 3.5).  Candidates, in search
 * order (ties go to the earlier): for each group size g of group_mask (bit i = g_i of {32, 64,
 * 128, 192, 288}, ascending), the non-MX members of palette_mask in palette order, and at g = 32
 * the MX members too (their own 32-element blocks); chameleon_group_candidates lists them.
 * scores (device, double [n_candidates]) = sum over channels c and input channels k of
 * e_k * (w - DQ(w))^2 with DQ the group-wise decode (fp16 scale, product rounded to fp16) or the
 * MX decode, e_k = energy[k] (device, double [K], e.g. chameleon_act_channel_energy sums over
 * calibration activations: the input-aware SQNR) or 1 when energy is NULL.  The SQNR argmax is
 * the score argmin (the signal term is the same for all candidates): chameleon_candidate_argmin.
 * Each element error is one fp32 fma, weighted and squared in fp32, summed in fp32 over 8
 * elements, then in fp64 in a fixed order.  K a multiple of 32, at most 256 groups per row.
 * ws (device) >= the size query. */
cham_status chameleon_group_candidates(uint32_t palette_mask, uint32_t group_mask, int* g_out, int* fmt_out,
                                       int cap, int* n_out);
cham_status chameleon_select_weight_groups_workspace_size(int N, int K, uint32_t palette_mask, uint32_t group_mask,
                                                          size_t* ws_bytes);
cham_status chameleon_select_weight_groups(const void* W, int N, int K, uint32_t palette_mask, uint32_t group_mask,
                                           const double* energy, double* scores, void* ws, size_t ws_bytes,
                                           void* stream);
/* Index of the first smallest of n scores (host); -1 when n <= 0 or scores is NULL. */
int chameleon_candidate_argmin(const double* scores, int n);

/* Activation energy per input channel for the input-aware SQNR: energy[k] += sum_m x[m, k]^2
 * (device, double [K]) over X (device, fp16 M x K, K a multiple of 8), so calls accumulate over
 * calibration tensors.  Deterministic (fixed summation order). */
cham_status chameleon_act_channel_energy(const void* X, int M, int K, double* energy, void* stream);

/* ------------------------------------------------------------------ a6: weight pack */

/* Packed-weight descriptor.  Channels are reordered (Sec. 5 proposes a permutation that groups
 * the channels of one format so that each group runs as its own GEMM) into two MMA classes, each
 * padded to 128-channel tiles:
 *   class 0 = 4-bit formats with an 8-bit tensor-core path (INT4-sym, INT4-asym, E2M1, MXINT4,
 *             MXFP4), class 1 = the rest (NF4, INT8-sym, INT8-asym, MXINT8);
 * inside a class in original channel order (a tile's output columns stay contiguous; the GEMM
 * decodes each channel in its own format).  Offsets are from the blob base, 256-byte aligned.
 * Blob regions:
 *   [0, 256)       a copy of this descriptor
 *   codes          per tile t (128 packed channels) and K-chunk c (64 elements): 128 * CB bytes,
 *                  CB = 64 (8-bit) or 32 (4-bit) bytes per channel, stored as CB/16 slabs of
 *                  128 x 16 bytes: slab j holds bytes [16j, 16j+16) of every channel's CB bytes.
 *                  8-bit: byte i = element i of the chunk (offset binary q + 128 for INT8-sym
 *                  and MXINT8, uint8 q for INT8-asym).  4-bit: each 32-bit word holds 8 elements
 *                  e0..e7, nibble j (bits 4j..4j+3) = e_{2j} for j < 4 and e_{2(j-4)+1} for j >= 4
 *                  (NF4 channels: nibble j = e_j); INT4-sym/MXINT4 offset binary q + 8, INT4-asym
 *                  q, NF4 level index, E2M1/MXFP4 bit pattern.  Elements k >= K hold the code of the value 0.  (Offset binary
 *                  lets the GEMM turn a code into its fp16 value with one byte permute and one
 *                  subtraction.)
 *   scale          float [Np]: per-channel scale s (1 for MX and padding)
 *   zero           uint8 [Np]: zero point z (asym formats, else 0)
 *   e8m0           uint8 [tiles][Kp/64][128][2]: the two E8M0 exponents of each channel's chunk
 *                  (MX formats; 127 otherwise).  Group-wise blobs (group > 0): the zero points
 *                  of the chunk's two 32-element blocks (asym formats, else 0)
 *   fmt            uint8 [Np]: format of each packed channel, 255 for padding
 *   perm           int32 [Np]: original channel of each packed channel, -1 for padding
 *   gscale         (group > 0 only) uint32 [tiles][Kp/64][128]: the fp16 scales of the chunk's
 *                  two 32-element blocks (block 0 in the low half), each its group's scale
 *                  rounded to fp16 (0 beyond K); the per-channel scale region then holds 1
 * with Np = 128 * (n_tiles[0] + n_tiles[1]) and Kp = K rounded up to 64.  A group-wise blob has
 * one non-MX format for every channel and a scale per run of `group` input channels (Sec. 3.5
 * forks); its weights decode to fp16(value(code) * scale16), the product rounded once. */
typedef struct {
  uint32_t magic;    /* 0x574D4843 ("CHMW") */
  uint32_t version;  /* 3 */
  int32_t N, K, Kp, bits;
  int32_t n_class[2];
  int32_t n_tiles[2];
  int32_t n_fmt[CHAM_W_NFORMATS];
  int32_t group;              /* 0: per-channel (or MX) formats; g > 0: group-wise, g input channels */
  uint64_t off_codes, off_scale, off_zero, off_e8m0, off_fmt, off_perm, bytes;
  uint64_t off_gscale;        /* group-wise blobs: the gscale region, else 0 */
  int32_t f16_only;           /* 0 (the plans' default): class-0 tiles multiply on the FP8 tensor cores
                                 when the activation format is E4M3, E5M2 or MXFP8 (see
                                 chameleon_linear); 1: every tile on fp16 MMAs.  The linear calls of
                                 one layer must see the same value (it fixes the workspace layout). */
  int32_t layout;             /* channel order inside each MMA class: 0 = original order (the class
                                 layout); 1 = format groups (chameleon_pack_plan_layout) */
  int32_t fold;               /* layout 1: a format with fewer channels than this shares its class's
                                 mixed tail group */
  uint8_t reserved[100];      /* pads the descriptor to 256 bytes */
} cham_wpack_desc;

/* Fill *desc for N x K weights whose selected formats are fmt_host (host, uint8 [N], all of one
 * bit width).  desc->bytes is the blob size. */
cham_status chameleon_pack_plan(int N, int K, const uint8_t* fmt_host, cham_wpack_desc* desc);

/* chameleon_pack_plan with a choice of channel order inside the MMA classes (Sec. 5: channels of
 * one format grouped behind a permutation).  layout 0 is chameleon_pack_plan: each class in
 * original channel order.  layout 1: format groups -- inside each class, the formats in palette
 * order (class 0: INT4-sym, INT4-asym, E2M1, MXINT4, MXFP4; class 1: NF4, INT8-sym, INT8-asym,
 * MXINT8), each format's channels in original order padded to whole 128-channel tiles, so that
 * every tile holds one format; formats with fewer than `fold` channels (fold >= 0) go together, in
 * original order, into one mixed tail group at the end of their class.  The GEMM calls take either
 * layout.  CHAM_ERR_INVALID_ARG as chameleon_pack_plan, or for layout outside 0..1 or fold < 0. */
cham_status chameleon_pack_plan_layout(int N, int K, const uint8_t* fmt_host, int layout, int fold,
                                       cham_wpack_desc* desc);

/* Selection (a5) and pack (a6) in one launch, for a palette whose members share one MMA class
 * (e.g. CHAM_PALETTE_W8): desc comes from chameleon_pack_plan_palette(N, K, palette_mask); the
 * warp that selects channel c's format encodes c right away.  Writes fmt_out (device, uint8 [N],
 * the formats chameleon_select_weight_formats would give) and the blob (device, as
 * chameleon_pack_weights would write it for those formats).  CHAM_ERR_INVALID_ARG when desc is not
 * a one-class plan of these N x K weights, or a palette member lies outside its class / width. */
cham_status chameleon_select_pack_palette(const void* W, int N, int K, uint32_t palette_mask,
                                          const cham_wpack_desc* desc, uint8_t* fmt_out, void* blob,
                                          size_t blob_bytes, int* dev_status, void* stream);

/* A group-wise plan (the DiT and few-step forks, Sec. 3.5): every channel in format fmt (a non-MX
 * format: INT8-sym, INT8-asym, INT4-sym, INT4-asym, NF4 or E2M1), one scale (and zero point) per
 * run of `group` input channels along K -- group a multiple of 32 with at most 256 groups per row
 * (the last group of a row is shorter when group does not divide K).  chameleon_pack_weights then
 * takes a device format array holding fmt for every channel.  CHAM_ERR_INVALID_ARG otherwise. */
cham_status chameleon_pack_plan_grouped(int N, int K, int fmt, int group, cham_wpack_desc* desc);

/* The same plan from the palette alone, for palettes whose members all share one MMA class (every
 * 8-bit palette; 4-bit palettes without NF4, or NF4 alone): the layout then depends only on N, K
 * and the bit width, so the selected formats need not be copied to the host and selection, pack
 * and the linear calls can run back to back on the stream (Sec. 5's permutation is the identity
 * up to padding).  desc->n_fmt[f] is -1 for every member (counts unknown on the host).  Returns
 * CHAM_ERR_UNSUPPORTED for a palette that spans both classes; CHAM_ERR_INVALID_ARG for an empty
 * mask, bits outside the 9 formats, mixed bit widths, or N, K <= 0 / K % 32 != 0.  Host-only. */
cham_status chameleon_pack_plan_palette(int N, int K, uint32_t palette_mask, cham_wpack_desc* desc);

/* Encode W (device, fp16 N x K) with each channel in fmt_dev[c] (device copy of the formats the
 * plan was made from) into blob (device, >= desc->bytes).  An MX channel whose dequantized values
 * are not all exact fp16 values sets *dev_status = CHAM_ERR_RANGE. */
cham_status chameleon_pack_weights(const void* W, const uint8_t* fmt_dev, const cham_wpack_desc* desc,
                                   void* blob, size_t blob_bytes, int* dev_status, void* stream);

/* ------------------------------------------------------------------ a7/a8: quantized linear */

/* Workspace (device) of the linear calls for M rows of the layer *desc in act_fmt: the activation
 * scales of up to CHAM_MAX_GROUPS row groups, the quantizer's range partials, the GEMM operands the
 * layer's tiles need -- the exact fp16 operand (M x K) for tiles on fp16 MMAs, the 1-byte codes
 * (M x K, plus for MXFP8 their E8M0 exponents chunk-major: [ceil(K/128)][round_up(M, 4)][4]) for
 * class-0 tiles on FP8 MMAs, neither for CHAM_A_FP16 -- and, when a GEMM launch splits K (a layer
 * whose 128-channel x token tiles are fewer than half the SMs and whose K spans at least 8
 * chunks), the fp32 partial sums of the K ranges, which a second kernel adds in order.  The size
 * depends on the current device's SM count. */
cham_status chameleon_linear_workspace_size(int M, const cham_wpack_desc* desc, int act_fmt,
                                            size_t* ws_bytes);

/* The kernels the linear calls launch for M rows of the layer *desc in act_fmt (host only, no GPU
 * work): *prepare_launches for chameleon_linear_prepare (is_static = 0, n_groups row groups) or
 * chameleon_linear_prepare_static (is_static = 1) -- 0 for CHAM_A_FP16, 1 for the static path and
 * the MX formats, 2 (range, encode) for a per-tensor format's dynamic scales -- and
 * *gemm_launches for chameleon_linear_gemm(_ex): 1, or 2 when the GEMM splits K (the partial sums'
 * reduction).  CHAM_ERR_INVALID_ARG as the size query, or for a NULL output pointer. */
cham_status chameleon_linear_launches(int M, const cham_wpack_desc* desc, int act_fmt, int n_groups, int is_static,
                                      int* prepare_launches, int* gemm_launches);

/* Y = DQ(Q_act_fmt(X)) . DQ(W)^T + bias: X (device, fp16 M x desc->K) is quantized in act_fmt
 * (= F[layer, bucket] resolved on the host, Alg. 2/3) with its own range, multiplied on tcgen05
 * tensor cores with the packed weights (device blob made from *desc, host), fp32 accumulation;
 * Y (device, fp32 M x desc->N) in original channel order.  bias (device, fp32 [N]) may be NULL.
 * act_fmt = CHAM_A_FP16 multiplies X itself (weight-only fork).  ws (device) >= the size query.
 * Which tensor cores multiply (Sec. 3.6: native FP8 and MX kernels): the class-0 tiles of a 4-bit
 * per-channel layout (INT4-sym, INT4-asym, E2M1, MXINT4, MXFP4 -- every decoded value an exact E4M3
 * number) against E4M3, E5M2 or MXFP8 activations run kind::mxf8f6f4 MMAs on the 1-byte codes,
 * with the MX exponents of both sides as block scale factors, unless desc->f16_only is set; every
 * other tile runs kind::f16 MMAs on exact fp16 operands.  Both give the same products; the sums
 * differ only in accumulation order. */
cham_status chameleon_linear(const void* X, int M, const cham_wpack_desc* desc, const void* blob,
                             int act_fmt, const float* bias, float* Y, void* ws, size_t ws_bytes,
                             int* dev_status, void* stream);

/* The two halves of chameleon_linear, for callers that schedule or time them separately.
 * chameleon_linear_prepare quantizes X (device, fp16 M x desc->K) in act_fmt into ws: the GEMM
 * operands that the layer *desc's tiles need (the exact fp16 value of every code, R13, and / or the
 * 1-byte codes, see chameleon_linear_workspace_size) plus the per-tensor scale; nothing for
 * CHAM_A_FP16.  chameleon_linear_gemm multiplies them (or X itself for CHAM_A_FP16; X may be NULL
 * otherwise) with the packed weights.  Same arguments, workspace and errors as chameleon_linear;
 * prepare and gemm of one layer take the same desc (its f16_only fixes which operands exist). */
cham_status chameleon_linear_prepare(const void* X, int M, const cham_wpack_desc* desc, int act_fmt, void* ws,
                                     size_t ws_bytes, int* dev_status, void* stream);
/* chameleon_linear_prepare on the static path of Alg. 2: the operand is quantized with *params
 * (host; see chameleon_act_quant_static for its checks and for MX / FP16, which ignore it) in
 * one pass.  Same workspace as chameleon_linear_prepare; chameleon_linear_gemm then multiplies it. */
cham_status chameleon_linear_prepare_static(const void* X, int M, const cham_wpack_desc* desc, int act_fmt,
                                            const cham_qparams* params, void* ws, size_t ws_bytes, int* dev_status,
                                            void* stream);
cham_status chameleon_linear_gemm(const void* X, int M, const cham_wpack_desc* desc, const void* blob,
                                  int act_fmt, const float* bias, float* Y, void* ws, size_t ws_bytes,
                                  int* dev_status, void* stream);

/* Per-sample dynamic scales (the DiT path scales each sample by its own range, Alg. 3): the M rows
 * of X form n_groups equal groups of M / n_groups consecutive rows (one sample each, e.g. its
 * tokens, or one half of a classifier-free-guidance pair), and each group of a per-tensor format
 * (0..2) is quantized with ScaleZP of its own range.  n_groups = 1 is chameleon_linear_prepare.
 * MX formats and FP16 have no per-tensor scale: for them n_groups is only checked.
 * CHAM_ERR_INVALID_ARG unless 1 <= n_groups <= CHAM_MAX_GROUPS and n_groups divides M; otherwise
 * as chameleon_linear_prepare (same workspace). */
cham_status chameleon_linear_prepare_groups(const void* X, int M, const cham_wpack_desc* desc, int act_fmt,
                                            int n_groups, void* ws, size_t ws_bytes, int* dev_status, void* stream);

/* chameleon_linear_gemm with the operand's row groups and a choice of output type.  n_groups must
 * be the one the operand was prepared with (1 after chameleon_linear_prepare or
 * chameleon_linear_prepare_static); row m uses the scale of group m / (M / n_groups).  y_type:
 * CHAM_Y_F32 (as chameleon_linear_gemm), CHAM_Y_F16 or CHAM_Y_BF16 -- the fp32 value
 * acc * (s_a * s_w) + bias rounded to nearest even into that type (beyond its range: +-Inf).
 * Y (device, M x desc->N of y_type, 16-byte aligned).  CHAM_ERR_INVALID_ARG for another y_type or
 * an n_groups that chameleon_linear_prepare_groups would reject. */
cham_status chameleon_linear_gemm_ex(const void* X, int M, const cham_wpack_desc* desc, const void* blob,
                                     int act_fmt, int n_groups, const float* bias, void* Y, int y_type, void* ws,
                                     size_t ws_bytes, int* dev_status, void* stream);

/* Test hook, not part of the method: the next chameleon_linear_gemm (or chameleon_linear) call
 * made by this host thread has the producer of the first CTA of its first GEMM launch withhold the
 * copies of that CTA's K-chunk number `chunk` (0-based over its work), so the decoders' bounded
 * wait for it runs out: the kernel records CHAM_ERR_TIMEOUT in the call's device status word,
 * drains its own copies and MMAs, releases tensor memory and returns within a few seconds, leaving
 * the context usable (the output of that call is undefined).  chunk = -1 cancels.  Host-only, no
 * GPU work. */
cham_status chameleon_debug_stall_next_gemm(int chunk);

/* chameleon_act_quant without a caller-supplied workspace.  The paper has no counterpart: this
 * entry point exists for callers that cannot allocate device memory when they quantize -- code
 * embedded in a host application or inference runtime that owns every device buffer and hands
 * its plugins only their inputs and outputs, or that forbids allocation once serving starts.
 * Same arguments, output layout and results as chameleon_act_quant, minus ws / ws_bytes.  The
 * per-tensor formats keep their range partials in a library-owned static device array of
 * 2048 x 16 bytes (32 KiB, held on every GPU that loads the library until exit); this fits any
 * M, K on GPUs with up to 256 SMs and returns CHAM_ERR_WORKSPACE (nothing launched) otherwise.
 * It calls no allocator.  The first call on a device looks up the array's address with that
 * device current: make it before any stream capture.  That address is kept until exit, so the
 * entry point must not be used on a device after cudaDeviceReset (the array may then move).  All calls share the array; calls whose
 * kernels overlap on the GPU (e.g. concurrent streams) race on it and give wrong results.
 * Errors are returned as status codes only (chameleon_last_error_detail is not updated). */
cham_status chameleon_act_quant_noalloc(const void* X, int M, int K, int fmt, void* qact, size_t qact_bytes,
                                        int* dev_status, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* CHAMELEON_H */
