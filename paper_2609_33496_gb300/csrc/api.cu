// api.cu -- the extern "C" entry points of libchameleon (include/chameleon.h).
//
// Host side only: argument validation, size queries, buffer carving, tensor-map encoding and
// kernel launches.  Nothing here allocates device memory or synchronises the device.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "act_quant.cuh"
#include "gemm.cuh"
#include "weights.cuh"

static_assert(sizeof(cham_wpack_desc) == 256, "descriptor is 256 bytes");
static_assert(sizeof(cham_qparams) == 16, "qparams is 16 bytes");

namespace {

thread_local char g_detail[512] = "";

cham_status fail(cham_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_detail, sizeof(g_detail), fmt, ap);
  va_end(ap);
  return s;
}

cham_status cuda_fail(cudaError_t e, const char* where) {
  return fail(CHAM_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// SM count of the current device, cached per device (host threads may race to fill an entry;
// they all store the same value).  152 (GB300) when the query fails: sizes then stay valid and
// the launch itself reports the CUDA error.
int num_sms_current() {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152;
  int n = cache[dev].load(std::memory_order_relaxed);
  if (n == 0) {
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 152;
    cache[dev].store(n, std::memory_order_relaxed);
  }
  return n;
}

// ---------------------------------------------------------------- NF4 levels (library's own)
// Quantile construction of NormalFloat-4 (QLoRA, cited in App. A.11): positive levels are the
// normal quantiles at 9 evenly spaced probabilities from delta to 1/2 (the last, 0, dropped),
// negative levels the negated quantiles at 8 probabilities from delta to 1/2 (zero dropped), plus
// one zero, all divided by the largest; delta = mean of 1 - 1/30 and 1 - 1/32.  The inverse
// normal CDF is solved here by bisection on Phi(x) = erfc(-x / sqrt 2) / 2; the levels are then
// rounded to fp16 (reading R9).
double phi_inv(double p) {
  double lo = -12.0, hi = 12.0;
  for (int i = 0; i < 200; ++i) {
    const double mid = 0.5 * (lo + hi);
    if (0.5 * std::erfc(-mid / std::sqrt(2.0)) < p) lo = mid;
    else hi = mid;
  }
  return 0.5 * (lo + hi);
}

uint16_t double_to_half_rne(double v) {  // finite |v| <= 65504, normal or zero range suffices here
  if (v == 0.0) return std::signbit(v) ? 0x8000u : 0u;
  const uint16_t sign = v < 0 ? 0x8000u : 0u;
  double a = std::fabs(v);
  int e;
  std::frexp(a, &e);
  e -= 1;                       // a in [2^e, 2^(e+1))
  if (e < -14) e = -14;         // subnormal binade
  const double quantum = std::ldexp(1.0, e - 10);
  double m = std::nearbyint(a / quantum);  // default rounding mode: nearest, ties to even
  if (m >= 2048.0) {           // rounded up into the next binade
    m /= 2.0;
    e += 1;
  }
  if (m < 1024.0) return static_cast<uint16_t>(sign | static_cast<uint16_t>(m));  // subnormal
  return static_cast<uint16_t>(sign | ((e + 15) << 10) | (static_cast<int>(m) - 1024));
}

double half_bits_to_double(uint16_t h) {
  const int e = (h >> 10) & 31, m = h & 1023;
  const double v = e == 0 ? std::ldexp(m, -24) : std::ldexp(1024 + m, e - 25);
  return (h & 0x8000u) ? -v : v;
}

const cham::NF4Table& nf4_table() {
  static cham::NF4Table t;
  static std::once_flag once;
  std::call_once(once, [] {
    const double delta = 0.5 * ((1.0 - 1.0 / 30.0) + (1.0 - 1.0 / 32.0));
    double v[16];
    int n = 0;
    for (int i = 0; i < 7; ++i) v[n++] = -phi_inv(delta + i * (0.5 - delta) / 7.0);
    v[n++] = 0.0;
    for (int i = 7; i >= 0; --i) v[n++] = phi_inv(delta + i * (0.5 - delta) / 8.0);
    const double vmax = phi_inv(delta);
    for (int i = 0; i < 16; ++i) t.level[i] = double_to_half_rne(v[i] / vmax);
    for (int i = 0; i < 15; ++i)
      t.mid[i] = static_cast<float>(0.5 * (half_bits_to_double(t.level[i]) + half_bits_to_double(t.level[i + 1])));
  });
  return t;
}

// ---------------------------------------------------------------- tensor map (TMA descriptor)
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// Row-major matrix rows x cols of fp16 (esize 2) or bytes (esize 1), box = 128 bytes of a row x
// box_rows rows, 128-byte swizzle.
cham_status make_act_map(CUtensorMap* map, const void* base, int rows, int cols, int box_rows, int esize) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return fail(CHAM_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * esize};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(128 / esize), static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(map, esize == 2 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8, 2,
                        const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(CHAM_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return CHAM_OK;
}

// ---------------------------------------------------------------- activation quantizer carving
struct ActLayout {
  size_t codes, params, e8m0, total;
};
ActLayout act_layout(int M, int K) {
  ActLayout L;
  const size_t n = static_cast<size_t>(M) * K;
  L.codes = 0;
  L.params = round_up(n, 256);
  L.e8m0 = L.params + 256;
  L.total = L.e8m0 + round_up(n / 32, 256);
  return L;
}

size_t range_ws_bytes(int64_t nvec) {
  return round_up(static_cast<size_t>(cham::range_grid(nvec, num_sms_current())) * sizeof(cham::RangePartial), 256);
}

cham_status check_act_args(const void* X, int M, int K, int fmt, bool allow_fp16) {
  if (M <= 0 || K <= 0) return fail(CHAM_ERR_INVALID_ARG, "M=%d K=%d must be positive", M, K);
  if (K % 32 != 0) return fail(CHAM_ERR_INVALID_ARG, "K=%d must be a multiple of 32", K);
  if (fmt < 0 || fmt > (allow_fp16 ? CHAM_A_FP16 : CHAM_A_MXINT8))
    return fail(CHAM_ERR_INVALID_ARG, "activation format %d is not valid here", fmt);
  if (X == nullptr || !aligned16(X)) return fail(CHAM_ERR_INVALID_ARG, "X must be a 16-byte aligned device pointer");
  return CHAM_OK;
}

// Parameters a caller hands to the static path (Alg. 2) must be those ScaleZP gives for that
// format: finite positive s and 1/s, z in the format's code range.
cham_status check_static_params(int fmt, const cham_qparams* p) {
  if (fmt > CHAM_A_E5M2) return CHAM_OK;  // MX formats and FP16 carry no per-tensor parameters
  if (p == nullptr) return fail(CHAM_ERR_INVALID_ARG, "static parameters are required for format %d", fmt);
  if (p->fmt != fmt) return fail(CHAM_ERR_INVALID_ARG, "parameters of format %d given for format %d", p->fmt, fmt);
  if (!std::isfinite(p->s) || !std::isfinite(p->inv) || !(p->s > 0.f) || !(p->inv > 0.f))
    return fail(CHAM_ERR_INVALID_ARG, "static scale s=%g inv=%g", p->s, p->inv);
  if (p->z < 0 || p->z > (fmt == CHAM_A_INT8_ASYM ? 255 : 0))
    return fail(CHAM_ERR_INVALID_ARG, "zero point %d out of range for format %d", p->z, fmt);
  return CHAM_OK;
}

cham::TensorParams tensor_params(const cham_qparams* p) {
  cham::TensorParams t{1.f, 1.f, 0};
  if (p != nullptr) t = cham::TensorParams{p->s, p->inv, p->z};
  return t;
}

// Formats of each MMA class (R15).
const int kClassOrder[2][5] = {{CHAM_W_INT4_SYM, CHAM_W_INT4_ASYM, CHAM_W_E2M1, CHAM_W_MXINT4, CHAM_W_MXFP4},
                               {CHAM_W_NF4, CHAM_W_INT8_SYM, CHAM_W_INT8_ASYM, CHAM_W_MXINT8, -1}};

cham_status check_desc(const cham_wpack_desc* d) {
  if (d == nullptr) return fail(CHAM_ERR_INVALID_ARG, "descriptor is NULL");
  if (d->magic != 0x574D4843u || d->version != 3) return fail(CHAM_ERR_INVALID_ARG, "not a packed-weight descriptor");
  if (d->N <= 0 || d->K <= 0 || d->K % 32 != 0 || (d->bits != 4 && d->bits != 8))
    return fail(CHAM_ERR_INVALID_ARG, "descriptor sizes are invalid");
  if (d->group < 0 || d->group % 32 != 0 || (d->group > 0 && (d->K + d->group - 1) / d->group > cham::kMaxRowGroups))
    return fail(CHAM_ERR_INVALID_ARG, "descriptor group size %d", d->group);
  if (d->f16_only != 0 && d->f16_only != 1) return fail(CHAM_ERR_INVALID_ARG, "descriptor f16_only %d", d->f16_only);
  if (d->layout < 0 || d->layout > 1 || d->fold < 0 || (d->layout == 1 && d->group > 0))
    return fail(CHAM_ERR_INVALID_ARG, "descriptor layout %d fold %d", d->layout, d->fold);
  return CHAM_OK;
}


// Which GEMM operands a layer's tiles need (Sec. 3.6): the class-0 tiles of a 4-bit per-channel
// layout run on FP8 MMAs against E4M3 / E5M2 / MXFP8 codes (unless the descriptor asks for fp16
// only) -- one launch of the FP8 kernel, whose NF4 tiles take its fp16 mainloop; every other layer
// runs on the fp16 kernel.  fp16 tiles need the exact fp16 operand (none for CHAM_A_FP16, which
// reads X).
struct OperandPlan {
  bool fp8;   // the FP8 kernel (1-byte codes, MXFP8: chunk-major exponents) over all tiles
  bool f16;   // some tiles multiply the fp16 operand (or X)
};
OperandPlan operand_plan(int M, const cham_wpack_desc* d, int act_fmt) {
  const bool fp8_act = act_fmt == CHAM_A_E4M3 || act_fmt == CHAM_A_E5M2 || act_fmt == CHAM_A_MXFP8;
  OperandPlan o;
  o.fp8 = fp8_act && d->bits == 4 && d->group == 0 && d->f16_only == 0 && d->n_tiles[0] > 0 && M > cham::kSmallM;
  o.f16 = !o.fp8 || d->n_tiles[1] > 0;
  return o;
}

// Byte offsets inside the linear workspace (each region 256-byte aligned): the activation scale
// per row group, the range partials, the fp16 operand, the 1-byte codes, the MXFP8 exponents
// chunk-major, then (gemm_plan) the split-K partial sums.
struct LinearWs {
  size_t scale, parts, operand, codes, e8, end;
  int mp;  // rows per chunk of the exponent region
};
LinearWs linear_ws(int M, const cham_wpack_desc* d, int act_fmt) {
  static_assert(cham::kMaxGroups == CHAM_MAX_GROUPS && cham::kMaxGroups * sizeof(float) <= 256, "scale slots");
  const int K = d->K;
  const int64_t nvec = static_cast<int64_t>(M) * K / 8;
  const int parts = std::max(cham::range_grid(nvec, num_sms_current()), cham::kMaxGroups);
  const OperandPlan o = operand_plan(M, d, act_fmt);
  LinearWs L{};
  L.scale = 0;
  L.parts = 256;
  // CHAM_A_FP16 multiplies X itself: no quantizer, only the scale slot precedes the partial sums
  size_t off = act_fmt == CHAM_A_FP16 ? 256 : 256 + round_up(static_cast<size_t>(parts) * sizeof(cham::RangePartial), 256);
  L.mp = (M + 3) / 4 * 4;
  const size_t mk = static_cast<size_t>(M) * K;
  L.operand = off;
  if (o.f16 && act_fmt != CHAM_A_FP16) off += round_up(mk * 2, 256);
  L.codes = off;
  if (o.fp8) off += round_up(mk, 256);
  L.e8 = off;
  if (o.fp8 && act_fmt == CHAM_A_MXFP8) off += round_up(static_cast<size_t>((K + 127) / 128) * L.mp * 4, 256);
  L.end = off;
  return L;
}

cham_status check_groups(int M, int n_groups) {
  if (n_groups < 1 || n_groups > CHAM_MAX_GROUPS || M % n_groups != 0)
    return fail(CHAM_ERR_INVALID_ARG, "n_groups=%d must be in 1..%d and divide M=%d", n_groups, CHAM_MAX_GROUPS, M);
  return CHAM_OK;
}

cham_status check_linear_common(int M, int K, int act_fmt, void* ws, size_t ws_bytes, size_t need) {
  if (M <= 0 || K <= 0 || K % 32 != 0) return fail(CHAM_ERR_INVALID_ARG, "M=%d K=%d", M, K);
  if (act_fmt < 0 || act_fmt > CHAM_A_FP16) return fail(CHAM_ERR_INVALID_ARG, "activation format %d", act_fmt);
  if (ws == nullptr || !aligned16(ws)) return fail(CHAM_ERR_INVALID_ARG, "ws must be a 16-byte aligned pointer");
  if (ws_bytes < need) return fail(CHAM_ERR_WORKSPACE, "workspace %zu < %zu bytes", ws_bytes, need);
  return CHAM_OK;
}

// The GEMM launch of a layer (the FP8 kernel over all tiles, or the fp16 kernel): token tile,
// split-K factor, and the partial-sum region after the operands.
struct GemmPlan {
  int bn, k_split;
  size_t partial, need;
};
GemmPlan gemm_plan(int M, const cham_wpack_desc* d, int act_fmt) {
  GemmPlan g{};
  const int num_sms = num_sms_current();
  const int ch_tiles = d->n_tiles[0] + d->n_tiles[1];
  if (M <= cham::kSmallM) {
    g.bn = 0;          // the weight-streaming kernel: no token tiles, no split-K partial sums
    g.k_split = 1;
  } else if (operand_plan(M, d, act_fmt).fp8) {
    g.bn = cham::gemm_pick_bn_f8(M, act_fmt == CHAM_A_MXFP8);
    g.k_split = cham::gemm_pick_split(ch_tiles * ((M + g.bn - 1) / g.bn), (d->Kp / 64 + 1) / 2, num_sms);
  } else {
    g.bn = cham::gemm_pick_bn(M, ch_tiles, num_sms);
    g.k_split = cham::gemm_pick_split(ch_tiles * ((M + g.bn - 1) / g.bn), d->Kp / 64, num_sms);
  }
  g.partial = linear_ws(M, d, act_fmt).end;
  g.need = g.partial + (g.k_split > 1 ? round_up(static_cast<size_t>(g.k_split) * M * 128 * ch_tiles * 4, 256) : 0);
  return g;
}

}  // namespace

extern "C" {

const char* chameleon_status_string(cham_status s) {
  switch (s) {
    case CHAM_OK: return "ok";
    case CHAM_ERR_INVALID_ARG: return "invalid argument";
    case CHAM_ERR_UNSUPPORTED: return "unsupported";
    case CHAM_ERR_WORKSPACE: return "workspace too small";
    case CHAM_ERR_NONFINITE: return "non-finite activation";
    case CHAM_ERR_TIMEOUT: return "device wait timed out";
    case CHAM_ERR_CUDA: return "CUDA error";
    case CHAM_ERR_RANGE: return "MX weight outside fp16";
    default: return "unknown status";
  }
}

const char* chameleon_last_error_detail(void) { return g_detail; }

int chameleon_version(void) { return 3; }

cham_status chameleon_check(const int* dev_status, void* stream) {
  if (dev_status == nullptr) return fail(CHAM_ERR_INVALID_ARG, "dev_status is NULL");
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
  int v = 0;
  e = cudaMemcpy(&v, dev_status, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "status copy");
  return v;
}

// ---------------------------------------------------------------- a1 and the LUT builder
int chameleon_bucket(int t, int T, int B) {
  if (T <= 0 || B <= 0 || t < 0) return -1;
  // floor(t / (T/B)) computed exactly in integers: floor(t * B / T)
  const long b = static_cast<long>(t) * B / T;
  return static_cast<int>(b < B - 1 ? b : B - 1);
}

cham_status chameleon_snr(int schedule, int T, double* snr_out) {
  if (T < 2 || snr_out == nullptr) return fail(CHAM_ERR_INVALID_ARG, "T must be >= 2 and snr_out non-NULL");
  if (schedule != CHAM_SCHEDULE_SCALED_LINEAR && schedule != CHAM_SCHEDULE_LINEAR)
    return fail(CHAM_ERR_INVALID_ARG, "unknown schedule %d", schedule);
  double abar = 1.0;
  for (int t = 0; t < T; ++t) {
    double beta;
    if (schedule == CHAM_SCHEDULE_SCALED_LINEAR) {
      const double a = std::sqrt(0.00085), b = std::sqrt(0.012);
      const double r = a + (b - a) * t / (T - 1);
      beta = r * r;
    } else {
      beta = 1e-4 + (0.02 - 1e-4) * t / (T - 1);
    }
    abar *= 1.0 - beta;
    snr_out[t] = abar / (1.0 - abar);
  }
  return CHAM_OK;
}

double chameleon_kurtosis(const double sums[5]) {
  const double n = sums[0];
  if (!(n > 0)) return 0.0;
  const double mu = sums[1] / n;
  const double m2 = sums[2] / n - mu * mu;
  const double m4 = sums[4] / n - 4.0 * mu * sums[3] / n + 6.0 * mu * mu * sums[2] / n - 3.0 * mu * mu * mu * mu;
  if (!(m2 > 0)) return 0.0;
  return m4 / (m2 * m2);
}

int chameleon_route(double kappa, double snr_b, int is_shortcut) {
  if (is_shortcut) return CHAM_A_MXFP8;
  if (kappa > 5.0 || snr_b < 0.2) return CHAM_A_E5M2;
  if (kappa <= 3.0 && snr_b > 2.0) return CHAM_A_INT8_ASYM;
  return CHAM_A_E4M3;
}

// ---------------------------------------------------------------- calibration power sums
cham_status chameleon_act_moments_workspace_size(int64_t count, size_t* ws_bytes) {
  if (count <= 0 || count % 8 != 0 || ws_bytes == nullptr)
    return fail(CHAM_ERR_INVALID_ARG, "count must be a positive multiple of 8");
  *ws_bytes = round_up(static_cast<size_t>(cham::range_grid(count / 8, num_sms_current())) * sizeof(cham::MomentPartial),
                       256);
  return CHAM_OK;
}

cham_status chameleon_act_moments(const void* X, int64_t count, double* out, void* ws, size_t ws_bytes,
                                  void* stream) {
  size_t need = 0;
  cham_status s = chameleon_act_moments_workspace_size(count, &need);
  if (s != CHAM_OK) return s;
  if (X == nullptr || out == nullptr || ws == nullptr || !aligned16(X) || !aligned16(ws))
    return fail(CHAM_ERR_INVALID_ARG, "null or misaligned pointer");
  if (ws_bytes < need) return fail(CHAM_ERR_WORKSPACE, "workspace %zu < %zu", ws_bytes, need);
  const int64_t nvec = count / 8;
  const int nparts = cham::range_grid(nvec, num_sms_current());
  cham::launch_act_moments(static_cast<const uint4*>(X), nvec, count, static_cast<cham::MomentPartial*>(ws), nparts,
                           out, static_cast<cudaStream_t>(stream));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "act_moments launch");
}

// ---------------------------------------------------------------- a2-a4
cham_status chameleon_act_quant_size(int M, int K, int fmt, size_t* qact_bytes, size_t* ws_bytes) {
  if (M <= 0 || K <= 0 || K % 32 != 0 || fmt < 0 || fmt > CHAM_A_MXINT8)
    return fail(CHAM_ERR_INVALID_ARG, "M=%d K=%d fmt=%d", M, K, fmt);
  const ActLayout L = act_layout(M, K);
  if (qact_bytes) *qact_bytes = L.total;
  if (ws_bytes) *ws_bytes = fmt <= CHAM_A_E5M2 ? range_ws_bytes(static_cast<int64_t>(M) * K / 8) : 0;
  return CHAM_OK;
}

cham_status chameleon_act_quant(const void* X, int M, int K, int fmt, void* qact, size_t qact_bytes, void* ws,
                                size_t ws_bytes, int* dev_status, void* stream) {
  cham_status s = check_act_args(X, M, K, fmt, false);
  if (s != CHAM_OK) return s;
  size_t need_q = 0, need_ws = 0;
  chameleon_act_quant_size(M, K, fmt, &need_q, &need_ws);
  if (qact == nullptr || !aligned16(qact)) return fail(CHAM_ERR_INVALID_ARG, "qact must be 16-byte aligned");
  if (qact_bytes < need_q) return fail(CHAM_ERR_WORKSPACE, "qact %zu < %zu bytes", qact_bytes, need_q);
  if (need_ws > 0 && (ws == nullptr || !aligned16(ws))) return fail(CHAM_ERR_INVALID_ARG, "ws must be 16-byte aligned");
  if (ws_bytes < need_ws) return fail(CHAM_ERR_WORKSPACE, "ws %zu < %zu bytes", ws_bytes, need_ws);
  const ActLayout L = act_layout(M, K);
  uint8_t* q = static_cast<uint8_t*>(qact);
  cham::ActQuantArgs a{};
  a.X = static_cast<const uint4*>(X);
  a.nvec = static_cast<int64_t>(M) * K / 8;
  a.num_sms = num_sms_current();
  a.parts = static_cast<cham::RangePartial*>(ws);
  a.nparts = cham::range_grid(a.nvec, a.num_sms);
  a.codes = reinterpret_cast<uint2*>(q + L.codes);
  a.deq = nullptr;
  a.e8m0 = fmt >= CHAM_A_MXFP8 ? q + L.e8m0 : nullptr;
  a.params = reinterpret_cast<cham_qparams*>(q + L.params);
  a.scale_out = nullptr;
  a.dev_status = dev_status;
  cham::launch_act_quant(fmt, a, true, false, static_cast<cudaStream_t>(stream));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "act_quant launch");
}

cham_status chameleon_scale_zp(int fmt, float lo, float hi, cham_qparams* out) {
  if (out == nullptr) return fail(CHAM_ERR_INVALID_ARG, "out is NULL");
  if (fmt < 0 || fmt > CHAM_A_E5M2) return fail(CHAM_ERR_INVALID_ARG, "ScaleZP is per-tensor: format %d", fmt);
  if (!std::isfinite(lo) || !std::isfinite(hi) || lo > hi)
    return fail(CHAM_ERR_INVALID_ARG, "range [%g, %g] must be finite and ordered", lo, hi);
  // The arithmetic of the quantizer's own ScaleZP, in the same fp32 operations and rounding.
  cham_qparams p{1.f, 0, 1.f, fmt};
  if (fmt == CHAM_A_INT8_ASYM) {
    const float lo_ = std::fmin(lo, 0.f), hi_ = std::fmax(hi, 0.f);
    const float d = hi_ - lo_;
    if (d != 0.f) {
      p.s = d / 255.f;
      p.inv = 255.f / d;
      const float zf = std::nearbyint(-lo_ * p.inv);
      p.z = zf < 0.f ? 0 : (zf > 255.f ? 255 : static_cast<int32_t>(zf));
    }
  } else {
    const float fmax = fmt == CHAM_A_E4M3 ? 448.f : 57344.f;
    const float amax = std::fmax(std::fabs(lo), std::fabs(hi));
    if (amax != 0.f) {
      p.s = amax / fmax;
      p.inv = fmax / amax;
    }
  }
  if (!std::isfinite(p.s) || !(p.inv > 0.f)) return fail(CHAM_ERR_INVALID_ARG, "range [%g, %g] too wide", lo, hi);
  *out = p;
  return CHAM_OK;
}

cham_status chameleon_act_quant_static(const void* X, int M, int K, int fmt, const cham_qparams* params, void* qact,
                                       size_t qact_bytes, int* dev_status, void* stream) {
  cham_status s = check_act_args(X, M, K, fmt, false);
  if (s != CHAM_OK) return s;
  s = check_static_params(fmt, params);
  if (s != CHAM_OK) return s;
  size_t need_q = 0;
  chameleon_act_quant_size(M, K, fmt, &need_q, nullptr);
  if (qact == nullptr || !aligned16(qact)) return fail(CHAM_ERR_INVALID_ARG, "qact must be 16-byte aligned");
  if (qact_bytes < need_q) return fail(CHAM_ERR_WORKSPACE, "qact %zu < %zu bytes", qact_bytes, need_q);
  const ActLayout L = act_layout(M, K);
  uint8_t* q = static_cast<uint8_t*>(qact);
  cham::ActQuantArgs a{};
  a.X = static_cast<const uint4*>(X);
  a.nvec = static_cast<int64_t>(M) * K / 8;
  a.num_sms = num_sms_current();
  a.codes = reinterpret_cast<uint2*>(q + L.codes);
  a.e8m0 = fmt >= CHAM_A_MXFP8 ? q + L.e8m0 : nullptr;
  a.params = reinterpret_cast<cham_qparams*>(q + L.params);
  a.dev_status = dev_status;
  a.use_static = true;
  a.stat = tensor_params(params);
  cham::launch_act_quant(fmt, a, true, false, static_cast<cudaStream_t>(stream));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "act_quant_static launch");
}

// ---------------------------------------------------------------- Eq. format-argmin (calibration)
namespace {
struct SseWs {
  size_t parts, sse;
  size_t total;
};
SseWs sse_ws(int64_t nvec) {
  const size_t n = static_cast<size_t>(cham::range_grid(nvec, num_sms_current()));
  SseWs L;
  L.parts = 0;
  L.sse = round_up(n * sizeof(cham::RangePartial), 256);
  L.total = L.sse + round_up(n * 5 * sizeof(double), 256);
  return L;
}
}  // namespace

cham_status chameleon_act_format_sse_workspace_size(int M, int K, size_t* ws_bytes) {
  if (M <= 0 || K <= 0 || K % 32 != 0 || ws_bytes == nullptr)
    return fail(CHAM_ERR_INVALID_ARG, "M=%d K=%d (K must be a multiple of 32)", M, K);
  *ws_bytes = sse_ws(static_cast<int64_t>(M) * K / 8).total;
  return CHAM_OK;
}

cham_status chameleon_act_format_sse(const void* X, int M, int K, double* sse, void* ws, size_t ws_bytes,
                                     int* dev_status, void* stream) {
  cham_status s = check_act_args(X, M, K, CHAM_A_INT8_ASYM, false);
  if (s != CHAM_OK) return s;
  if (sse == nullptr || reinterpret_cast<uintptr_t>(sse) % 8 != 0)
    return fail(CHAM_ERR_INVALID_ARG, "sse must be an 8-byte aligned device pointer");
  const int64_t nvec = static_cast<int64_t>(M) * K / 8;
  const SseWs L = sse_ws(nvec);
  if (ws == nullptr || !aligned16(ws)) return fail(CHAM_ERR_INVALID_ARG, "ws must be 16-byte aligned");
  if (ws_bytes < L.total) return fail(CHAM_ERR_WORKSPACE, "ws %zu < %zu bytes", ws_bytes, L.total);
  uint8_t* w = static_cast<uint8_t*>(ws);
  cham::launch_act_format_sse(static_cast<const uint4*>(X), nvec, reinterpret_cast<cham::RangePartial*>(w + L.parts),
                              cham::range_grid(nvec, num_sms_current()), reinterpret_cast<double*>(w + L.sse), sse,
                              dev_status, static_cast<cudaStream_t>(stream));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "act_format_sse launch");
}

int chameleon_act_format_argmin(const double* sse) {
  if (sse == nullptr) return -1;
  int best = 0;
  for (int f = 1; f < 5; ++f)
    if (sse[f] < sse[best]) best = f;
  return best;
}

// ---------------------------------------------------------------- a5
cham_status chameleon_select_weight_formats(const void* W, int N, int K, uint32_t palette_mask, uint8_t* fmt_out,
                                            double* sse_out, void* stream) {
  if (N <= 0 || K <= 0 || K % 32 != 0) return fail(CHAM_ERR_INVALID_ARG, "N=%d K=%d (K must be a multiple of 32)", N, K);
  if (palette_mask == 0 || (palette_mask & ~0x1FFu) != 0) return fail(CHAM_ERR_INVALID_ARG, "palette mask 0x%x", palette_mask);
  if ((palette_mask & CHAM_PALETTE_W8) && (palette_mask & CHAM_PALETTE_W4))
    return fail(CHAM_ERR_INVALID_ARG, "palette mixes 8-bit and 4-bit formats");
  if (W == nullptr || !aligned16(W) || fmt_out == nullptr) return fail(CHAM_ERR_INVALID_ARG, "null or misaligned pointer");
  cham::launch_select(static_cast<const __half*>(W), N, K, palette_mask, fmt_out, sse_out, nf4_table(),
                      static_cast<cudaStream_t>(stream));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "select launch");
}

// ---------------------------------------------------------------- (g, f) search (Sec. 3.5 forks)
namespace {
const int kGroupSizes[5] = {32, 64, 128, 192, 288};

int group_candidates(uint32_t palette_mask, uint32_t group_mask, cham::GroupCand* out, int cap) {
  int n = 0;
  for (int i = 0; i < 5; ++i) {
    if (!((group_mask >> i) & 1u)) continue;
    for (int f = 0; f < CHAM_W_NFORMATS; ++f) {
      if (!((palette_mask >> f) & 1u)) continue;
      if (cham::w_is_mx(f) && kGroupSizes[i] != 32) continue;
      if (n < cap) out[n] = cham::GroupCand{kGroupSizes[i], f};
      ++n;
    }
  }
  return n;
}

cham_status check_group_search(int N, int K, uint32_t palette_mask, uint32_t group_mask) {
  if (N <= 0 || K <= 0 || K % 32 != 0) return fail(CHAM_ERR_INVALID_ARG, "N=%d K=%d (K must be a multiple of 32)", N, K);
  if (palette_mask == 0 || (palette_mask & ~0x1FFu) != 0) return fail(CHAM_ERR_INVALID_ARG, "palette mask 0x%x", palette_mask);
  if ((palette_mask & CHAM_PALETTE_W8) && (palette_mask & CHAM_PALETTE_W4))
    return fail(CHAM_ERR_INVALID_ARG, "palette mixes 8-bit and 4-bit formats");
  if (group_mask == 0 || (group_mask & ~0x1Fu) != 0) return fail(CHAM_ERR_INVALID_ARG, "group mask 0x%x", group_mask);
  for (int i = 0; i < 5; ++i)
    if (((group_mask >> i) & 1u) && (K + kGroupSizes[i] - 1) / kGroupSizes[i] > cham::kMaxRowGroups)
      return fail(CHAM_ERR_INVALID_ARG, "K=%d has more than %d groups of %d", K, cham::kMaxRowGroups, kGroupSizes[i]);
  cham::GroupCand c[cham::kMaxCands];
  if (group_candidates(palette_mask, group_mask, c, cham::kMaxCands) == 0)
    return fail(CHAM_ERR_INVALID_ARG, "no (g, f) candidate: palette 0x%x, groups 0x%x", palette_mask, group_mask);
  return CHAM_OK;
}

size_t group_search_ws(int N, int K, int n_cand) {
  return round_up(static_cast<size_t>(K) * 4, 256) + round_up(static_cast<size_t>(N) * n_cand * 8, 256);
}
}  // namespace

cham_status chameleon_group_candidates(uint32_t palette_mask, uint32_t group_mask, int* g_out, int* fmt_out, int cap,
                                       int* n_out) {
  if (n_out == nullptr || cap < 0 || (cap > 0 && (g_out == nullptr || fmt_out == nullptr)))
    return fail(CHAM_ERR_INVALID_ARG, "null output");
  cham::GroupCand c[cham::kMaxCands];
  const int n = group_candidates(palette_mask & 0x1FFu, group_mask & 0x1Fu, c, cham::kMaxCands);
  for (int i = 0; i < n && i < cap; ++i) {
    g_out[i] = c[i].g;
    fmt_out[i] = c[i].f;
  }
  *n_out = n;
  return CHAM_OK;
}

cham_status chameleon_select_weight_groups_workspace_size(int N, int K, uint32_t palette_mask, uint32_t group_mask,
                                                          size_t* ws_bytes) {
  cham_status s = check_group_search(N, K, palette_mask, group_mask);
  if (s != CHAM_OK) return s;
  if (ws_bytes == nullptr) return fail(CHAM_ERR_INVALID_ARG, "ws_bytes is NULL");
  cham::GroupCand c[cham::kMaxCands];
  *ws_bytes = group_search_ws(N, K, group_candidates(palette_mask, group_mask, c, cham::kMaxCands));
  return CHAM_OK;
}

cham_status chameleon_select_weight_groups(const void* W, int N, int K, uint32_t palette_mask, uint32_t group_mask,
                                           const double* energy, double* scores, void* ws, size_t ws_bytes,
                                           void* stream) {
  cham_status s = check_group_search(N, K, palette_mask, group_mask);
  if (s != CHAM_OK) return s;
  if (W == nullptr || !aligned16(W) || scores == nullptr || ws == nullptr || !aligned16(ws))
    return fail(CHAM_ERR_INVALID_ARG, "null or misaligned pointer");
  cham::GroupSearchArgs a{};
  a.n_cand = group_candidates(palette_mask, group_mask, a.cand, cham::kMaxCands);
  const size_t need = group_search_ws(N, K, a.n_cand);
  if (ws_bytes < need) return fail(CHAM_ERR_WORKSPACE, "ws %zu < %zu bytes", ws_bytes, need);
  uint8_t* w = static_cast<uint8_t*>(ws);
  a.W = static_cast<const __half*>(W);
  a.N = N;
  a.K = K;
  a.energy = energy;
  a.energy32 = reinterpret_cast<float*>(w);
  a.parts = reinterpret_cast<double*>(w + round_up(static_cast<size_t>(K) * 4, 256));
  a.scores = scores;
  cham::launch_select_groups(a, nf4_table(), static_cast<cudaStream_t>(stream));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "group search launch");
}

int chameleon_candidate_argmin(const double* scores, int n) {
  if (scores == nullptr || n <= 0) return -1;
  int best = 0;
  for (int i = 1; i < n; ++i)
    if (scores[i] < scores[best]) best = i;
  return best;
}

cham_status chameleon_act_channel_energy(const void* X, int M, int K, double* energy, void* stream) {
  if (M <= 0 || K <= 0 || K % 8 != 0 || X == nullptr || !aligned16(X) || energy == nullptr)
    return fail(CHAM_ERR_INVALID_ARG, "M=%d K=%d (K a multiple of 8, X 16-byte aligned)", M, K);
  cham::launch_channel_energy(static_cast<const __half*>(X), M, K, energy, static_cast<cudaStream_t>(stream));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "channel energy launch");
}

// ---------------------------------------------------------------- a6
}  // extern "C"
namespace {
void finish_plan(cham_wpack_desc* d, int N, int K, int bits);

// The packed groups of a plan, in slot order.  Layout 0: one group per MMA class.  Layout 1: per
// class, each format with at least `fold` channels in palette order, then the class's tail of the
// formats with fewer.  group_of[f] is -1 for a format without channels.
struct PackGroups {
  int n;
  int cls[cham::kMaxPackGroups], count[cham::kMaxPackGroups];
  int8_t group_of[CHAM_W_NFORMATS];
};
PackGroups pack_groups(const cham_wpack_desc* d) {
  PackGroups g{};
  for (int f = 0; f < CHAM_W_NFORMATS; ++f) g.group_of[f] = -1;
  for (int cls = 0; cls < 2; ++cls) {
    if (d->layout != 1) {
      g.cls[g.n] = cls;
      g.count[g.n] = d->n_class[cls];
      for (int j = 0; j < 5; ++j)
        if (kClassOrder[cls][j] >= 0) g.group_of[kClassOrder[cls][j]] = static_cast<int8_t>(g.n);
      ++g.n;
      continue;
    }
    int tail = 0;
    for (int j = 0; j < 5; ++j) {
      const int f = kClassOrder[cls][j];
      if (f < 0 || d->n_fmt[f] <= 0) continue;
      if (d->n_fmt[f] >= d->fold) {
        g.cls[g.n] = cls;
        g.count[g.n] = d->n_fmt[f];
        g.group_of[f] = static_cast<int8_t>(g.n++);
      } else {
        tail += d->n_fmt[f];
      }
    }
    if (tail > 0) {
      for (int j = 0; j < 5; ++j) {
        const int f = kClassOrder[cls][j];
        if (f >= 0 && d->n_fmt[f] > 0 && d->n_fmt[f] < d->fold) g.group_of[f] = static_cast<int8_t>(g.n);
      }
      g.cls[g.n] = cls;
      g.count[g.n++] = tail;
    }
  }
  return g;
}
}  // namespace
extern "C" {

cham_status chameleon_pack_plan(int N, int K, const uint8_t* fmt_host, cham_wpack_desc* d) {
  return chameleon_pack_plan_layout(N, K, fmt_host, 0, 0, d);
}

cham_status chameleon_pack_plan_layout(int N, int K, const uint8_t* fmt_host, int layout, int fold,
                                       cham_wpack_desc* d) {
  if (N <= 0 || K <= 0 || K % 32 != 0 || fmt_host == nullptr || d == nullptr)
    return fail(CHAM_ERR_INVALID_ARG, "N=%d K=%d (K must be a multiple of 32)", N, K);
  if (layout < 0 || layout > 1 || fold < 0) return fail(CHAM_ERR_INVALID_ARG, "layout %d fold %d", layout, fold);
  std::memset(d, 0, sizeof(*d));
  int bits = 0;
  for (int c = 0; c < N; ++c) {
    const int f = fmt_host[c];
    if (f >= CHAM_W_NFORMATS) return fail(CHAM_ERR_INVALID_ARG, "channel %d has format %d", c, f);
    const int b = cham::wbits(f);
    if (bits != 0 && b != bits) return fail(CHAM_ERR_INVALID_ARG, "formats of mixed bit width");
    bits = b;
    d->n_fmt[f] += 1;
  }
  for (int cls = 0; cls < 2; ++cls)
    for (int j = 0; j < 5; ++j)
      if (kClassOrder[cls][j] >= 0) d->n_class[cls] += d->n_fmt[kClassOrder[cls][j]];
  d->layout = layout;
  d->fold = fold;
  finish_plan(d, N, K, bits);
  return CHAM_OK;
}

// A plan from the palette alone: when every member shares one MMA class, the packed layout
// depends only on N, K and the bit width (no device -> host copy of the selected formats).
cham_status chameleon_pack_plan_palette(int N, int K, uint32_t palette_mask, cham_wpack_desc* d) {
  if (N <= 0 || K <= 0 || K % 32 != 0 || d == nullptr)
    return fail(CHAM_ERR_INVALID_ARG, "N=%d K=%d (K must be a multiple of 32)", N, K);
  if (palette_mask == 0 || (palette_mask & ~0x1FFu) != 0) return fail(CHAM_ERR_INVALID_ARG, "palette mask 0x%x", palette_mask);
  int bits = 0, cls = -1;
  for (int f = 0; f < CHAM_W_NFORMATS; ++f) {
    if (!((palette_mask >> f) & 1u)) continue;
    if (bits != 0 && cham::wbits(f) != bits) return fail(CHAM_ERR_INVALID_ARG, "palette mixes 8-bit and 4-bit formats");
    bits = cham::wbits(f);
    if (cls >= 0 && cham::w_class(f) != cls)
      return fail(CHAM_ERR_UNSUPPORTED, "palette 0x%x spans both MMA classes: plan from the selected formats", palette_mask);
    cls = cham::w_class(f);
  }
  std::memset(d, 0, sizeof(*d));
  for (int f = 0; f < CHAM_W_NFORMATS; ++f)
    if ((palette_mask >> f) & 1u) d->n_fmt[f] = -1;  // per-format counts are not known on the host
  d->n_class[cls] = N;
  finish_plan(d, N, K, bits);
  return CHAM_OK;
}

cham_status chameleon_pack_plan_grouped(int N, int K, int fmt, int group, cham_wpack_desc* d) {
  if (N <= 0 || K <= 0 || K % 32 != 0 || d == nullptr)
    return fail(CHAM_ERR_INVALID_ARG, "N=%d K=%d (K must be a multiple of 32)", N, K);
  if (fmt < 0 || fmt >= CHAM_W_NFORMATS || cham::w_is_mx(fmt))
    return fail(CHAM_ERR_INVALID_ARG, "format %d has no group-wise form", fmt);
  if (group < 32 || group % 32 != 0 || (K + group - 1) / group > cham::kMaxRowGroups)
    return fail(CHAM_ERR_INVALID_ARG, "group %d (a multiple of 32, at most %d groups per row)", group,
                cham::kMaxRowGroups);
  std::memset(d, 0, sizeof(*d));
  d->n_fmt[fmt] = N;
  d->n_class[cham::w_class(fmt)] = N;
  d->group = group;
  finish_plan(d, N, K, cham::wbits(fmt));
  return CHAM_OK;
}

}  // extern "C"

namespace {
void finish_plan(cham_wpack_desc* d, int N, int K, int bits) {
  d->magic = 0x574D4843u;
  d->version = 3;
  d->N = N;
  d->K = K;
  d->Kp = static_cast<int>(round_up(K, 64));
  d->bits = bits;
  for (int cls = 0; cls < 2; ++cls) {
    if (d->layout == 1) {
      const PackGroups g = pack_groups(d);
      d->n_tiles[cls] = 0;
      for (int i = 0; i < g.n; ++i)
        if (g.cls[i] == cls) d->n_tiles[cls] += (g.count[i] + 127) / 128;
    } else {
      d->n_tiles[cls] = (d->n_class[cls] + 127) / 128;
    }
  }
  const size_t tiles = static_cast<size_t>(d->n_tiles[0] + d->n_tiles[1]);
  const size_t np = tiles * 128, chunks = d->Kp / 64;
  size_t off = 256;
  d->off_codes = off;
  off = round_up(off + tiles * chunks * 128 * (bits == 8 ? 64 : 32), 256);
  d->off_scale = off;
  off = round_up(off + np * 4, 256);
  d->off_zero = off;
  off = round_up(off + np, 256);
  d->off_e8m0 = off;
  off = round_up(off + tiles * chunks * 128 * 2, 256);
  d->off_fmt = off;
  off = round_up(off + np, 256);
  d->off_perm = off;
  off = round_up(off + np * 4, 256);
  if (d->group > 0) {
    d->off_gscale = off;
    off = round_up(off + tiles * chunks * 128 * 4, 256);
  }
  d->bytes = off;
}
}  // namespace

namespace {
cham::PackArgs pack_args(const cham_wpack_desc* d, const void* W, const uint8_t* fmt_dev, void* blob, int* dev_status) {
  uint8_t* b = static_cast<uint8_t*>(blob);
  cham::PackArgs a{};
  a.W = static_cast<const __half*>(W);
  a.fmt_dev = fmt_dev;
  a.N = d->N;
  a.K = d->K;
  a.Kp = d->Kp;
  a.bits = d->bits;
  a.n_chunks = d->Kp / 64;
  a.n_packed = 128 * (d->n_tiles[0] + d->n_tiles[1]);
  a.cls_base[0] = 0;
  a.cls_base[1] = 128 * d->n_tiles[0];
  a.cls_count[0] = d->n_class[0];
  a.cls_count[1] = d->n_class[1];
  const PackGroups g = pack_groups(d);
  a.n_groups = g.n;
  int base = 0;
  for (int i = 0; i < g.n; ++i) {
    a.group_base[i] = base;
    a.group_count[i] = g.count[i];
    base += 128 * ((g.count[i] + 127) / 128);
  }
  for (int f = 0; f < CHAM_W_NFORMATS; ++f) a.group_of_fmt[f] = g.group_of[f];
  a.codes = b + d->off_codes;
  a.scale = reinterpret_cast<float*>(b + d->off_scale);
  a.zero = b + d->off_zero;
  a.e8m0 = b + d->off_e8m0;
  a.fmtp = b + d->off_fmt;
  a.perm = reinterpret_cast<int32_t*>(b + d->off_perm);
  a.dev_status = dev_status;
  // one MMA class in original order: slot = channel, no ranking pass (not for format groups)
  a.one_class = d->layout != 0 ? -1 : (d->n_class[0] == 0 ? 1 : (d->n_class[1] == 0 ? 0 : -1));
  a.group = d->group;
  a.gscale = d->group > 0 ? reinterpret_cast<uint32_t*>(b + d->off_gscale) : nullptr;
  a.desc = *d;
  a.desc_out = reinterpret_cast<cham_wpack_desc*>(b);
  return a;
}
}  // namespace

extern "C" {

cham_status chameleon_pack_weights(const void* W, const uint8_t* fmt_dev, const cham_wpack_desc* d, void* blob,
                                   size_t blob_bytes, int* dev_status, void* stream) {
  cham_status s = check_desc(d);
  if (s != CHAM_OK) return s;
  if (W == nullptr || fmt_dev == nullptr || blob == nullptr || !aligned16(W) || !aligned16(blob))
    return fail(CHAM_ERR_INVALID_ARG, "null or misaligned pointer");
  if (blob_bytes < d->bytes) return fail(CHAM_ERR_WORKSPACE, "blob %zu < %llu bytes", blob_bytes,
                                          static_cast<unsigned long long>(d->bytes));
  cham::launch_pack(pack_args(d, W, fmt_dev, blob, dev_status), nf4_table(), static_cast<cudaStream_t>(stream));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "pack launch");
}

cham_status chameleon_select_pack_palette(const void* W, int N, int K, uint32_t palette_mask,
                                          const cham_wpack_desc* d, uint8_t* fmt_out, void* blob, size_t blob_bytes,
                                          int* dev_status, void* stream) {
  cham_status s = check_desc(d);
  if (s != CHAM_OK) return s;
  if (d->N != N || d->K != K || d->group != 0 || d->layout != 0 || (d->n_class[0] != 0 && d->n_class[1] != 0))
    return fail(CHAM_ERR_INVALID_ARG, "descriptor is not a one-class plan of %d x %d weights", N, K);
  if (palette_mask == 0 || (palette_mask & ~0x1FFu) != 0) return fail(CHAM_ERR_INVALID_ARG, "palette mask 0x%x", palette_mask);
  const int cls = d->n_class[0] == 0 ? 1 : 0;
  for (int f = 0; f < CHAM_W_NFORMATS; ++f)
    if (((palette_mask >> f) & 1u) && (cham::w_class(f) != cls || cham::wbits(f) != d->bits))
      return fail(CHAM_ERR_INVALID_ARG, "palette 0x%x does not match the plan's class and width", palette_mask);
  if (W == nullptr || fmt_out == nullptr || blob == nullptr || !aligned16(W) || !aligned16(blob))
    return fail(CHAM_ERR_INVALID_ARG, "null or misaligned pointer");
  if (blob_bytes < d->bytes) return fail(CHAM_ERR_WORKSPACE, "blob %zu < %llu bytes", blob_bytes,
                                          static_cast<unsigned long long>(d->bytes));
  cham::PackArgs a = pack_args(d, W, nullptr, blob, dev_status);
  a.fmt_out = fmt_out;
  cham::launch_select_pack(a, palette_mask, nf4_table(), static_cast<cudaStream_t>(stream));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "select+pack launch");
}

// ---------------------------------------------------------------- a7/a8
// Workspace: [0, 256) the per-tensor scale s_a; [256, 256 + R) range partials; then the M x K
// fp16 activation operand (exact values of the codes, R13); then, when the GEMM splits K, its
// fp32 partial sums.
cham_status chameleon_linear_workspace_size(int M, const cham_wpack_desc* d, int act_fmt, size_t* ws_bytes) {
  cham_status s = check_desc(d);
  if (s != CHAM_OK) return s;
  if (M <= 0 || act_fmt < 0 || act_fmt > CHAM_A_FP16 || ws_bytes == nullptr)
    return fail(CHAM_ERR_INVALID_ARG, "M=%d act_fmt=%d", M, act_fmt);
  *ws_bytes = gemm_plan(M, d, act_fmt).need;
  return CHAM_OK;
}

cham_status chameleon_linear_launches(int M, const cham_wpack_desc* d, int act_fmt, int n_groups, int is_static,
                                      int* prepare_launches, int* gemm_launches) {
  cham_status s = check_desc(d);
  if (s != CHAM_OK) return s;
  if (M <= 0 || act_fmt < 0 || act_fmt > CHAM_A_FP16 || prepare_launches == nullptr || gemm_launches == nullptr)
    return fail(CHAM_ERR_INVALID_ARG, "M=%d act_fmt=%d", M, act_fmt);
  s = check_groups(M, n_groups);
  if (s != CHAM_OK) return s;
  *prepare_launches = act_fmt == CHAM_A_FP16 ? 0 : (is_static || act_fmt >= CHAM_A_MXFP8 ? 1 : 2);
  *gemm_launches = gemm_plan(M, d, act_fmt).k_split > 1 ? 2 : 1;
  return CHAM_OK;
}

}  // extern "C"


namespace {
// The prepare calls (Alg. 3 dynamic per tensor or per sample, or Alg. 2 static): quantize X into
// the operands the layer's tiles need (operand_plan) -- one quantizer pass writes both when both
// kernels run.
cham_status prepare_common(const void* X, int M, const cham_wpack_desc* d, int act_fmt, int n_groups,
                           const cham_qparams* params, bool is_static, void* ws, size_t ws_bytes, int* dev_status,
                           void* stream) {
  cham_status s = check_desc(d);
  if (s != CHAM_OK) return s;
  const int K = d->K;
  s = check_act_args(X, M, K, act_fmt, true);
  if (s != CHAM_OK) return s;
  s = check_groups(M, n_groups);
  if (s != CHAM_OK) return s;
  if (is_static) {
    s = check_static_params(act_fmt, params);
    if (s != CHAM_OK) return s;
  }
  const LinearWs L = linear_ws(M, d, act_fmt);
  s = check_linear_common(M, K, act_fmt, ws, ws_bytes, L.end);
  if (s != CHAM_OK) return s;
  if (act_fmt == CHAM_A_FP16) return CHAM_OK;
  const OperandPlan o = operand_plan(M, d, act_fmt);
  uint8_t* w = static_cast<uint8_t*>(ws);
  cham::ActQuantArgs a{};
  a.X = static_cast<const uint4*>(X);
  a.nvec = static_cast<int64_t>(M) * K / 8;
  a.num_sms = num_sms_current();
  a.codes = o.fp8 ? reinterpret_cast<uint2*>(w + L.codes) : nullptr;
  a.kperm = o.fp8;  // the FP8 GEMM operand in the weight codes' group order
  a.deq = o.f16 ? reinterpret_cast<uint4*>(w + L.operand) : nullptr;
  a.e8m0 = nullptr;
  if (o.fp8 && act_fmt == CHAM_A_MXFP8) {
    a.e8cm = w + L.e8;
    a.kblocks = K / 32;
    a.cm_plane = static_cast<int64_t>(L.mp) * 4;
  }
  a.params = nullptr;
  a.scale_out = act_fmt <= CHAM_A_E5M2 ? reinterpret_cast<float*>(w + L.scale) : nullptr;
  a.dev_status = dev_status;
  if (is_static) {
    a.use_static = true;
    a.stat = tensor_params(params);
  } else {
    a.parts = reinterpret_cast<cham::RangePartial*>(w + L.parts);
    a.n_groups = act_fmt <= CHAM_A_E5M2 ? n_groups : 1;
    a.nparts = cham::group_grid(a.nvec, a.n_groups, a.num_sms);
  }
  cham::launch_act_quant(act_fmt, a, a.codes != nullptr, a.deq != nullptr, static_cast<cudaStream_t>(stream));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "linear_prepare launch");
}
}  // namespace

extern "C" {

cham_status chameleon_linear_prepare(const void* X, int M, const cham_wpack_desc* d, int act_fmt, void* ws,
                                     size_t ws_bytes, int* dev_status, void* stream) {
  return prepare_common(X, M, d, act_fmt, 1, nullptr, false, ws, ws_bytes, dev_status, stream);
}

cham_status chameleon_linear_prepare_groups(const void* X, int M, const cham_wpack_desc* d, int act_fmt,
                                            int n_groups, void* ws, size_t ws_bytes, int* dev_status, void* stream) {
  return prepare_common(X, M, d, act_fmt, n_groups, nullptr, false, ws, ws_bytes, dev_status, stream);
}

cham_status chameleon_linear_prepare_static(const void* X, int M, const cham_wpack_desc* d, int act_fmt,
                                            const cham_qparams* params, void* ws, size_t ws_bytes, int* dev_status,
                                            void* stream) {
  return prepare_common(X, M, d, act_fmt, 1, params, true, ws, ws_bytes, dev_status, stream);
}

namespace {
// set by chameleon_debug_stall_next_gemm, taken by the next GEMM call of the same host thread
thread_local int g_stall_next_gemm = -1;
}  // namespace

cham_status chameleon_debug_stall_next_gemm(int chunk) {
  if (chunk < -1) return fail(CHAM_ERR_INVALID_ARG, "chunk %d", chunk);
  g_stall_next_gemm = chunk;
  return CHAM_OK;
}

cham_status chameleon_linear_gemm(const void* X, int M, const cham_wpack_desc* d, const void* blob, int act_fmt,
                                  const float* bias, float* Y, void* ws, size_t ws_bytes, int* dev_status,
                                  void* stream) {
  return chameleon_linear_gemm_ex(X, M, d, blob, act_fmt, 1, bias, Y, CHAM_Y_F32, ws, ws_bytes, dev_status, stream);
}

cham_status chameleon_linear_gemm_ex(const void* X, int M, const cham_wpack_desc* d, const void* blob, int act_fmt,
                                     int n_groups, const float* bias, void* Y, int y_type, void* ws,
                                     size_t ws_bytes, int* dev_status, void* stream) {
  cham_status s = check_desc(d);
  if (s != CHAM_OK) return s;
  if (y_type < CHAM_Y_F32 || y_type > CHAM_Y_BF16) return fail(CHAM_ERR_INVALID_ARG, "y_type %d", y_type);
  s = check_groups(M, n_groups);
  if (s != CHAM_OK) return s;
  const int K = d->K;
  const GemmPlan plan = gemm_plan(M, d, act_fmt);
  s = check_linear_common(M, K, act_fmt, ws, ws_bytes, plan.need);
  if (s != CHAM_OK) return s;
  if (act_fmt == CHAM_A_FP16 && (X == nullptr || !aligned16(X)))
    return fail(CHAM_ERR_INVALID_ARG, "X must be a 16-byte aligned device pointer");
  if (blob == nullptr || Y == nullptr || !aligned16(blob) || !aligned16(Y) || (bias != nullptr && !aligned16(bias)))
    return fail(CHAM_ERR_INVALID_ARG, "null or misaligned pointer");
  uint8_t* w = static_cast<uint8_t*>(ws);
  const LinearWs L = linear_ws(M, d, act_fmt);
  const OperandPlan o = operand_plan(M, d, act_fmt);
  const float* act_scale = act_fmt <= CHAM_A_E5M2 ? reinterpret_cast<const float*>(w + L.scale) : nullptr;
  const uint8_t* b = static_cast<const uint8_t*>(blob);
  const int tiles = d->n_tiles[0] + d->n_tiles[1];
  cham::GemmArgs g{};
  g.codes = b + d->off_codes;
  g.wscale = reinterpret_cast<const float*>(b + d->off_scale);
  g.wzero = b + d->off_zero;
  g.we8m0 = b + d->off_e8m0;
  g.wgscale = d->group > 0 ? reinterpret_cast<const uint32_t*>(b + d->off_gscale) : nullptr;
  g.wfmt = b + d->off_fmt;
  g.perm = reinterpret_cast<const int32_t*>(b + d->off_perm);
  g.bias = bias;
  g.act_scale = act_scale;
  g.Y = Y;
  g.y_type = y_type;
  g.rows_per_group = act_fmt <= CHAM_A_E5M2 ? M / n_groups : M;
  g.M = M;
  g.N = d->N;
  g.bits = d->bits;
  g.Np = 128 * tiles;
  g.nk64 = d->Kp / 64;
  g.kblocks = K / 32;
  g.stall_chunk = g_stall_next_gemm;
  g_stall_next_gemm = -1;
  g.dev_status = dev_status;
  const cham::NF4Table& nf4 = nf4_table();
  for (int r = 0; r < 4; ++r) {
    g.nf4_lo[r] = g.nf4_hi[r] = 0;
    for (int k = 0; k < 4; ++k) {
      g.nf4_lo[r] |= static_cast<uint32_t>(nf4.level[4 * r + k] & 0xFFu) << (8 * k);
      g.nf4_hi[r] |= static_cast<uint32_t>(nf4.level[4 * r + k] >> 8) << (8 * k);
    }
  }
  const int num_sms = num_sms_current();
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  g.tile0 = 0;
  g.n_ch_tiles = tiles;
  g.k_split = plan.k_split;
  g.partial = plan.k_split > 1 ? reinterpret_cast<float*>(w + plan.partial) : nullptr;
  if (M <= cham::kSmallM) {
    // a handful of tokens: weight streaming on the CUDA cores (one cluster per 64 channels)
    const void* operand = act_fmt == CHAM_A_FP16 ? X : static_cast<const void*>(w + L.operand);
    g.n_chunks = g.nk64;
    const cudaError_t e = cham::launch_gemm_small(static_cast<const __half*>(operand), g,
                                                  cham::gemm_small_split(tiles, g.nk64, num_sms), st);
    return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "small-M gemm launch");
  }
  CUtensorMap map16;
  if (o.f16) {
    const void* operand = act_fmt == CHAM_A_FP16 ? X : static_cast<const void*>(w + L.operand);
    s = make_act_map(&map16, operand, M, K, plan.bn, 2);
    if (s != CHAM_OK) return s;
  }
  if (o.fp8) {
    // class-0 tiles on FP8 MMAs (the 1-byte codes, K-major rows of K bytes), NF4 tiles on fp16
    CUtensorMap map8;
    s = make_act_map(&map8, w + L.codes, M, K, plan.bn, 1);
    if (s != CHAM_OK) return s;
    g.f8_tiles = d->n_tiles[0];
    g.n_chunks = (g.nk64 + 1) / 2;
    g.b_fmt = act_fmt == CHAM_A_E5M2 ? 1 : 0;
    if (act_fmt == CHAM_A_MXFP8) {
      g.act_e8 = w + L.e8;
      g.act_mp = L.mp;
      g.act_e8_plane = static_cast<int64_t>(L.mp) * 4;
    }
    const cudaError_t e = cham::launch_gemm_f8(map8, o.f16 ? map16 : map8, g, num_sms, plan.bn, st);
    return e == cudaSuccess ? CHAM_OK : cuda_fail(e, "fp8 gemm launch");
  }
  g.n_chunks = g.nk64;
  const cudaError_t e = cham::launch_gemm_f16(map16, g, num_sms, plan.bn, st);
  if (e != cudaSuccess) return cuda_fail(e, "gemm launch");
  return CHAM_OK;
}

cham_status chameleon_linear(const void* X, int M, const cham_wpack_desc* d, const void* blob, int act_fmt,
                             const float* bias, float* Y, void* ws, size_t ws_bytes, int* dev_status, void* stream) {
  cham_status s = check_desc(d);
  if (s != CHAM_OK) return s;
  s = chameleon_linear_prepare(X, M, d, act_fmt, ws, ws_bytes, dev_status, stream);
  if (s != CHAM_OK) return s;
  return chameleon_linear_gemm(X, M, d, blob, act_fmt, bias, Y, ws, ws_bytes, dev_status, stream);
}

}  // extern "C"
