// noalloc.cu -- chameleon_act_quant_noalloc: the activation quantizer with its scratch in a
// file-scope device array, for callers that cannot allocate device memory at call time.
//
// The per-tensor formats (INT8-asym, E4M3, E5M2) reduce the tensor's range in two launches and
// need one 16-byte partial per CTA of the first launch between them.  chameleon_act_quant takes
// that scratch from the caller's `ws`; this variant keeps it in g_range_scratch below instead, so
// the caller passes only X, the output buffer and the status word.
//
// Limits and sharing rules:
//   * capacity: kScratchParts partials (32 KiB).  The range pass launches at most 8 CTAs per SM, so
//     any M and K fit on GPUs with up to 256 SMs; a request that would need more partials is
//     rejected with CHAM_ERR_WORKSPACE before anything is launched.
//   * every GPU that loads the library holds the array until the process exits.
//   * all calls share the array.  Nothing in it has to start at zero: the first launch of a call
//     overwrites every partial the second launch reads.  Calls whose kernels overlap on the GPU
//     (for example on two streams at once) race on the array and produce wrong scales.
//   * the first call on a device looks up the array's device address for that device (with that
//     device current); make that first call before any stream capture.  The address is kept for
//     the life of the process: after cudaDeviceReset the module is loaded again and the array may
//     move, so the entry point must not be called on a device that has been reset.
#include <cuda_runtime.h>

#include <mutex>

#include "act_quant.cuh"

namespace {

constexpr int kScratchParts = 2048;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) cham::RangePartial g_range_scratch[kScratchParts];

// Device address of g_range_scratch on the current device, looked up once per device.
cham_status scratch_address(cham::RangePartial** out) {
  static std::mutex mu;
  static cham::RangePartial* addr[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return CHAM_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return CHAM_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(mu);
  if (addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_range_scratch);
    if (e != cudaSuccess) return CHAM_ERR_CUDA;
    addr[dev] = static_cast<cham::RangePartial*>(p);
  }
  *out = addr[dev];
  return CHAM_OK;
}

}  // namespace

extern "C" {

cham_status chameleon_act_quant_noalloc(const void* X, int M, int K, int fmt, void* qact, size_t qact_bytes,
                                        int* dev_status, void* stream) {
  if (M <= 0 || K <= 0 || K % 32 != 0) return CHAM_ERR_INVALID_ARG;
  if (fmt < CHAM_A_INT8_ASYM || fmt > CHAM_A_MXINT8) return CHAM_ERR_INVALID_ARG;
  if (X == nullptr || qact == nullptr || (reinterpret_cast<uintptr_t>(X) & 15u) != 0 ||
      (reinterpret_cast<uintptr_t>(qact) & 15u) != 0)
    return CHAM_ERR_INVALID_ARG;
  const size_t n = static_cast<size_t>(M) * K;
  const size_t params_off = (n + 255) / 256 * 256;
  const size_t e8_off = params_off + 256;
  const size_t need = e8_off + (n / 32 + 255) / 256 * 256;
  if (qact_bytes < need) return CHAM_ERR_WORKSPACE;

  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return CHAM_ERR_CUDA;
  const int64_t nvec = static_cast<int64_t>(n / 8);
  const int nparts = cham::range_grid(nvec, sms);
  if (fmt <= CHAM_A_E5M2 && nparts > kScratchParts)
    return CHAM_ERR_WORKSPACE;
  cham::RangePartial* scratch = nullptr;
  cham_status s = scratch_address(&scratch);
  if (s != CHAM_OK) return s;

  uint8_t* q = static_cast<uint8_t*>(qact);
  cham::ActQuantArgs a{};
  a.X = static_cast<const uint4*>(X);
  a.nvec = nvec;
  a.num_sms = sms;
  a.parts = scratch;
  a.nparts = nparts;
  a.codes = reinterpret_cast<uint2*>(q);
  a.deq = nullptr;
  a.e8m0 = fmt >= CHAM_A_MXFP8 ? q + e8_off : nullptr;
  a.params = reinterpret_cast<cham_qparams*>(q + params_off);
  a.scale_out = nullptr;
  a.dev_status = dev_status;
  cham::launch_act_quant(fmt, a, true, false, static_cast<cudaStream_t>(stream));
  e = cudaGetLastError();
  if (e != cudaSuccess) return CHAM_ERR_CUDA;
  return CHAM_OK;
}

}  // extern "C"
