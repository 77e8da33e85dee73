"""ctypes binding of libchameleon (include/chameleon.h): argument marshalling only.

Every step of the quantized linear runs in the library's CUDA kernels; this module only turns torch
tensors into pointers, allocates the buffers the size queries ask for (through torch) and raises
when a call fails.  There is no fallback: without the built library every call raises.
"""
import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libchameleon.so")

# status codes
OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_WORKSPACE, ERR_NONFINITE, ERR_TIMEOUT, ERR_CUDA, ERR_RANGE = range(8)
# activation formats (Sec. 3.2 codes) and the fp16 operand of the weight-only fork
A_INT8_ASYM, A_E4M3, A_E5M2, A_MXFP8, A_MXINT8, A_FP16 = range(6)
# weight formats in palette order
(W_INT8_SYM, W_INT8_ASYM, W_MXINT8, W_INT4_SYM, W_INT4_ASYM, W_NF4, W_E2M1, W_MXINT4,
 W_MXFP4) = range(9)
PALETTE_W8 = 0x007
PALETTE_W4 = 0x1F8
SCHEDULE_SCALED_LINEAR, SCHEDULE_LINEAR = 0, 1
Y_F32, Y_F16, Y_BF16 = 0, 1, 2
MAX_GROUPS = 64

EXPORTS = [
    "chameleon_status_string", "chameleon_last_error_detail", "chameleon_version",
    "chameleon_bucket", "chameleon_snr", "chameleon_kurtosis", "chameleon_route",
    "chameleon_act_moments_workspace_size", "chameleon_act_moments",
    "chameleon_act_quant_size", "chameleon_act_quant",
    "chameleon_select_weight_formats", "chameleon_pack_plan", "chameleon_pack_plan_layout",
    "chameleon_pack_plan_palette", "chameleon_pack_weights",
    "chameleon_linear_workspace_size", "chameleon_linear_launches", "chameleon_linear", "chameleon_linear_prepare",
    "chameleon_linear_gemm", "chameleon_act_quant_noalloc", "chameleon_debug_stall_next_gemm",
    "chameleon_scale_zp", "chameleon_act_quant_static", "chameleon_linear_prepare_static",
    "chameleon_linear_prepare_groups", "chameleon_linear_gemm_ex",
    "chameleon_act_format_sse_workspace_size", "chameleon_act_format_sse", "chameleon_act_format_argmin",
    "chameleon_pack_plan_grouped", "chameleon_group_candidates", "chameleon_select_weight_groups_workspace_size",
    "chameleon_select_weight_groups", "chameleon_candidate_argmin", "chameleon_act_channel_energy",
    "chameleon_select_pack_palette", "chameleon_check",
]


class WPackDesc(ctypes.Structure):
    """cham_wpack_desc (256 bytes)."""
    _fields_ = [("magic", ctypes.c_uint32), ("version", ctypes.c_uint32),
                ("N", ctypes.c_int32), ("K", ctypes.c_int32), ("Kp", ctypes.c_int32),
                ("bits", ctypes.c_int32), ("n_class", ctypes.c_int32 * 2),
                ("n_tiles", ctypes.c_int32 * 2), ("n_fmt", ctypes.c_int32 * 9),
                ("group", ctypes.c_int32),
                ("off_codes", ctypes.c_uint64), ("off_scale", ctypes.c_uint64),
                ("off_zero", ctypes.c_uint64), ("off_e8m0", ctypes.c_uint64),
                ("off_fmt", ctypes.c_uint64), ("off_perm", ctypes.c_uint64),
                ("bytes", ctypes.c_uint64), ("off_gscale", ctypes.c_uint64),
                ("f16_only", ctypes.c_int32), ("layout", ctypes.c_int32), ("fold", ctypes.c_int32),
                ("reserved", ctypes.c_uint8 * 100)]


assert ctypes.sizeof(WPackDesc) == 256


class QParams(ctypes.Structure):
    """cham_qparams: per-tensor scale s, zero point z, 1/s as the quantizer multiplies, format."""
    _fields_ = [("s", ctypes.c_float), ("z", ctypes.c_int32), ("inv", ctypes.c_float), ("fmt", ctypes.c_int32)]


assert ctypes.sizeof(QParams) == 16

_lib = None


class ChameleonError(RuntimeError):
    def __init__(self, status, detail):
        super().__init__("chameleon status %d (%s): %s" % (status, STATUS_NAMES.get(status, "?"), detail))
        self.status = status


STATUS_NAMES = {OK: "ok", ERR_INVALID_ARG: "invalid argument", ERR_UNSUPPORTED: "unsupported",
                ERR_WORKSPACE: "workspace too small", ERR_NONFINITE: "non-finite activation",
                ERR_TIMEOUT: "device wait timed out", ERR_CUDA: "CUDA error",
                ERR_RANGE: "MX weight outside fp16"}


def lib():
    """The loaded library (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError("libchameleon.so is not built: run `python -m paper_2609_33496_gb300.build` "
                           "(there is no fallback path)")
    L = ctypes.CDLL(LIB_PATH)
    vp, i32, i64, u32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_uint32, ctypes.c_size_t
    psz = ctypes.POINTER(ctypes.c_size_t)
    pdesc = ctypes.POINTER(WPackDesc)
    sig = {
        "chameleon_status_string": (ctypes.c_char_p, [i32]),
        "chameleon_last_error_detail": (ctypes.c_char_p, []),
        "chameleon_version": (i32, []),
        "chameleon_bucket": (i32, [i32, i32, i32]),
        "chameleon_snr": (i32, [i32, i32, ctypes.POINTER(ctypes.c_double)]),
        "chameleon_kurtosis": (ctypes.c_double, [ctypes.POINTER(ctypes.c_double)]),
        "chameleon_route": (i32, [ctypes.c_double, ctypes.c_double, i32]),
        "chameleon_act_moments_workspace_size": (i32, [i64, psz]),
        "chameleon_act_moments": (i32, [vp, i64, vp, vp, sz, vp]),
        "chameleon_act_quant_size": (i32, [i32, i32, i32, psz, psz]),
        "chameleon_act_quant": (i32, [vp, i32, i32, i32, vp, sz, vp, sz, vp, vp]),
        "chameleon_select_weight_formats": (i32, [vp, i32, i32, u32, vp, vp, vp]),
        "chameleon_pack_plan": (i32, [i32, i32, vp, pdesc]),
        "chameleon_pack_plan_layout": (i32, [i32, i32, vp, i32, i32, pdesc]),
        "chameleon_pack_plan_palette": (i32, [i32, i32, ctypes.c_uint32, pdesc]),
        "chameleon_pack_weights": (i32, [vp, vp, pdesc, vp, sz, vp, vp]),
        "chameleon_linear_workspace_size": (i32, [i32, pdesc, i32, psz]),
        "chameleon_linear_launches": (i32, [i32, pdesc, i32, i32, i32, ctypes.POINTER(ctypes.c_int),
                                            ctypes.POINTER(ctypes.c_int)]),
        "chameleon_linear": (i32, [vp, i32, pdesc, vp, i32, vp, vp, vp, sz, vp, vp]),
        "chameleon_linear_prepare": (i32, [vp, i32, pdesc, i32, vp, sz, vp, vp]),
        "chameleon_linear_gemm": (i32, [vp, i32, pdesc, vp, i32, vp, vp, vp, sz, vp, vp]),
        "chameleon_act_quant_noalloc": (i32, [vp, i32, i32, i32, vp, sz, vp, vp]),
        "chameleon_debug_stall_next_gemm": (i32, [i32]),
        "chameleon_scale_zp": (i32, [i32, ctypes.c_float, ctypes.c_float, ctypes.POINTER(QParams)]),
        "chameleon_act_quant_static": (i32, [vp, i32, i32, i32, ctypes.POINTER(QParams), vp, sz, vp, vp]),
        "chameleon_linear_prepare_static": (i32, [vp, i32, pdesc, i32, ctypes.POINTER(QParams), vp, sz, vp, vp]),
        "chameleon_linear_prepare_groups": (i32, [vp, i32, pdesc, i32, i32, vp, sz, vp, vp]),
        "chameleon_linear_gemm_ex": (i32, [vp, i32, pdesc, vp, i32, i32, vp, vp, i32, vp, sz, vp, vp]),
        "chameleon_act_format_sse_workspace_size": (i32, [i32, i32, psz]),
        "chameleon_act_format_sse": (i32, [vp, i32, i32, vp, vp, sz, vp, vp]),
        "chameleon_act_format_argmin": (i32, [ctypes.POINTER(ctypes.c_double)]),
        "chameleon_pack_plan_grouped": (i32, [i32, i32, i32, i32, pdesc]),
        "chameleon_group_candidates": (i32, [u32, u32, vp, vp, i32, ctypes.POINTER(ctypes.c_int)]),
        "chameleon_select_weight_groups_workspace_size": (i32, [i32, i32, u32, u32, psz]),
        "chameleon_select_weight_groups": (i32, [vp, i32, i32, u32, u32, vp, vp, vp, sz, vp]),
        "chameleon_candidate_argmin": (i32, [ctypes.POINTER(ctypes.c_double), i32]),
        "chameleon_act_channel_energy": (i32, [vp, i32, i32, vp, vp]),
        "chameleon_select_pack_palette": (i32, [vp, i32, i32, u32, pdesc, vp, vp, sz, vp, vp]),
        "chameleon_check": (i32, [vp, vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def status_string(status):
    """The library's name for a status code."""
    return lib().chameleon_status_string(status).decode()


def version():
    """The library's ABI version (2: descriptors with group-wise weights)."""
    return lib().chameleon_version()


def check(status):
    """Raise ChameleonError (with the library's detail line) unless status is CHAM_OK."""
    if status != OK:
        raise ChameleonError(status, lib().chameleon_last_error_detail().decode())


def device_status(dev_status, stream=None):
    """Synchronise the stream and return the device status word (0 = ok) without raising."""
    return lib().chameleon_check(_ptr(dev_status), _stream(stream))


def _ptr(t):
    """Device address of a tensor the library reads or writes as one dense buffer."""
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors passed to libchameleon must be contiguous (got strides %s)" % (t.stride(),))
    if not t.is_cuda:
        raise ValueError("tensors passed to libchameleon must be CUDA tensors (got one on %s)" % (t.device,))
    return ctypes.c_void_p(t.data_ptr())


def _typed(t, dtype_name, what):
    """_ptr of t after checking its element type (None passes through)."""
    if t is not None and str(t.dtype) != "torch." + dtype_name:
        raise TypeError("%s must be a %s tensor (got %s)" % (what, dtype_name, t.dtype))
    return _ptr(t)


def _half(t, what):
    return _typed(t, "float16", what)


def _f32(t, what):
    return _typed(t, "float32", what)


def _stream(stream):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _bytes(n, device):
    import torch
    return torch.empty(max(int(n), 16), dtype=torch.uint8, device=device)


# ------------------------------------------------------------------ host helpers
def bucket(t, T=1000, B=10):
    """Timestep bucket b = min(floor(t / (T/B)), B - 1) (Alg. 2, Alg. 3); -1 for invalid input."""
    return lib().chameleon_bucket(int(t), int(T), int(B))


def snr(schedule=SCHEDULE_SCALED_LINEAR, T=1000):
    """SNR(t) = abar_t / (1 - abar_t) for t = 0..T-1 of a noise schedule (host, float64 [T])."""
    out = np.zeros(T, dtype=np.float64)
    check(lib().chameleon_snr(schedule, T, out.ctypes.data_as(ctypes.POINTER(ctypes.c_double))))
    return out


def kurtosis(sums):
    """kappa = m4 / m2^2 from the power sums {n, S1, S2, S3, S4} (the first five of act_moments)."""
    arr = (ctypes.c_double * 5)(*[float(s) for s in sums[:5]])
    return lib().chameleon_kurtosis(arr)


def route(kappa, snr_b, is_shortcut=False):
    """The activation format the routing rule picks for kurtosis kappa at SNR(t_b) (Sec. 3.3)."""
    return lib().chameleon_route(float(kappa), float(snr_b), int(bool(is_shortcut)))


# ------------------------------------------------------------------ calibration sums
def act_moments(X, out=None, stream=None):
    """Alg. 1 accumulator {n, S1..S4, min, max} of the fp16 tensor X, added into `out` (a
    7-element float64 CUDA tensor; a fresh one when None)."""
    import torch
    if out is None:
        out = torch.tensor([0, 0, 0, 0, 0, float("inf"), float("-inf")], dtype=torch.float64, device=X.device)
    n = X.numel()
    ws_b = ctypes.c_size_t()
    check(lib().chameleon_act_moments_workspace_size(n, ctypes.byref(ws_b)))
    ws = _bytes(ws_b.value, X.device)
    check(lib().chameleon_act_moments(_half(X, "X"), n, _ptr(out), _ptr(ws), ws_b.value, _stream(stream)))
    return out


# ------------------------------------------------------------------ a2-a4
def act_quant_size(M, K, fmt):
    """(qact bytes, workspace bytes) of chameleon_act_quant for an M x K tensor in format fmt."""
    q, w = ctypes.c_size_t(), ctypes.c_size_t()
    check(lib().chameleon_act_quant_size(M, K, fmt, ctypes.byref(q), ctypes.byref(w)))
    return q.value, w.value


def act_quant(X, fmt, dev_status=None, stream=None, qact=None, ws=None):
    """Quantize fp16 X (M x K, CUDA) in activation format fmt.  Returns the raw qact byte buffer
    (layout of include/chameleon.h) and the device status word.  qact and ws may be passed in for
    reuse (uint8 CUDA tensors of at least the size query's bytes)."""
    import torch
    M, K = X.shape
    qb, wb = act_quant_size(M, K, fmt)
    if qact is None or qact.numel() < qb:
        qact = _bytes(qb, X.device)
    if ws is None or ws.numel() < wb:
        ws = _bytes(wb, X.device)
    if dev_status is None:
        dev_status = torch.zeros(1, dtype=torch.int32, device=X.device)
    check(lib().chameleon_act_quant(_half(X, "X"), M, K, fmt, _ptr(qact), qact.numel(), _ptr(ws), ws.numel(),
                                    _ptr(dev_status), _stream(stream)))
    return qact, dev_status


def scale_zp(fmt, lo, hi):
    """ScaleZP of a per-tensor activation format from the range [lo, hi] (host only)."""
    p = QParams()
    check(lib().chameleon_scale_zp(fmt, lo, hi, ctypes.byref(p)))
    return p


def _pref(params):
    return None if params is None else ctypes.byref(params)


def act_quant_static(X, fmt, params, dev_status=None, stream=None):
    """Quantize fp16 X with fixed per-tensor parameters (a QParams from scale_zp of a calibration
    range); MX formats ignore params.  Returns the qact byte buffer and the device status word."""
    import torch
    M, K = X.shape
    qb, _ = act_quant_size(M, K, fmt)
    qact = _bytes(qb, X.device)
    if dev_status is None:
        dev_status = torch.zeros(1, dtype=torch.int32, device=X.device)
    check(lib().chameleon_act_quant_static(_half(X, "X"), M, K, fmt, _pref(params), _ptr(qact), qb, _ptr(dev_status),
                                           _stream(stream)))
    return qact, dev_status


def split_qact(qact, M, K):
    """Views of a qact buffer: codes (M x K uint8), params (s, z, inv, fmt), e8m0 (M x K/32)."""
    import torch
    n = M * K
    P = (n + 255) // 256 * 256
    codes = qact[:n].view(M, K)
    pbytes = qact[P:P + 16].cpu().numpy().tobytes()
    s, inv = np.frombuffer(pbytes[0:4], np.float32)[0], np.frombuffer(pbytes[8:12], np.float32)[0]
    z, fmt = int(np.frombuffer(pbytes[4:8], np.int32)[0]), int(np.frombuffer(pbytes[12:16], np.int32)[0])
    e8 = qact[P + 256:P + 256 + n // 32].view(M, K // 32)
    return codes, {"s": s, "z": z, "inv": inv, "fmt": fmt}, e8


# ------------------------------------------------------------------ Eq. format-argmin
def act_format_sse(X, out=None, dev_status=None, stream=None):
    """SSE of the five activation formats on fp16 X (M x K, CUDA), added to `out` (5 float64 on the
    device; zeros when not given).  Returns (out, dev_status)."""
    import torch
    M, K = X.shape
    if out is None:
        out = torch.zeros(5, dtype=torch.float64, device=X.device)
    if dev_status is None:
        dev_status = torch.zeros(1, dtype=torch.int32, device=X.device)
    w = ctypes.c_size_t()
    check(lib().chameleon_act_format_sse_workspace_size(M, K, ctypes.byref(w)))
    ws = _bytes(w.value, X.device)
    check(lib().chameleon_act_format_sse(_half(X, "X"), M, K, _ptr(out), _ptr(ws), w.value, _ptr(dev_status),
                                         _stream(stream)))
    return out, dev_status


def act_format_argmin(sse_host):
    """First format of the activation palette with the least error (host)."""
    a = (ctypes.c_double * 5)(*[float(v) for v in sse_host])
    return lib().chameleon_act_format_argmin(a)


# ------------------------------------------------------------------ a5
def select_weight_formats(W, palette_mask, want_sse=False, stream=None, fmt_out=None):
    """fmt_out: optional uint8 device tensor of N elements to write the formats into."""
    import torch
    N, K = W.shape
    fmt = torch.empty(N, dtype=torch.uint8, device=W.device) if fmt_out is None else fmt_out
    if fmt.numel() != N or fmt.dtype != torch.uint8 or not fmt.is_contiguous():
        raise ValueError("fmt_out must be a contiguous uint8 tensor of N elements")
    sse = torch.empty((N, 9), dtype=torch.float64, device=W.device) if want_sse else None
    check(lib().chameleon_select_weight_formats(_half(W, "W"), N, K, palette_mask, _ptr(fmt), _ptr(sse),
                                                _stream(stream)))
    return fmt, sse


# ------------------------------------------------------------------ a6
def pack_plan_palette(N, K, palette_mask):
    """Packed layout for N x K weights whose palette shares one MMA class (no host copy of the
    selected formats needed); the formats are written by the selection on the device."""
    d = WPackDesc()
    check(lib().chameleon_pack_plan_palette(N, K, palette_mask, ctypes.byref(d)))
    return d


GROUP_SIZES = (32, 64, 128, 192, 288)


def group_mask(groups):
    """Bit mask of group sizes (bit i = GROUP_SIZES[i])."""
    return sum(1 << GROUP_SIZES.index(g) for g in groups)


def pack_plan_grouped(N, K, fmt, group):
    """Plan of a group-wise blob: every channel in fmt, one scale per `group` input channels."""
    d = WPackDesc()
    check(lib().chameleon_pack_plan_grouped(N, K, fmt, group, ctypes.byref(d)))
    return d


def group_candidates(palette_mask, gmask):
    """The (g, f) candidates of a search, in search order."""
    n = ctypes.c_int()
    g = (ctypes.c_int * 64)()
    f = (ctypes.c_int * 64)()
    check(lib().chameleon_group_candidates(palette_mask, gmask, g, f, 64, ctypes.byref(n)))
    return [(g[i], f[i]) for i in range(n.value)]


def select_weight_groups(W, palette_mask, gmask, energy=None, stream=None):
    """Scores (device float64, one per candidate) of the per-linear (g, f) search."""
    import torch
    N, K = W.shape
    w = ctypes.c_size_t()
    check(lib().chameleon_select_weight_groups_workspace_size(N, K, palette_mask, gmask, ctypes.byref(w)))
    ws = _bytes(w.value, W.device)
    scores = torch.empty(len(group_candidates(palette_mask, gmask)), dtype=torch.float64, device=W.device)
    check(lib().chameleon_select_weight_groups(_half(W, "W"), N, K, palette_mask, gmask, _ptr(energy), _ptr(scores),
                                               _ptr(ws), w.value, _stream(stream)))
    return scores


def candidate_argmin(scores_host):
    """Index of the first smallest (g, f) search score (host list or array)."""
    a = (ctypes.c_double * len(scores_host))(*[float(v) for v in scores_host])
    return lib().chameleon_candidate_argmin(a, len(scores_host))


def act_channel_energy(X, energy=None, stream=None):
    """energy[k] += sum_m X[m, k]^2 (device float64 [K], zeros when not given)."""
    import torch
    M, K = X.shape
    if energy is None:
        energy = torch.zeros(K, dtype=torch.float64, device=X.device)
    check(lib().chameleon_act_channel_energy(_half(X, "X"), M, K, _ptr(energy), _stream(stream)))
    return energy


def pack_plan(N, K, fmt_host, layout=0, fold=0):
    """Packed layout (cham_wpack_desc) for N x K weights with the selected formats fmt_host (host
    uint8 [N]); layout 1 groups the channels of each format (formats with fewer than `fold`
    channels share their class's tail group)."""
    f = np.ascontiguousarray(np.asarray(fmt_host, dtype=np.uint8))
    d = WPackDesc()
    check(lib().chameleon_pack_plan_layout(N, K, f.ctypes.data_as(ctypes.c_void_p), layout, fold, ctypes.byref(d)))
    return d


def select_pack_palette(W, palette_mask, desc, fmt_out=None, blob=None, dev_status=None, stream=None):
    """Selection and pack in one launch for a one-class palette plan (pack_plan_palette).  Returns
    (fmt device uint8 [N], blob, dev_status)."""
    import torch
    N, K = W.shape
    if fmt_out is None:
        fmt_out = torch.empty(N, dtype=torch.uint8, device=W.device)
    if blob is None or blob.numel() < desc.bytes:
        blob = _bytes(desc.bytes, W.device)
    if dev_status is None:
        dev_status = torch.zeros(1, dtype=torch.int32, device=W.device)
    check(lib().chameleon_select_pack_palette(_half(W, "W"), N, K, palette_mask, ctypes.byref(desc), _ptr(fmt_out),
                                              _ptr(blob), blob.numel(), _ptr(dev_status), _stream(stream)))
    return fmt_out, blob, dev_status


def pack_weights(W, fmt_dev, desc, dev_status=None, stream=None, blob=None):
    """Encode each channel of W (fp16 N x K, CUDA) in its format fmt_dev (uint8 [N], CUDA) into the
    packed blob desc describes.  Returns (blob, dev_status)."""
    import torch
    if blob is None or blob.numel() < desc.bytes:
        blob = _bytes(desc.bytes, W.device)
    if dev_status is None:
        dev_status = torch.zeros(1, dtype=torch.int32, device=W.device)
    check(lib().chameleon_pack_weights(_half(W, "W"), _ptr(fmt_dev), ctypes.byref(desc), _ptr(blob), blob.numel(),
                                       _ptr(dev_status), _stream(stream)))
    return blob, dev_status


# ------------------------------------------------------------------ a7/a8
def linear_workspace_size(M, desc, act_fmt):
    """Workspace bytes of chameleon_linear for M rows, the packed weights desc and act_fmt."""
    w = ctypes.c_size_t()
    check(lib().chameleon_linear_workspace_size(M, ctypes.byref(desc), act_fmt, ctypes.byref(w)))
    return w.value


def linear_launches(M, desc, act_fmt, n_groups=1, is_static=False):
    """(prepare launches, gemm launches): the kernels chameleon_linear_prepare* and
    chameleon_linear_gemm* launch for M rows of the layer desc in act_fmt (host only)."""
    p, g = ctypes.c_int(), ctypes.c_int()
    check(lib().chameleon_linear_launches(M, ctypes.byref(desc), act_fmt, n_groups, int(bool(is_static)),
                                          ctypes.byref(p), ctypes.byref(g)))
    return p.value, g.value


def linear(X, desc, blob, act_fmt, bias=None, Y=None, ws=None, dev_status=None, stream=None):
    """Y = DQ(Q_act_fmt(X)) DQ(W)^T + bias on the GPU.  Buffers may be passed in for reuse."""
    import torch
    M = X.shape[0]
    need = linear_workspace_size(M, desc, act_fmt)
    if ws is None or ws.numel() < need:
        ws = _bytes(need, X.device)
    if Y is None:
        Y = torch.empty((M, desc.N), dtype=torch.float32, device=X.device)
    if dev_status is None:
        dev_status = torch.zeros(1, dtype=torch.int32, device=X.device)
    check(lib().chameleon_linear(_half(X, "X"), M, ctypes.byref(desc), _ptr(blob), act_fmt, _f32(bias, "bias"),
                                 _f32(Y, "Y"), _ptr(ws), ws.numel(), _ptr(dev_status), _stream(stream)))
    return Y, dev_status


def linear_static(X, desc, blob, act_fmt, params, bias=None, Y=None, ws=None, dev_status=None, stream=None):
    """linear with the activation quantized by fixed parameters (linear_prepare_static, then
    linear_gemm on the same stream)."""
    import torch
    M = X.shape[0]
    need = linear_workspace_size(M, desc, act_fmt)
    if ws is None or ws.numel() < need:
        ws = _bytes(need, X.device)
    if Y is None:
        Y = torch.empty((M, desc.N), dtype=torch.float32, device=X.device)
    if dev_status is None:
        dev_status = torch.zeros(1, dtype=torch.int32, device=X.device)
    linear_prepare_static(X, desc, act_fmt, params, ws, dev_status, stream)
    linear_gemm(X, desc, blob, act_fmt, bias, Y, ws, dev_status, stream)
    return Y, dev_status


def _y_type(Y):
    import torch
    t = {torch.float32: Y_F32, torch.float16: Y_F16, torch.bfloat16: Y_BF16}.get(Y.dtype)
    if t is None:
        raise ValueError("Y must be float32, float16 or bfloat16")
    return t


def linear_prepare_groups(X, desc, act_fmt, n_groups, ws, dev_status, stream=None):
    """First half of linear with per-sample scales: rows in n_groups equal groups, each quantized
    with the ScaleZP of its own range, into the operands the layer desc's tiles need."""
    check(lib().chameleon_linear_prepare_groups(_half(X, "X"), X.shape[0], ctypes.byref(desc), act_fmt, n_groups,
                                                _ptr(ws), ws.numel(), _ptr(dev_status), _stream(stream)))


def linear_gemm_ex(X, desc, blob, act_fmt, n_groups, bias, Y, ws, dev_status, stream=None):
    """Second half of linear with the operand's row groups; the output type is Y's dtype."""
    check(lib().chameleon_linear_gemm_ex(_half(X, "X"), X.shape[0], ctypes.byref(desc), _ptr(blob), act_fmt,
                                         n_groups, _f32(bias, "bias"), _ptr(Y), _y_type(Y), _ptr(ws), ws.numel(),
                                         _ptr(dev_status), _stream(stream)))


def linear_ex(X, desc, blob, act_fmt, n_groups=1, y_dtype=None, bias=None, Y=None, ws=None, dev_status=None,
              stream=None):
    """linear with per-sample activation scales (n_groups) and an fp32 / fp16 / bf16 output."""
    import torch
    M = X.shape[0]
    need = linear_workspace_size(M, desc, act_fmt)
    if ws is None or ws.numel() < need:
        ws = _bytes(need, X.device)
    if Y is None:
        Y = torch.empty((M, desc.N), dtype=y_dtype or torch.float32, device=X.device)
    if dev_status is None:
        dev_status = torch.zeros(1, dtype=torch.int32, device=X.device)
    linear_prepare_groups(X, desc, act_fmt, n_groups, ws, dev_status, stream)
    linear_gemm_ex(X, desc, blob, act_fmt, n_groups, bias, Y, ws, dev_status, stream)
    return Y, dev_status


def debug_stall_next_gemm(chunk):
    """Test hook: the next GEMM launch withholds one K-chunk so its bounded waits run out."""
    check(lib().chameleon_debug_stall_next_gemm(chunk))


def linear_prepare(X, desc, act_fmt, ws, dev_status, stream=None):
    """First half of linear: quantize X into the workspace operands the layer desc's tiles need."""
    check(lib().chameleon_linear_prepare(_half(X, "X"), X.shape[0], ctypes.byref(desc), act_fmt, _ptr(ws),
                                         ws.numel(), _ptr(dev_status), _stream(stream)))


def linear_prepare_static(X, desc, act_fmt, params, ws, dev_status, stream=None):
    """First half of linear on the static path: quantize X with fixed parameters (QParams)."""
    check(lib().chameleon_linear_prepare_static(_half(X, "X"), X.shape[0], ctypes.byref(desc), act_fmt,
                                                _pref(params), _ptr(ws), ws.numel(), _ptr(dev_status),
                                                _stream(stream)))


def linear_gemm(X, desc, blob, act_fmt, bias, Y, ws, dev_status, stream=None):
    """Second half of linear: the tcgen05 GEMM on the prepared operand."""
    check(lib().chameleon_linear_gemm(_half(X, "X"), X.shape[0], ctypes.byref(desc), _ptr(blob), act_fmt,
                                      _f32(bias, "bias"), _f32(Y, "Y"), _ptr(ws), ws.numel(), _ptr(dev_status),
                                      _stream(stream)))


def act_quant_noalloc(X, fmt, qact, dev_status, stream=None):
    """chameleon_act_quant without a workspace, for callers that cannot allocate at call time:
    the caller passes the output buffer `qact` (sized by act_quant_size) and the status word; the
    range partials live in a static device array inside the library.  Returns the raw status."""
    M, K = X.shape
    return lib().chameleon_act_quant_noalloc(_half(X, "X"), M, K, fmt, _ptr(qact), qact.numel(), _ptr(dev_status),
                                             _stream(stream))
