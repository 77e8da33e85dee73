"""Number formats of the Chameleon palette, written from their definitions.

Test infrastructure (see ``oracle/__init__``).  Passages followed:
  * activation palette and codes 0..4 -- Sec. 3.2 (F_a, numbered 0 to 4 in the runtime LUT);
  * weight palettes F_w^(8), F_w^(4) -- Sec. 3.2;
  * INT8-asym, E4M3, E5M2, MX, 4-bit codes -- App. A.11 (the number-format appendix);
  * ScaleZP -- App. A.7 (shared helper of Alg. 1 and Alg. 3);
  * clamp before the FP8 cast -- App. A.7, implementation note (ii);
  * MX shared exponent floor(log2 max|x|) with an E8M0 byte -- Sec. 3.6, App. A.11, App. A.12.

Readings of passages the paper leaves open (numbered R1..R17 across the project):
  R1  MX shared exponent: X = floor(log2 amax) - emax_elem with emax_elem = 8 (E4M3 body),
      2 (E2M1 body), 0 (integer bodies) -- the OCP rule the paper says it follows exactly.
  R2  all-zero MX block: E8M0 byte 0; the element codes are the encodings of the zero elements
      (sign of zero kept for FP bodies).
  R3  MX integer bodies are symmetric: MXINT8 codes in [-127, 127] (value code * 2^-6),
      MXINT4 codes in [-7, 7] (value code * 2^-2).
  R4  INT-asym uses the zero-inclusive range lo' = min(lo, 0), hi' = max(hi, 0).
  R5  round() is round-to-nearest, ties to even, everywhere.
  R6  x/s is evaluated as x * inv with inv = (levels / range) by one correctly rounded fp32
      division; the fp32 product is rounded before the format rounding (two steps).
  R7  degenerate range (amax == 0 or hi' == lo'): s = 1, inv = 1, z = 0.
  R8  symmetric integer ranges are [-127, 127] and [-7, 7]; s = amax / 127 or amax / 7.
  R10 weight granularity: per output channel for INT8/INT4 sym/asym, NF4 and E2M1; 32-element
      blocks along K with an E8M0 exponent for the MX formats.
"""
import numpy as np

# ---------------------------------------------------------------- format codes (Sec. 3.2)
A_INT8_ASYM, A_E4M3, A_E5M2, A_MXFP8, A_MXINT8, A_FP16 = 0, 1, 2, 3, 4, 5
ACT_FORMATS = (A_INT8_ASYM, A_E4M3, A_E5M2, A_MXFP8, A_MXINT8)

W_INT8_SYM, W_INT8_ASYM, W_MXINT8 = 0, 1, 2
W_INT4_SYM, W_INT4_ASYM, W_NF4, W_E2M1, W_MXINT4, W_MXFP4 = 3, 4, 5, 6, 7, 8
W8_PALETTE = (W_INT8_SYM, W_INT8_ASYM, W_MXINT8)
W4_PALETTE = (W_INT4_SYM, W_INT4_ASYM, W_NF4, W_E2M1, W_MXINT4, W_MXFP4)
W_BITS = {W_INT8_SYM: 8, W_INT8_ASYM: 8, W_MXINT8: 8, W_INT4_SYM: 4, W_INT4_ASYM: 4,
          W_NF4: 4, W_E2M1: 4, W_MXINT4: 4, W_MXFP4: 4}
W_IS_MX = {f: f in (W_MXINT8, W_MXINT4, W_MXFP4) for f in W_BITS}

MX_BLOCK = 32  # MX formats: 32-element blocks sharing one 8-bit exponent (Sec. 3.2)

# ---------------------------------------------------------------- binary minifloats (App. A.11)
# name: (exponent bits, mantissa bits, bias, largest finite magnitude)
FP_SPECS = {
    "e4m3": (4, 3, 7, 448.0),      # max 448, smallest normal 2^-6, no infinities (App. A.11)
    "e5m2": (5, 2, 15, 57344.0),   # max 57344, smallest normal 2^-14 (App. A.11)
    "e2m1": (2, 1, 1, 6.0),        # {0, +-0.5, +-1, +-1.5, +-2, +-3, +-4, +-6}
}


def fp_round(v, name):
    """Round float64 values (holding fp32 numbers) to the nearest value of the minifloat `name`,
    ties to even mantissa (R5), saturating at the largest finite magnitude (App. A.7 note (ii):
    clamp to the representable range before the cast).  Returns float64 grid values; the sign
    of zero is kept."""
    ebits, mbits, bias, vmax = FP_SPECS[name]
    v = np.asarray(v, dtype=np.float64)
    a = np.abs(v)
    emin = 1 - bias
    _, ex = np.frexp(a)                     # a = m * 2^ex, m in [0.5, 1)
    e = np.maximum(ex - 1, emin)            # binade of a, floored at the subnormal binade
    quantum = np.ldexp(1.0, e - mbits)      # spacing of the grid inside that binade
    r = np.rint(a / quantum) * quantum      # exact power-of-two scaling, RNE on the integer
    r = np.minimum(r, vmax)
    return np.copysign(r, v)


def fp_encode(r, name):
    """Bit pattern (sign | exponent | mantissa) of grid values produced by fp_round."""
    ebits, mbits, bias, _ = FP_SPECS[name]
    r = np.asarray(r, dtype=np.float64)
    a = np.abs(r)
    emin = 1 - bias
    _, ex = np.frexp(a)
    e = ex - 1
    normal = a >= np.ldexp(1.0, emin)
    ef = np.where(normal, e + bias, 0)
    mf_normal = (np.ldexp(a, -np.where(normal, e, 0)) - 1.0) * (1 << mbits)
    mf_sub = np.ldexp(a, -(emin - mbits))
    mf = np.where(normal, mf_normal, mf_sub)
    sign = np.signbit(r).astype(np.int64)
    code = (sign << (ebits + mbits)) | (ef.astype(np.int64) << mbits) | mf.astype(np.int64)
    return code


def fp_decode(code, name):
    """Value of each bit pattern; NaN for the NaN encodings (E4M3 S.1111.111, E5M2 exponent
    all ones) -- App. A.11."""
    ebits, mbits, bias, _ = FP_SPECS[name]
    code = np.asarray(code, dtype=np.int64)
    sign = (code >> (ebits + mbits)) & 1
    ef = (code >> mbits) & ((1 << ebits) - 1)
    mf = code & ((1 << mbits) - 1)
    emin = 1 - bias
    val = np.where(ef == 0,
                   np.ldexp(mf.astype(np.float64), emin - mbits),
                   np.ldexp(1.0 + mf / float(1 << mbits), ef - bias))
    if name == "e4m3":
        val = np.where((ef == 15) & (mf == 7), np.nan, val)
    elif name == "e5m2":
        val = np.where(ef == 31, np.nan, val)   # E5M2 keeps IEEE inf/NaN encodings
    return np.where(sign == 1, -val, val)


def fp_quantize(v, name):
    """RNE + saturate + encode in one call."""
    return fp_encode(fp_round(v, name), name)


# ---------------------------------------------------------------- E8M0 shared exponent
def floor_log2(a):
    """floor(log2 a) of positive float32/float64 values, read exactly from the exponent."""
    _, ex = np.frexp(np.asarray(a, dtype=np.float64))
    return ex - 1


def e8m0_byte(X):
    """E8M0 byte of a power-of-two exponent X: X + 127, clamped to [0, 254] (255 is NaN)."""
    return np.clip(np.asarray(X, dtype=np.int64) + 127, 0, 254)


# ---------------------------------------------------------------- integer helpers
def rne(v):
    """Round to nearest integer, ties to even (R5)."""
    return np.rint(np.asarray(v, dtype=np.float64))


def _f32(v):
    return np.asarray(v, dtype=np.float32)


# ---------------------------------------------------------------- ScaleZP (App. A.7)
def scale_zp_asym(lo, hi, levels):
    """ScaleZP for an asymmetric integer format with `levels` steps (255 for INT8, 15 for INT4):
    s = (hi - lo) / levels, z = round(-lo / s) (App. A.7), with the zero-inclusive range (R4),
    x/s as x*inv (R6) and the degenerate range rule (R7).  Returns fp32 (s, inv) and int z."""
    lo = np.float32(min(np.float32(lo), np.float32(0.0)))
    hi = np.float32(max(np.float32(hi), np.float32(0.0)))
    d = np.float32(hi - lo)
    if d == 0:
        return np.float32(1.0), np.float32(1.0), 0
    s = np.float32(d / np.float32(levels))
    inv = np.float32(np.float32(levels) / d)
    z = int(rne(np.float32(np.float32(-lo) * inv)))
    z = min(max(z, 0), levels)
    return s, inv, z


def scale_sym(amax, fmax):
    """Symmetric scale: s = amax / fmax, inv = fmax / amax (App. A.7 for FP8 with fmax = 448 or
    57344; R8 for symmetric integers with fmax = 127 or 7; E2M1 with fmax = 6)."""
    amax = np.float32(amax)
    if amax == 0:
        return np.float32(1.0), np.float32(1.0)
    return np.float32(amax / np.float32(fmax)), np.float32(np.float32(fmax) / amax)


def scale_zp(fmt, lo, hi):
    """ScaleZP of a per-tensor activation format from an observed range (App. A.7; the helper of
    Alg. 1 and Alg. 3): INT8-asym by scale_zp_asym, E4M3 / E5M2 by scale_sym of max(|lo|, |hi|).
    Returns fp32 (s, inv) and int z."""
    if fmt == A_INT8_ASYM:
        return scale_zp_asym(lo, hi, 255)
    if fmt in (A_E4M3, A_E5M2):
        amax = max(abs(np.float32(lo)), abs(np.float32(hi)))
        s, inv = scale_sym(amax, 448.0 if fmt == A_E4M3 else 57344.0)
        return s, inv, 0
    raise ValueError("ScaleZP is defined for the per-tensor formats 0..2, not %r" % (fmt,))


# ---------------------------------------------------------------- activation quantizer
def act_quant(X, fmt, lo=None, hi=None):
    """Quantize one activation tensor X (fp16, M x K, K contiguous) in activation format `fmt`.
    Per-tensor formats take ScaleZP of a range: by default X's own range -- the dynamic path of
    Alg. 3 (lo, hi = min, max of the tensor); with `lo`, `hi` given, that range -- the UNet /
    few-step path of Alg. 2, whose (s, z) are ScaleZP of the calibration range stored by Alg. 1
    (values outside it clamp to the extreme codes).  MX formats ignore lo, hi.  Returns a dict:
      codes  uint8 M x K  (INT8-asym: q; E4M3/E5M2/MXFP8: FP8 bit pattern; MXINT8: int8 byte)
      s, z   per-tensor fp32 scale and integer zero point (MX: s = 1, z = 0, App. A.7)
      e8m0   uint8 M x K/32 for the MX formats, else None
    """
    X = np.asarray(X)
    x = X.astype(np.float32)
    M, K = x.shape
    out = {"fmt": fmt, "e8m0": None, "s": np.float32(1.0), "z": 0}
    if fmt in (A_INT8_ASYM, A_E4M3, A_E5M2) and lo is None:
        lo = x.min() if x.size else np.float32(0)
        hi = x.max() if x.size else np.float32(0)
    if fmt == A_INT8_ASYM:
        s, inv, z = scale_zp(fmt, lo, hi)
        q = rne(_f32(x * inv)) + z
        out.update(codes=np.clip(q, 0, 255).astype(np.uint8), s=s, z=z, inv=inv)
    elif fmt in (A_E4M3, A_E5M2):
        name = "e4m3" if fmt == A_E4M3 else "e5m2"
        s, inv, _ = scale_zp(fmt, lo, hi)
        out.update(codes=fp_quantize(_f32(x * inv), name).astype(np.uint8), s=s, z=0, inv=inv)
    elif fmt in (A_MXFP8, A_MXINT8):
        assert K % MX_BLOCK == 0
        codes, e8 = mx_quant_rows(x, "e4m3" if fmt == A_MXFP8 else "int8")
        out.update(codes=codes, e8m0=e8)
    else:
        raise ValueError("unknown activation format %r" % (fmt,))
    return out


def act_dequant(q):
    """DQ of act_quant's output as float64 (the GEMM operand of the reference)."""
    fmt = q["fmt"]
    c = q["codes"]
    if fmt == A_INT8_ASYM:
        return (c.astype(np.float64) - q["z"]) * np.float64(q["s"])
    if fmt == A_E4M3:
        return fp_decode(c, "e4m3") * np.float64(q["s"])
    if fmt == A_E5M2:
        return fp_decode(c, "e5m2") * np.float64(q["s"])
    if fmt == A_MXFP8:
        return mx_dequant_rows(c, q["e8m0"], "e4m3")
    if fmt == A_MXINT8:
        return mx_dequant_rows(c, q["e8m0"], "int8")
    raise ValueError(fmt)


def act_quant_per_sample(X, fmt, n_groups):
    """Per-sample dynamic scaling of the DiT path (Alg. 3 with min/max taken over one sample): the
    M rows of X form n_groups equal groups of consecutive rows, and each group is quantized by
    act_quant with its own range.  Returns the list of the groups' act_quant outputs."""
    X = np.asarray(X)
    M = X.shape[0]
    if n_groups < 1 or M % n_groups:
        raise ValueError("n_groups must divide M")
    R = M // n_groups
    return [act_quant(X[g * R:(g + 1) * R], fmt) for g in range(n_groups)]


def act_dequant_per_sample(qs):
    """DQ of act_quant_per_sample's output: the groups' dequantized rows stacked in order."""
    return np.vstack([act_dequant(q) for q in qs])


# ---------------------------------------------------------------- MX blocks (App. A.11/A.12)
# element body: (emax_elem used by R1, integer scale exponent of the body)
MX_BODIES = {"e4m3": 8, "e2m1": 2, "int8": 0, "int4": 0}


def mx_quant_rows(x, body):
    """Quantize each 32-element block along the last axis of the fp32 array x (rows x K):
    amax = max|x_i|; shared exponent X = floor(log2 amax) - emax_elem (R1); element
    v_i = x_i * 2^-X (exact); body code of v_i (R3 for integer bodies); E8M0 byte X + 127.
    Returns (codes as uint8 bytes, rows x K; e8m0 uint8, rows x K/32).  4-bit bodies return the
    code as a small integer in an uint8 (two's complement nibble for int4, E2M1 pattern)."""
    x = np.asarray(x, dtype=np.float32)
    R, K = x.shape
    xb = x.reshape(R, K // MX_BLOCK, MX_BLOCK).astype(np.float64)
    amax = np.abs(xb).max(axis=2)
    zero = amax == 0
    X = np.where(zero, -127, floor_log2(np.where(zero, 1.0, amax)) - MX_BODIES[body])
    byte = e8m0_byte(X)
    Xeff = byte - 127                                   # exponent actually encoded
    # all-zero block (R2): byte 0 and v = x itself (all zeros, sign kept)
    v = np.where(zero[..., None], xb, np.ldexp(xb, -Xeff[..., None]))
    if body == "e4m3":
        codes = fp_quantize(v, "e4m3")
    elif body == "e2m1":
        codes = fp_quantize(v, "e2m1")
    elif body == "int8":
        codes = np.clip(rne(v * 64.0), -127, 127).astype(np.int64) & 0xFF
    elif body == "int4":
        codes = np.clip(rne(v * 4.0), -7, 7).astype(np.int64) & 0xF
    else:
        raise ValueError(body)
    return codes.reshape(R, K).astype(np.uint8), byte.astype(np.uint8)


def mx_element_value(codes, body):
    """Value of MX element codes before the block scale."""
    c = np.asarray(codes, dtype=np.int64)
    if body == "e4m3":
        return fp_decode(c, "e4m3")
    if body == "e2m1":
        return fp_decode(c, "e2m1")
    if body == "int8":
        return np.where(c >= 128, c - 256, c).astype(np.float64) * 2.0 ** -6
    if body == "int4":
        return np.where(c >= 8, c - 16, c).astype(np.float64) * 2.0 ** -2
    raise ValueError(body)


def mx_dequant_rows(codes, e8m0, body):
    """DQ of mx_quant_rows: element value * 2^(byte - 127), float64."""
    R, K = codes.shape
    val = mx_element_value(codes, body).reshape(R, K // MX_BLOCK, MX_BLOCK)
    X = e8m0.astype(np.int64) - 127
    return np.ldexp(val, X[..., None]).reshape(R, K)


# ---------------------------------------------------------------- weight codecs (Sec. 3.4)
def weight_quant(W, fmt, nf4_levels=None):
    """Quantize every output channel (row) of W (fp16, N x K) in weight format `fmt` at the
    granularity of R10.  Returns a dict with
      codes  int64 N x K  -- INT formats: the signed/unsigned integer q; NF4: level index 0..15;
                             E2M1: 4-bit pattern; MX formats: body code byte/nibble
      s      fp32 [N] per-channel scale (1 for MX), z int64 [N] zero point (asym only, else 0)
      e8m0   uint8 N x K/32 (MX only)
    """
    w = np.asarray(W).astype(np.float32)
    N, K = w.shape
    s = np.ones(N, dtype=np.float32)
    z = np.zeros(N, dtype=np.int64)
    out = {"fmt": fmt, "s": s, "z": z, "e8m0": None}
    amax = np.abs(w).max(axis=1) if K else np.zeros(N, np.float32)
    if fmt in (W_INT8_SYM, W_INT4_SYM):
        qmax = 127 if fmt == W_INT8_SYM else 7
        codes = np.zeros((N, K), dtype=np.int64)
        for c in range(N):
            s[c], inv = scale_sym(amax[c], qmax)
            codes[c] = np.clip(rne(_f32(w[c] * inv)), -qmax, qmax)
        out["codes"] = codes
    elif fmt in (W_INT8_ASYM, W_INT4_ASYM):
        levels = 255 if fmt == W_INT8_ASYM else 15
        codes = np.zeros((N, K), dtype=np.int64)
        for c in range(N):
            s[c], inv, z[c] = scale_zp_asym(w[c].min(), w[c].max(), levels)
            codes[c] = np.clip(rne(_f32(w[c] * inv)) + z[c], 0, levels)
        out["codes"] = codes
    elif fmt == W_E2M1:
        codes = np.zeros((N, K), dtype=np.int64)
        for c in range(N):
            s[c], inv = scale_sym(amax[c], 6.0)
            codes[c] = fp_quantize(_f32(w[c] * inv), "e2m1")
        out["codes"] = codes
    elif fmt == W_NF4:
        assert nf4_levels is not None
        L = np.asarray(nf4_levels, dtype=np.float64)
        mids = (L[:-1] + L[1:]) / 2.0                     # fp64 midpoints ...
        mids32 = mids.astype(np.float32)                  # ... rounded to fp32
        codes = np.zeros((N, K), dtype=np.int64)
        for c in range(N):
            sc = np.float32(amax[c]) if amax[c] != 0 else np.float32(1.0)
            s[c] = sc
            v = _f32(w[c] / sc)                           # correctly rounded fp32 division
            # level index = number of midpoints strictly below v (ties go to the lower level)
            codes[c] = (mids32[None, :] < v[:, None]).sum(axis=1)
        out["codes"] = codes
    elif fmt in (W_MXINT8, W_MXINT4, W_MXFP4):
        body = {W_MXINT8: "int8", W_MXINT4: "int4", W_MXFP4: "e2m1"}[fmt]
        codes, e8 = mx_quant_rows(w, body)
        out["codes"] = codes.astype(np.int64)
        out["e8m0"] = e8
    else:
        raise ValueError(fmt)
    return out


def weight_dequant(q, nf4_levels=None):
    """DQ of weight_quant's output, float64 N x K."""
    fmt = q["fmt"]
    c = q["codes"]
    s = q["s"].astype(np.float64)[:, None]
    if fmt in (W_INT8_SYM, W_INT4_SYM):
        return c.astype(np.float64) * s
    if fmt in (W_INT8_ASYM, W_INT4_ASYM):
        return (c - q["z"][:, None]).astype(np.float64) * s
    if fmt == W_E2M1:
        return fp_decode(c, "e2m1") * s
    if fmt == W_NF4:
        L = np.asarray(nf4_levels, dtype=np.float64)
        return L[c] * s
    body = {W_MXINT8: "int8", W_MXINT4: "int4", W_MXFP4: "e2m1"}[fmt]
    return mx_dequant_rows(c.astype(np.uint8), q["e8m0"], body)


# ---------------------------------------------------------------- group-wise weight formats (Sec. 3.5 forks)
GROUP_SIZES = (32, 64, 128, 192, 288)


def group_bounds(K, g):
    """[k0, k1) of each group of one row: runs of g consecutive input channels, the last one
    shorter when g does not divide K (reading R24)."""
    return [(k0, min(k0 + g, K)) for k0 in range(0, K, g)]


def weight_quant_grouped(W, fmt, g, nf4_levels=None):
    """Group-wise quantization of a non-MX weight format (the DiT and few-step forks, Sec. 3.5):
    every run of g input channels of every output channel is quantized by the format's own rule
    (weight_quant applied to that slice: its scale, and zero point for asym, from the group's
    statistics).  Returns {"fmt", "g", "groups": [(k0, k1, weight_quant dict)]}."""
    if W_IS_MX[fmt]:
        raise ValueError("MX formats carry their own 32-element blocks")
    W = np.asarray(W)
    return {"fmt": fmt, "g": g,
            "groups": [(k0, k1, weight_quant(W[:, k0:k1], fmt, nf4_levels)) for k0, k1 in group_bounds(W.shape[1], g)]}


def weight_dequant_grouped(q, nf4_levels=None):
    """DQ of weight_quant_grouped's output (R24): the code's value times the group scale stored as
    fp16 (the weights' own type), the product rounded once to fp16.  float64 N x K."""
    N = q["groups"][0][2]["codes"].shape[0]
    K = q["groups"][-1][1]
    out = np.zeros((N, K))
    for k0, k1, qq in q["groups"]:
        s16 = qq["s"].astype(np.float16).astype(np.float64)
        v = weight_dequant(dict(qq, s=np.ones_like(qq["s"])), nf4_levels)  # the codes' values
        out[:, k0:k1] = (v * s16[:, None]).astype(np.float16)    # exact product, one rounding
    return out
