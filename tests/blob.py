"""Host-side reader of the packed-weight blob layout declared in include/chameleon.h (test helper:
it only re-indexes bytes, it computes nothing of the method)."""
import numpy as np

CLASS0 = (3, 4, 6, 7, 8)


def desc_fields(blob_bytes):
    hdr = np.frombuffer(blob_bytes[:256], dtype=np.uint8)
    i32 = hdr[:80].view(np.int32)
    u64 = hdr[80:144].view(np.uint64)
    keys = ["off_codes", "off_scale", "off_zero", "off_e8m0", "off_fmt", "off_perm", "bytes", "off_gscale"]
    d = {"magic": int(hdr[:4].view(np.uint32)[0]), "N": int(i32[2]), "K": int(i32[3]),
         "Kp": int(i32[4]), "bits": int(i32[5]), "n_class": [int(i32[6]), int(i32[7])],
         "n_tiles": [int(i32[8]), int(i32[9])], "n_fmt": [int(v) for v in i32[10:19]],
         "version": int(hdr[4:8].view(np.uint32)[0]), "group": int(i32[19])}
    d.update({k: int(v) for k, v in zip(keys, u64)})
    return d


def unpack(blob_bytes):
    """Per original channel: fmt, codes (int64 [K], the logical code values), scale, zero, e8m0
    ([K/32] bytes), plus the packed order."""
    b = np.frombuffer(blob_bytes, dtype=np.uint8)
    d = desc_fields(blob_bytes)
    N, K, Kp, bits = d["N"], d["K"], d["Kp"], d["bits"]
    tiles = d["n_tiles"][0] + d["n_tiles"][1]
    Np, nch = 128 * tiles, Kp // 64
    fmt = b[d["off_fmt"]:d["off_fmt"] + Np]
    perm = b[d["off_perm"]:d["off_perm"] + 4 * Np].view(np.int32)
    scale = b[d["off_scale"]:d["off_scale"] + 4 * Np].view(np.float32)
    zero = b[d["off_zero"]:d["off_zero"] + Np]
    e8 = b[d["off_e8m0"]:d["off_e8m0"] + tiles * nch * 256].reshape(tiles, nch, 128, 2)
    gsc = None
    if d["group"] > 0:   # group-wise blob: fp16 scale of each 32-element block
        gsc = b[d["off_gscale"]:d["off_gscale"] + tiles * nch * 512].view(np.float16).reshape(tiles, nch, 128, 2)
    CB = 64 if bits == 8 else 32
    codes_raw = b[d["off_codes"]:d["off_codes"] + tiles * nch * 128 * CB].reshape(tiles, nch, CB // 16, 128, 16)
    # per slot: bytes of each chunk in order
    per_slot = codes_raw.transpose(0, 3, 1, 2, 4).reshape(tiles * 128, nch * CB)
    out = {}
    for p in range(Np):
        c = int(perm[p])
        if c < 0:
            continue
        raw = per_slot[p]
        if bits == 8:
            vals = raw[:K].astype(np.int64)
        else:
            words = raw.view(np.uint32)
            vals = np.zeros(Kp, dtype=np.int64)
            nib = [(words >> (4 * j)) & 0xF for j in range(8)]
            if int(fmt[p]) == 5:            # NF4: nibble j = element j
                for j in range(8):
                    vals[j::8] = nib[j]
            else:
                for j in range(4):
                    vals[2 * j::8] = nib[j]
                    vals[2 * j + 1::8] = nib[4 + j]
            vals = vals[:K]
        f = int(fmt[p])
        t, r = divmod(p, 128)
        e8c = e8[t, :, r, :].reshape(-1)[:K // 32]
        # symmetric integer codes are stored in offset binary; the oracle keeps INT8/INT4-sym
        # signed and MXINT8/MXINT4 as two's-complement bytes / nibbles
        if f == 0:                      # INT8-sym: q + 128
            vals = vals - 128
        elif f == 2:                    # MXINT8: (q + 128) -> q & 0xFF
            vals = vals ^ 0x80
        elif f == 3:                    # INT4-sym: q + 8
            vals = vals - 8
        elif f == 7:                    # MXINT4: (q + 8) -> q & 0xF
            vals = vals ^ 0x8
        out[c] = {"fmt": f, "codes": vals, "s": np.float32(scale[p]), "z": int(zero[p]), "e8m0": e8c,
                  "slot": p}
        if gsc is not None:
            out[c]["gscale16"] = gsc[t, :, r, :].reshape(-1)[:K // 32]
    return d, out
