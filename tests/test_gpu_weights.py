"""GPU weight-format selection (a5) and pack (a6) against the oracle."""
import numpy as np
import pytest

from oracle import formats as F
from oracle import select as SEL
from paper_2609_33496_gb300 import workloads as WL
from gpu_common import lib_module, cuda, host
from blob import unpack

pytestmark = pytest.mark.gpu
TURBO = (1 << F.W_INT4_ASYM) | (1 << F.W_NF4) | (1 << F.W_E2M1) | (1 << F.W_MXINT4) | (1 << F.W_MXFP4)


@pytest.fixture(scope="module")
def cl():
    return lib_module()


def gpu_select(cl, W, mask):
    import torch
    fmt, sse = cl.select_weight_formats(cuda(W), mask, want_sse=True)
    torch.cuda.synchronize()
    return host(fmt), host(sse)


def check_selection(cl, W, mask):
    fmt_g, sse_g = gpu_select(cl, W, mask)
    fmt_o, sse_o, pal = SEL.select_formats(W, mask)
    for j, f in enumerate(pal):
        np.testing.assert_allclose(sse_g[:, f], sse_o[:, j], rtol=1e-6, atol=1e-30)
    nonmember = [f for f in range(9) if f not in pal]
    assert np.all(np.isinf(sse_g[:, nonmember]))
    diff = np.nonzero(fmt_g != fmt_o)[0]
    for c in diff:   # a different choice only where the oracle's two best errors are a near-tie
        assert SEL.near_tie(sse_o[c]), (c, fmt_g[c], fmt_o[c], sse_o[c])
    return fmt_g, fmt_o


@pytest.mark.parametrize("mask", [0x007, 0x1F8, TURBO])
def test_select_single_layer(cl, mask):
    _, W, _ = WL.single_layer()
    check_selection(cl, W, mask)


@pytest.mark.parametrize("mask", [0x007, 0x1F8])
def test_select_mixed_distributions(cl, mask):
    W = WL.weight_mix(np.random.default_rng(3), 300, 320)
    fmt_g, _ = check_selection(cl, W, mask)
    assert len(np.unique(fmt_g)) >= 2


def test_select_constructed_channels(cl):
    K = 64
    ints = np.tile(np.arange(-7, 8), 5)[:K].astype(np.float64)
    W = np.stack([ints * 2.0 ** -9, np.zeros(K), np.ones(K) * 0.01]).astype(np.float16)
    fmt_g, fmt_o = check_selection(cl, W, 0x1F8)
    assert fmt_g[0] == F.W_INT4_SYM and fmt_g[1] == F.W_INT4_SYM


def unpack_blob(cl, W, fmt, layout=0, fold=0):
    import torch
    d = cl.pack_plan(W.shape[0], W.shape[1], fmt, layout, fold)
    blob, st = cl.pack_weights(cuda(W), cuda(fmt), d)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return unpack(host(blob).tobytes())


@pytest.mark.parametrize("layout,fold", [(0, 0), (1, 0), (1, 40)])
@pytest.mark.parametrize("mask,K", [(0x007, 320), (0x1F8, 320), (0x1F8, 96), (0x007, 160)])
def test_pack_matches_oracle_codes(cl, mask, K, layout, fold):
    W = WL.weight_mix(np.random.default_rng(K), 261, K)
    fmt_o, _, pal = SEL.select_formats(W, mask)
    fmt = fmt_o.copy()
    fmt[::7] = pal[-1]          # make sure every palette member appears
    fmt[1::7] = pal[0]
    desc, got = unpack_blob(cl, W, fmt, layout, fold)
    ref = SEL.quantize_selected(W, fmt)
    assert sorted(got) == list(range(W.shape[0]))
    for c, r in enumerate(ref):
        g = got[c]
        assert g["fmt"] == r["fmt"]
        np.testing.assert_array_equal(g["codes"], r["codes"], err_msg="channel %d fmt %d" % (c, r["fmt"]))
        if F.W_IS_MX[r["fmt"]]:
            np.testing.assert_array_equal(g["e8m0"], r["e8m0"])
        else:
            assert np.float32(g["s"]).tobytes() == np.float32(r["s"]).tobytes()
            assert g["z"] == r["z"]


@pytest.mark.parametrize("fold", [0, 30])
def test_pack_format_groups_order(cl, fold):
    """Layout 1: inside each class the formats in palette order, each in original channel order and
    padded to whole tiles (every tile one format); formats with fewer than `fold` channels share the
    class's tail group, in original order, after the class's own groups."""
    W = WL.weight_mix(np.random.default_rng(19), 400, 96)
    g = np.random.default_rng(2)
    fmt = np.concatenate([np.full(n, f) for f, n in ((3, 140), (4, 20), (5, 150), (6, 10), (7, 60), (8, 20))])
    fmt = fmt[g.permutation(len(fmt))].astype(np.uint8)
    desc, got = unpack_blob(cl, W, fmt, 1, fold)
    order0, order1 = [3, 4, 6, 7, 8], [5]
    counts = {f: int((fmt == f).sum()) for f in range(9)}
    expect, base = {}, 0
    for cls_order in (order0, order1):
        own = [f for f in cls_order if counts[f] >= max(fold, 1)]
        tail = [f for f in cls_order if 0 < counts[f] < fold]
        for grp in [[f] for f in own] + ([tail] if tail else []):
            chans = [c for c in range(len(fmt)) if fmt[c] in grp]
            for r, c in enumerate(chans):
                expect[c] = base + r
            base += 128 * (-(-len(chans) // 128))
    assert {c: g_["slot"] for c, g_ in got.items()} == expect
    assert desc["n_tiles"][0] + desc["n_tiles"][1] == base // 128


def test_pack_permutation_groups_classes(cl):
    W = WL.weight_mix(np.random.default_rng(9), 200, 64)
    fmt = np.random.default_rng(1).choice(np.arange(3, 9), 200).astype(np.uint8)
    desc, got = unpack_blob(cl, W, fmt)
    slots = sorted((g["slot"], c, g["fmt"]) for c, g in got.items())
    keys = [(0 if f in (3, 4, 6, 7, 8) else 1, c) for _, c, f in slots]
    assert keys == sorted(keys)                      # class 0 first, original order inside a class
    class1_first = min(g["slot"] for g in got.values() if g["fmt"] == F.W_NF4)
    assert class1_first == 128 * desc["n_tiles"][0]


@pytest.mark.parametrize("mask,K", [(0x007, 320), ((1 << F.W_INT4_ASYM) | (1 << F.W_E2M1) | (1 << F.W_MXINT4) | (1 << F.W_MXFP4), 96)])
def test_palette_plan_packs_the_same_blob(cl, mask, K):
    """A blob packed from the palette-only plan equals the one packed from the host plan of the
    selected formats, except for the per-format counts in its header copy."""
    import torch
    W = WL.weight_mix(np.random.default_rng(11), 260, K)
    Wd = cuda(W)
    fmt, _ = cl.select_weight_formats(Wd, mask)
    d_host = cl.pack_plan(W.shape[0], K, host(fmt))
    d_pal = cl.pack_plan_palette(W.shape[0], K, mask)
    assert d_host.bytes == d_pal.bytes
    b_host, st1 = cl.pack_weights(Wd, fmt, d_host)
    b_pal, st2 = cl.pack_weights(Wd, fmt, d_pal)
    torch.cuda.synchronize()
    assert int(st1.item()) == 0 and int(st2.item()) == 0
    a, b = host(b_host), host(b_pal)
    d = d_host
    tiles = d.n_tiles[0] + d.n_tiles[1]
    np_, chunks, cb = 128 * tiles, d.Kp // 64, 64 if d.bits == 8 else 32
    regions = [(d.off_codes, tiles * chunks * 128 * cb), (d.off_scale, 4 * np_), (d.off_zero, np_),
               (d.off_e8m0, tiles * chunks * 256), (d.off_fmt, np_), (d.off_perm, 4 * np_)]
    for off, n in regions:                             # the bytes the pack defines (gaps are not written)
        assert np.array_equal(a[off:off + n], b[off:off + n]), off
    assert np.array_equal(a[:40], b[:40]) and np.array_equal(a[76:256], b[76:256])
    n_fmt = slice(40, 40 + 4 * 9)                      # int32 n_fmt[9] in the descriptor copy
    assert np.all(b[n_fmt].view(np.int32)[[f for f in range(9) if (mask >> f) & 1]] == -1)


@pytest.mark.parametrize("mask,K", [(0x007, 320), (0x007, 1280), ((1 << 4) | (1 << 6) | (1 << 7) | (1 << 8), 96),
                                    (1 << 5, 64)])
def test_fused_select_pack_equals_the_two_launches(cl, mask, K):
    """chameleon_select_pack_palette gives the formats of chameleon_select_weight_formats and the
    blob chameleon_pack_weights writes for them from the same palette plan, byte for byte."""
    import torch
    W = WL.weight_mix(np.random.default_rng(K + mask), 300, K)
    Wd = cuda(W)
    d = cl.pack_plan_palette(W.shape[0], K, mask)
    fmt_ref, _ = cl.select_weight_formats(Wd, mask)
    b_ref, st1 = cl.pack_weights(Wd, fmt_ref, d)
    fmt, b, st2 = cl.select_pack_palette(Wd, mask, d)
    torch.cuda.synchronize()
    assert int(st1.item()) == 0 and int(st2.item()) == 0
    np.testing.assert_array_equal(host(fmt), host(fmt_ref))
    a, c = host(b_ref), host(b)
    tiles = d.n_tiles[0] + d.n_tiles[1]
    np_, chunks, cb = 128 * tiles, d.Kp // 64, 64 if d.bits == 8 else 32
    for off, n in [(0, 256), (d.off_codes, tiles * chunks * 128 * cb), (d.off_scale, 4 * np_), (d.off_zero, np_),
                   (d.off_e8m0, tiles * chunks * 256), (d.off_fmt, np_), (d.off_perm, 4 * np_)]:
        assert np.array_equal(a[off:off + n], c[off:off + n]), off


@pytest.mark.parametrize("layer", range(len(WL.SDXL_PROJ_LAYERS)))
def test_fused_select_pack_against_oracle_on_benchmark_weights(cl, layer):
    """The fused selection + pack the benchmark's step runs (chameleon_select_pack_palette, W8
    palette), checked directly against the oracle on the ten SDXL projection weights the benchmark
    packs: formats equal except at oracle near-ties, and the blob's codes, scales, zero points and
    E8M0 bytes of each channel equal the oracle's encoding of the format the kernel chose.  Layers
    with more than 1280 channels are checked on 1024 seeded channels."""
    import torch
    name, M, K, N = WL.SDXL_PROJ_LAYERS[layer]
    W, _ = WL.sdxl_layer_weights(layer)
    d = cl.pack_plan_palette(N, K, cl.PALETTE_W8)
    fmt_d, blob, st = cl.select_pack_palette(cuda(W), cl.PALETTE_W8, d)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    fmt_g = host(fmt_d)
    rows = np.arange(N) if N <= 1280 else np.sort(np.random.default_rng(layer).choice(N, 1024, replace=False))
    fmt_o, sse_o, _ = SEL.select_formats(W[rows], cl.PALETTE_W8)
    for i in np.nonzero(fmt_g[rows] != fmt_o)[0]:
        assert SEL.near_tie(sse_o[i]), (name, rows[i], fmt_g[rows[i]], fmt_o[i])
    _, got = unpack(host(blob).tobytes())
    ref = SEL.quantize_selected(W[rows], fmt_g[rows])
    for c, r in zip(rows, ref):
        g = got[int(c)]
        assert g["fmt"] == r["fmt"] == fmt_g[c]
        np.testing.assert_array_equal(g["codes"], r["codes"], err_msg="%s channel %d" % (name, c))
        if F.W_IS_MX[r["fmt"]]:
            np.testing.assert_array_equal(g["e8m0"], r["e8m0"])
        else:
            assert np.float32(g["s"]).tobytes() == np.float32(r["s"]).tobytes() and g["z"] == r["z"]
