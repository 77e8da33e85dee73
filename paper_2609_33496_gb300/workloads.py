"""Seeded synthetic inputs shaped like the paper's workloads (stand-ins for SDXL / PixArt-alpha
activations and weights; no checkpoint or dataset is used).  Holds no arithmetic of the method:
only value distributions, shapes and seeds.  Shared by the tests, the benchmark and the oracle's
callers.

Seeds: 20260000 + 1000 * config + index.  Values are drawn in float64 and rounded to fp16.
"""
import numpy as np

SEED_BASE = 20260000

# SDXL-UNet attention / FFN projections at batch 2 with classifier-free guidance:
# (name, M tokens, K in-features, N out-features)
SDXL_PROJ_LAYERS = (
    [("down1.attn.%s" % n, 8192, 640, 640) for n in ("q", "k", "v", "out")]
    + [("down2.attn.%s" % n, 2048, 1280, 1280) for n in ("q", "k", "v", "out")]
    + [("down2.ff.geglu_in", 2048, 1280, 10240), ("down2.ff.out", 2048, 5120, 1280)]
)

# Student-t degrees of freedom of the activations per timestep bucket b = 0..9 (None = Gaussian):
# near-Gaussian at high SNR (b = 0), heavy-tailed at low SNR (b = 9), App. A.3 phases.
NU_SCHEDULE = (None, 30, 20, 12, 9, 7, 6, 5, 4, 3)


def rng(config, index=0):
    return np.random.default_rng(SEED_BASE + 1000 * config + index)


def to_fp16(x):
    return np.asarray(x, dtype=np.float64).astype(np.float16)


def student_t(g, nu, shape):
    return g.standard_normal(shape) if nu is None else g.standard_t(nu, shape)


def single_layer(seed_index=0, M=256, K=320, N=320, n_outliers=4, outlier_gain=20.0):
    """Single linear layer: X = 0.5 * StudentT(3), W ~ N(0, 0.02^2) with `n_outliers` output
    channels scaled by `outlier_gain`, bias ~ N(0, 0.02^2)."""
    g = rng(1, seed_index)
    X = to_fp16(0.5 * g.standard_t(3, (M, K)))
    W = g.normal(0.0, 0.02, (N, K))
    if n_outliers:
        rows = g.choice(N, n_outliers, replace=False)
        W[rows] *= outlier_gain
    bias = g.normal(0.0, 0.02, N).astype(np.float32)
    return X, to_fp16(W), bias


def channel_jitter(g, K, sigma=0.1):
    """Per-input-channel scale c_k = exp(sigma * N(0, 1))."""
    return np.exp(sigma * g.standard_normal(K))


def sdxl_layer_weights(layer_index):
    name, M, K, N = SDXL_PROJ_LAYERS[layer_index]
    g = rng(2, layer_index)
    W = to_fp16(g.normal(0.0, 0.02, (N, K)))
    bias = g.normal(0.0, 0.02, N).astype(np.float32)
    return W, bias


def sdxl_layer_activation(layer_index, bucket, rows=None):
    """Activation of projection layer `layer_index` at timestep bucket `bucket`:
    StudentT(nu_b) * c_k with a per-layer channel jitter c_k.  `rows` limits M (smaller tests)."""
    name, M, K, N = SDXL_PROJ_LAYERS[layer_index]
    if rows is not None:
        M = rows
    c = channel_jitter(rng(2, 100 + layer_index), K)
    g = rng(2, 200 + 10 * layer_index + bucket)
    return to_fp16(student_t(g, NU_SCHEDULE[bucket], (M, K)) * c[None, :])


def weight_mix(g, N, K, scale=0.02):
    """Weights with per-channel distribution diversity (round-robin Gaussian, Laplace, uniform,
    Student-t nu=4, sparse outliers) so that a format argmin yields a mix."""
    W = np.empty((N, K))
    for n in range(N):
        kind = n % 5
        if kind == 0:
            W[n] = g.normal(0, scale, K)
        elif kind == 1:
            W[n] = g.laplace(0, scale / np.sqrt(2), K)
        elif kind == 2:
            W[n] = g.uniform(-scale * np.sqrt(3), scale * np.sqrt(3), K)
        elif kind == 3:
            W[n] = g.standard_t(4, K) * scale / np.sqrt(2)
        else:
            W[n] = g.normal(0, scale, K)
            idx = g.choice(K, max(1, K // 64), replace=False)
            W[n, idx] *= 12.0
    return to_fp16(W)


# Representative layer shapes (M, K, N) of the wider workloads, batch 2 unless stated:
# * SDXL UNet step at 1024^2 (latent 128^2): time embedding (M = 2), text cross-attention K/V
#   (M = 2 x 77), the 1280-wide transformer stage, a 640-wide 1x1 conv and the 32768-token stage;
# * PixArt-alpha DiT (hidden 1152, MLP 4608, 4096 tokens, 120 caption tokens);
# * SDXL-Turbo weight-only at batch 1 / 8 / 16: M = b, 77 b and b x HW rows.
UNET_W4A8_SHAPES = ((2, 320, 1280), (154, 2048, 1280), (2048, 5120, 1280), (8192, 1920, 640),
                    (32768, 960, 320))
PIXART_W4A8_SHAPES = ((240, 1152, 1152), (8192, 1152, 4608), (8192, 4608, 1152), (240, 4096, 1152))
TURBO_W4A16_SHAPES = ((1, 320, 1280), (16, 1280, 1280), (616, 2048, 640), (8192, 640, 640))
# The 22 distinct (M, K, N) of the linear and 1x1-conv GEMMs of one SDXL-architecture UNet step at
# 1024^2 (latent 128^2, batch 2): time embedding and its projections (M = 2), text cross-attention
# K/V (M = 154), and the 32^2 / 64^2 / 128^2 stages (M = 2048 / 8192 / 32768).
UNET_STEP_SHAPES = ((2, 320, 1280), (2, 1280, 320), (2, 1280, 640), (2, 1280, 1280), (2, 2816, 1280),
                    (154, 2048, 640), (154, 2048, 1280), (2048, 640, 1280), (2048, 1280, 1280),
                    (2048, 1920, 1280), (2048, 2560, 1280), (2048, 5120, 1280), (2048, 1280, 10240),
                    (8192, 320, 640), (8192, 640, 640), (8192, 960, 640), (8192, 1280, 640),
                    (8192, 1920, 640), (8192, 2560, 640), (8192, 640, 5120), (32768, 640, 320),
                    (32768, 960, 320))
# The distinct GEMMs of one PixArt-alpha XL/2 block at 1024^2, batch 2 (4096 tokens, 120 caption
# tokens per sample): self q/k/v/out and cross q/out, cross k/v, MLP fc1 and fc2, and the caption
# projection.
PIXART_STEP_SHAPES = ((8192, 1152, 1152), (240, 1152, 1152), (8192, 1152, 4608), (8192, 4608, 1152),
                      (240, 4096, 1152))


def pixart_layer_activation(index, bucket):
    """Input of PixArt-alpha block GEMM `index` (PIXART_STEP_SHAPES) at timestep bucket `bucket`:
    StudentT(nu_b) * c_k as for the SDXL projections, the two samples of the batch drawn together."""
    M, K, N = PIXART_STEP_SHAPES[index]
    c = channel_jitter(rng(4, 100 + index), K)
    g = rng(4, 200 + 10 * index + bucket)
    return to_fp16(student_t(g, NU_SCHEDULE[bucket], (M, K)) * c[None, :])


def pixart_layer_weights(index):
    M, K, N = PIXART_STEP_SHAPES[index]
    g = rng(4, 300 + index)
    return weight_mix(g, N, K), g.normal(0.0, 0.02, N).astype(np.float32)


def turbo_batch_shapes(b):
    """SDXL-Turbo weight-only rows at batch b (512^2, one step): the time-embedding projection
    (M = b), text cross-attention K/V (M = 77 b) and a 32^2-stage projection (M = 1024 b)."""
    return ((b, 320, 1280), (77 * b, 2048, 1280), (1024 * b, 1280, 1280))


def config_layer(config, index, M, K, N, nu=7):
    """X fp16 M x K = StudentT(nu) * c_k (config 2's mid-bucket distribution with channel
    jitter), weights with per-channel distribution diversity, bias N(0, 0.02^2)."""
    g = rng(config, index)
    c = channel_jitter(g, K)
    X = to_fp16(student_t(g, nu, (M, K)) * c[None, :])
    W = weight_mix(g, N, K)
    bias = g.normal(0.0, 0.02, N).astype(np.float32)
    return X, W, bias


# ------------------------------------------------------------------ PixArt-alpha DiT, whole model
# PixArt-alpha XL/2 at 1024^2, batch 2 (4096 image tokens and 120 caption tokens per sample): the
# caption projection (two linears on the 240 caption tokens), then 28 blocks of ten linears each --
# self-attention q, k, v, out; cross-attention q, k, v (k and v on the caption tokens), out; MLP fc1
# and fc2 -- 282 GEMMs per sampler step.  Each entry: (name, M, K, N, input); linears that read the
# same tensor in the network share an input key: q, k and v read the normalised hidden state of
# the self-attention, cross k and v the caption tokens; cross q and fc1 read their own normalised
# states.
PIXART_BLOCKS = 28
PIXART_CAPTION_LINEARS = (("caption.fc1", 240, 4096, 1152, "caption"),
                          ("caption.fc2", 240, 1152, 1152, "caption_hidden"))
PIXART_BLOCK_LINEARS = (("self.q", 8192, 1152, 1152, "hidden_sa"), ("self.k", 8192, 1152, 1152, "hidden_sa"),
                        ("self.v", 8192, 1152, 1152, "hidden_sa"), ("self.out", 8192, 1152, 1152, "attn"),
                        ("cross.q", 8192, 1152, 1152, "hidden_ca"), ("cross.k", 240, 1152, 1152, "text"),
                        ("cross.v", 240, 1152, 1152, "text"), ("cross.out", 8192, 1152, 1152, "cross_attn"),
                        ("mlp.fc1", 8192, 1152, 4608, "hidden_mlp"), ("mlp.fc2", 8192, 4608, 1152, "mlp"))
PIXART_INPUTS = {"caption": (240, 4096), "caption_hidden": (240, 1152), "hidden_sa": (8192, 1152),
                 "attn": (8192, 1152), "hidden_ca": (8192, 1152), "text": (240, 1152),
                 "cross_attn": (8192, 1152), "hidden_mlp": (8192, 1152), "mlp": (8192, 4608)}
PIXART_SAMPLER_T = tuple(999 - 50 * i for i in range(20))   # 20 steps, two per timestep bucket


def pixart_model_linears():
    """The 282 linears of one PixArt-alpha sampler step, in execution order: (name, M, K, N, input)."""
    out = [tuple(L) for L in PIXART_CAPTION_LINEARS]
    for b in range(PIXART_BLOCKS):
        out += [("block%d.%s" % (b, n), M, K, N, x) for (n, M, K, N, x) in PIXART_BLOCK_LINEARS]
    return out


def pixart_model_gemms():
    """The GEMM launches of one sampler step.  Linears that read the same input tensor are stacked
    along N into one GEMM -- each output channel keeps its own weights, format and bias, and the
    shared input is quantized once, so the outputs are those of the separate linears: q, k, v of a
    block (consecutive), and the cross-attention k and v of all 28 blocks, which read the same
    caption tokens (they depend on nothing the blocks compute, so the one GEMM runs where block 0's
    would).  Entries: (names, M, K, N, input, [indices into pixart_model_linears()]); 171 GEMMs."""
    out = []
    text_at = None
    for i, (name, M, K, N, x) in enumerate(pixart_model_linears()):
        short = name.split(".", 1)[1] if name.startswith("block") else name
        if x == "text" and text_at is not None:
            names, _, _, n0, _, idx = out[text_at]
            out[text_at] = (names + (name,), M, K, n0 + N, x, idx + [i])
        elif out and out[-1][4] == x and out[-1][1] == M and out[-1][2] == K and short in ("self.k", "self.v"):
            names, _, _, n0, _, idx = out[-1]
            out[-1] = (names + (name,), M, K, n0 + N, x, idx + [i])
        else:
            if x == "text":
                text_at = len(out)
            out.append(((name,), M, K, N, x, [i]))
    return out


def weight_mix_rows(g, N, K, scale=0.02):
    """The weight_mix distributions (channel n: kind n % 5 of Gaussian, Laplace, uniform, Student-t
    nu = 4, Gaussian with K/64 outliers x12), drawn kind by kind for all rows at once."""
    W = np.empty((N, K))
    rows = [np.arange(k, N, 5) for k in range(5)]
    W[rows[0]] = g.normal(0, scale, (len(rows[0]), K))
    W[rows[1]] = g.laplace(0, scale / np.sqrt(2), (len(rows[1]), K))
    W[rows[2]] = g.uniform(-scale * np.sqrt(3), scale * np.sqrt(3), (len(rows[2]), K))
    W[rows[3]] = g.standard_t(4, (len(rows[3]), K)) * scale / np.sqrt(2)
    W[rows[4]] = g.normal(0, scale, (len(rows[4]), K))
    n_out = max(1, K // 64)
    for r in rows[4]:
        W[r, g.choice(K, n_out, replace=False)] *= 12.0
    return to_fp16(W)


def pixart_model_weights(layer_index):
    """Weights (per-channel distribution diversity, config 3's recipe) and bias of linear
    `layer_index` of pixart_model_linears()."""
    _, M, K, N, _ = pixart_model_linears()[layer_index]
    g = rng(4, 1000 + layer_index)
    return weight_mix_rows(g, N, K), g.normal(0.0, 0.02, N).astype(np.float32)


def pixart_model_input(key, bucket):
    """Input tensor `key` (PIXART_INPUTS) at timestep bucket `bucket`: StudentT(nu_b) * c_k with the
    per-bucket nu of the SDXL projections (heavier tails at high noise) and per-channel jitter."""
    M, K = PIXART_INPUTS[key]
    i = sorted(PIXART_INPUTS).index(key)
    c = channel_jitter(rng(4, 2000 + i), K)
    return to_fp16(student_t(rng(4, 2100 + 10 * i + bucket), NU_SCHEDULE[bucket], (M, K)) * c[None, :])
