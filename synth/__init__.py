"""Seeded synthetic inputs and workload shapes for the FlashDecoder streaming decoder.

Shared by the CPU oracle (``oracle/``) and by the CUDA path's tests and benchmark. It holds
only workload shapes, random draws and the order of tensors in the weight blob; none of the
decoder's arithmetic lives here.

Random draws use numpy's Philox4x64-10 counter-based generator (Salmon et al., SC'11), keyed
by ``(seed, tensor index)`` so every tensor can be drawn on its own and the same key gives the
same numbers on every platform.

Workload shapes follow the paper: Wan2.1 latents (16 channels, 8x spatial, Sec. 4.3
"Generalization Across Latent Spaces") folded by PixelUnshuffle(2) so a 480p frame gives
30x52 = 1560 tokens and a 720p frame 45x80 = 3600 tokens; head dimension 64 (Table
"Model scaling": D/N = 64 for every model size); KV groups from the L and XL rows of that
table; two temporal-refinement blocks (Sec. 3.4 "Step 2"); a 4x temporal factor.
"""
from __future__ import annotations

import dataclasses
from concurrent.futures import ThreadPoolExecutor

import numpy as np

__all__ = [
    "FDConfig", "PRESETS", "weight_layout", "make_weights", "make_latents",
    "normal", "to_bf16_values", "frames_of_chunk", "make_target_pixels",
]


@dataclasses.dataclass(frozen=True)
class FDConfig:
    """Decoder shape. Field names follow the paper's notation (Sec. 3, Algorithm 1)."""

    latent_channels: int = 16      # C'
    latent_h: int = 8              # H'
    latent_w: int = 8              # W'
    patch: int = 1                 # PixelUnshuffle factor p applied to the latent
    hidden: int = 256              # D
    heads: int = 4                 # N
    kv_groups: int = 2             # G
    mlp_ratio: int = 4
    mlp_gated: bool = False        # MLP: False = Linear, GELU, Linear; True = gated SiLU
    qk_norm: bool = False          # per-head RMSNorm on Q and K instead of on K and V
    mlp_fp8: bool = False          # MLP GEMMs in FP8 (e4m3) with static scales
    first_chunk_frames: int = 0    # 1: chunk 0 emits one frame (causal frame count, Fig. 2)
    rope_mode: str = "abs"         # temporal RoPE index: "abs" (t L_frm offset) or "window"
    n_blocks: int = 2              # backbone blocks
    n_refine: int = 0              # temporal-refinement blocks
    window: int = 2                # W_frm, counts the current chunk
    r_t: int = 1                   # temporal upsampling factor
    vae_spatial: int = 8           # pixels per latent cell side
    out_channels: int = 3          # C
    out_u8: bool = False           # pixels as uint8 instead of fp32
    norm_eps: float = 1e-6
    rope_base: float = 10000.0
    # workload (not model) fields
    name: str = "tiny"
    chunks: int = 2
    streams: int = 1
    latent_mode: str = "iid"       # "iid" N(0,1) or "ar1" (rho = 0.9 along time)
    latent_seed: int = 0
    weight_seed: int = 1000

    # ---- derived shapes -------------------------------------------------
    @property
    def head_dim(self) -> int:
        return self.hidden // self.heads

    @property
    def c_in(self) -> int:
        return self.latent_channels * self.patch * self.patch

    @property
    def grid_h(self) -> int:
        return self.latent_h // self.patch

    @property
    def grid_w(self) -> int:
        return self.latent_w // self.patch

    @property
    def tokens(self) -> int:           # L_frm
        return self.grid_h * self.grid_w

    @property
    def r_s(self) -> int:              # pixels per token side
        return self.vae_spatial * self.patch

    @property
    def head_out(self) -> int:         # C * r_s^2
        return self.out_channels * self.r_s * self.r_s

    @property
    def out_h(self) -> int:
        return self.grid_h * self.r_s

    @property
    def out_w(self) -> int:
        return self.grid_w * self.r_s

    @property
    def frames_per_chunk(self) -> int:
        return self.r_t

    @property
    def qkv_out(self) -> int:
        return (self.heads + 2 * self.kv_groups) * self.head_dim

    def replace(self, **kw) -> "FDConfig":
        return dataclasses.replace(self, **kw)


# Workload presets. The first five are the benchmark's configurations; the rest are
# small parity cases (several tiles and a ragged tail, oracle time in seconds).
PRESETS: dict[str, FDConfig] = {
    # 16x8x8 latent, patch 1, 2 blocks, D=256, 4 heads, head 3x8x8 px/token, 2 chunks
    "tiny": FDConfig(),
    # 480p: 16x60x104 latent, patch 2 -> 1560 tokens, 24 blocks, D=1024, 16 heads, W=4
    "480p": FDConfig(latent_h=60, latent_w=104, patch=2, hidden=1024, heads=16, kv_groups=4,
                     n_blocks=24, n_refine=2, window=4, r_t=4, name="480p", chunks=16),
    # 720p: 16x90x160 latent -> 3600 tokens, uint8 output
    "720p": FDConfig(latent_h=90, latent_w=160, patch=2, hidden=1024, heads=16, kv_groups=4,
                     n_blocks=24, n_refine=2, window=4, r_t=4, out_u8=True, name="720p",
                     chunks=32),
    # 480p x 8 independent streams; stream s draws its latents with seed s
    "480p_x8": FDConfig(latent_h=60, latent_w=104, patch=2, hidden=1024, heads=16,
                        kv_groups=4, n_blocks=24, n_refine=2, window=4, r_t=4,
                        name="480p_x8", chunks=16, streams=8),
    # 720p wide model, long stream: D=1536, 24 heads (G=3), 32 blocks, W=8, AR(1) latents
    "720p_wide": FDConfig(latent_h=90, latent_w=160, patch=2, hidden=1536, heads=24,
                          kv_groups=3, n_blocks=32, n_refine=2, window=8, r_t=4, out_u8=True,
                          name="720p_wide", chunks=128, latent_mode="ar1"),
    # the 720p wide model's structure (D=1536, 24 heads / 3 KV groups, 32 + 2 blocks, W=8,
    # AR(1) latents, uint8) on a 10x13-token frame, 10 chunks: the W=8 window fills and evicts
    "wide_small": FDConfig(latent_h=20, latent_w=26, patch=2, hidden=1536, heads=24,
                           kv_groups=3, n_blocks=32, n_refine=2, window=8, r_t=4, out_u8=True,
                           name="wide_small", chunks=10, latent_mode="ar1"),
    # the 720p token count (3600 tokens, 14400 refined) at reduced depth (2 + 1 blocks), 5
    # chunks: the W = 4 rings of both stacks fill and evict
    "720p_d3": FDConfig(latent_h=90, latent_w=160, patch=2, hidden=1024, heads=16, kv_groups=4,
                        n_blocks=2, n_refine=1, window=4, r_t=4, out_u8=True, name="720p_d3",
                        chunks=5),
    # the 720p wide model's shapes (3600 tokens, D=1536, 24 heads / 3 KV groups, W=8, AR(1)
    # latents, uint8) at reduced depth (2 + 1 blocks), 2 chunks (chunk 1 attends to chunk 0)
    "720p_wide_d3": FDConfig(latent_h=90, latent_w=160, patch=2, hidden=1536, heads=24,
                             kv_groups=3, n_blocks=2, n_refine=1, window=8, r_t=4, out_u8=True,
                             name="720p_wide_d3", chunks=2, latent_mode="ar1"),
    # the 480p token grid (60x104 latents, 1560 tokens: 1664 padded rows, 3120 refined rows per
    # chunk) at reduced width and depth, for the training step's parity at the product's token
    # count (the fp64 oracle's backward stays within seconds)
    "train_480p_grid": FDConfig(latent_h=60, latent_w=104, patch=2, hidden=256, heads=4,
                                kv_groups=2, n_blocks=2, n_refine=1, window=2, r_t=2,
                                name="train_480p_grid", chunks=3),
    # degenerate window W=1: every chunk attends to itself only (no temporal context)
    "tiny_w1": FDConfig(window=1, n_refine=1, r_t=2, name="tiny_w1", chunks=3),
    # refinement exercised at tiny size: r_t=2, one refinement block, 3 chunks
    "tiny_rt": FDConfig(r_t=2, n_refine=1, name="tiny_rt", chunks=3),
    # several M tiles with ragged tails: 10x13=130 tokens (4L = 520), W=3 so eviction runs
    "small": FDConfig(latent_h=20, latent_w=26, patch=2, hidden=256, heads=4, kv_groups=2,
                      n_blocks=2, n_refine=1, window=3, r_t=4, name="small", chunks=5),
    # same, uint8 output and G=1 (multi-query)
    "small_u8": FDConfig(latent_h=20, latent_w=26, patch=2, hidden=256, heads=4, kv_groups=1,
                         n_blocks=1, n_refine=1, window=2, r_t=4, out_u8=True,
                         name="small_u8", chunks=4),
    # FP8 MLPs (static scales) at small size and at 480p
    "small_fp8": FDConfig(latent_h=20, latent_w=26, patch=2, hidden=256, heads=4, kv_groups=2,
                          n_blocks=2, n_refine=1, window=3, r_t=4, mlp_fp8=True,
                          name="small_fp8", chunks=5),
    "480p_fp8": FDConfig(latent_h=60, latent_w=104, patch=2, hidden=1024, heads=16,
                         kv_groups=4, n_blocks=24, n_refine=2, window=4, r_t=4, mlp_fp8=True,
                         name="480p_fp8", chunks=16),
    # gated (XL-layout) MLP in FP8 at tiny size, with refinement
    "tiny_gated_fp8": FDConfig(latent_channels=48, latent_h=10, latent_w=13, vae_spatial=16,
                               mlp_gated=True, mlp_fp8=True, n_refine=1, r_t=2,
                               name="tiny_gated_fp8", chunks=3),
    # the causal frame count of Fig. 2 (T' latents -> 1 + r_t (T' - 1) frames), r_t = 4
    "small_f1": FDConfig(latent_h=20, latent_w=26, patch=2, hidden=256, heads=4, kv_groups=2,
                         n_blocks=2, n_refine=1, window=3, r_t=4, first_chunk_frames=1,
                         name="small_f1", chunks=3),
    # the QK-norm reading of "KV-norm" at tiny size, with refinement
    "tiny_qk": FDConfig(qk_norm=True, n_refine=1, r_t=2, name="tiny_qk", chunks=3),
    # XL layout at tiny size: 48-channel 16x latent, patch 1, gated-SiLU MLP, refinement
    "tiny_gated": FDConfig(latent_channels=48, latent_h=10, latent_w=13, vae_spatial=16,
                           mlp_gated=True, n_refine=1, r_t=2, name="tiny_gated", chunks=3),
    # the XL layout at tiny size with the rest of XL's stream rules: W=2, r_t=4 and the
    # one-frame first chunk (training-step parity of the gated MLP under the causal frame count)
    "tiny_xl": FDConfig(latent_channels=48, latent_h=10, latent_w=13, vae_spatial=16,
                        mlp_gated=True, n_refine=1, window=2, r_t=4, first_chunk_frames=1,
                        name="tiny_xl", chunks=3),
    # FlashDecoder-XL as the paper's configuration table gives it: Wan2.2 latents (48
    # channels, 16x spatial), patch 1, D=1536, 24 heads / 3 KV groups, 20 + 2 blocks, W=2,
    # r_t=4, gated-SiLU MLP 4x; 480p (30x52 latent), 720p (45x80), 1080p (68x120)
    "xl_480p": FDConfig(latent_channels=48, latent_h=30, latent_w=52, vae_spatial=16,
                        hidden=1536, heads=24, kv_groups=3, mlp_gated=True, n_blocks=20,
                        n_refine=2, window=2, r_t=4, name="xl_480p", chunks=16),
    "xl_720p": FDConfig(latent_channels=48, latent_h=45, latent_w=80, vae_spatial=16,
                        hidden=1536, heads=24, kv_groups=3, mlp_gated=True, n_blocks=20,
                        n_refine=2, window=2, r_t=4, out_u8=True, name="xl_720p", chunks=16),
    # the XL layout with FP8 MLPs (the paper's lossy "XL-Opt" setting, Sec. 4.6)
    "xl_480p_fp8": FDConfig(latent_channels=48, latent_h=30, latent_w=52, vae_spatial=16,
                            hidden=1536, heads=24, kv_groups=3, mlp_gated=True, mlp_fp8=True,
                            n_blocks=20, n_refine=2, window=2, r_t=4, name="xl_480p_fp8",
                            chunks=16),
    "xl_720p_fp8": FDConfig(latent_channels=48, latent_h=45, latent_w=80, vae_spatial=16,
                            hidden=1536, heads=24, kv_groups=3, mlp_gated=True, mlp_fp8=True,
                            n_blocks=20, n_refine=2, window=2, r_t=4, out_u8=True,
                            name="xl_720p_fp8", chunks=16),
    "xl_1080p": FDConfig(latent_channels=48, latent_h=68, latent_w=120, vae_spatial=16,
                         hidden=1536, heads=24, kv_groups=3, mlp_gated=True, n_blocks=20,
                         n_refine=2, window=2, r_t=4, out_u8=True, name="xl_1080p", chunks=8),
}


def weight_layout(cfg: FDConfig) -> list[tuple[str, tuple[int, ...], str]]:
    """Tensors of the weight blob in blob order: (name, shape, kind).

    kind is "w" (linear weight, stored [out][in]), "b" (bias) or "g" (RMSNorm gain).
    The same order is documented in include/flashdec.h.
    """
    D, Dh, N, G = cfg.hidden, cfg.head_dim, cfg.heads, cfg.kv_groups
    Dm = cfg.mlp_ratio * D
    D1 = 2 * Dm if cfg.mlp_gated else Dm  # gated: gate rows, then up rows
    out: list[tuple[str, tuple[int, ...], str]] = [
        ("embed.w", (D, cfg.c_in), "w"), ("embed.b", (D,), "b")]

    def block(prefix: str) -> None:
        out.extend([
            (f"{prefix}.norm1.g", (D,), "g"),
            (f"{prefix}.qkv.w", ((N + 2 * G) * Dh, D), "w"),
            (f"{prefix}.qkv.b", ((N + 2 * G) * Dh,), "b"),
            (f"{prefix}.knorm.g", (Dh,), "g"),
            (f"{prefix}.{'qnorm' if cfg.qk_norm else 'vnorm'}.g", (Dh,), "g"),
            (f"{prefix}.out.w", (D, N * Dh), "w"),
            (f"{prefix}.out.b", (D,), "b"),
            (f"{prefix}.norm2.g", (D,), "g"),
            (f"{prefix}.mlp1.w", (D1, D), "w"),
            (f"{prefix}.mlp1.b", (D1,), "b"),
            (f"{prefix}.mlp2.w", (D, Dm), "w"),
            (f"{prefix}.mlp2.b", (D,), "b"),
        ])

    for b in range(cfg.n_blocks):
        block(f"blocks.{b}")
    out.extend([("normf.g", (D,), "g"), ("tup.w", (cfg.r_t * D, D), "w"),
                ("tup.b", (cfg.r_t * D,), "b")])
    for b in range(cfg.n_refine):
        block(f"refine.{b}")
    out.extend([("normh.g", (D,), "g"), ("head1.w", (D, D), "w"), ("head1.b", (D,), "b"),
                ("head2.w", (cfg.head_out, D), "w"), ("head2.b", (cfg.head_out,), "b")])
    return out


def normal(seed: int, stream: int, n: int, dtype=np.float32) -> np.ndarray:
    """n standard-normal draws from Philox4x64-10 keyed by (seed, stream)."""
    key = (int(seed) << 32) | (int(stream) & 0xFFFFFFFF)
    gen = np.random.Generator(np.random.Philox(key=key))
    return gen.standard_normal(n, dtype=dtype)


def to_bf16_values(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even); returned as fp32.

    Plain bit manipulation of IEEE binary32 (sign, 8-bit exponent, top 7 mantissa bits
    kept), used only to make the random weights exactly representable in bf16 so the
    oracle and the CUDA path start from identical weight values.
    """
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) & np.uint32(0xFFFF0000)
    return r.view(np.float32)


def make_weights(cfg: FDConfig, seed: int | None = None, std: float = 0.02,
                 threads: int = 8) -> dict[str, np.ndarray]:
    """Random-init weights: linears and biases N(0, std^2), gains 1 + N(0, std^2).

    Every value is rounded to bf16 so both sides use the same numbers.
    """
    seed = cfg.weight_seed if seed is None else seed
    layout = weight_layout(cfg)

    def one(i: int) -> tuple[str, np.ndarray]:
        name, shape, kind = layout[i]
        n = int(np.prod(shape))
        x = normal(seed, i, n) * np.float32(std)
        if kind == "g":
            x = x + np.float32(1.0)
        return name, to_bf16_values(x).reshape(shape)

    with ThreadPoolExecutor(max_workers=max(1, threads)) as ex:
        return dict(ex.map(one, range(len(layout))))


def make_latents(cfg: FDConfig, chunks: int | None = None, seed: int | None = None,
                 mode: str | None = None, rho: float = 0.9) -> np.ndarray:
    """Latent chunks, fp32 [chunks][C'][H'][W'] (one latent frame per chunk).

    "iid": N(0,1). "ar1": z_0 = e_0, z_t = rho z_{t-1} + sqrt(1 - rho^2) e_t, elementwise.
    """
    chunks = cfg.chunks if chunks is None else chunks
    seed = cfg.latent_seed if seed is None else seed
    mode = cfg.latent_mode if mode is None else mode
    per = cfg.latent_channels * cfg.latent_h * cfg.latent_w
    e = normal(seed, 0x7FFF0000, chunks * per).reshape(
        chunks, cfg.latent_channels, cfg.latent_h, cfg.latent_w)
    if mode == "iid":
        return e
    if mode != "ar1":
        raise ValueError(f"unknown latent mode {mode!r}")
    z = np.empty_like(e)
    a = np.float32(rho)
    b = np.float32(np.sqrt(1.0 - rho * rho))
    z[0] = e[0]
    for t in range(1, chunks):
        z[t] = a * z[t - 1] + b * e[t]
    return z


def frames_of_chunk(cfg: FDConfig, t: int) -> int:
    """Output frames of chunk t: r_t, or 1 for chunk 0 under the causal count of Fig. 2."""
    return 1 if t == 0 and cfg.first_chunk_frames == 1 else cfg.r_t


def make_target_pixels(cfg: FDConfig, chunks: int | None = None, seed: int = 77,
                       min_abs: float = 0.0) -> list[np.ndarray]:
    """Synthetic ground-truth video for a training step: per chunk fp32
    [C][frames][H][W] with values in [-1, 1] (normalised pixels). Magnitudes are uniform on
    [min_abs, 1] with a random sign (min_abs = 0: uniform on [-1, 1])."""
    chunks = cfg.chunks if chunks is None else chunks
    out = []
    for t in range(chunks):
        shape = (cfg.out_channels, frames_of_chunk(cfg, t), cfg.out_h, cfg.out_w)
        n = int(np.prod(shape))
        key = (int(seed) << 32) | (0x7FFE0000 + t)
        gen = np.random.Generator(np.random.Philox(key=key))
        mag = gen.uniform(min_abs, 1.0, n).astype(np.float32)
        sign = np.where(gen.integers(0, 2, n) == 1, np.float32(1.0), np.float32(-1.0))
        out.append((mag * sign).reshape(shape))
    return out
