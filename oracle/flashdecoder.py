"""FlashDecoder streaming decode: plain fp64 CPU oracle.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s
CPU-baseline / reference arm may import this module. The CUDA library never calls it, and it
shares no code with the CUDA path; the only thing both sides use is the seeded input module
``synth``.

Everything here is written straight from the paper, in fp64 with PyTorch CPU tensors:
  * Sec. 3.2 "Base Architecture": pre-RMSNorm before each sublayer, GQA attention, KV-norm,
    3D-RoPE applied separately on the temporal and spatial (H' x W') axes.
  * Eq. (projection): latent frame -> L_frm tokens in raster order -> Linear_{C'->D}.
  * Sec. 4.3 "Generalization Across Latent Spaces": PixelUnshuffle(2) on 8x latents.
  * Sec. 3.3, Eq. (kv_cache), Algorithm 1: frame-by-frame decoding with a rolling cache of the
    last W_frm frames, kept literally as concat(tail_{(W-1)L}(K), K_t).
  * Eq. (temporal_upsample): Linear_{D -> r_t D}, channels reinterpreted as r_t frames.
  * Sec. 3.4 "Step 2": temporal-refinement blocks with window r_t W_frm.
  * Sec. 3.4 "Step 3": 2-layer MLP D -> C r_s^2, then PixelShuffle(r_s).

Readings where the paper leaves a choice (each listed in the design notes):
  R3  KV-norm = RMSNorm over the head dimension of K and of V (learned gain of length D_h,
      shared by all groups), applied before RoPE; Q is not normalised. Option qk_norm: the
      usual QK-norm instead, on Q and K (gains qnorm.g, knorm.g), V not normalised.
  R4  3D-RoPE bands: D_h split [temporal | height | width] = [D_h - 2*2*floor(D_h/6) | 2*floor(D_h/6)
      | 2*floor(D_h/6)] dims (24/20/20 at D_h = 64); rotation of interleaved pairs
      (2i, 2i+1) by angle pos * base^(-2i/d_band).
  R5  "RoPE offset t*L_frm": chunk t has temporal coordinate t (backbone) or t*r_t + tau
      (refinement); "relative to the window" (Sec. 4.3 "Long Video Decoding") is the
      rope_mode="window" option and gives the same scores in exact arithmetic.
  R6  Reshape after temporal upsampling: channel block tau (channels tau*D .. tau*D + D - 1)
      becomes refined frame tau; refined token tau*L + l.
  R7  MLP = Linear(D, 4D) -> GELU (erf form) -> Linear(4D, D); biases on every linear (R13).
      Gated option (the XL layout): Linear(D, 4D) gate and Linear(D, 4D) up, SiLU(gate) * up,
      then Linear(4D, D); the first weight stores the gate rows, then the up rows.
      FP8 option (Sec. 4.6, "static-calibrated FP8 quantization of all MLP layers"): both MLP
      matrix products take e4m3 operands with power-of-two scales fixed before decoding:
      per weight row s = 2^ceil(log2(max|w| / 448)); the MLP input u = RMSNorm(h) g obeys
      |u_i| <= sqrt(D) max|g|, its scale s_u covers that; the MLP hidden a = GELU(z) obeys
      |a_j| <= max(1, max_j 1.125 sqrt(D) max|g| ||w1_j|| + |b1_j|), its scale s_h covers that.
      With the gated MLP, a_j = SiLU(z_gate_j) z_up_j and |SiLU(x)| <= max(|x|, 0.28) (SiLU is
      below x for x > 0 and its negative branch never reaches -0.2785), so
      |a_j| <= max(B_gate_j, 0.28) B_up_j with B the same per-row bound on |z|.
      So no value leaves the e4m3 range (448) for any input.
  R8  Head MLP: Linear(D, D) -> GELU -> Linear(D, C r_s^2).
  R9  Pixels clamped to [-1, 1]; uint8 = round-half-even(fl32(fl32(x + 1) * 127.5)).
  R12 RMSNorm with a learned gain before the temporal upsampling and before the head.
  R16 Frame count: every chunk emits r_t frames; option first_chunk_frames = 1 follows Fig. 2's
      causal count (T' latent frames -> 1 + r_t (T' - 1) frames): chunk 0 emits refined frame
      tau = 0 only (the paper does not say which one is kept); nothing else changes.
  R14 RMSNorm: x / sqrt(mean(x^2) + eps) * g with eps = 1e-6.
"""
from __future__ import annotations

import contextlib
import math

import numpy as np
import torch

F64 = torch.float64

# Multiply-add counter: every matrix product below adds 2*M*N*K here (used to pin the
# closed-form cost model against the work this oracle actually performs).
FLOPS = {"gemm": 0, "attn": 0}


def reset_flops() -> None:
    FLOPS["gemm"] = 0
    FLOPS["attn"] = 0


# Operand rounding (off by default): the computation stays fp64, but the operands of every
# matrix product are first rounded to the storage precision of "bf16 compute, fp32
# accumulate": Linear inputs to bf16 (round to nearest even), attention Q and K to bf16 and
# V to fp16. With it on, the oracle measures the rounding noise that precision alone causes,
# which is what a floating-point tolerance for a given model size can be derived from.
_OPERAND_ROUNDING = [False]


@contextlib.contextmanager
def operand_rounding():
    prev = _OPERAND_ROUNDING[0]
    _OPERAND_ROUNDING[0] = True
    try:
        yield
    finally:
        _OPERAND_ROUNDING[0] = prev


def _round(x: torch.Tensor, dtype) -> torch.Tensor:
    return x.to(dtype).to(F64) if _OPERAND_ROUNDING[0] else x


def _t(x) -> torch.Tensor:
    return torch.as_tensor(np.asarray(x), dtype=F64) if not torch.is_tensor(x) else x.to(F64)


# --------------------------------------------------------------------------------------
# Elementary operators
# --------------------------------------------------------------------------------------
def rms_norm(x: torch.Tensor, g: torch.Tensor, eps: float) -> torch.Tensor:
    """RMSNorm (Sec. 3.2, Zhang & Sennrich): x / sqrt(mean(x^2) + eps) * g, last axis."""
    return x / torch.sqrt((x * x).mean(dim=-1, keepdim=True) + eps) * g


def gelu(x: torch.Tensor) -> torch.Tensor:
    """GELU, exact erf form: x * Phi(x) = 0.5 x (1 + erf(x / sqrt 2))."""
    return 0.5 * x * (1.0 + torch.erf(x / math.sqrt(2.0)))


def e4m3(x: torch.Tensor) -> torch.Tensor:
    """Round to the nearest FP8 E4M3 value (OCP: 3 mantissa bits, bias 7, largest 448,
    subnormals down to 2^-9), ties to even."""
    return x.to(torch.float8_e4m3fn).to(F64)


def pow2_ceil(x: float) -> float:
    """Smallest power of two >= x (x > 0), exactly."""
    m, e = math.frexp(x)          # x = m 2^e, 0.5 <= m < 1
    return math.ldexp(1.0, e - 1) if m == 0.5 else math.ldexp(1.0, e)


def fp8_weight(w: torch.Tensor) -> torch.Tensor:
    """Per-row FP8 quantisation of a Linear weight [out][in], returned dequantised."""
    amax = w.abs().max(dim=1).values
    s = torch.tensor([pow2_ceil(float(a) / 448.0) if a > 0 else 1.0 for a in amax], dtype=F64)
    return e4m3(w / s[:, None]) * s[:, None]


def fp8_mlp_scales(g2: torch.Tensor, w1_deq: torch.Tensor, b1: torch.Tensor,
                   gated: bool = False):
    """Static activation scales (s_u, s_h) of one FP8 MLP from its weights (see R7)."""
    D = g2.shape[0]
    gmax = float(g2.abs().max())
    s_u = pow2_ceil(math.sqrt(D) * gmax / 448.0)
    bz = 1.125 * math.sqrt(D) * gmax * w1_deq.norm(dim=1) + b1.abs()   # |z_j| <= bz_j
    if gated:
        dm = bz.shape[0] // 2
        bound = float((torch.clamp(bz[:dm], min=0.28) * bz[dm:]).max())
    else:
        bound = float(bz.max())
    s_h = pow2_ceil(max(bound, 1.0) / 448.0)
    return s_u, s_h


def silu(x: torch.Tensor) -> torch.Tensor:
    """SiLU (swish): x * sigmoid(x) = x / (1 + exp(-x))."""
    return x / (1.0 + torch.exp(-x))


def linear(x: torch.Tensor, w: torch.Tensor, b: torch.Tensor | None) -> torch.Tensor:
    """y = x W^T + b with W stored [out][in] (Eq. projection and every other Linear)."""
    FLOPS["gemm"] += 2 * x.shape[0] * w.shape[0] * w.shape[1]
    y = _round(x, torch.bfloat16) @ w.T
    return y if b is None else y + b


def pixel_unshuffle(z: torch.Tensor, p: int) -> torch.Tensor:
    """Latent frame [C'][H'][W'] -> tokens [L][C' p^2] (Sec. 4.3, Eq. projection).

    Token l = h*(W'/p) + w in raster order; channel c*p^2 + i*p + j holds z[c][h*p+i][w*p+j]
    (PixelUnshuffle's channel order).
    """
    C, H, W = z.shape
    t = z.reshape(C, H // p, p, W // p, p).permute(1, 3, 0, 2, 4)  # [h][w][c][i][j]
    return t.reshape((H // p) * (W // p), C * p * p)


def pixel_shuffle(F: torch.Tensor, frames: int, gh: int, gw: int, C: int, rs: int) -> torch.Tensor:
    """Head features [frames*L][C r_s^2] -> pixels [C][frames][gh*r_s][gw*r_s] (Sec. 3.4).

    pix[c][tau][h*r_s+i][w*r_s+j] = F[tau*L + h*gw + w][c*r_s^2 + i*r_s + j]
    (PixelShuffle, Shi et al. 2016).
    """
    t = F.reshape(frames, gh, gw, C, rs, rs).permute(3, 0, 1, 4, 2, 5)  # [c][tau][h][i][w][j]
    return t.reshape(C, frames, gh * rs, gw * rs)


def rope_bands(dh: int) -> list[tuple[int, int]]:
    """(offset, width) of the temporal, height and width bands of 3D-RoPE (reading R4)."""
    ds = 2 * (dh // 6)
    dt = dh - 2 * ds
    return [(0, dt), (dt, ds), (dt + ds, ds)]


def rope(x: torch.Tensor, pos_f, pos_y, pos_x, base: float) -> torch.Tensor:
    """3D-RoPE on x [..., L, D_h]; pos_* are the L tokens' temporal / row / column indices.

    Each band rotates its interleaved pairs (2i, 2i+1) by the angle pos * base^(-2i/d_band)
    (RoFormer, Su et al.), one band per axis (Sec. 3.2).
    """
    out = x.clone()
    dh = x.shape[-1]
    for (off, d), pos in zip(rope_bands(dh), (pos_f, pos_y, pos_x)):
        i = torch.arange(d // 2, dtype=F64)
        theta = base ** (-2.0 * i / d)
        ang = _t(pos)[:, None] * theta[None, :]
        c, s = torch.cos(ang), torch.sin(ang)
        a = x[..., off:off + d:2]
        b = x[..., off + 1:off + d:2]
        out[..., off:off + d:2] = a * c - b * s
        out[..., off + 1:off + d:2] = a * s + b * c
    return out


def attention(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor,
              allowed: torch.Tensor | None = None, rows: int = 2048) -> torch.Tensor:
    """GQA attention softmax(q k^T / sqrt(D_h)) v (Sec. 3.2, Eq. kv_cache).

    q [N][Lq][D_h]; k, v [G][Lk][D_h]; query head n reads KV group n // (N/G).
    ``allowed`` [Lq][Lk] (optional) marks visible keys; streaming decode needs none
    (Sec. 3.3 "Attention Pattern"). The softmax is row-wise, so query rows are taken
    ``rows`` at a time only to bound memory.
    """
    N, Lq, dh = q.shape
    G, Lk, _ = k.shape
    q, k, v = _round(q, torch.bfloat16), _round(k, torch.bfloat16), _round(v, torch.float16)
    out = torch.empty_like(q)
    scale = 1.0 / math.sqrt(dh)
    for n in range(N):
        g = n // (N // G)
        for r0 in range(0, Lq, rows):
            r1 = min(Lq, r0 + rows)
            s = (q[n, r0:r1] @ k[g].T) * scale
            if allowed is not None:
                s = s.masked_fill(~allowed[r0:r1], float("-inf"))
            s = s - s.max(dim=-1, keepdim=True).values
            p = torch.exp(s)
            out[n, r0:r1] = (p @ v[g]) / p.sum(dim=-1, keepdim=True)
        FLOPS["attn"] += 4 * Lq * Lk * dh
    return out


def quantize_u8(pix: np.ndarray | torch.Tensor) -> np.ndarray:
    """uint8 code of clamped pixels (reading R9), decided in fp32 like the kernel.

    q = round_half_even(fl32(fl32(clamp(x, -1, 1) + 1) * 127.5)); NaN -> 0.
    """
    x = np.asarray(pix.numpy() if torch.is_tensor(pix) else pix).astype(np.float32)
    x = np.where(np.isnan(x), np.float32(-1.0), x)
    x = np.minimum(np.maximum(x, np.float32(-1.0)), np.float32(1.0))
    a = (x + np.float32(1.0)).astype(np.float32)
    b = (a * np.float32(127.5)).astype(np.float32)
    return np.rint(b).astype(np.uint8)


# --------------------------------------------------------------------------------------
# Transformer block (Sec. 3.2) with the rolling cache of Sec. 3.3 / Algorithm 1
# --------------------------------------------------------------------------------------
def _block_qkv(h, w, p, cfg, pos):
    """Pre-norm, QKV projection, KV-norm (R3) and 3D-RoPE for one block."""
    N, G, dh = cfg.heads, cfg.kv_groups, cfg.head_dim
    L = h.shape[0]
    u = rms_norm(h, w[p + "norm1.g"], cfg.norm_eps)
    qkv = linear(u, w[p + "qkv.w"], w[p + "qkv.b"])
    q = qkv[:, :N * dh].reshape(L, N, dh).transpose(0, 1)
    k = qkv[:, N * dh:(N + G) * dh].reshape(L, G, dh).transpose(0, 1)
    v = qkv[:, (N + G) * dh:].reshape(L, G, dh).transpose(0, 1)
    k = rms_norm(k, w[p + "knorm.g"], cfg.norm_eps)
    if cfg.qk_norm:
        q = rms_norm(q, w[p + "qnorm.g"], cfg.norm_eps)
    else:
        v = rms_norm(v, w[p + "vnorm.g"], cfg.norm_eps)
    if pos is not None:
        q = rope(q, *pos, cfg.rope_base)
        k = rope(k, *pos, cfg.rope_base)
    return q, k, v


def _block_rest(h, o, w, p, cfg):
    """Output projection + residual, then pre-norm MLP + residual (Sec. 3.2, R7)."""
    L = h.shape[0]
    o = o.transpose(0, 1).reshape(L, -1)
    h = h + linear(o, w[p + "out.w"], w[p + "out.b"])
    u = rms_norm(h, w[p + "norm2.g"], cfg.norm_eps)
    if getattr(cfg, "mlp_fp8", False):
        w1, w2 = fp8_weight(w[p + "mlp1.w"]), fp8_weight(w[p + "mlp2.w"])
        s_u, s_h = fp8_mlp_scales(w[p + "norm2.g"], w1, w[p + "mlp1.b"], cfg.mlp_gated)
        z = linear(e4m3(u / s_u) * s_u, w1, w[p + "mlp1.b"])
        if cfg.mlp_gated:
            dm = z.shape[1] // 2
            a = silu(z[:, :dm]) * z[:, dm:]
        else:
            a = gelu(z)
        return h + linear(e4m3(a / s_h) * s_h, w2, w[p + "mlp2.b"])
    z = linear(u, w[p + "mlp1.w"], w[p + "mlp1.b"])
    if cfg.mlp_gated:
        dm = z.shape[1] // 2
        a = silu(z[:, :dm]) * z[:, dm:]
    else:
        a = gelu(z)
    return h + linear(a, w[p + "mlp2.w"], w[p + "mlp2.b"])


def _positions(cfg, frames: list[int], tokens_per_frame: int):
    """Temporal / row / column index of each token of the listed frames (raster order)."""
    l = torch.arange(tokens_per_frame)
    f = torch.cat([torch.full((tokens_per_frame,), fr, dtype=F64) for fr in frames])
    y = (l // cfg.grid_w).to(F64).repeat(len(frames))
    x = (l % cfg.grid_w).to(F64).repeat(len(frames))
    return f, y, x


class StreamingDecoder:
    """Algorithm 1, one latent frame per call to ``decode_chunk``.

    ``rope_mode="abs"``: keys are rotated once, at their absolute temporal index, when they
    enter the cache. ``rope_mode="window"``: the cache keeps un-rotated keys and every step
    re-rotates the whole window with temporal indices counted from the window's first frame
    (Sec. 4.3 "Long Video Decoding").
    """

    def __init__(self, cfg, weights: dict, rope_mode: str = "abs", detach_cache: bool = False):
        self.cfg = cfg
        self.w = {k: _t(v) for k, v in weights.items()}
        if rope_mode not in ("abs", "window"):
            raise ValueError(rope_mode)
        self.rope_mode = rope_mode
        # training option (oracle/training.py): keep the cached K / V out of the autograd
        # graph, so a chunk's gradient stops at the cache; no effect on the values
        self.detach_cache = detach_cache
        self.reset()

    def reset(self) -> None:
        """Algorithm 1 initialisation: empty caches, empty output."""
        cfg = self.cfg
        empty = lambda: torch.zeros(cfg.kv_groups, 0, cfg.head_dim, dtype=F64)
        self.kB = [empty() for _ in range(cfg.n_blocks)]
        self.vB = [empty() for _ in range(cfg.n_blocks)]
        self.kR = [empty() for _ in range(cfg.n_refine)]
        self.vR = [empty() for _ in range(cfg.n_refine)]
        self.t = 0

    # one stack of blocks (backbone B or refinement R) over the frames of chunk t
    def _stack(self, h, prefix, n, kc, vc, frames, tail):
        cfg = self.cfg
        L = cfg.tokens
        window_rel = self.rope_mode == "window"
        pos_new = _positions(cfg, frames, L)
        for b in range(n):
            p = f"{prefix}.{b}."
            q, k, v = _block_qkv(h, self.w, p, cfg, None if window_rel else pos_new)
            # cache update: concat(tail_{(W-1) L}(K), K_t)  (Algorithm 1)
            K = torch.cat([kc[b][:, max(0, kc[b].shape[1] - tail):], k], dim=1)
            V = torch.cat([vc[b][:, max(0, vc[b].shape[1] - tail):], v], dim=1)
            kc[b], vc[b] = (K.detach(), V.detach()) if self.detach_cache else (K, V)
            if window_rel:
                n_frames = K.shape[1] // L             # frames now in the window
                first = frames[-1] + 1 - n_frames      # absolute index of the oldest one
                K = rope(K, *_positions(cfg, list(range(n_frames)), L), cfg.rope_base)
                q = rope(q, *_positions(cfg, [fr - first for fr in frames], L),
                         cfg.rope_base)
            o = attention(q, K, V)
            h = _block_rest(h, o, self.w, p, cfg)
        return h

    def decode_chunk(self, z_t, clamp: bool = True) -> torch.Tensor:
        """Decode latent frame z_t [C'][H'][W'] -> clamped pixels [C][r_t][H][W] (fp64).
        clamp=False returns the head's output before the clamp (the training loss's input)."""
        cfg, w, t = self.cfg, self.w, self.t
        L, D, rt = cfg.tokens, cfg.hidden, cfg.r_t
        # Project (Eq. projection, with PixelUnshuffle(p) of Sec. 4.3)
        x0 = pixel_unshuffle(_t(z_t), cfg.patch)
        h = linear(x0, w["embed.w"], w["embed.b"])
        # Backbone B with temporal index t, cache tail (W-1) L
        h = self._stack(h, "blocks", cfg.n_blocks, self.kB, self.vB, [t],
                        (cfg.window - 1) * L)
        # Temporal upsampling (Eq. temporal_upsample) and channel -> time reshape (R6)
        y = rms_norm(h, w["normf.g"], cfg.norm_eps)
        e = linear(y, w["tup.w"], w["tup.b"])                       # [L][r_t D]
        hf = e.reshape(L, rt, D).transpose(0, 1).reshape(rt * L, D)  # token tau*L + l
        # Temporal refinement R: frames t*r_t + tau, cache tail r_t (W-1) L
        hf = self._stack(hf, "refine", cfg.n_refine, self.kR, self.vR,
                         [t * rt + tau for tau in range(rt)], rt * (cfg.window - 1) * L)
        # Spatial upsampling: MLP D -> C r_s^2, PixelShuffle(r_s), clamp (R8, R9)
        y = rms_norm(hf, w["normh.g"], cfg.norm_eps)
        F = linear(gelu(linear(y, w["head1.w"], w["head1.b"])), w["head2.w"], w["head2.b"])
        pix = pixel_shuffle(F, rt, cfg.grid_h, cfg.grid_w, cfg.out_channels, cfg.r_s)
        if t == 0 and getattr(cfg, "first_chunk_frames", 0) == 1:
            pix = pix[:, :1]                                        # R16
        self.t += 1
        return pix.clamp(-1.0, 1.0) if clamp else pix


def decode_stream(cfg, weights, latents, rope_mode: str = "abs") -> list[torch.Tensor]:
    """Algorithm 1 over all latent frames: list of per-chunk pixel tensors."""
    dec = StreamingDecoder(cfg, weights, rope_mode)
    return [dec.decode_chunk(z) for z in latents]


# --------------------------------------------------------------------------------------
# Full-sequence pass under the block sliding-window mask (Sec. 3.3 "Training-Inference
# Consistency"): all chunks at once, query chunk i sees key chunk j iff i - W < j <= i.
# Streaming decode must equal this pass; it is the check that the rolling cache is right.
# --------------------------------------------------------------------------------------
def chunk_mask(chunk_of_tok: torch.Tensor, window: int) -> torch.Tensor:
    i = chunk_of_tok[:, None]
    j = chunk_of_tok[None, :]
    return (j <= i) & (j > i - window)


def decode_full_masked(cfg, weights, latents, clamp: bool = True) -> list[torch.Tensor]:
    w = {k: _t(v) for k, v in weights.items()}
    T = len(latents)
    L, D, rt = cfg.tokens, cfg.hidden, cfg.r_t

    def stack(h, prefix, n, frames_per_chunk):
        tok_per_chunk = frames_per_chunk * L
        chunk_of = torch.arange(T * tok_per_chunk) // tok_per_chunk
        allowed = chunk_mask(chunk_of, cfg.window)
        frames = list(range(T * frames_per_chunk))
        pos = _positions(cfg, frames, L)
        for b in range(n):
            p = f"{prefix}.{b}."
            q, k, v = _block_qkv(h, w, p, cfg, pos)
            o = attention(q, k, v, allowed)
            h = _block_rest(h, o, w, p, cfg)
        return h

    h = torch.cat([linear(pixel_unshuffle(_t(z), cfg.patch), w["embed.w"], w["embed.b"])
                   for z in latents])
    h = stack(h, "blocks", cfg.n_blocks, 1)
    y = rms_norm(h, w["normf.g"], cfg.norm_eps)
    e = linear(y, w["tup.w"], w["tup.b"])
    hf = torch.cat([e[c * L:(c + 1) * L].reshape(L, rt, D).transpose(0, 1).reshape(rt * L, D)
                    for c in range(T)])
    hf = stack(hf, "refine", cfg.n_refine, rt)
    y = rms_norm(hf, w["normh.g"], cfg.norm_eps)
    F = linear(gelu(linear(y, w["head1.w"], w["head1.b"])), w["head2.w"], w["head2.b"])
    out = [pixel_shuffle(F[c * rt * L:(c + 1) * rt * L], rt, cfg.grid_h, cfg.grid_w,
                         cfg.out_channels, cfg.r_s) for c in range(T)]
    if clamp:
        out = [o.clamp(-1.0, 1.0) for o in out]
    if getattr(cfg, "first_chunk_frames", 0) == 1:
        out[0] = out[0][:, :1]                                      # R16
    return out


# --------------------------------------------------------------------------------------
# Closed forms used to check the accounting (Sec. 3.3 "Complexity Analysis", Eq. kv_cache)
# --------------------------------------------------------------------------------------
def kv_cache_elems(cfg) -> dict:
    """Cache size per layer: G x (W L) x D_h for K and for V (Eq. kv_cache), backbone and
    refinement (capacity r_t W L, Sec. 3.3)."""
    per_b = 2 * cfg.kv_groups * cfg.window * cfg.tokens * cfg.head_dim
    per_r = 2 * cfg.kv_groups * cfg.r_t * cfg.window * cfg.tokens * cfg.head_dim
    return {"backbone_per_layer": per_b, "refine_per_layer": per_r}
