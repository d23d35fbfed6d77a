"""Algorithmic work of one decoded chunk, per kernel kind.

FLOPs count 2 per multiply-add of the method's own contractions (Sec. 3.3 "Complexity
Analysis": attention over the c_t = min(t+1, W) cached chunks only); bytes count each HBM
operand of the bandwidth-bound kernels once.
"""
from __future__ import annotations

DH = 64


def window_chunks(cfg, t: int) -> int:
    return min(t + 1, cfg.window)


def chunk_flops(cfg, t: int) -> dict[str, int]:
    L, D, N, G = cfg.tokens, cfg.hidden, cfg.heads, cfg.kv_groups
    R = cfg.r_t * L
    c = window_chunks(cfg, t)
    qkv_out = (N + 2 * G) * DH
    Dm = cfg.mlp_ratio * D

    def block(rows: int, keys: int) -> dict[str, int]:
        return {"qkv": 2 * rows * D * qkv_out, "attn": 4 * rows * keys * DH * N,
                "out": 2 * rows * N * DH * D,
                "mlp1": 2 * rows * D * Dm * (2 if cfg.mlp_gated else 1),  # gated: gate + up
                "mlp2": 2 * rows * Dm * D}

    f = {"embed": 2 * L * cfg.c_in * D, "qkv": 0, "attn_backbone": 0, "attn_refine": 0,
         "out": 0, "mlp1": 0, "mlp2": 0, "tup": 2 * L * D * cfg.r_t * D,
         "head1": 2 * R * D * D, "head2": 2 * R * D * cfg.head_out}
    for rows, keys, n, akey in ((L, c * L, cfg.n_blocks, "attn_backbone"),
                                (R, c * R, cfg.n_refine, "attn_refine")):
        b = block(rows, keys)
        f["qkv"] += n * b["qkv"]
        f[akey] += n * b["attn"]
        for k in ("out", "mlp1", "mlp2"):
            f[k] += n * b[k]
    return f


def chunk_bytes(cfg, t: int) -> dict[str, int]:
    """HBM bytes of the bandwidth-bound kernels (read once + write once)."""
    L, D, R = cfg.tokens, cfg.hidden, cfg.r_t * cfg.tokens
    out_elem = 1 if cfg.out_u8 else 4
    norm_rows = 2 * cfg.n_blocks * L + 2 * cfg.n_refine * R + L + R
    return {
        "unshuffle": cfg.latent_channels * cfg.latent_h * cfg.latent_w * 4 + L * cfg.c_in * 2,
        "rmsnorm": norm_rows * D * (4 + 2),
        "pixel": R * cfg.head_out * (4 + out_elem),
    }


def stream_flops(cfg, chunks: int) -> int:
    return sum(sum(chunk_flops(cfg, t).values()) for t in range(chunks))


def training_step_flops(cfg, chunks: int) -> dict[str, int]:
    """Contraction FLOPs of one streaming training step over `chunks` latent frames (the
    forward passes of Algorithm 1, the L1 pixel loss, every parameter's gradient). Each
    product's backward is two products of its size (the input and the weight gradient; in
    attention dQ and dK for the scores, dP and dV for P V), except the patch-embedding, whose
    input is the latent and needs no gradient."""
    fwd = stream_flops(cfg, chunks)
    emb = sum(chunk_flops(cfg, t)["embed"] for t in range(chunks))
    return {"forward": fwd, "backward": 2 * fwd - emb}


def training_kind_flops(cfg, chunks: int) -> dict[str, int]:
    """training_step_flops split by the kernel kinds of the GPU step (enum fd_train_kind): the
    linears' forward products, their input gradients (none for the patch-embedding), their weight
    gradients, and the attention's products (S and P V forward, dP, dQ, dK, dV backward: three
    times the forward's; the step's recomputation of S is not counted)."""
    lin = emb = att = 0
    for t in range(chunks):
        f = chunk_flops(cfg, t)
        a = f["attn_backbone"] + f["attn_refine"]
        att += a
        lin += sum(f.values()) - a
        emb += f["embed"]
    return {"linear": lin, "dgrad": lin - emb, "wgrad": lin, "attn_gemm": 3 * att}
