"""Explicit backward pass of the FlashDecoder training step: plain fp64 CPU oracle.

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: only ``tests/`` may import it. It
shares no code with the CUDA path.

Each function below is the derivative of one forward operator written out by the chain rule,
with no automatic differentiation: these are the per-operator references that backward kernels
are checked against. ``training_step_explicit`` composes them into the gradient of the
training step of ``oracle.training`` (L1 pixel loss of a clip, reading T3), computed over the
whole clip at once under the block sliding-window mask (query chunk i sees key chunks
i - W < j <= i). Streaming training through the rolling cache has exactly this gradient
(Sec. 3.3 "Training--Inference Consistency", reading T2; pinned in the tests), and the one-pass
form is the one a GPU runs with all chunks in flight.

Notation: y = f(x) forward, dy = dL/dy coming in, dx = dL/dx going out. All tensors fp64.
"""
from __future__ import annotations

import math

import numpy as np
import torch

from .flashdecoder import (F64, _positions, attention, chunk_mask, gelu, linear, pixel_shuffle,
                           pixel_unshuffle, rms_norm, rope, silu)


# --------------------------------------------------------------------------------------
# Operators
# --------------------------------------------------------------------------------------
def linear_bwd(x: torch.Tensor, w: torch.Tensor, dy: torch.Tensor, need_dx: bool = True):
    """y = x W^T + b (W [out][in]): dx = dy W, dW = dy^T x, db = sum over rows of dy."""
    dx = dy @ w if need_dx else None
    return dx, dy.T @ x, dy.sum(dim=0)


def rms_norm_bwd(x: torch.Tensor, g: torch.Tensor, eps: float, dy: torch.Tensor):
    """y = x r g with r = (mean(x^2) + eps)^(-1/2) over the last axis (length n).
    With e = dy * g:  dx = r e - x r^3 (sum_j e_j x_j) / n;  dg = sum over rows of dy x r."""
    n = x.shape[-1]
    r = 1.0 / torch.sqrt((x * x).mean(dim=-1, keepdim=True) + eps)
    e = dy * g
    dx = r * e - x * r ** 3 * (e * x).sum(dim=-1, keepdim=True) / n
    dg = (dy * x * r).reshape(-1, n).sum(dim=0)
    return dx, dg


def gelu_bwd(z: torch.Tensor, da: torch.Tensor) -> torch.Tensor:
    """a = z Phi(z):  da/dz = Phi(z) + z phi(z), phi the standard normal density."""
    Phi = 0.5 * (1.0 + torch.erf(z / math.sqrt(2.0)))
    phi = torch.exp(-0.5 * z * z) / math.sqrt(2.0 * math.pi)
    return da * (Phi + z * phi)


def swiglu_bwd(z: torch.Tensor, da: torch.Tensor) -> torch.Tensor:
    """a = SiLU(z_gate) z_up with z = [z_gate | z_up] (gate columns first, reading R7):
    d z_gate = da z_up SiLU'(z_gate), SiLU'(x) = s(x) (1 + x (1 - s(x))), s the logistic;
    d z_up = da SiLU(z_gate)."""
    dm = z.shape[1] // 2
    zg, zu = z[:, :dm], z[:, dm:]
    s = 1.0 / (1.0 + torch.exp(-zg))
    return torch.cat([da * zu * s * (1.0 + zg * (1.0 - s)), da * silu(zg)], dim=1)


def rope_bwd(dy: torch.Tensor, pos_f, pos_y, pos_x, base: float) -> torch.Tensor:
    """RoPE rotates each pair by an angle; the transpose of a rotation is the rotation by the
    negated angle, i.e. RoPE at the negated positions."""
    neg = lambda p: -torch.as_tensor(np.asarray(p), dtype=F64) if not torch.is_tensor(p) else -p
    return rope(dy, neg(pos_f), neg(pos_y), neg(pos_x), base)


def attention_bwd(q, k, v, do, allowed=None):
    """O = softmax(q k^T / sqrt(D_h)) v per query head, head n reading KV group n // (N/G)
    (q [N][Lq][D_h], k, v [G][Lk][D_h]). With P the softmax and S the scaled scores:
      dV = P^T dO,  dP = dO V^T,  delta = rowsum(dO * O),  dS = P (dP - delta),
      dQ = dS K / sqrt(D_h),  dK = dS^T Q / sqrt(D_h);
    a group's dK, dV sum over the heads reading it."""
    N, Lq, dh = q.shape
    G = k.shape[0]
    scale = 1.0 / math.sqrt(dh)
    dq = torch.zeros_like(q)
    dk = torch.zeros_like(k)
    dv = torch.zeros_like(v)
    for n in range(N):
        g = n // (N // G)
        s = (q[n] @ k[g].T) * scale
        if allowed is not None:
            s = s.masked_fill(~allowed, float("-inf"))
        p = torch.exp(s - s.max(dim=-1, keepdim=True).values)
        p = p / p.sum(dim=-1, keepdim=True)
        o = p @ v[g]
        dv[g] += p.T @ do[n]
        dp = do[n] @ v[g].T
        delta = (do[n] * o).sum(dim=-1, keepdim=True)
        ds = p * (dp - delta)
        dq[n] = ds @ k[g] * scale
        dk[g] += ds.T @ q[n] * scale
    return dq, dk, dv


def pixel_shuffle_bwd(dpix: torch.Tensor, frames: int, gh: int, gw: int, C: int,
                      rs: int) -> torch.Tensor:
    """Inverse permutation of the pixel shuffle (Sec. 3.4 Step 3): pixel
    (c, tau, h r_s + i, w r_s + j) came from F[tau L + h gw + w][c r_s^2 + i r_s + j]."""
    t = dpix.reshape(C, frames, gh, rs, gw, rs).permute(1, 2, 4, 0, 3, 5)  # [tau][h][w][c][i][j]
    return t.reshape(frames * gh * gw, C * rs * rs)


def l1_bwd(pix: torch.Tensor, target, total: int) -> torch.Tensor:
    """L = sum |pix - x| / total:  dL/dpix = sign(pix - x) / total."""
    return torch.sign(pix - torch.as_tensor(np.asarray(target), dtype=F64)) / total


# --------------------------------------------------------------------------------------
# One block (Sec. 3.2) forward with saved activations, and its backward
# --------------------------------------------------------------------------------------
def _block_fwd(h, w, p, cfg, pos, allowed):
    N, G, dh = cfg.heads, cfg.kv_groups, cfg.head_dim
    L = h.shape[0]
    sv = {"h": h}
    u = rms_norm(h, w[p + "norm1.g"], cfg.norm_eps)
    qkv = linear(u, w[p + "qkv.w"], w[p + "qkv.b"])
    q0 = qkv[:, :N * dh].reshape(L, N, dh).transpose(0, 1)
    k0 = qkv[:, N * dh:(N + G) * dh].reshape(L, G, dh).transpose(0, 1)
    v0 = qkv[:, (N + G) * dh:].reshape(L, G, dh).transpose(0, 1)
    k1 = rms_norm(k0, w[p + "knorm.g"], cfg.norm_eps)
    if cfg.qk_norm:
        q1, v1 = rms_norm(q0, w[p + "qnorm.g"], cfg.norm_eps), v0
    else:
        q1, v1 = q0, rms_norm(v0, w[p + "vnorm.g"], cfg.norm_eps)
    q2, k2 = rope(q1, *pos, cfg.rope_base), rope(k1, *pos, cfg.rope_base)
    o = attention(q2, k2, v1, allowed)
    of = o.transpose(0, 1).reshape(L, -1)
    hm = h + linear(of, w[p + "out.w"], w[p + "out.b"])
    u2 = rms_norm(hm, w[p + "norm2.g"], cfg.norm_eps)
    z = linear(u2, w[p + "mlp1.w"], w[p + "mlp1.b"])
    if cfg.mlp_gated:
        dm = z.shape[1] // 2
        a = silu(z[:, :dm]) * z[:, dm:]
    else:
        a = gelu(z)
    ho = hm + linear(a, w[p + "mlp2.w"], w[p + "mlp2.b"])
    sv.update(u=u, q0=q0, k0=k0, v0=v0, q1=q1, k1=k1, v1=v1, q2=q2, k2=k2, of=of, hm=hm, u2=u2,
              z=z, a=a)
    return ho, sv


def _block_bwd(dho, sv, w, p, cfg, pos, allowed, grads):
    N, G, dh = cfg.heads, cfg.kv_groups, cfg.head_dim
    L = dho.shape[0]
    # MLP and its residual
    da, grads[p + "mlp2.w"], grads[p + "mlp2.b"] = linear_bwd(sv["a"], w[p + "mlp2.w"], dho)
    dz = swiglu_bwd(sv["z"], da) if cfg.mlp_gated else gelu_bwd(sv["z"], da)
    du2, grads[p + "mlp1.w"], grads[p + "mlp1.b"] = linear_bwd(sv["u2"], w[p + "mlp1.w"], dz)
    dhm_n, grads[p + "norm2.g"] = rms_norm_bwd(sv["hm"], w[p + "norm2.g"], cfg.norm_eps, du2)
    dhm = dho + dhm_n
    # attention output projection and its residual
    dof, grads[p + "out.w"], grads[p + "out.b"] = linear_bwd(sv["of"], w[p + "out.w"], dhm)
    do = dof.reshape(L, N, dh).transpose(0, 1)
    dq2, dk2, dv1 = attention_bwd(sv["q2"], sv["k2"], sv["v1"], do, allowed)
    dq1, dk1 = rope_bwd(dq2, *pos, cfg.rope_base), rope_bwd(dk2, *pos, cfg.rope_base)
    dk0, grads[p + "knorm.g"] = rms_norm_bwd(sv["k0"], w[p + "knorm.g"], cfg.norm_eps, dk1)
    if cfg.qk_norm:
        dq0, grads[p + "qnorm.g"] = rms_norm_bwd(sv["q0"], w[p + "qnorm.g"], cfg.norm_eps, dq1)
        dv0 = dv1
    else:
        dq0 = dq1
        dv0, grads[p + "vnorm.g"] = rms_norm_bwd(sv["v0"], w[p + "vnorm.g"], cfg.norm_eps, dv1)
    dqkv = torch.cat([dq0.transpose(0, 1).reshape(L, N * dh),
                      dk0.transpose(0, 1).reshape(L, G * dh),
                      dv0.transpose(0, 1).reshape(L, G * dh)], dim=1)
    du, grads[p + "qkv.w"], grads[p + "qkv.b"] = linear_bwd(sv["u"], w[p + "qkv.w"], dqkv)
    dh_n, grads[p + "norm1.g"] = rms_norm_bwd(sv["h"], w[p + "norm1.g"], cfg.norm_eps, du)
    return dhm + dh_n


# --------------------------------------------------------------------------------------
# The whole step
# --------------------------------------------------------------------------------------
def training_step_explicit(cfg, weights: dict, latents, targets):
    """(loss, {parameter name: dL/dparameter}) of the L1 training step over a clip, by the
    explicit backward above (no autograd)."""
    if getattr(cfg, "mlp_fp8", False):
        raise ValueError("the training step is defined for the bf16-valued decoder")
    with torch.no_grad():
        w = {k: torch.as_tensor(np.asarray(v), dtype=F64) for k, v in weights.items()}
        T = len(latents)
        L, D, rt = cfg.tokens, cfg.hidden, cfg.r_t
        grads: dict[str, torch.Tensor] = {}

        def stack_setup(frames_per_chunk):
            tok = frames_per_chunk * L
            allowed = chunk_mask(torch.arange(T * tok) // tok, cfg.window)
            pos = _positions(cfg, list(range(T * frames_per_chunk)), L)
            return allowed, pos

        # ---- forward, saving what the backward reads
        x0 = torch.cat([pixel_unshuffle(torch.as_tensor(np.asarray(z), dtype=F64), cfg.patch)
                        for z in latents])
        h = linear(x0, w["embed.w"], w["embed.b"])
        allowB, posB = stack_setup(1)
        savedB = []
        for b in range(cfg.n_blocks):
            h, sv = _block_fwd(h, w, f"blocks.{b}.", cfg, posB, allowB)
            savedB.append(sv)
        hB = h
        y = rms_norm(hB, w["normf.g"], cfg.norm_eps)
        e = linear(y, w["tup.w"], w["tup.b"])                            # [T L][r_t D]
        hf = torch.cat([e[c * L:(c + 1) * L].reshape(L, rt, D).transpose(0, 1).reshape(rt * L, D)
                        for c in range(T)])
        allowR, posR = stack_setup(rt)
        savedR = []
        for b in range(cfg.n_refine):
            hf, sv = _block_fwd(hf, w, f"refine.{b}.", cfg, posR, allowR)
            savedR.append(sv)
        hR = hf
        yh = rms_norm(hR, w["normh.g"], cfg.norm_eps)
        z1 = linear(yh, w["head1.w"], w["head1.b"])
        a1 = gelu(z1)
        F = linear(a1, w["head2.w"], w["head2.b"])
        pix = [pixel_shuffle(F[c * rt * L:(c + 1) * rt * L], rt, cfg.grid_h, cfg.grid_w,
                             cfg.out_channels, cfg.r_s) for c in range(T)]
        if getattr(cfg, "first_chunk_frames", 0) == 1:
            pix[0] = pix[0][:, :1]                                       # reading R16
        total = sum(p.numel() for p in pix)
        loss = sum((p - torch.as_tensor(np.asarray(x), dtype=F64)).abs().sum()
                   for p, x in zip(pix, targets)) / total

        # ---- backward
        dF = []
        for c in range(T):
            dp = l1_bwd(pix[c], targets[c], total)
            if dp.shape[1] != rt:                                        # one-frame chunk 0
                full = torch.zeros(dp.shape[0], rt, *dp.shape[2:], dtype=F64)
                full[:, :dp.shape[1]] = dp
                dp = full
            dF.append(pixel_shuffle_bwd(dp, rt, cfg.grid_h, cfg.grid_w, cfg.out_channels,
                                        cfg.r_s))
        dF = torch.cat(dF)
        da1, grads["head2.w"], grads["head2.b"] = linear_bwd(a1, w["head2.w"], dF)
        dz1 = gelu_bwd(z1, da1)
        dyh, grads["head1.w"], grads["head1.b"] = linear_bwd(yh, w["head1.w"], dz1)
        dhf, grads["normh.g"] = rms_norm_bwd(hR, w["normh.g"], cfg.norm_eps, dyh)
        for b in reversed(range(cfg.n_refine)):
            dhf = _block_bwd(dhf, savedR[b], w, f"refine.{b}.", cfg, posR, allowR, grads)
        # channel block tau of token l <- refined token tau L + l (reading R6), per chunk
        de = torch.cat([dhf[c * rt * L:(c + 1) * rt * L].reshape(rt, L, D).transpose(0, 1)
                        .reshape(L, rt * D) for c in range(T)])
        dy, grads["tup.w"], grads["tup.b"] = linear_bwd(y, w["tup.w"], de)
        dh, grads["normf.g"] = rms_norm_bwd(hB, w["normf.g"], cfg.norm_eps, dy)
        for b in reversed(range(cfg.n_blocks)):
            dh = _block_bwd(dh, savedB[b], w, f"blocks.{b}.", cfg, posB, allowB, grads)
        _, grads["embed.w"], grads["embed.b"] = linear_bwd(x0, w["embed.w"], dh, need_dx=False)
    return float(loss), grads
