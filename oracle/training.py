"""FlashDecoder streaming training step: plain fp64 CPU oracle.

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: only ``tests/`` may import it. It
shares no code with the CUDA path.

What one training step computes, from the paper:
  * Sec. 3.3 "Training--Inference Consistency": training follows the decoding protocol, T'
    sequential forward passes (Algorithm 1, one latent frame per pass) through the rolling
    cache, with no attention mask. The decode itself is ``StreamingDecoder``.
  * Sec. 3.5, Eq. (loss): the objective is lambda_L1 L1(x_hat, x) + lambda_LPIPS LPIPS +
    lambda_adv L_adv, with lambda_L1 = 1 in every stage of the supplementary hyper-parameter
    table. Only the pixel term is computed here: LPIPS needs a pretrained feature network and
    the adversarial term a trained 3D PatchGAN discriminator, neither of which is part of the
    decoder.
  * The gradient of that loss with respect to every decoder parameter, by reverse-mode
    differentiation of the fp64 oracle (PyTorch autograd as the differentiation routine).

Readings where the paper leaves a choice:
  T1  The loss takes the decoder's output before the clamp to [-1, 1] of reading R9 (the clamp
      is the display step of decoding; its derivative would be zero wherever it is active).
  T2  Gradients flow through the cache: the K / V a pass appends stay in the autograd graph,
      so the loss of frame t reaches the parameters through the passes of frames
      t - W + 1 .. t - 1 as well. The step's gradient is then the gradient of the same function
      that one pass over the whole clip under the block sliding-window mask computes, which is
      the consistency Sec. 3.3 claims. Option ``detach_cache``: the cache is kept out of the
      graph, so each pass's backward covers that pass alone (memory O(W L) per pass), a
      truncated gradient that differs from the full one whenever W > 1.
  T3  L1 = mean over every decoded pixel of every frame of the clip of |x_hat - x|.
"""
from __future__ import annotations

import numpy as np
import torch

from .flashdecoder import F64, StreamingDecoder, decode_full_masked


def leaf_weights(weights: dict) -> dict[str, torch.Tensor]:
    """Decoder parameters as fp64 leaf tensors that collect gradients."""
    return {k: torch.as_tensor(np.asarray(v), dtype=F64).clone().requires_grad_(True)
            for k, v in weights.items()}


def l1_loss(pixels: list[torch.Tensor], targets) -> torch.Tensor:
    """Mean absolute error over every pixel of every frame (reading T3)."""
    total = sum(p.numel() for p in pixels)
    err = sum((p - torch.as_tensor(np.asarray(x), dtype=F64)).abs().sum()
              for p, x in zip(pixels, targets))
    return err / total


def streaming_outputs(cfg, w: dict, latents, detach_cache: bool = False) -> list[torch.Tensor]:
    """Unclamped outputs of the T' sequential passes (Algorithm 1), graph kept (reading T2)."""
    dec = StreamingDecoder(cfg, w, detach_cache=detach_cache)
    return [dec.decode_chunk(z, clamp=False) for z in latents]


def streaming_loss(cfg, w: dict, latents, targets, detach_cache: bool = False) -> torch.Tensor:
    return l1_loss(streaming_outputs(cfg, w, latents, detach_cache), targets)


def masked_loss(cfg, w: dict, latents, targets) -> torch.Tensor:
    """The same loss from one pass over the whole clip under the block sliding-window mask
    (the masked training that Sec. 3.3 compares streaming training with)."""
    return l1_loss(decode_full_masked(cfg, w, latents, clamp=False), targets)


def gradients(loss: torch.Tensor, w: dict) -> dict[str, torch.Tensor]:
    names = list(w)
    g = torch.autograd.grad(loss, [w[n] for n in names], allow_unused=True)
    return {n: (torch.zeros_like(w[n]) if gi is None else gi) for n, gi in zip(names, g)}


def training_step(cfg, weights: dict, latents, targets, detach_cache: bool = False):
    """One streaming training step: (loss, {parameter name: dL/dparameter}), fp64."""
    w = leaf_weights(weights)
    loss = streaming_loss(cfg, w, latents, targets, detach_cache)
    return float(loss.detach()), gradients(loss, w)
