"""Strength of the oracle's pins: plant a plausible mistake in the oracle (on the CPU, by
replacing one of its functions for the duration of a test) and check that at least one pin of
tests/test_oracle_pins.py fails. A mistake no pin catches would mean the oracle is only
checked against itself there. CPU only."""
import contextlib
import math

import numpy as np
import pytest
import torch

import oracle
import oracle.flashdecoder as fd
import test_oracle_pins as pins

F64 = torch.float64


@contextlib.contextmanager
def planted(name, fn):
    """Replace oracle function `name` everywhere the pins and the decoder look it up."""
    saved = getattr(fd, name)
    setattr(fd, name, fn)
    had = hasattr(oracle, name)
    if had:
        saved_pkg = getattr(oracle, name)
        setattr(oracle, name, fn)
    try:
        yield
    finally:
        setattr(fd, name, saved)
        if had:
            setattr(oracle, name, saved_pkg)


def caught(*checks):
    for check in checks:
        try:
            check()
        except AssertionError:
            return True
    return False


# ---------------------------------------------------------------- the planted mistakes
def _rms_eps_outside(x, g, eps):
    return x / (torch.sqrt((x * x).mean(dim=-1, keepdim=True)) + eps) * g


def _gelu_tanh(x):
    return 0.5 * x * (1 + torch.tanh(math.sqrt(2 / math.pi) * (x + 0.044715 * x ** 3)))


def _linear_no_bias(x, w, b):
    fd.FLOPS["gemm"] += 2 * x.shape[0] * w.shape[0] * w.shape[1]
    return x @ w.T


_orig_shuffle = fd.pixel_shuffle
_orig_unshuffle = fd.pixel_unshuffle
_orig_rope = fd.rope
_orig_attention = fd.attention
_orig_stack = fd.StreamingDecoder._stack
_orig_quantize = fd.quantize_u8
_orig_mask = fd.chunk_mask


def _shuffle_ij_swapped(F, frames, gh, gw, C, rs):
    t = F.reshape(frames, gh, gw, C, rs, rs).permute(3, 0, 1, 5, 2, 4)
    return t.reshape(C, frames, gh * rs, gw * rs)


def _unshuffle_channel_last(z, p):
    C, H, W = z.shape
    t = z.reshape(C, H // p, p, W // p, p).permute(1, 3, 2, 4, 0)
    return t.reshape((H // p) * (W // p), C * p * p)


def _rope_backwards(x, pos_f, pos_y, pos_x, base):
    neg = lambda p: -fd._t(p)
    return _orig_rope(x, neg(pos_f), neg(pos_y), neg(pos_x), base)


def _rope_bands_uneven(dh):
    return [(0, 20), (20, 22), (42, 22)]


def _attention_unscaled(q, k, v, allowed=None, rows=2048):
    return _orig_attention(q * math.sqrt(q.shape[-1]), k, v, allowed, rows)


def _attention_groups_interleaved(q, k, v, allowed=None, rows=2048):
    N, G = q.shape[0], k.shape[0]
    perm = [n % G * (N // G) + n // G for n in range(N)]  # head n reads group n % G
    out = _orig_attention(q[perm], k, v, allowed, rows)
    inv = [0] * N
    for i, pn in enumerate(perm):
        inv[pn] = i
    return out[inv]


def _stack_tail(delta_chunks):
    def stack(self, h, prefix, n, kc, vc, frames, tail):
        rows = len(frames) * self.cfg.tokens
        return _orig_stack(self, h, prefix, n, kc, vc, frames, max(0, tail + delta_chunks * rows))
    return stack


def _block_qkv_v_unnormalised(h, w, p, cfg, pos):
    q, k, v = _orig_block_qkv(h, w, p, cfg, pos)
    L = h.shape[0]
    u = fd.rms_norm(h, w[p + "norm1.g"], cfg.norm_eps)
    qkv = fd.linear(u, w[p + "qkv.w"], w[p + "qkv.b"])
    v_raw = qkv[:, (cfg.heads + cfg.kv_groups) * 64:].reshape(L, cfg.kv_groups, 64).transpose(0, 1)
    return q, k, v_raw


_orig_block_qkv = fd._block_qkv
_orig_block_rest = fd._block_rest


def _block_rest_no_attention(h, o, w, p, cfg):
    return _orig_block_rest(h, torch.zeros_like(o), w, p, cfg)


def _quantize_half_up(pix):
    x = np.asarray(pix.numpy() if torch.is_tensor(pix) else pix).astype(np.float32)
    x = np.where(np.isnan(x), np.float32(-1.0), x)
    x = np.clip(x, -1.0, 1.0).astype(np.float32)
    b = ((x + np.float32(1.0)).astype(np.float32) * np.float32(127.5)).astype(np.float32)
    return np.floor(b + 0.5).astype(np.uint8)


def _mask_one_too_many(chunk_of_tok, window):
    return _orig_mask(chunk_of_tok, window + 1)


# every mistake with the pins expected to see it
MUTATIONS = [
    ("RMSNorm eps outside the square root", "rms_norm", _rms_eps_outside,
     [pins.test_rms_norm_matches_library_and_closed_form]),
    ("GELU tanh approximation instead of erf", "gelu", _gelu_tanh,
     [pins.test_gelu_matches_library_and_identities]),
    ("linear layer without its bias", "linear", _linear_no_bias,
     [pins.test_linear_is_x_wt_plus_b, pins.test_identity_blocks_reduce_to_closed_form]),
    ("pixel shuffle with i and j swapped", "pixel_shuffle", _shuffle_ij_swapped,
     [pins.test_pixel_shuffle_matches_library_and_inverts_unshuffle]),
    ("pixel unshuffle with the channel last", "pixel_unshuffle", _unshuffle_channel_last,
     [pins.test_pixel_unshuffle_matches_library_and_index_formula]),
    ("RoPE rotating by the negated angle", "rope", _rope_backwards,
     [pins.test_rope_matches_complex_rotation_and_is_relative]),
    ("RoPE bands split 20 / 22 / 22", "rope_bands", _rope_bands_uneven,
     [pins.test_rope_bands_at_head_dim_64]),
    ("attention without the 1/sqrt(D_h) scale", "attention", _attention_unscaled,
     [pins.test_attention_brute_force_gqa]),
    ("GQA head n reading group n % G", "attention", _attention_groups_interleaved,
     [pins.test_attention_brute_force_gqa]),
    ("V left without its KV-norm", "_block_qkv", _block_qkv_v_unnormalised,
     [pins.test_uniform_attention_decode_closed_form]),
    ("attention output not added to the residual", "_block_rest", _block_rest_no_attention,
     [pins.test_uniform_attention_decode_closed_form]),
    ("uint8 rounding half up instead of half to even", "quantize_u8", _quantize_half_up,
     [pins.test_quantize_u8_special_values]),
    ("block mask one chunk too wide", "chunk_mask", _mask_one_too_many,
     [pins.test_fig2_visibility_golden]),
]


@pytest.mark.parametrize("what,name,fn,checks", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_a_planted_mistake_fails_a_pin(what, name, fn, checks):
    with planted(name, fn):
        assert caught(*checks), f"no pin caught: {what}"
    # and with the oracle restored the same pins pass
    for check in checks:
        check()


@pytest.mark.parametrize("delta", [1, -1], ids=["cache one chunk too long", "one too short"])
def test_a_wrong_cache_window_fails_a_pin(delta):
    fd.StreamingDecoder._stack = _stack_tail(delta)
    try:
        assert caught(lambda: pins.test_streaming_equals_masked_full_sequence("small"),
                      pins.test_eviction_one_block)
    finally:
        fd.StreamingDecoder._stack = _orig_stack


# ---------------------------------------------------------------- training-step oracle
import test_oracle_training as tpins  # noqa: E402
from oracle import backward as bw  # noqa: E402
from oracle import training as tr  # noqa: E402

_orig_l1 = tr.l1_loss
_orig_streaming_outputs = tr.streaming_outputs


def _l1_sum_not_mean(pixels, targets):
    return _orig_l1(pixels, targets) * sum(p.numel() for p in pixels)


def _outputs_cache_detached(cfg, w, latents, detach_cache=False):
    return _orig_streaming_outputs(cfg, w, latents, True)


TRAIN_MUTATIONS = [
    ("L1 summed instead of averaged", "l1_loss", _l1_sum_not_mean,
     [tpins.test_last_layer_gradient_closed_form]),
    ("gradient stopped at the cache", "streaming_outputs", _outputs_cache_detached,
     [lambda: tpins.test_streaming_gradients_equal_masked_full_sequence("tiny_rt")]),
]


@pytest.mark.parametrize("what,name,fn,checks", TRAIN_MUTATIONS, ids=[m[0] for m in TRAIN_MUTATIONS])
def test_a_planted_training_mistake_fails_a_pin(what, name, fn, checks):
    saved = getattr(tr, name)
    setattr(tr, name, fn)
    try:
        assert caught(*checks), f"no pin caught: {what}"
    finally:
        setattr(tr, name, saved)


_orig_rms_bwd = bw.rms_norm_bwd
_orig_attn_bwd = bw.attention_bwd


def _rms_bwd_no_projection(x, g, eps, dy):
    r = 1.0 / torch.sqrt((x * x).mean(dim=-1, keepdim=True) + eps)
    dx, dg = _orig_rms_bwd(x, g, eps, dy)
    return r * dy * g, dg                  # the term through r dropped


def _attn_bwd_no_delta(q, k, v, do, allowed=None):
    N, Lq, dh = q.shape
    G = k.shape[0]
    scale = 1.0 / math.sqrt(dh)
    dq, dk, dv = torch.zeros_like(q), torch.zeros_like(k), torch.zeros_like(v)
    for n in range(N):
        g = n // (N // G)
        s = (q[n] @ k[g].T) * scale
        if allowed is not None:
            s = s.masked_fill(~allowed, float("-inf"))
        p = torch.softmax(s, dim=-1)
        dv[g] += p.T @ do[n]
        ds = p * (do[n] @ v[g].T)          # the softmax's - delta term dropped
        dq[n] = ds @ k[g] * scale
        dk[g] += ds.T @ q[n] * scale
    return dq, dk, dv


BWD_MUTATIONS = [
    ("RMSNorm backward without the normaliser's term", "rms_norm_bwd", _rms_bwd_no_projection),
    ("attention backward without delta", "attention_bwd", _attn_bwd_no_delta),
]


@pytest.mark.parametrize("what,name,fn", BWD_MUTATIONS, ids=[m[0] for m in BWD_MUTATIONS])
def test_a_planted_backward_mistake_fails_a_pin(what, name, fn):
    import test_oracle_backward as bpins
    saved = getattr(bw, name)
    setattr(bw, name, fn)
    try:
        assert caught(lambda: bpins.test_explicit_step_equals_autograd_step("tiny_rt")), what
    finally:
        setattr(bw, name, saved)


# ---------------------------------------------------------------- mistakes inside decode_chunk
def _mutant_decode_chunk(old, new):
    """decode_chunk with one line of its source replaced (a planted mistake)."""
    import inspect
    import textwrap
    src = textwrap.dedent(inspect.getsource(fd.StreamingDecoder.decode_chunk))
    assert src.count(old) == 1, old
    ns = {}
    exec(compile(src.replace(old, new), "<mutant>", "exec"), vars(fd), ns)
    return ns["decode_chunk"]


CHUNK_MUTATIONS = [
    ("upsampled channels read token-major (reading R6 broken)",
     "hf = e.reshape(L, rt, D).transpose(0, 1).reshape(rt * L, D)",
     "hf = e.reshape(rt * L, D)",
     pins.test_identity_blocks_reduce_to_closed_form),
    ("refined frames all at temporal index t",
     "[t * rt + tau for tau in range(rt)]",
     "[t for tau in range(rt)]",
     lambda: pins.test_streaming_equals_masked_full_sequence("tiny_rt")),
]


@pytest.mark.parametrize("what,old,new,check", CHUNK_MUTATIONS, ids=[m[0] for m in CHUNK_MUTATIONS])
def test_a_planted_mistake_in_the_chunk_step_fails_a_pin(what, old, new, check):
    saved = fd.StreamingDecoder.decode_chunk
    fd.StreamingDecoder.decode_chunk = _mutant_decode_chunk(old, new)
    try:
        assert caught(check), f"no pin caught: {what}"
    finally:
        fd.StreamingDecoder.decode_chunk = saved
    check()
