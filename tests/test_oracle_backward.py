"""Pins of the explicit backward oracle (oracle/backward.py): every operator's hand-written
derivative against PyTorch's automatic differentiation of the forward operator (a library
routine), against central differences, and against closed forms; the composed step against
the autograd step of oracle/training.py. CPU only."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from oracle import backward as bw
from oracle import training as tr

F64 = torch.float64


def rnd(*shape, seed=0, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return torch.randn(*shape, generator=g, dtype=F64) * scale


def vjp(f, inputs, dy):
    """Autograd's vector-Jacobian product of f at inputs with cotangent dy."""
    xs = [x.clone().requires_grad_(True) for x in inputs]
    return torch.autograd.grad(f(*xs), xs, dy)


def close(a, b, tol=1e-12):
    return float((a - b).abs().max()) <= tol * (float(b.abs().max()) + 1e-300)


def test_linear_bwd_matches_autograd():
    x, w, b, dy = rnd(7, 12, seed=1), rnd(5, 12, seed=2), rnd(5, seed=3), rnd(7, 5, seed=4)
    want = vjp(lambda x, w, b: x @ w.T + b, [x, w, b], dy)
    got = bw.linear_bwd(x, w, dy)
    assert all(close(g, t) for g, t in zip(got, want))


@pytest.mark.parametrize("shape", [(6, 32), (3, 9, 64)])
def test_rms_norm_bwd_matches_autograd_and_differences(shape):
    x, g, dy = rnd(*shape, seed=5), 1 + rnd(shape[-1], seed=6, scale=0.1), rnd(*shape, seed=7)
    want = vjp(lambda x, g: oracle.rms_norm(x, g, 1e-6), [x, g], dy)
    got = bw.rms_norm_bwd(x, g, 1e-6, dy)
    assert close(got[0], want[0]) and close(got[1], want[1])
    # one coordinate by central differences
    idx = (0,) * (len(shape) - 1) + (3,)
    eps = 1e-6
    xp, xm = x.clone(), x.clone()
    xp[idx] += eps
    xm[idx] -= eps
    fd = float(((oracle.rms_norm(xp, g, 1e-6) - oracle.rms_norm(xm, g, 1e-6)) * dy).sum()) / (2 * eps)
    assert fd == pytest.approx(float(got[0][idx]), rel=1e-7)


def test_gelu_bwd_matches_autograd_and_closed_form():
    z = torch.linspace(-6, 6, 241, dtype=F64)
    da = rnd(241, seed=8)
    assert close(bw.gelu_bwd(z, da), vjp(oracle.gelu, [z], da)[0])
    # GELU'(0) = 1/2, and GELU'(z) -> 1 / 0 far on the positive / negative side
    one = torch.ones(1, dtype=F64)
    assert float(bw.gelu_bwd(torch.zeros(1, dtype=F64), one)) == pytest.approx(0.5, abs=1e-15)
    assert float(bw.gelu_bwd(torch.full((1,), 9.0, dtype=F64), one)) == pytest.approx(1.0, abs=1e-12)
    assert abs(float(bw.gelu_bwd(torch.full((1,), -9.0, dtype=F64), one))) < 1e-12


def test_swiglu_bwd_matches_autograd():
    z, da = rnd(5, 16, seed=9, scale=3.0), rnd(5, 8, seed=10)
    f = lambda z: oracle.silu(z[:, :8]) * z[:, 8:]
    assert close(bw.swiglu_bwd(z, da), vjp(f, [z], da)[0])


def test_rope_bwd_is_the_inverse_rotation():
    pos = (torch.tensor([0.0, 3.0, 7.0], dtype=F64), torch.tensor([1.0, 2.0, 5.0], dtype=F64),
           torch.tensor([4.0, 0.0, 9.0], dtype=F64))
    x, dy = rnd(2, 3, 64, seed=11), rnd(2, 3, 64, seed=12)
    f = lambda x: oracle.rope(x, *pos, 10000.0)
    assert close(bw.rope_bwd(dy, *pos, 10000.0), vjp(f, [x], dy)[0])
    # a rotation's transpose undoes it
    assert close(bw.rope_bwd(f(x), *pos, 10000.0), x, 1e-13)


@pytest.mark.parametrize("masked", [False, True])
def test_attention_bwd_matches_autograd(masked):
    N, G, Lq, Lk = 4, 2, 6, 9
    q, k, v = rnd(N, Lq, 64, seed=13), rnd(G, Lk, 64, seed=14), rnd(G, Lk, 64, seed=15)
    do = rnd(N, Lq, 64, seed=16)
    allowed = None
    if masked:  # query row i sees keys <= i + 3 (every row keeps at least one key)
        allowed = torch.arange(Lk)[None, :] <= torch.arange(Lq)[:, None] + 3
    want = vjp(lambda q, k, v: oracle.attention(q, k, v, allowed), [q, k, v], do)
    got = bw.attention_bwd(q, k, v, do, allowed)
    assert all(close(g, t) for g, t in zip(got, want))


def test_attention_bwd_with_one_key_closed_form():
    """One key: the softmax is 1, O = v for every query, so dV sums dO over the group's heads
    and queries, and dQ, dK vanish."""
    q, k, v = rnd(4, 5, 64, seed=17), rnd(2, 1, 64, seed=18), rnd(2, 1, 64, seed=19)
    do = rnd(4, 5, 64, seed=20)
    dq, dk, dv = bw.attention_bwd(q, k, v, do)
    assert float(dq.abs().max()) < 1e-14 and float(dk.abs().max()) < 1e-14
    for g in range(2):
        assert close(dv[g, 0], do[2 * g:2 * g + 2].sum(dim=(0, 1)))


def test_pixel_shuffle_bwd_is_the_adjoint():
    """<shuffle(F), P> = <F, shuffle_bwd(P)> for the permutation (no autograd involved)."""
    frames, gh, gw, C, rs = 2, 3, 4, 3, 8
    F = rnd(frames * gh * gw, C * rs * rs, seed=21)
    P = rnd(C, frames, gh * rs, gw * rs, seed=22)
    lhs = float((oracle.pixel_shuffle(F, frames, gh, gw, C, rs) * P).sum())
    rhs = float((F * bw.pixel_shuffle_bwd(P, frames, gh, gw, C, rs)).sum())
    assert lhs == pytest.approx(rhs, rel=1e-13)


def test_l1_bwd_is_the_sign_over_the_count():
    pix = torch.tensor([[0.5, -0.2], [0.1, 0.9]], dtype=F64)
    x = np.array([[0.0, 0.3], [0.1, -1.0]])
    assert torch.equal(bw.l1_bwd(pix, x, 8), torch.tensor([[1, -1], [0, 1]], dtype=F64) / 8)


@pytest.mark.parametrize("name", ["tiny", "tiny_rt", "small", "tiny_gated", "tiny_qk",
                                  "small_f1", "tiny_xl"])
def test_explicit_step_equals_autograd_step(name):
    """The hand-written backward over the whole clip (masked one-pass form) gives the
    streaming step's loss and every gradient, to rounding."""
    cfg = synth.PRESETS[name]
    if name == "small":
        cfg = cfg.replace(chunks=4)
    w, z, x = synth.make_weights(cfg), synth.make_latents(cfg), synth.make_target_pixels(cfg)
    la, ga = tr.training_step(cfg, w, z, x)
    le, ge = bw.training_step_explicit(cfg, w, z, x)
    assert le == pytest.approx(la, rel=1e-13)
    assert set(ge) == set(ga)
    for k in ga:
        assert close(ge[k], ga[k], 1e-11), k


def test_explicit_step_refuses_the_fp8_option():
    cfg = synth.PRESETS["small_fp8"]
    with pytest.raises(ValueError):
        bw.training_step_explicit(cfg, synth.make_weights(cfg), synth.make_latents(cfg),
                                  synth.make_target_pixels(cfg))
