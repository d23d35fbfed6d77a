"""Pins of the streaming training-step oracle (oracle/training.py) to things other than
itself: central finite differences of the loss (independent of autograd), the masked
full-sequence training pass (Sec. 3.3 "Training--Inference Consistency"), a closed form for
the last layer's gradient, and the degenerate window W = 1. CPU only."""
import numpy as np
import pytest
import torch

import oracle
import synth
from oracle import training as tr

F64 = torch.float64


def _setup(name, chunks=None, min_abs=0.0, **kw):
    cfg = synth.PRESETS[name].replace(**kw)
    chunks = cfg.chunks if chunks is None else chunks
    cfg = cfg.replace(chunks=chunks)
    w = synth.make_weights(cfg)
    z = synth.make_latents(cfg)
    x = synth.make_target_pixels(cfg, min_abs=min_abs)
    return cfg, w, z, x


def _direction(w, seed=5):
    """A random direction over every parameter, scaled like the parameters (std 0.02)."""
    g = torch.Generator().manual_seed(seed)
    return {k: torch.randn(np.asarray(v).shape, generator=g, dtype=F64) * 0.02
            for k, v in w.items()}


def _shift(w, d, eps):
    return {k: torch.as_tensor(np.asarray(v), dtype=F64) + eps * d[k] for k, v in w.items()}


def _dot(g, d):
    return sum(float((g[k] * d[k]).sum()) for k in g)


@pytest.mark.parametrize("name", ["tiny", "tiny_rt", "small", "tiny_gated", "tiny_qk",
                                  "small_f1"])
def test_streaming_gradients_equal_masked_full_sequence(name):
    """Sec. 3.3: streaming training (T' passes through the rolling cache, gradients through
    the cache, reading T2) optimises the same function as one masked pass over the clip, so
    loss and every parameter gradient agree up to summation order."""
    cfg, w, z, x = _setup(name, chunks=4 if name == "small" else None)
    ws = tr.leaf_weights(w)
    ls = tr.streaming_loss(cfg, ws, z, x)
    gs = tr.gradients(ls, ws)
    wm = tr.leaf_weights(w)
    lm = tr.masked_loss(cfg, wm, z, x)
    gm = tr.gradients(lm, wm)
    assert float(ls.detach()) == pytest.approx(float(lm.detach()), rel=1e-12)
    for k in gs:
        scale = float(gm[k].abs().max()) + 1e-30
        assert float((gs[k] - gm[k]).abs().max()) <= 1e-9 * scale, k


@pytest.mark.parametrize("name", ["tiny_rt", "tiny_gated"])
def test_gradient_matches_central_differences(name):
    """<dL/dtheta, d> against (L(theta + eps d) - L(theta - eps d)) / (2 eps), in fp64, for a
    random direction d over all parameters. The targets keep every residual at least 0.26 away
    from zero (|x| >= 0.6, |x_hat| <= 0.34 on these cases), so no |.| kink lies within
    +-eps d and the difference quotient has only its O(eps^2) error."""
    cfg, w, z, x = _setup(name, min_abs=0.6)
    loss, g = tr.training_step(cfg, w, z, x)
    out = tr.streaming_outputs(cfg, {k: torch.as_tensor(np.asarray(v), dtype=F64)
                                     for k, v in w.items()}, z)
    assert min(float((o - torch.as_tensor(t, dtype=F64)).abs().min())
               for o, t in zip(out, x)) > 0.2
    d = _direction(w)
    eps = 1e-4
    with torch.no_grad():
        lp = float(tr.streaming_loss(cfg, _shift(w, d, eps), z, x))
        lm = float(tr.streaming_loss(cfg, _shift(w, d, -eps), z, x))
    fd = (lp - lm) / (2 * eps)
    an = _dot(g, d)
    assert abs(an) > 1e-4                       # a direction the loss actually changes along
    assert fd == pytest.approx(an, rel=1e-6)


def test_single_parameter_derivatives_match_central_differences():
    """Entries of the gradient of single weights deep in the network (first block's QKV,
    attention output, refinement MLP, embedding) against one-coordinate differences."""
    cfg, w, z, x = _setup("tiny_rt", min_abs=0.6)
    _, g = tr.training_step(cfg, w, z, x)
    rng = np.random.default_rng(3)
    for name in ["embed.w", "blocks.0.qkv.w", "blocks.0.knorm.g", "blocks.1.out.w",
                 "refine.0.mlp1.w", "tup.b", "normh.g"]:
        shape = np.asarray(w[name]).shape
        idx = tuple(int(rng.integers(0, s)) for s in shape)
        eps = 1e-4
        vals = []
        for sgn in (1, -1):
            w2 = {k: torch.as_tensor(np.asarray(v), dtype=F64).clone() for k, v in w.items()}
            w2[name][idx] += sgn * eps
            with torch.no_grad():
                vals.append(float(tr.streaming_loss(cfg, w2, z, x)))
        fd = (vals[0] - vals[1]) / (2 * eps)
        an = float(g[name][idx])
        # 1e-11: the rounding of L (about 0.6) at fp64, divided by 2 eps, with a margin
        assert abs(fd - an) <= 1e-6 * abs(an) + 1e-11, (name, idx, fd, an)


def test_last_layer_gradient_closed_form():
    """For L = mean |x_hat - x| the head's last bias gets
    dL/db2[j] = (1 / P) sum over the pixels fed by output channel j of sign(x_hat - x),
    with channel j = c r_s^2 + i r_s + jj feeding pixel (c, tau, h r_s + i, w r_s + jj) of every
    token (PixelShuffle, Sec. 3.4). Computed here with numpy indexing, not autograd."""
    cfg, w, z, x = _setup("tiny_rt", min_abs=0.6)
    _, g = tr.training_step(cfg, w, z, x)
    with torch.no_grad():
        out = tr.streaming_outputs(cfg, {k: torch.as_tensor(np.asarray(v), dtype=F64)
                                         for k, v in w.items()}, z)
    rs, C = cfg.r_s, cfg.out_channels
    P = sum(o.numel() for o in out)
    want = np.zeros(C * rs * rs)
    for o, t in zip(out, x):
        s = np.sign(o.numpy() - t)                      # [C][frames][H][W]
        for c in range(C):
            for i in range(rs):
                for jj in range(rs):
                    want[c * rs * rs + i * rs + jj] += s[c, :, i::rs, jj::rs].sum()
    want /= P
    assert np.allclose(g["head2.b"].numpy(), want, rtol=0, atol=1e-15)


def test_detached_cache_is_the_truncated_gradient():
    """Option detach_cache (reading T2): the gradient is the sum over passes of each pass's
    gradient with the cache it read held constant. Pinned by central differences of exactly
    that objective: pass t re-run with perturbed weights on the cache state the unperturbed
    stream left before it. With W = 1 (no cache across passes) it equals the full gradient;
    with W = 2 it does not."""
    cfg, w, z, x = _setup("tiny_rt", min_abs=0.6)
    _, gd = tr.training_step(cfg, w, z, x, detach_cache=True)
    _, gf = tr.training_step(cfg, w, z, x)
    assert max(float((gd[k] - gf[k]).abs().max()) for k in gd) > 1e-8
    # cache state before each pass, from the unperturbed stream
    w0 = {k: torch.as_tensor(np.asarray(v), dtype=F64) for k, v in w.items()}
    dec = oracle.StreamingDecoder(cfg, w0)
    states = []
    with torch.no_grad():
        for t in range(cfg.chunks):
            states.append(([k.clone() for k in dec.kB], [v.clone() for v in dec.vB],
                           [k.clone() for k in dec.kR], [v.clone() for v in dec.vR], dec.t))
            dec.decode_chunk(z[t])
    P = sum(np.asarray(t).size for t in x)

    def frozen_loss(wp):
        total = 0.0
        for t in range(cfg.chunks):
            d2 = oracle.StreamingDecoder(cfg, wp)
            kB, vB, kR, vR, d2.t = states[t]
            d2.kB, d2.vB, d2.kR, d2.vR = list(kB), list(vB), list(kR), list(vR)
            o = d2.decode_chunk(z[t], clamp=False)
            total += float((o - torch.as_tensor(x[t], dtype=F64)).abs().sum())
        return total / P

    d = _direction(w)
    an = _dot(gd, d)
    assert abs(an) > 1e-4                       # a direction the loss actually changes along
    eps = 1e-4
    with torch.no_grad():
        fd = (frozen_loss(_shift(w, d, eps)) - frozen_loss(_shift(w, d, -eps))) / (2 * eps)
    assert fd == pytest.approx(an, rel=1e-6)
    # W = 1: nothing crosses passes, both gradients coincide
    cfg1, w1, z1, x1 = _setup("tiny_w1")
    _, a = tr.training_step(cfg1, w1, z1, x1, detach_cache=True)
    _, b = tr.training_step(cfg1, w1, z1, x1)
    for k in a:
        assert torch.equal(a[k], b[k]), k


def test_causal_training_gradient_of_a_frame_ignores_later_frames():
    """The loss of frame t alone has a gradient that does not depend on later latents
    (temporal causality by processing order, Sec. 3.3)."""
    cfg, w, z, x = _setup("tiny_rt")
    z2 = z.copy()
    z2[2] = -z[2]
    ga, gb = [], []
    for lat, acc in ((z, ga), (z2, gb)):
        ws = tr.leaf_weights(w)
        outs = tr.streaming_outputs(cfg, ws, lat)
        loss = tr.l1_loss(outs[:2], x[:2])         # frames of chunks 0 and 1 only
        acc.append(tr.gradients(loss, ws))
    for k in ga[0]:
        assert torch.equal(ga[0][k], gb[0][k]), k


@pytest.mark.parametrize("name", ["tiny_rt", "small", "tiny_gated"])
def test_training_cost_model_matches_counted_products(name):
    """costs.training_step_flops against the products the oracle's step actually runs, as
    PyTorch's FlopCounterMode counts them (forward and autograd's backward separately)."""
    from torch.utils.flop_counter import FlopCounterMode

    from paper_2607_14898_gb300 import costs
    cfg, w, z, x = _setup(name)
    ws = tr.leaf_weights(w)
    fwd, bwd = FlopCounterMode(display=False), FlopCounterMode(display=False)
    with fwd:
        loss = tr.streaming_loss(cfg, ws, z, x)
    with bwd:
        tr.gradients(loss, ws)
    want = costs.training_step_flops(cfg, cfg.chunks)
    assert fwd.get_total_flops() == want["forward"]
    assert bwd.get_total_flops() == want["backward"]


def test_target_pixels_are_seeded_normalised_frames():
    """Synthetic ground truth: one [C][frames][H][W] array per chunk in [-1, 1] (one frame
    for chunk 0 under the causal frame count), magnitudes at least min_abs, same seed same
    values."""
    cfg = synth.PRESETS["small_f1"]
    a, b = synth.make_target_pixels(cfg, min_abs=0.6), synth.make_target_pixels(cfg, min_abs=0.6)
    assert [x.shape for x in a] == [(3, 1, 160, 208)] + [(3, 4, 160, 208)] * (cfg.chunks - 1)
    for x, y in zip(a, b):
        assert np.array_equal(x, y) and x.dtype == np.float32
        assert float(np.abs(x).min()) >= 0.6 and float(np.abs(x).max()) <= 1.0
        assert abs(float((x > 0).mean()) - 0.5) < 0.02          # both signs, evenly
    c = synth.make_target_pixels(cfg, seed=78)
    assert not np.array_equal(c[1], synth.make_target_pixels(cfg)[1])
