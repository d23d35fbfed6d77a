"""Pins of the CPU oracle to things other than itself (library routines, brute force, closed
forms, the paper's worked example, invariants of the method). CPU only."""
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as tF

import oracle
import synth

F64 = torch.float64
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rnd(*shape, seed=0, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return torch.randn(*shape, generator=g, dtype=F64) * scale


# ---------------------------------------------------------------- elementary operators
def test_rms_norm_matches_library_and_closed_form():
    x, g = rnd(7, 33, seed=1), rnd(33, seed=2)
    ref = tF.rms_norm(x, (33,), weight=g, eps=1e-6)
    assert torch.allclose(oracle.rms_norm(x, g, 1e-6), ref, rtol=1e-12, atol=1e-12)
    # [3, 4]: mean square 12.5
    y = oracle.rms_norm(torch.tensor([3.0, 4.0], dtype=F64), torch.ones(2, dtype=F64), 0.0)
    assert torch.allclose(y, torch.tensor([3.0, 4.0], dtype=F64) / math.sqrt(12.5))


def test_gelu_matches_library_and_identities():
    x = torch.linspace(-8, 8, 1001, dtype=F64)
    assert torch.allclose(oracle.gelu(x), tF.gelu(x, approximate="none"), atol=1e-14)
    assert torch.allclose(oracle.gelu(x) - oracle.gelu(-x), x, atol=1e-12)  # Phi(x)+Phi(-x)=1
    assert oracle.gelu(torch.tensor(1.0, dtype=F64)).item() == pytest.approx(
        0.5 * (1 + math.erf(1 / math.sqrt(2))), rel=1e-15)


def test_silu_matches_library_and_identities():
    x = torch.linspace(-30, 30, 2001, dtype=torch.float64)
    assert torch.allclose(oracle.silu(x), tF.silu(x), rtol=0, atol=1e-15)
    # silu(x) - silu(-x) = x (sigmoid(x) + sigmoid(-x) = 1); silu(0) = 0; tails -> x and -> 0
    assert torch.allclose(oracle.silu(x) - oracle.silu(-x), x, rtol=0, atol=1e-12)
    assert float(oracle.silu(torch.tensor(0.0, dtype=torch.float64))) == 0.0
    big = torch.tensor([40.0, -40.0], dtype=torch.float64)
    assert torch.allclose(oracle.silu(big), torch.tensor([40.0, 0.0], dtype=torch.float64),
                          atol=1e-15)


def test_gated_mlp_worked_example():
    """Gated MLP of the XL layout on a hand-computed case: out-projection zero, h = (1, 1) so
    the pre-norm leaves it at (1, 1) / sqrt(1 + eps); gate row (1, 0), up row (0, 2) give
    SiLU(g) * u; down rows (1) and (-1) with bias (0.5, 0)."""
    from oracle.flashdecoder import _block_rest

    class Cfg:
        norm_eps = 1e-6
        mlp_gated = True

    f = lambda v: torch.tensor(v, dtype=torch.float64)
    w = {"x.out.w": torch.zeros(2, 2, dtype=torch.float64), "x.out.b": f([0.0, 0.0]),
         "x.norm2.g": f([1.0, 1.0]), "x.mlp1.w": f([[1.0, 0.0], [0.0, 2.0]]),
         "x.mlp1.b": f([0.0, 0.0]), "x.mlp2.w": f([[1.0], [-1.0]]), "x.mlp2.b": f([0.5, 0.0])}
    h = f([[1.0, 1.0]])
    o = torch.zeros(1, 1, 2, dtype=torch.float64)
    s = 1.0 / math.sqrt(1.0 + 1e-6)
    a = s / (1.0 + math.exp(-s)) * (2.0 * s)
    got = _block_rest(h, o, w, "x.", Cfg)
    assert torch.allclose(got, f([[1.0 + a + 0.5, 1.0 - a]]), rtol=0, atol=1e-14)


def test_xl_parameter_count_fits_the_gated_mlp():
    """FlashDecoder-XL is listed with 769.3 M parameters (Table "Model scaling", D = 1536,
    N = 24, G = 3, 20 blocks). With the configuration table's 2 refinement blocks and 48
    latent channels, the gated 3-matrix 4x MLP comes within 3 % of it; the 2-matrix MLP falls
    more than 200 M short."""
    count = lambda cfg: sum(int(np.prod(s)) for _, s, _ in synth.weight_layout(cfg))
    xl = synth.PRESETS["xl_480p"]
    assert abs(count(xl) - 769.3e6) < 0.03 * 769.3e6
    assert 769.3e6 - count(xl.replace(mlp_gated=False)) > 200e6


def test_operand_rounding_rounds_to_nearest_even_and_is_off_by_default():
    """The test-only operand rounding: Linear inputs to bf16, attention Q, K to bf16 and V to
    fp16, round to nearest even (as the library's dtype conversions); off outside the context."""
    x = torch.tensor([[1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -9, -3.0 + 2.0 ** -10]],
                     dtype=torch.float64)
    w = torch.eye(3, dtype=torch.float64)
    assert torch.equal(oracle.linear(x, w, None), x)
    with oracle.operand_rounding():
        # ties go to even: 1 + 2^-8 -> 1 (bf16 spacing 2^-7), 1 + 3 2^-9 -> 1 + 2^-7
        want = torch.tensor([[1.0, 1.0 + 2.0 ** -7, -3.0]], dtype=torch.float64)
        assert torch.equal(oracle.linear(x, w, None), want)
        v = torch.tensor([[[1.0 + 2.0 ** -11, 2.0]]], dtype=torch.float64)
        q = torch.zeros(1, 1, 1, dtype=torch.float64)
        k = torch.zeros(1, 1, 1, dtype=torch.float64)
        # one key: the output is V, rounded to fp16 (1 + 2^-11 is a tie between 1 and 1 + 2^-10)
        assert float(oracle.attention(q, k, v[:, :, :1])[0, 0, 0]) == 1.0
    assert torch.equal(oracle.linear(x, w, None), x)


def test_qk_norm_bounds_every_score():
    """QK-norm option: with unit gains every query and key head vector has length sqrt(D_h), so
    by Cauchy-Schwarz every scaled score q.k / sqrt(D_h) lies in [-sqrt(D_h), sqrt(D_h)] = [-8, 8],
    whatever the activations; V keeps its scale. KV-norm normalises V instead of Q."""
    from oracle.flashdecoder import _block_qkv
    base = synth.PRESETS["tiny_qk"]
    Dh, N, G, D = base.head_dim, base.heads, base.kv_groups, base.hidden
    torch.manual_seed(0)
    h = torch.randn(16, D, dtype=torch.float64) * 3
    w = {"x.norm1.g": torch.ones(D, dtype=torch.float64),
         "x.qkv.w": torch.randn((N + 2 * G) * Dh, D, dtype=torch.float64) * 5,
         "x.qkv.b": torch.zeros((N + 2 * G) * Dh, dtype=torch.float64),
         "x.knorm.g": torch.ones(Dh, dtype=torch.float64),
         "x.qnorm.g": torch.ones(Dh, dtype=torch.float64),
         "x.vnorm.g": torch.ones(Dh, dtype=torch.float64)}
    for qk in (True, False):
        cfg = base.replace(qk_norm=qk, norm_eps=0.0)
        q, k, v = _block_qkv(h, w, "x.", cfg, None)
        qn, kn, vn = (x.norm(dim=-1) for x in (q, k, v))
        assert torch.allclose(kn, torch.full_like(kn, math.sqrt(Dh)), atol=1e-9)
        if qk:
            assert torch.allclose(qn, torch.full_like(qn, math.sqrt(Dh)), atol=1e-9)
            s = torch.einsum("nld,nmd->nlm", q, k.repeat_interleave(N // G, 0)) / math.sqrt(Dh)
            assert float(s.abs().max()) <= math.sqrt(Dh) + 1e-9
            assert float(vn.max()) > 2 * math.sqrt(Dh)   # V left as projected
        else:
            assert torch.allclose(vn, torch.full_like(vn, math.sqrt(Dh)), atol=1e-9)
            assert float(qn.max()) > 2 * math.sqrt(Dh)


def test_e4m3_rounding_worked_values():
    """FP8 E4M3 (3 mantissa bits, exponent bias 7, max 448, subnormal step 2^-9), ties to even,
    on values worked out by hand: 1 + 2^-4 lies halfway between 1 and 1.125 -> 1 (even
    mantissa); 1.1875 halfway between 1.125 and 1.25 -> 1.25; 3 * 2^-10 halfway between the
    subnormals 2^-9 and 2^-8 -> 2^-8; 2^-10 halfway between 0 and 2^-9 -> 0; 449 -> 448."""
    cases = [(0.5, 0.5), (1.0625, 1.0), (1.1875, 1.25), (-1.0625, -1.0), (13.0, 13.0),
             (448.0, 448.0), (449.0, 448.0), (2.0 ** -9, 2.0 ** -9), (3 * 2.0 ** -10, 2.0 ** -8),
             (2.0 ** -10, 0.0), (248.0, 256.0), (0.0, 0.0)]
    x = torch.tensor([c[0] for c in cases], dtype=torch.float64)
    assert oracle.e4m3(x).tolist() == [c[1] for c in cases]


def test_pow2_ceil_is_exact():
    assert [oracle.pow2_ceil(v) for v in (3.0, 4.0, 0.3, 1.0, 4.000001, 2.0 ** -20)] == \
        [4.0, 4.0, 0.5, 1.0, 8.0, 2.0 ** -20]


def test_fp8_static_scales_never_overflow_and_are_tight():
    """The static MLP scales keep every scaled FP8 operand within the e4m3 range (448) for any
    input, including a row whose RMSNorm puts all its weight in one coordinate (|u_i| =
    sqrt(D) g_i, the bound), and that row uses more than half of the range."""
    from oracle.flashdecoder import gelu, linear
    cfg = synth.PRESETS["small_fp8"]
    w = {k: torch.from_numpy(v).to(torch.float64) for k, v in synth.make_weights(cfg).items()}
    D = cfg.hidden
    g2, w1, b1 = w["blocks.0.norm2.g"], oracle.fp8_weight(w["blocks.0.mlp1.w"]), w["blocks.0.mlp1.b"]
    s_u, s_h = oracle.fp8_mlp_scales(g2, w1, b1)
    h = torch.randn(64, D, dtype=torch.float64) * 3
    i = int(g2.abs().argmax())
    h[0] = 0.0
    h[0, i] = 5.0                                 # one-hot row: |u_i| = sqrt(D) |g_i|
    u = oracle.rms_norm(h, g2, 0.0)
    assert float((u / s_u).abs().max()) <= 448.0
    assert float((u[0] / s_u).abs().max()) > 224.0
    a = gelu(linear(oracle.e4m3(u / s_u) * s_u, w1, b1))
    assert float((a / s_h).abs().max()) <= 448.0
    # the FP8 MLP output differs from the exact one by FP8-sized amounts, not more
    w2 = w["blocks.0.mlp2.w"]
    exact = linear(gelu(linear(u, w["blocks.0.mlp1.w"], b1)), w2, None)
    q = linear(oracle.e4m3(a / s_h) * s_h, oracle.fp8_weight(w2), None)
    rel = float((q - exact).norm() / exact.norm())
    assert 1e-3 < rel < 0.1, rel


def test_silu_bound_used_by_the_gated_fp8_scale():
    """|SiLU(x)| <= max(|x|, 0.28): SiLU lies below x for x > 0, and its negative branch has
    its minimum near x = -1.2785 at about -0.2785 (so the 0.28 floor is nearly reached)."""
    x = torch.linspace(-40.0, 40.0, 400001, dtype=F64)
    y = oracle.silu(x)
    assert bool((y.abs() <= torch.clamp(x.abs(), min=0.28)).all())
    assert -0.2786 < float(y.min()) < -0.2784
    assert abs(float(x[int(y.argmin())]) + 1.2785) < 1e-3


def test_gated_fp8_scales_never_overflow():
    """The gated FP8 MLP's hidden scale covers SiLU(gate) * up for any input: adversarial
    one-hot rows that put all of u into the coordinate with the largest gain, and random
    rows, stay within the e4m3 range after scaling; the FP8 gated MLP differs from the exact
    one by FP8-sized amounts."""
    from oracle.flashdecoder import linear
    cfg = synth.PRESETS["tiny_gated_fp8"]
    w = {k: torch.from_numpy(v).to(torch.float64) for k, v in synth.make_weights(cfg).items()}
    D = cfg.hidden
    g2, b1 = w["blocks.0.norm2.g"], w["blocks.0.mlp1.b"]
    w1 = oracle.fp8_weight(w["blocks.0.mlp1.w"])
    s_u, s_h = oracle.fp8_mlp_scales(g2, w1, b1, gated=True)
    h = torch.randn(64, D, dtype=torch.float64) * 3
    for r, i in enumerate(g2.abs().argsort(descending=True)[:8].tolist()):
        h[r] = 0.0
        h[r, i] = (-1.0) ** r * 5.0
    u = oracle.rms_norm(h, g2, 0.0)
    assert float((u / s_u).abs().max()) <= 448.0
    z = linear(oracle.e4m3(u / s_u) * s_u, w1, b1)
    dm = z.shape[1] // 2
    a = oracle.silu(z[:, :dm]) * z[:, dm:]
    assert float((a / s_h).abs().max()) <= 448.0
    w2 = w["blocks.0.mlp2.w"]
    zx = linear(u, w["blocks.0.mlp1.w"], b1)
    exact = linear(oracle.silu(zx[:, :dm]) * zx[:, dm:], w2, None)
    q = linear(oracle.e4m3(a / s_h) * s_h, oracle.fp8_weight(w2), None)
    rel = float((q - exact).norm() / exact.norm())
    assert 1e-3 < rel < 0.2, rel


def test_linear_is_x_wt_plus_b():
    x, w, b = rnd(5, 7, seed=3), rnd(4, 7, seed=4), rnd(4, seed=5)
    brute = torch.tensor([[sum(x[i, k] * w[j, k] for k in range(7)) + b[j] for j in range(4)]
                          for i in range(5)], dtype=F64)
    assert torch.allclose(oracle.linear(x, w, b), brute, atol=1e-12)


def test_pixel_unshuffle_matches_library_and_index_formula():
    C, H, W, p = 3, 6, 8, 2
    z = rnd(C, H, W, seed=6)
    tok = oracle.pixel_unshuffle(z, p)                       # [L][C p^2]
    lib = tF.pixel_unshuffle(z[None], p)[0]                   # [C p^2][H/p][W/p]
    assert torch.equal(tok, lib.reshape(C * p * p, -1).T)
    for l in range((H // p) * (W // p)):
        h, w_ = divmod(l, W // p)
        for c in range(C):
            for i in range(p):
                for j in range(p):
                    assert tok[l, c * p * p + i * p + j] == z[c, h * p + i, w_ * p + j]


def test_pixel_shuffle_matches_library_and_inverts_unshuffle():
    frames, gh, gw, C, rs = 2, 3, 4, 3, 4
    L = gh * gw
    F = rnd(frames * L, C * rs * rs, seed=7)
    pix = oracle.pixel_shuffle(F, frames, gh, gw, C, rs)
    assert pix.shape == (C, frames, gh * rs, gw * rs)
    for tau in range(frames):
        lib = tF.pixel_shuffle(F[tau * L:(tau + 1) * L].T.reshape(1, C * rs * rs, gh, gw), rs)[0]
        assert torch.equal(pix[:, tau], lib)
        # PixelShuffle o PixelUnshuffle = identity on one frame
        assert torch.equal(oracle.pixel_unshuffle(pix[:, tau], rs), F[tau * L:(tau + 1) * L])
    # one element by the index formula
    c, tau, h, i, w_, j = 2, 1, 2, 3, 1, 0
    assert pix[c, tau, h * rs + i, w_ * rs + j] == F[tau * L + h * gw + w_, c * rs * rs + i * rs + j]


# ---------------------------------------------------------------- 3D-RoPE
def test_rope_bands_at_head_dim_64():
    assert oracle.rope_bands(64) == [(0, 24), (24, 20), (44, 20)]


def test_rope_matches_complex_rotation_and_is_relative():
    dh, L, base = 64, 9, 10000.0
    x = rnd(2, L, dh, seed=8)
    f = torch.arange(L, dtype=F64) * 3
    y = torch.arange(L, dtype=F64) % 4
    xx = torch.arange(L, dtype=F64) // 2
    r = oracle.rope(x, f, y, xx, base)
    # complex form: (x_2i + i x_2i+1) * exp(i pos theta_i), band by band
    for (off, d), pos in zip(oracle.rope_bands(dh), (f, y, xx)):
        th = torch.tensor([base ** (-2.0 * k / d) for k in range(d // 2)], dtype=F64)
        zc = torch.complex(x[..., off:off + d:2], x[..., off + 1:off + d:2])
        rot = zc * torch.exp(1j * pos[:, None] * th[None, :])
        assert torch.allclose(r[..., off:off + d:2], rot.real, atol=1e-12)
        assert torch.allclose(r[..., off + 1:off + d:2], rot.imag, atol=1e-12)
    # rotations keep norms; zero position is the identity
    assert torch.allclose(r.norm(dim=-1), x.norm(dim=-1), atol=1e-12)
    z0 = torch.zeros(L, dtype=F64)
    assert torch.allclose(oracle.rope(x, z0, z0, z0, base), x)
    # <R_a q, R_b k> depends on a - b only, on every axis
    q, k = rnd(1, 1, dh, seed=9), rnd(1, 1, dh, seed=10)
    def dot(a, b):
        pa = [torch.tensor([v], dtype=F64) for v in a]
        pb = [torch.tensor([v], dtype=F64) for v in b]
        return (oracle.rope(q, *pa, base) * oracle.rope(k, *pb, base)).sum().item()
    assert dot((5, 2, 7), (3, 1, 4)) == pytest.approx(dot((12, 4, 9), (10, 3, 6)), abs=1e-10)
    assert dot((5, 2, 7), (3, 1, 4)) != pytest.approx(dot((5, 2, 7), (4, 1, 4)), abs=1e-6)


# ---------------------------------------------------------------- attention
def test_attention_brute_force_gqa():
    """Naive softmax attention with explicit exp / sum loops, tiny Lq x Lk, 4 heads on 2
    KV groups."""
    N, G, Lq, Lk, dh = 4, 2, 5, 13, 8
    q, k, v = rnd(N, Lq, dh, seed=11), rnd(G, Lk, dh, seed=12), rnd(G, Lk, dh, seed=13)
    out = oracle.attention(q, k, v)
    for n in range(N):
        g = n // (N // G)
        for i in range(Lq):
            s = [sum(q[n, i, d].item() * k[g, j, d].item() for d in range(dh)) / math.sqrt(dh)
                 for j in range(Lk)]
            e = [math.exp(x) for x in s]
            tot = sum(e)
            for d in range(dh):
                o = sum(e[j] * v[g, j, d].item() for j in range(Lk)) / tot
                assert out[n, i, d].item() == pytest.approx(o, rel=1e-10, abs=1e-12)


def test_attention_matches_library_sdpa_and_gqa_special_cases():
    N, G, Lq, Lk, dh = 6, 3, 17, 40, 16
    q, k, v = rnd(N, Lq, dh, seed=14), rnd(G, Lk, dh, seed=15), rnd(G, Lk, dh, seed=16)
    ref = tF.scaled_dot_product_attention(q, k.repeat_interleave(N // G, 0),
                                          v.repeat_interleave(N // G, 0))
    assert torch.allclose(oracle.attention(q, k, v), ref, atol=1e-12)
    # G = N is MHA: duplicating each KV head N/G times and using G' = N changes nothing
    kd, vd = k.repeat_interleave(N // G, 0), v.repeat_interleave(N // G, 0)
    assert torch.allclose(oracle.attention(q, kd, vd), oracle.attention(q, k, v), atol=1e-12)
    # G = 1 is MQA: every head reads the single group
    o1 = oracle.attention(q, k[:1], v[:1])
    for n in range(N):
        assert torch.allclose(o1[n], oracle.attention(q[n:n + 1], k[:1], v[:1])[0], atol=1e-12)
    # row blocking does not change the result
    assert torch.allclose(oracle.attention(q, k, v, rows=3), oracle.attention(q, k, v), atol=1e-13)
    # a mask equals dropping the masked keys
    allowed = torch.zeros(Lq, Lk, dtype=torch.bool)
    allowed[:, 10:30] = True
    assert torch.allclose(oracle.attention(q, k, v, allowed),
                          oracle.attention(q, k[:, 10:30], v[:, 10:30]), atol=1e-12)


# ---------------------------------------------------------------- pixel quantisation
def test_quantize_u8_special_values():
    x = np.array([-1.0, 1.0, 0.0, -2.0, 3.0, np.nan, np.inf, -np.inf,
                  -1.0 + 1 / 255, 0.5 / 127.5 - 1.0, 1.5 / 127.5 - 1.0], dtype=np.float32)
    q = oracle.quantize_u8(x)
    # (x+1)*127.5: -1 -> 0, 1 -> 255, 0 -> 127.5 -> 128 (ties to even), NaN -> 0
    assert list(q[:8]) == [0, 255, 128, 0, 255, 0, 255, 0]
    assert q[8] == 0 or q[8] == 1
    # exact .5 ties go to even codes (the fp32 products land on 0.5 / 1.5 or next to them)
    a = (np.float32(x[9]) + np.float32(1)).astype(np.float32) * np.float32(127.5)
    assert q[9] == np.rint(np.float32(a))
    every = np.arange(256, dtype=np.float32) / np.float32(127.5) - np.float32(1)
    assert np.all(np.abs(oracle.quantize_u8(every).astype(int) - np.arange(256)) <= 1)


# ---------------------------------------------------------------- streaming decode invariants
def _setup(name, **kw):
    cfg = synth.PRESETS[name].replace(**kw)
    return cfg, synth.make_weights(cfg), synth.make_latents(cfg)


def test_fig2_visibility_golden():
    """Fig. 2(a): at W=2, z0 alone, z1 sees [z0, z1], z2 sees [z1, z2]."""
    rows = {}
    with open(os.path.join(GOLDEN, "fig2_visibility.txt")) as fh:
        for line in fh:
            line = line.split("#")[0].strip()
            if line.startswith("window"):
                W = int(line.split()[1])
            elif line:
                a, b = line.split(":")
                rows[int(a)] = [int(x) for x in b.split()]
    m = oracle.chunk_mask(torch.arange(3), W)
    for i, seen in rows.items():
        assert [j for j in range(3) if m[i, j]] == seen
    # the streaming cache holds exactly those chunks after each step
    cfg, w, z = _setup("tiny", window=W, chunks=3, n_blocks=1)
    dec = oracle.StreamingDecoder(cfg, w)
    keys_of_chunk = []
    for t in range(3):
        dec.decode_chunk(z[t])
        K = dec.kB[0]
        keys_of_chunk.append(K[:, -cfg.tokens:].clone())
        want = rows[t]
        assert K.shape[1] == len(want) * cfg.tokens
        for slot, c in enumerate(want):
            assert torch.equal(K[:, slot * cfg.tokens:(slot + 1) * cfg.tokens], keys_of_chunk[c])


@pytest.mark.parametrize("name", ["tiny", "tiny_rt", "small", "small_u8", "tiny_qk", "tiny_gated",
                                  "small_fp8", "tiny_gated_fp8"])
def test_streaming_equals_masked_full_sequence(name):
    """Sec. 3.3: sequential decoding with the rolling cache equals one pass under the block
    sliding-window mask (the paper's training-inference consistency)."""
    cfg, w, z = _setup(name)
    a = oracle.decode_stream(cfg, w, z)
    b = oracle.decode_full_masked(cfg, w, z)
    for x, y in zip(a, b):
        assert torch.allclose(x, y, atol=1e-12)


def test_causality_later_chunks_do_not_matter():
    cfg, w, z = _setup("small")
    base = oracle.decode_stream(cfg, w, z)
    z2 = z.copy()
    z2[3:] = synth.make_latents(cfg, seed=77)[3:]
    pert = oracle.decode_stream(cfg, w, z2)
    for t in range(3):
        assert torch.equal(base[t], pert[t])
    assert not torch.allclose(base[3], pert[3])
    # same for the masked full-sequence pass
    fb = oracle.decode_full_masked(cfg, w, z2)
    for t in range(3):
        assert torch.allclose(fb[t], base[t], atol=1e-12)


def test_eviction_one_block():
    """One block, no refinement: chunk t's output ignores chunks <= t - W (evicted, Fig. 2a);
    with two blocks the receptive field grows and it does change."""
    W = 2
    cfg, w, z = _setup("tiny", window=W, chunks=4, n_blocks=1)
    z2 = z.copy()
    z2[0] = -z[0] + 0.5
    a, b = oracle.decode_stream(cfg, w, z), oracle.decode_stream(cfg, w, z2)
    assert torch.allclose(a[2], b[2], atol=1e-13) and torch.allclose(a[3], b[3], atol=1e-13)
    assert not torch.allclose(a[1], b[1])
    cfg2 = cfg.replace(n_blocks=2)
    w2 = synth.make_weights(cfg2)
    a, b = oracle.decode_stream(cfg2, w2, z), oracle.decode_stream(cfg2, w2, z2)
    assert not torch.allclose(a[2], b[2])       # reaches chunk 0 through block 1's cache
    assert torch.allclose(a[3], b[3], atol=1e-13)


def test_window_of_one_chunk_decodes_each_chunk_alone():
    """Degenerate window W = 1: every layer attends to the current chunk only, and RoPE scores
    depend only on position differences (Sec. 3.2), so chunk t decodes exactly as if it were
    chunk 0 of a new stream, whatever came before."""
    cfg, w, z = _setup("tiny_w1")
    stream = oracle.decode_stream(cfg, w, z)
    for t in range(cfg.chunks):
        alone = oracle.decode_stream(cfg, w, z[t:t + 1])[0]
        assert torch.allclose(stream[t], alone, atol=1e-12)
    assert not torch.allclose(stream[0], stream[1])   # the chunks themselves differ


@pytest.mark.parametrize("name", ["tiny_rt", "small"])
def test_window_relative_rope_equals_absolute(name):
    """Sec. 4.3: RoPE positions relative to the window give the same scores."""
    cfg, w, z = _setup(name)
    a = oracle.decode_stream(cfg, w, z, rope_mode="abs")
    b = oracle.decode_stream(cfg, w, z, rope_mode="window")
    for x, y in zip(a, b):
        assert torch.allclose(x, y, atol=1e-10)


def test_identity_blocks_reduce_to_closed_form():
    """With zero out-projections and zero second MLP layers every block is the identity, and
    the decoder reduces to head(upsample(RMS(embed(z)))) written with plain numpy."""
    cfg, w, z = _setup("small", chunks=2)
    for k in list(w):
        if k.endswith(("out.w", "out.b", "mlp2.w", "mlp2.b")):
            w[k] = np.zeros_like(w[k])
    got = oracle.decode_stream(cfg, w, z)
    L, D, rt, rs, p = cfg.tokens, cfg.hidden, cfg.r_t, cfg.r_s, cfg.patch
    ww = {k: v.astype(np.float64) for k, v in w.items()}
    erf = np.vectorize(math.erf)
    for t in range(2):
        x0 = np.zeros((L, cfg.c_in))
        for c in range(cfg.latent_channels):
            for yy in range(cfg.latent_h):
                for xx in range(cfg.latent_w):
                    l = (yy // p) * cfg.grid_w + xx // p
                    x0[l, c * p * p + (yy % p) * p + xx % p] = z[t, c, yy, xx]
        h = x0 @ ww["embed.w"].T + ww["embed.b"]
        def rms(a, g):
            return a / np.sqrt((a ** 2).mean(-1, keepdims=True) + cfg.norm_eps) * g
        e = rms(h, ww["normf.g"]) @ ww["tup.w"].T + ww["tup.b"]
        hf = np.concatenate([e[:, tau * D:(tau + 1) * D] for tau in range(rt)])
        y = rms(hf, ww["normh.g"])
        a1 = y @ ww["head1.w"].T + ww["head1.b"]
        F = (0.5 * a1 * (1 + erf(a1 / math.sqrt(2)))) @ ww["head2.w"].T + ww["head2.b"]
        pix = np.zeros((3, rt, cfg.out_h, cfg.out_w))
        for tau in range(rt):
            for l in range(L):
                hh, w_ = divmod(l, cfg.grid_w)
                blk = F[tau * L + l].reshape(3, rs, rs)
                pix[:, tau, hh * rs:(hh + 1) * rs, w_ * rs:(w_ + 1) * rs] = blk
        assert np.allclose(got[t].numpy(), np.clip(pix, -1, 1), atol=1e-12)


def test_output_shapes_follow_compression_factors():
    """8x spatial per latent cell, r_t frames per chunk: 480p -> 480x832, 720p -> 720x1280."""
    for name, hw in [("480p", (480, 832)), ("720p", (720, 1280)), ("720p_wide", (720, 1280))]:
        cfg = synth.PRESETS[name]
        assert (cfg.out_h, cfg.out_w) == hw and cfg.r_s == 16 and cfg.head_out == 768
        F = torch.zeros(cfg.r_t * cfg.tokens, cfg.head_out, dtype=F64)
        pix = oracle.pixel_shuffle(F, cfg.r_t, cfg.grid_h, cfg.grid_w, 3, cfg.r_s)
        assert tuple(pix.shape) == (3, 4) + hw
    assert synth.PRESETS["480p"].tokens == 1560 and synth.PRESETS["720p"].tokens == 3600
    cfg, w, z = _setup("tiny")
    assert tuple(oracle.decode_stream(cfg, w, z)[0].shape) == (3, 1, 64, 64)


def test_causal_frame_count_of_fig2():
    """Fig. 2 caption: at r_t = 4, 3 latent frames decode to 9 output frames (1 + r_t (T'-1)).
    With first_chunk_frames = 1 chunk 0 keeps refined frame 0 only; every other output, and
    chunk 0's kept frame, equal the r_t-frames-per-chunk decode of the same stream."""
    cfg, w, z = _setup("small_f1")
    got = oracle.decode_stream(cfg, w, z)
    assert cfg.r_t == 4 and len(got) == 3
    assert sum(p.shape[1] for p in got) == 9
    full = oracle.decode_stream(cfg.replace(first_chunk_frames=0), w, z)
    assert torch.equal(got[0], full[0][:, :1])
    for a, b in zip(got[1:], full[1:]):
        assert torch.equal(a, b)
    masked = oracle.decode_full_masked(cfg, w, z)
    for a, b in zip(got, masked):
        assert a.shape == b.shape and torch.allclose(a, b, atol=1e-12)


def test_kv_cache_size_formula():
    """Eq. kv_cache: G x (W L) x D_h per layer for K and V; refinement r_t W L (Sec. 3.3)."""
    cfg = synth.PRESETS["480p"]
    e = oracle.kv_cache_elems(cfg)
    assert e["backbone_per_layer"] == 2 * 4 * 4 * 1560 * 64
    assert e["refine_per_layer"] == 4 * e["backbone_per_layer"]
    cfg, w, z = _setup("small")
    dec = oracle.StreamingDecoder(cfg, w)
    for t in range(cfg.chunks):
        dec.decode_chunk(z[t])
    assert dec.kB[0].numel() + dec.vB[0].numel() == oracle.kv_cache_elems(cfg)["backbone_per_layer"]
    assert dec.kR[0].numel() + dec.vR[0].numel() == oracle.kv_cache_elems(cfg)["refine_per_layer"]


def test_weights_and_latents_are_seeded_and_bf16_exact():
    cfg = synth.PRESETS["tiny"]
    a, b = synth.make_weights(cfg), synth.make_weights(cfg)
    for k in a:
        assert np.array_equal(a[k], b[k])
        bf = torch.from_numpy(a[k]).to(torch.bfloat16).float().numpy()
        assert np.array_equal(bf, a[k])       # exactly representable in bf16
    z = synth.make_latents(synth.PRESETS["720p_wide"].replace(latent_h=4, latent_w=4), chunks=400)
    c = np.corrcoef(z[:-1].ravel(), z[1:].ravel())[0, 1]
    assert abs(c - 0.9) < 0.02                  # AR(1), rho = 0.9


def test_uniform_attention_decode_closed_form():
    """With the query projection zeroed every score is 0, so attention averages the values of
    the cached window: head n returns the mean over the window's keys of group n // (N/G)'s
    normalised V (KV-norm, Sec. 3.2). The whole stream (cache windows, out-projection,
    residuals, MLPs, temporal upsampling, refinement, head) is then written here with plain
    numpy and compared with the oracle."""
    cfg, w, z = _setup("tiny_rt", chunks=3)
    N, G, dh, D, L, rt = cfg.heads, cfg.kv_groups, 64, cfg.hidden, cfg.tokens, cfg.r_t
    hpg = N // G
    for k in list(w):
        if k.endswith("qkv.w") or k.endswith("qkv.b"):
            w[k] = w[k].copy()
            w[k][:N * dh] = 0.0                        # Q = 0 (and RoPE of 0 is 0)
    got = oracle.decode_stream(cfg, w, z)
    ww = {k: v.astype(np.float64) for k, v in w.items()}
    erf = np.vectorize(math.erf)
    eps = cfg.norm_eps

    def rms(a, g):
        return a / np.sqrt((a ** 2).mean(-1, keepdims=True) + eps) * g

    def gelu(a):
        return 0.5 * a * (1 + erf(a / math.sqrt(2)))

    def stack(h, prefix, n, cache, t, per_chunk):
        for b in range(n):
            p = f"{prefix}.{b}."
            qkv = rms(h, ww[p + "norm1.g"]) @ ww[p + "qkv.w"].T + ww[p + "qkv.b"]
            v = qkv[:, (N + G) * dh:].reshape(-1, G, dh)
            v = rms(v, ww[p + "vnorm.g"])                                 # [rows][G][64]
            cache.setdefault(p, []).append(v)
            window = np.concatenate(cache[p][max(0, t - cfg.window + 1):t + 1])
            mean_v = window.mean(axis=0)                                  # [G][64]
            o = np.concatenate([mean_v[n_ // hpg] for n_ in range(N)])    # [N * 64]
            h = h + o @ ww[p + "out.w"].T + ww[p + "out.b"]
            u2 = rms(h, ww[p + "norm2.g"])
            h = h + gelu(u2 @ ww[p + "mlp1.w"].T + ww[p + "mlp1.b"]) @ ww[p + "mlp2.w"].T + ww[p + "mlp2.b"]
        return h

    cache = {}
    for t in range(cfg.chunks):
        x0 = oracle.pixel_unshuffle(torch.from_numpy(z[t]).double(), cfg.patch).numpy()
        h = x0 @ ww["embed.w"].T + ww["embed.b"]
        h = stack(h, "blocks", cfg.n_blocks, cache, t, L)
        e = rms(h, ww["normf.g"]) @ ww["tup.w"].T + ww["tup.b"]
        hf = np.concatenate([e[:, tau * D:(tau + 1) * D] for tau in range(rt)])
        hf = stack(hf, "refine", cfg.n_refine, cache, t, rt * L)
        F = gelu(rms(hf, ww["normh.g"]) @ ww["head1.w"].T + ww["head1.b"]) @ ww["head2.w"].T + ww["head2.b"]
        pix = oracle.pixel_shuffle(torch.from_numpy(F), rt, cfg.grid_h, cfg.grid_w,
                                   cfg.out_channels, cfg.r_s).numpy()
        assert np.allclose(got[t].numpy(), np.clip(pix, -1, 1), atol=1e-12), t
