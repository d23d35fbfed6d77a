"""Per-kernel parity of the CUDA path against the oracle's functions (through the C ABI's
kernel-level entry points), on identical bf16-exact inputs."""
import math

import numpy as np
import pytest
import torch

import oracle
from helpers import assert_close_scaled, bf16_values, dev, f64, randn

pytestmark = pytest.mark.gpu

fdp = pytest.importorskip("paper_2607_14898_gb300.flashdec")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    fdp.lib()


def err_word():
    return torch.zeros(1, dtype=torch.int32, device="cuda")


def check_err(err):
    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"kernel reported error bits {int(err.item())}"


def linear_case(M, N, K, seed):
    A = bf16_values(randn((M, K), seed, 1.0))
    W = bf16_values(randn((N, K), seed + 1, 1.0 / math.sqrt(K)))
    b = randn((N,), seed + 2, 0.1)
    return A, W, b


# ------------------------------------------------------------------ tcgen05 GEMM
@pytest.mark.parametrize("M,N,K,bn", [
    (130, 256, 256, 128),     # ragged M (2 tiles), one K tile of 4 x 64
    (520, 768, 1024, 192),    # 192-wide tiles
    (64, 192, 16, 64),        # K < 64 (tiny patch-embed), zero-filled K tail
    (520, 1024, 256, 256),    # 256-wide tiles
    (1560, 1536, 1024, 128),  # 480p QKV shape: 13 x 12 tiles, persistent (> 1 tile per CTA)
    (1560, 1024, 4096, 0),    # 480p MLP-down shape, library tile choice (96-wide tiles)
    (1560, 1024, 1024, 96),   # 480p out-projection shape: 13 x 11 tiles of 96, ragged N
    (300, 608, 512, 96),      # ragged M and N with 96-wide tiles
    (6240, 768, 1024, 0),     # 480p head layer 2 on r_t L tokens
    (200, 256, 192, 128),     # odd number of K blocks: the last two-block stage is half past K
    (130, 320, 128, 64),      # exactly one two-block stage
])
def test_linear_f32(M, N, K, bn):
    A, W, b = linear_case(M, N, K, seed=M + N + K)
    out = torch.zeros(M, N, device="cuda")
    err = err_word()
    fdp.op_linear(fdp.EPI_F32, dev(A, torch.bfloat16), dev(W, torch.bfloat16), dev(b), out,
                  bn=bn, err=err)
    check_err(err)
    want = oracle.linear(f64(A), f64(W), f64(b))
    assert_close_scaled(out, want, 2e-5, "linear f32")


@pytest.mark.parametrize("M,N,K,bn", [
    (1560, 4096, 1024, 256),  # 480p MLP layer 1 shape: 7 pair tiles of 256 rows, ragged last
    (1560, 1024, 4096, 128),  # 480p MLP layer 2 shape, long K
    (300, 608, 512, 96),      # ragged M and N; the second CTA of the last pair has no rows
    (6240, 1536, 1024, 192),  # refinement QKV shape, several tiles per pair (persistent)
    (130, 256, 64, 128),      # one K block
    (520, 512, 320, 256),     # odd number of K blocks on pairs
])
def test_linear_cta_pairs(M, N, K, bn):
    """256-row tiles on CTA pairs (tcgen05 cta_group::2; each CTA holds half of W) compute the
    same products as single CTAs: fp32, residual and GELU epilogues against the oracle, and
    bit-identical to the single-CTA launch of the same width."""
    A, W, b = linear_case(M, N, K, seed=M + 5 * N + K)
    Ad, Wd, bd = dev(A, torch.bfloat16), dev(W, torch.bfloat16), dev(b)
    err = err_word()
    out = {}
    for pair in (1, 2):
        o = torch.zeros(M, N, device="cuda")
        fdp.op_linear(fdp.EPI_F32, Ad, Wd, bd, o, bn=bn, err=err, pair=pair)
        check_err(err)
        out[pair] = o
    want = oracle.linear(f64(A), f64(W), f64(b))
    assert_close_scaled(out[2], want, 2e-5, f"pair linear f32 bn={bn}")
    assert torch.equal(out[1], out[2])
    h = torch.ones(M, N, device="cuda")
    fdp.op_linear(fdp.EPI_RESID, Ad, Wd, bd, h, bn=bn, err=err, pair=2)
    check_err(err)
    assert torch.equal(h, out[1] + 1.0)
    if bn % 64 == 0:
        g1 = torch.zeros(M, N, dtype=torch.bfloat16, device="cuda")
        g2 = torch.zeros(M, N, dtype=torch.bfloat16, device="cuda")
        fdp.op_linear(fdp.EPI_GELU, Ad, Wd, bd, g1, bn=bn, err=err, pair=1)
        fdp.op_linear(fdp.EPI_GELU, Ad, Wd, bd, g2, bn=bn, err=err, pair=2)
        check_err(err)
        assert torch.equal(g1, g2)


@pytest.mark.parametrize("frames_in,frames,gh,gw,C,rs,u8", [
    (4, 4, 30, 52, 3, 16, False),  # 480p refinement rows -> 4 fp32 frames
    (4, 4, 45, 80, 3, 16, True),   # 720p, uint8 codes
    (4, 1, 6, 7, 3, 16, False),    # first chunk of a one-frame-first stream: frame 0 only
    (2, 2, 9, 11, 3, 8, True),     # rs 8 (four pixel rows per 32 columns), ragged tiles
])
def test_linear_pixel_equals_linear_then_pixel_head(frames_in, frames, gh, gw, C, rs, u8):
    """The pixel shuffle folded into head layer 2's epilogue gives the bits of the two-launch
    path (fd_op_linear's F, then fd_op_pixel_head), fp32 and uint8, including outputs past the
    clamp (the inputs are scaled so that some pre-activations leave [-1, 1])."""
    L = gh * gw
    M, K, N = frames_in * L, 256, C * rs * rs
    A, W, b = linear_case(M, N, K, seed=M + N)
    Ad, Wd, bd = dev(A, torch.bfloat16), dev(W * 3.0, torch.bfloat16), dev(b)
    err = err_word()
    F = torch.zeros(M, N, device="cuda")
    fdp.op_linear(fdp.EPI_F32, Ad, Wd, bd, F, err=err, bn=256)
    shape = (C, frames, gh * rs, gw * rs)
    dtype = torch.uint8 if u8 else torch.float32
    want = torch.zeros(shape, dtype=dtype, device="cuda")
    code = 2 if u8 else 0  # FD_DTYPE_U8 / FD_DTYPE_F32
    fdp.op_pixel_head(F, frames, gh, gw, C, rs, code, want)
    got = torch.full(shape, 7, dtype=dtype, device="cuda")
    fdp.op_linear_pixel(Ad, Wd, bd, frames, gh, gw, C, rs, code, got, err=err)
    check_err(err)
    assert float((F.abs() > 1).float().mean()) > 0.01  # the clamp is exercised
    assert torch.equal(got, want)


def test_gelu_epilogue_is_the_exact_erf_gelu_at_bf16():
    """The GELU epilogue evaluates erf with Abramowitz & Stegun 7.1.26 (error <= 1.5e-7): on a
    grid of pre-activations from -8 to 8 (A holds x in one column, W picks it, the bias shifts
    it) every bf16 output is within one bf16 step of bf16(GELU(z)) computed in fp64 with the
    exact erf (or, in the far negative tail, within 1e-6 of the exact value), and at least 99 %
    of the outputs above 1e-3 in magnitude are equal to it (the rest are round-to-nearest
    ties decided by the last fp32 bits)."""
    M, N, K = 512, 64, 64
    x = bf16_values(np.linspace(-8.0, 8.0, M).astype(np.float32))
    A = np.zeros((M, K), np.float32)
    A[:, 0] = x
    W = np.zeros((N, K), np.float32)
    W[:, 0] = 1.0
    b = ((np.arange(N) - 32) / 32.0).astype(np.float32)
    out = torch.zeros(M, N, dtype=torch.bfloat16, device="cuda")
    err = err_word()
    fdp.op_linear(fdp.EPI_GELU, dev(A, torch.bfloat16), dev(W, torch.bfloat16), dev(b), out,
                  err=err)
    check_err(err)
    z = f64(x)[:, None] + f64(b)[None, :]
    exact = oracle.gelu(z)
    want = exact.to(torch.bfloat16)
    got = out.cpu()
    big = exact.abs() > 1e-3
    steps = (got.view(torch.int16).int() - want.view(torch.int16).int()).abs()
    assert int(steps[big].max()) <= 1
    assert float((steps[big] == 0).double().mean()) >= 0.99
    assert bool(((steps <= 1) | ((f64(got) - exact).abs() <= 1e-6)).all())


@pytest.mark.parametrize("M,Dm,K,bn", [
    (520, 512, 256, 0),     # ragged M, library tile choice
    (130, 256, 1024, 128),  # 128-wide tiles: one 64-wide output slab per tile
    (300, 576, 512, 256),   # 256-wide tiles; the last tile holds only 128 gate / up columns
])
def test_linear_swiglu(M, Dm, K, bn):
    """Gated MLP layer 1 of the XL layout: out = SiLU(A Wg^T + bg) * (A Wu^T + bu), with the
    gate and up rows interleaved in blocks of 32 as the epilogue expects."""
    A = bf16_values(randn((M, K), M + K, 1.0))
    Wg = bf16_values(randn((Dm, K), M + 1, 1.0 / math.sqrt(K)))
    Wu = bf16_values(randn((Dm, K), M + 2, 1.0 / math.sqrt(K)))
    bg, bu = randn((Dm,), M + 3, 0.1), randn((Dm,), M + 4, 0.1)
    blocks = lambda g, u: np.concatenate(
        [np.concatenate([g[32 * j:32 * j + 32], u[32 * j:32 * j + 32]]) for j in range(Dm // 32)])
    W, b = blocks(Wg, Wu), blocks(bg, bu)
    out = torch.zeros(M, Dm, dtype=torch.bfloat16, device="cuda")
    err = err_word()
    fdp.op_linear(fdp.EPI_SWIGLU, dev(A, torch.bfloat16), dev(W, torch.bfloat16), dev(b), out,
                  bn=bn, err=err)
    check_err(err)
    want = oracle.silu(oracle.linear(f64(A), f64(Wg), f64(bg))) * \
        oracle.linear(f64(A), f64(Wu), f64(bu))
    assert_close_scaled(out.float(), want, 8e-3, "swiglu")


def e4m3_codes(x):
    """fp64 values -> (e4m3 codes as uint8, the values they stand for)."""
    q = torch.as_tensor(x, dtype=torch.float64).to(torch.float8_e4m3fn)
    return q.view(torch.uint8), q.to(torch.float64)


def assert_e4m3_close(got_codes, want_values, what):
    """e4m3 outputs computed in fp32 (GPU) vs fp64 (oracle): equal codes except where the exact
    value sits at a rounding boundary, and then one step apart (relative 2^-3, or one
    subnormal step)."""
    got = got_codes.cpu().view(torch.float8_e4m3fn).to(torch.float64)
    want = want_values.to(torch.float8_e4m3fn).to(torch.float64)
    diff = (got - want).abs()
    assert float((diff > 0).double().mean()) < 0.01, f"{what}: too many codes differ"
    assert bool((diff <= 2.0 ** -3 * want.abs() + 2.0 ** -9).all()), f"{what}: more than a step"


@pytest.mark.parametrize("M,N,K,bn", [
    (520, 1024, 256, 0),     # ragged M, library tile choice
    (1560, 1024, 4096, 96),  # 480p MLP-down shape, 96-wide tiles, 32 K-blocks of 128
    (300, 640, 208, 128),    # K not a multiple of 128: zero-filled K tail
    (260, 512, 384, 128),    # odd number of 128-element K blocks (two per stage)
])
def test_linear_e4m3_fp32_epilogues(M, N, K, bn):
    """FP8 MLP products (Sec. 4.6): e4m3 operands make every product exact, so the fp32 and
    residual epilogues match the oracle's dequantised matrix product to fp32 accumulation."""
    torch.manual_seed(M + N + K)
    a_c, a = e4m3_codes(torch.randn(M, K, dtype=torch.float64) * 3)
    w_c, wv = e4m3_codes(torch.randn(N, K, dtype=torch.float64) * 40)
    cs = torch.tensor([2.0 ** -int(e) for e in torch.randint(4, 12, (N,))], dtype=torch.float32)
    b = torch.randn(N, dtype=torch.float32) * 0.1
    want = oracle.linear(a, wv, None) * cs.double() + b.double()
    err = err_word()
    out = torch.zeros(M, N, device="cuda")
    fdp.op_linear_e4m3(fdp.EPI_F32, a_c.cuda(), w_c.cuda(), cs.cuda(), b.cuda(), out, bn=bn,
                       err=err)
    check_err(err)
    assert_close_scaled(out, want, 2e-5, "e4m3 linear f32")
    h0 = torch.randn(M, N, dtype=torch.float32)
    h = h0.cuda()
    fdp.op_linear_e4m3(fdp.EPI_RESID, a_c.cuda(), w_c.cuda(), cs.cuda(), b.cuda(), h, bn=bn,
                       err=err)
    check_err(err)
    assert_close_scaled(h, h0.double() + want, 2e-5, "e4m3 linear residual")


def test_linear_e4m3_gelu_to_e4m3_and_rmsnorm_e4m3():
    """The two FP8 producers of the MLP: GELU epilogue to e4m3 (layer 1 output) and RMSNorm to
    e4m3 (layer 1 input), each against the oracle's rounding of the same formula."""
    M, N, K = 520, 1024, 512
    torch.manual_seed(5)
    a_c, a = e4m3_codes(torch.randn(M, K, dtype=torch.float64) * 2)
    w_c, wv = e4m3_codes(torch.randn(N, K, dtype=torch.float64) * 30)
    cs = torch.full((N,), 2.0 ** -10, dtype=torch.float32)
    b = torch.randn(N, dtype=torch.float32) * 0.1
    z = oracle.linear(a, wv, None) * cs.double() + b.double()
    for bn in (128, 256):
        out = torch.zeros(M, N, dtype=torch.uint8, device="cuda")
        err = err_word()
        fdp.op_linear_e4m3(fdp.EPI_GELU, a_c.cuda(), w_c.cuda(), cs.cuda(), b.cuda(), out,
                           out_scale=32.0, bn=bn, err=err)
        check_err(err)
        assert_e4m3_close(out, oracle.gelu(z) * 32.0, f"gelu e4m3 bn={bn}")
    D = 1024
    h = torch.from_numpy(randn((M, D), 9, 2.0))
    g = torch.from_numpy(bf16_values(1 + randn((D,), 10, 0.1)))
    u = torch.zeros(M, D, dtype=torch.uint8, device="cuda")
    fdp.op_rmsnorm_e4m3(h.cuda(), g.cuda(), 1e-6, 8.0, u)
    torch.cuda.synchronize()
    assert_e4m3_close(u, oracle.rms_norm(h.double(), g.double(), 1e-6) * 8.0, "rmsnorm e4m3")


def test_linear_e4m3_swiglu_to_e4m3():
    """The FP8 gated MLP's layer 1: gate and up rows interleaved in blocks of 32 as for the
    bf16 gated epilogue, out = e4m3(SiLU(g) u out_scale) against the oracle's rounding of the
    same formula; two launches in a row give the same codes."""
    M, Dm, K = 300, 512, 384
    torch.manual_seed(11)
    a_c, a = e4m3_codes(torch.randn(M, K, dtype=torch.float64) * 2)
    wg_c, wg = e4m3_codes(torch.randn(Dm, K, dtype=torch.float64) * 30)
    wu_c, wu = e4m3_codes(torch.randn(Dm, K, dtype=torch.float64) * 30)
    csg = torch.full((Dm,), 2.0 ** -10, dtype=torch.float32)
    csu = torch.full((Dm,), 2.0 ** -11, dtype=torch.float32)
    bg, bu = torch.randn(Dm) * 0.1, torch.randn(Dm) * 0.1
    blocks = lambda g, u: torch.cat([torch.cat([g[32 * j:32 * j + 32], u[32 * j:32 * j + 32]])
                                     for j in range(Dm // 32)])
    W, cs, b = blocks(wg_c, wu_c), blocks(csg, csu), blocks(bg, bu)
    zg = oracle.linear(a, wg, None) * csg.double() + bg.double()
    zu = oracle.linear(a, wu, None) * csu.double() + bu.double()
    want = oracle.silu(zg) * zu * 4.0
    outs = []
    for _ in range(2):
        out = torch.zeros(M, Dm, dtype=torch.uint8, device="cuda")
        err = err_word()
        fdp.op_linear_e4m3(fdp.EPI_SWIGLU, a_c.cuda(), W.contiguous().cuda(), cs.cuda(),
                           b.cuda(), out, out_scale=4.0, err=err)
        check_err(err)
        assert_e4m3_close(out, want, "swiglu e4m3")
        outs.append(out.cpu())
    assert torch.equal(outs[0], outs[1])


def test_linear_resid_gelu_tup():
    M, N, K, D = 520, 1024, 256, 256
    A, W, b = linear_case(M, N, K, seed=11)
    Ad, Wd, bd = dev(A, torch.bfloat16), dev(W, torch.bfloat16), dev(b)
    want = oracle.linear(f64(A), f64(W), f64(b))
    err = err_word()
    # residual: h += A W^T + b
    h0 = randn((M, N), 99)
    h = dev(h0)
    fdp.op_linear(fdp.EPI_RESID, Ad, Wd, bd, h, err=err)
    check_err(err)
    assert_close_scaled(h, f64(h0) + want, 2e-5, "residual")
    # GELU -> bf16
    g = torch.zeros(M, N, dtype=torch.bfloat16, device="cuda")
    fdp.op_linear(fdp.EPI_GELU, Ad, Wd, bd, g, err=err)
    check_err(err)
    assert_close_scaled(g.float(), oracle.gelu(want), 8e-3, "gelu")
    # temporal upsampling reshape: column tau*D + d of row l -> row tau*M + l
    o = torch.zeros(N // D * M, D, device="cuda")
    fdp.op_linear(fdp.EPI_TUP, Ad, Wd, bd, o, tup_hidden=D, err=err)
    check_err(err)
    rt = N // D
    want_t = want.reshape(M, rt, D).transpose(0, 1).reshape(rt * M, D)
    assert_close_scaled(o, want_t, 2e-5, "tup")


# ------------------------------------------------------------------ fused QKV epilogue
class Cfg:
    def __init__(self, **kw):
        self.__dict__.update(kw)


@pytest.mark.parametrize("heads,groups,grid_h,grid_w,fpc,window,t,K,bn,qk", [
    (4, 2, 10, 13, 4, 3, 5, 256, 128, False),    # refinement-like: 4 frames per chunk, ragged
    (16, 4, 30, 52, 1, 4, 7, 1024, 192, False),  # 480p backbone block, 192-wide tiles
    (16, 4, 30, 52, 1, 4, 7, 1024, 256, False),  # same, 256-wide tiles
    (24, 3, 3, 5, 1, 8, 130, 1536, 64, False),   # wide model, long stream (large temporal index)
    (4, 2, 8, 8, 4, 2, 40000, 256, 0, False),    # very long stream: temporal index 160000
    (16, 4, 30, 52, 1, 4, 7, 1024, 192, True),   # QK-norm instead of KV-norm
    (4, 2, 10, 13, 4, 3, 5, 256, 128, True),     # QK-norm, refinement-like
])
def test_qkv_fused(heads, groups, grid_h, grid_w, fpc, window, t, K, bn, qk):
    dh, eps, base = 64, 1e-6, 10000.0
    tokens = grid_h * grid_w
    M = fpc * tokens
    N = (heads + 2 * groups) * dh
    A, W, b = linear_case(M, N, K, seed=heads * 7 + t)
    kg = bf16_values(1 + randn((dh,), 5, 0.1))
    vg = bf16_values(1 + randn((dh,), 6, 0.1))
    pitch = -(-window * M // 128) * 128
    q_out = torch.zeros(M, heads * dh, dtype=torch.bfloat16, device="cuda")
    k_ring = torch.zeros(groups, pitch, dh, dtype=torch.bfloat16, device="cuda")
    vt_ring = torch.zeros(groups, dh, pitch, dtype=torch.float16, device="cuda")
    err = err_word()
    rope_t = torch.zeros(fpc, 12, 2, device="cuda")
    fdp.op_rope_table(t, fpc, base, rope_t)
    fdp.op_qkv(dev(A, torch.bfloat16), dev(W, torch.bfloat16), dev(b), dev(kg), dev(vg), heads,
               groups, tokens, grid_w, fpc, window, t, eps, base, rope_t, q_out, k_ring, vt_ring,
               pitch, bn=bn, err=err, qk_norm=qk)
    check_err(err)
    # oracle: Linear, KV-norm (or QK-norm, vg then Q's gain), 3D-RoPE at (t*fpc + row // tokens,
    # y, x)
    qkv = oracle.linear(f64(A), f64(W), f64(b))
    q = qkv[:, :heads * dh].reshape(M, heads, dh).transpose(0, 1)
    k = qkv[:, heads * dh:(heads + groups) * dh].reshape(M, groups, dh).transpose(0, 1)
    v = qkv[:, (heads + groups) * dh:].reshape(M, groups, dh).transpose(0, 1)
    k = oracle.rms_norm(k, f64(kg), eps)
    if qk:
        q = oracle.rms_norm(q, f64(vg), eps)
    else:
        v = oracle.rms_norm(v, f64(vg), eps)
    r = torch.arange(M)
    pos = ((t * fpc + r // tokens).double(), ((r % tokens) // grid_w).double(),
           ((r % tokens) % grid_w).double())
    q = oracle.rope(q, *pos, base)
    k = oracle.rope(k, *pos, base)
    assert_close_scaled(q_out.float().reshape(M, heads, dh).transpose(0, 1), q, 1e-2, "Q")
    slot = t % window
    kr = k_ring.float()[:, slot * M:(slot + 1) * M]
    vr = vt_ring.float()[:, :, slot * M:(slot + 1) * M].transpose(1, 2)
    assert_close_scaled(kr, k, 1e-2, "K ring slot")
    assert_close_scaled(vr, v, 1e-2, "V ring slot")
    # nothing outside the slot was written
    mask = torch.ones(pitch, dtype=torch.bool)
    mask[slot * M:(slot + 1) * M] = False
    assert float(k_ring.float()[:, mask].abs().max()) == 0.0
    assert float(vt_ring.float()[:, :, mask].abs().max()) == 0.0


# ------------------------------------------------------------------ attention
def attention_case(Lq, heads, groups, pitch, n_keys, seed, qscale=1.5):
    dh = 64
    q = bf16_values(randn((Lq, heads * dh), seed, qscale))
    k = bf16_values(randn((groups, pitch, dh), seed + 1))
    v = randn((groups, pitch, dh), seed + 2).astype(np.float16).astype(np.float32)  # fp16 V
    # entries past n_keys hold large stale values: they must not leak in
    k[:, n_keys:] *= 50
    v[:, n_keys:] *= 50
    return q, k, v


def run_attention(q, k, v, heads, groups, pitch, n_keys, parts=0, runs=1):
    Lq = q.shape[0]
    vt = np.ascontiguousarray(np.transpose(v, (0, 2, 1)))
    ws_bytes = fdp.attention_workspace_bytes(Lq, heads, groups, n_keys, parts)
    # the workspace starts as NaN garbage: the call must clear what it relies on
    ws = torch.full((max(1, ws_bytes // 4),), float("nan"), device="cuda")
    err = err_word()
    outs = []
    for _ in range(runs):
        out = torch.zeros(Lq, heads * 64, dtype=torch.bfloat16, device="cuda")
        fdp.op_attention(dev(q, torch.bfloat16), dev(k, torch.bfloat16), dev(vt, torch.float16),
                         heads, groups, pitch, n_keys, out, parts=parts, workspace=ws, err=err)
        outs.append(out)
    check_err(err)
    return outs[0].float().cpu() if runs == 1 else [o.float().cpu() for o in outs]


# parts = CTAs of the persistent launch: each takes an equal run of the (tile pair, key block)
# units, so runs start and end inside pairs and partial results are combined
@pytest.mark.parametrize("Lq,heads,groups,n_keys,parts", [
    (520, 4, 2, 520, 1),      # one CTA takes every pair: many segments, no partials
    (520, 4, 2, 1300, 1),     # ragged last key block
    (520, 4, 2, 1300, 3),     # runs of ~37 blocks: partial first / last pairs, whole pairs between
    (520, 4, 2, 1300, 25),    # runs of ~4 blocks: each pair cut into 3-4 partials
    (130, 4, 1, 390, 2),      # multi-query (G = 1)
    (128, 4, 4, 128, 1),      # MHA (G = N): one tile per group, second tile of each pair empty
    (128, 4, 4, 128, 7),      # more CTAs than units: some CTAs have nothing to do
    (520, 4, 2, 1300, 200),   # 110 units on 200 CTAs: a pair's parts lie between empty CTAs
    (300, 3, 3, 700, 0),      # N/G = 1 with 3 query tiles: last pair half out of range
    (300, 4, 2, 700, 5),      # Lq % 8 != 0: heads padded to 304 rows in the packed space
    (64, 2, 1, 1, 1),         # a single key
])
def test_attention_small(Lq, heads, groups, n_keys, parts):
    pitch = max(128, -(-n_keys // 128) * 128 + 128)
    q, k, v = attention_case(Lq, heads, groups, pitch, n_keys, seed=Lq + n_keys)
    got = run_attention(q, k, v, heads, groups, pitch, n_keys, parts)
    qh = f64(q).reshape(Lq, heads, 64).transpose(0, 1)
    want = oracle.attention(qh, f64(k)[:, :n_keys], f64(v)[:, :n_keys])
    assert_close_scaled(got.reshape(Lq, heads, 64).transpose(0, 1), want, 1.5e-2, "attention")


@pytest.mark.parametrize("Lq,heads,groups,n_keys", [
    (6240, 16, 4, 24960),    # 480p refinement, steady state (4 chunks x 4 frames x 1560)
    (1560, 16, 4, 6240),     # 480p backbone, steady state
    (3600, 16, 4, 14400),    # 720p backbone, steady state
    (14400, 16, 4, 57600),   # 720p refinement, steady state (4 chunks x 4 frames x 3600)
    (3600, 24, 3, 28800),    # 720p wide model backbone: 8 heads per group, W = 8 chunks
    (14400, 24, 3, 115200),  # 720p wide model refinement: 32 frames of 3600 keys
    (8160, 24, 3, 16320),    # XL layout at 1080p, backbone (W = 2)
    (32640, 24, 3, 65280),   # XL layout at 1080p, refinement: the largest packed row space
])
def test_attention_full_size_sampled(Lq, heads, groups, n_keys):
    """The launch configuration of the decode (one CTA per SM); two launches in a row on one
    workspace give identical bits (the combine order is fixed and the counters are reset)."""
    pitch = -(-n_keys // 128) * 128
    q, k, v = attention_case(Lq, heads, groups, pitch, n_keys, seed=7, qscale=1.0)
    got, again = run_attention(q, k, v, heads, groups, pitch, n_keys, runs=2)
    assert torch.equal(got, again)
    rows = np.random.default_rng(0).choice(Lq, 48, replace=False)
    rows = np.concatenate([rows, [0, Lq - 1]])
    qh = f64(q[rows]).reshape(len(rows), heads, 64).transpose(0, 1)
    want = oracle.attention(qh, f64(k)[:, :n_keys], f64(v)[:, :n_keys])
    assert_close_scaled(got[rows].reshape(len(rows), heads, 64).transpose(0, 1), want, 1.5e-2,
                        "attention sampled rows")


# ------------------------------------------------------------------ cache append (bit-exact)
def test_kv_append_ring_indexing_bit_exact():
    """After appending chunk t, ring slot s holds chunk j with j = s mod W, t-W < j <= t, bit
    for bit equal to the nearest-even rounding of its fp32 K (bf16) and V (fp16)."""
    G, rows, W, dh = 3, 200, 3, 64
    pitch = -(-W * rows // 128) * 128
    k_ring = torch.zeros(G, pitch, dh, dtype=torch.bfloat16, device="cuda")
    vt_ring = torch.zeros(G, dh, pitch, dtype=torch.float16, device="cuda")
    chunks = []
    for t in range(7):
        k = randn((G, rows, dh), 100 + t)
        v = randn((G, rows, dh), 200 + t)
        chunks.append((k, v))
        fdp.op_kv_append(dev(k), dev(v), W, t, pitch, k_ring, vt_ring)
        torch.cuda.synchronize()
        kr = k_ring.view(torch.int16).cpu().numpy()
        vr = vt_ring.view(torch.int16).cpu().numpy()
        for j in range(max(0, t - W + 1), t + 1):
            s = j % W
            kb = torch.from_numpy(chunks[j][0]).to(torch.bfloat16).view(torch.int16).numpy()
            vb = torch.from_numpy(chunks[j][1]).to(torch.float16).view(torch.int16).numpy()
            assert np.array_equal(kr[:, s * rows:(s + 1) * rows], kb), (t, j)
            assert np.array_equal(vr[:, :, s * rows:(s + 1) * rows], vb.transpose(0, 2, 1)), (t, j)
        assert not kr[:, W * rows:].any()   # padding rows never written


# ------------------------------------------------------------------ RMSNorm, unshuffle, head
def test_rmsnorm():
    M, D = 1560, 1024
    h = randn((M, D), 3, 2.0)
    g = bf16_values(1 + randn((D,), 4, 0.02))
    u = torch.zeros(M, D, dtype=torch.bfloat16, device="cuda")
    fdp.op_rmsnorm(dev(h), dev(g), 1e-6, u)
    torch.cuda.synchronize()
    assert_close_scaled(u.float(), oracle.rms_norm(f64(h), f64(g), 1e-6), 8e-3, "rmsnorm")


@pytest.mark.parametrize("C,H,W,p", [(16, 60, 104, 2), (16, 8, 8, 1)])
def test_unshuffle_bit_exact(C, H, W, p):
    z = randn((C, H, W), 8)
    x0 = torch.zeros((H // p) * (W // p), C * p * p, dtype=torch.bfloat16, device="cuda")
    fdp.op_unshuffle(dev(z), p, x0)
    torch.cuda.synchronize()
    want = oracle.pixel_unshuffle(torch.from_numpy(z), p).to(torch.bfloat16)
    assert torch.equal(x0.cpu().view(torch.int16), want.view(torch.int16))


@pytest.mark.parametrize("frames,gh,gw,rs,u8", [(4, 30, 52, 16, False), (4, 45, 80, 16, True),
                                                (1, 8, 8, 8, False), (2, 3, 5, 8, True)])
def test_pixel_head_bit_exact(frames, gh, gw, rs, u8):
    C = 3
    L = gh * gw
    F = randn((frames * L, C * rs * rs), 9, 0.7)
    # exact quantisation ties, the clamp limits, out-of-range values and NaN
    special = np.array([-1.0, 1.0, 0.0, 2.5, -7.0, np.nan, 1 / 255.0 - 1.0,
                        np.float32(0.5) / np.float32(127.5) - 1.0], dtype=np.float32)
    F.reshape(-1)[:special.size] = special
    out = torch.zeros(C, frames, gh * rs, gw * rs, dtype=torch.uint8 if u8 else torch.float32,
                      device="cuda")
    fdp.op_pixel_head(dev(F), frames, gh, gw, C, rs, fdp.DTYPE_U8 if u8 else fdp.DTYPE_F32, out)
    torch.cuda.synchronize()
    pix = oracle.pixel_shuffle(torch.from_numpy(F).double(), frames, gh, gw, C, rs)
    if u8:
        want = oracle.quantize_u8(pix.float().numpy())
        assert np.array_equal(out.cpu().numpy(), want)
    else:
        pf = pix.float().numpy()
        want = np.clip(np.where(np.isnan(pf), -1.0, pf), -1, 1).astype(np.float32)
        assert np.array_equal(out.cpu().numpy(), want)
