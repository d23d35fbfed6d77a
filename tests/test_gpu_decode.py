"""End-to-end parity of fd_decode_chunk (C ABI) with the CPU oracle, chunk by chunk, plus
properties that hold at any size (determinism, causality, cache indexing)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from helpers import dev, f64, pixel_errors

pytestmark = pytest.mark.gpu

fdp = pytest.importorskip("paper_2607_14898_gb300.flashdec")

# Tolerance on pixels in [-1, 1]: bf16 compute with fp32 accumulation against the fp64 oracle.
MAX_ABS, MEAN_ABS = 2e-2, 2e-3
# The XL layout (D = 1536, gated MLP) is outside the configurations that bar was set for: with
# its operands rounded to bf16 / fp16 (oracle.operand_rounding) the fp64 oracle itself moves by
# max-abs 1.6e-2, mean-abs 2.4e-3 on 480p chunk 0 (the L model at 480p: 5.6e-3 / 8.4e-4), so no
# bf16-operand computation of it meets 2e-3. Its bar is derived from that noise.
XL_MAX_ABS, XL_MEAN_ABS = 2e-2, 3e-3


@pytest.fixture(scope="module", autouse=True)
def _setup(torch_threads):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    fdp.lib()


def gpu_stream(cfg, w, z, chunks=None, reset_and_repeat=False):
    chunks = cfg.chunks if chunks is None else chunks
    W = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    dec = fdp.Decoder(cfg, W)
    shape = (cfg.out_channels, cfg.r_t, cfg.out_h, cfg.out_w)
    dt = torch.uint8 if cfg.out_u8 else torch.float32
    runs = []
    for _ in range(2 if reset_and_repeat else 1):
        outs = []
        for t in range(chunks):
            f1 = t == 0 and getattr(cfg, "first_chunk_frames", 0) == 1  # one frame (Fig. 2)
            pix = torch.empty((shape[0], 1) + shape[2:] if f1 else shape, dtype=dt, device="cuda")
            dec.decode_chunk(dev(z[t]), pix)
            outs.append(pix)
        torch.cuda.synchronize()
        assert dec.sync_status() == fdp.FD_OK
        runs.append([p.cpu() for p in outs])
        dec.reset()
    dec.close()
    W.close()
    return runs if reset_and_repeat else runs[0]


def compare(cfg, got, want, what, max_abs=MAX_ABS, mean_abs=MEAN_ABS):
    for t, (g, o) in enumerate(zip(got, want)):
        if cfg.out_u8:
            wc = oracle.quantize_u8(o.float().numpy()).astype(np.int32)
            gc = g.numpy().astype(np.int32)
            d = np.abs(gc - wc)
            print(f"{what} chunk {t}: max code diff {d.max()} mean {d.mean() / 127.5:.3e}")
            assert d.max() <= 3, f"{what} chunk {t}: max code diff {d.max()}"
            assert d.mean() / 127.5 <= mean_abs, f"{what} chunk {t}: mean {d.mean() / 127.5:.2e}"
        else:
            mx, mean = pixel_errors(g, o)
            print(f"{what} chunk {t}: max-abs {mx:.3e} mean-abs {mean:.3e}")
            assert mx <= max_abs and mean <= mean_abs, \
                f"{what} chunk {t}: max-abs {mx:.3e} mean-abs {mean:.3e}"


@pytest.mark.parametrize("name", ["tiny", "tiny_rt", "small", "small_u8", "tiny_gated",
                                  "tiny_qk", "small_fp8", "small_f1", "tiny_gated_fp8",
                                  "tiny_w1"])
def test_decode_matches_oracle(name):
    cfg = synth.PRESETS[name]
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    want = oracle.decode_stream(cfg, w, z)
    got = gpu_stream(cfg, w, z)
    compare(cfg, got, want, name)


def test_decode_deterministic_after_reset():
    cfg = synth.PRESETS["small"]
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    a, b = gpu_stream(cfg, w, z, reset_and_repeat=True)
    for x, y in zip(a, b):
        assert torch.equal(x, y)


def test_reset_orders_a_decode_on_another_stream():
    """fd_reset enqueues its clears on the stream of the handle's last call (A). Stream A is
    held busy by a sleep kernel when the reset is enqueued, and the next chunk is decoded on
    stream B at once: it must still be chunk 0 of a new stream (the decode waits for the reset's
    event), bit for bit the chunk 0 of a fresh decode, and the chunk after it chunk 1."""
    cfg = synth.PRESETS["tiny_rt"]
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    fresh = gpu_stream(cfg, w, z, chunks=2)
    W = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    dec = fdp.Decoder(cfg, W)
    shape = (cfg.out_channels, cfg.r_t, cfg.out_h, cfg.out_w)
    a, b = torch.cuda.Stream(), torch.cuda.Stream()
    for t in range(2):
        dec.decode_chunk(dev(z[t]), torch.empty(shape, device="cuda"), a)
    torch.cuda.synchronize()
    lat = [dev(z[t]) for t in range(2)]
    got = [torch.empty(shape, device="cuda") for _ in range(2)]
    torch.cuda.synchronize()
    with torch.cuda.stream(a):
        torch.cuda._sleep(200_000_000)      # about 0.1 s of stream A
    dec.reset()                             # clears enqueued on A, behind the sleep
    for t in range(2):
        dec.decode_chunk(lat[t], got[t], b)
    torch.cuda.synchronize()
    assert dec.sync_status() == fdp.FD_OK
    assert dec.chunk_index == 2
    for t in range(2):
        assert torch.equal(got[t].cpu(), fresh[t]), t
    dec.close()
    W.close()


def test_decode_chunks_concurrent_streams_match_single_stream_decodes():
    """fd_decode_chunks runs independent streams (one weights object, three handles, seeds s)
    concurrently on forked streams; each stream's pixels are bit-identical to decoding it alone
    with fd_decode_chunk, chunk after chunk, and the caller's stream sees all of them."""
    cfg = synth.PRESETS["small"]
    w = synth.make_weights(cfg)
    zs = [synth.make_latents(cfg, seed=s) for s in range(3)]
    alone = [gpu_stream(cfg, w, z) for z in zs]
    W = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    decs = [fdp.Decoder(cfg, W) for _ in zs]
    stream = torch.cuda.Stream()
    shape = (cfg.out_channels, cfg.r_t, cfg.out_h, cfg.out_w)
    got = [[] for _ in zs]
    with torch.cuda.stream(stream):
        for t in range(cfg.chunks):
            lat = [dev(z[t]) for z in zs]
            pix = [torch.empty(shape, device="cuda") for _ in zs]
            fdp.decode_chunks(decs, lat, pix, stream)
            copies = [p.to("cpu", non_blocking=False) for p in pix]  # ordered on `stream`
            for s, c in enumerate(copies):
                got[s].append(c)
    torch.cuda.synchronize()
    for d in decs:
        assert d.sync_status() == fdp.FD_OK
        d.close()
    W.close()
    for s in range(len(zs)):
        for t in range(cfg.chunks):
            assert torch.equal(got[s][t], alone[s][t]), (s, t)


def test_state_save_load_resumes_the_stream_bit_exactly():
    """Checkpoint / resume: decode chunks 0..k-1, save the state, load it into a fresh handle
    (same configuration and weights) and decode chunks k.. there: every pixel equals the
    uninterrupted stream's, and the saving handle continues unaffected. A state of another
    configuration, a wrong size or a damaged header is refused."""
    cfg = synth.PRESETS["small"]          # W = 3: the resumed chunks evict saved ones
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    want = gpu_stream(cfg, w, z)
    W = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    a = fdp.Decoder(cfg, W)
    shape = (cfg.out_channels, cfg.r_t, cfg.out_h, cfg.out_w)
    k = 2
    for t in range(k):
        a.decode_chunk(dev(z[t]), torch.empty(shape, device="cuda"))
    buf = torch.empty(a.state_bytes(), dtype=torch.uint8).pin_memory()
    a.save_state(buf)
    torch.cuda.synchronize()
    b = fdp.Decoder(cfg, W)
    b.load_state(buf)
    assert b.chunk_index == k
    for t in range(k, cfg.chunks):
        pa, pb = torch.empty(shape, device="cuda"), torch.empty(shape, device="cuda")
        a.decode_chunk(dev(z[t]), pa)
        b.decode_chunk(dev(z[t]), pb)
        torch.cuda.synchronize()
        assert torch.equal(pb.cpu(), want[t]), t
        assert torch.equal(pa.cpu(), want[t]), t
    assert a.sync_status() == fdp.FD_OK and b.sync_status() == fdp.FD_OK
    L = fdp.lib()
    other = synth.PRESETS["small"].replace(window=2)
    c = fdp.Decoder(other, fdp.Weights(other, fdp.pack_blob(other, synth.make_weights(other))))
    assert L.fd_load_state(c.handle, fdp._ptr(buf), a.state_bytes(), None) == 1  # size differs
    bad = buf.clone()
    bad[0] = ord("X")
    assert L.fd_load_state(b.handle, fdp._ptr(bad), b.state_bytes(), None) == 1
    for d in (a, b, c):
        d.close()
    W.close()


def test_decode_causality_on_gpu():
    """Outputs of chunks < 3 are bit-identical when chunks >= 3 change."""
    cfg = synth.PRESETS["small"]
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    z2 = z.copy()
    z2[3:] = synth.make_latents(cfg, seed=5)[3:]
    a, b = gpu_stream(cfg, w, z), gpu_stream(cfg, w, z2)
    for t in range(3):
        assert torch.equal(a[t], b[t])
    assert not torch.equal(a[3], b[3])


def test_ring_slots_hold_the_window():
    """After chunk t, ring slot s of the first backbone layer holds chunk j = s mod W of the
    last W chunks: the same keys as the oracle's concat(tail) cache, slot by slot."""
    cfg = synth.PRESETS["small"]  # W = 3, 5 chunks: slots wrap around
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    ref = oracle.StreamingDecoder(cfg, w)
    Wt = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    dec = fdp.Decoder(cfg, Wt)
    L, G, Wn = cfg.tokens, cfg.kv_groups, cfg.window
    for t in range(cfg.chunks):
        ref.decode_chunk(z[t])
        pix = torch.empty(3, cfg.r_t, cfg.out_h, cfg.out_w, device="cuda")
        dec.decode_chunk(dev(z[t]), pix)
        kbits, vbits = dec.read_ring(0, 0, G, Wn, L)
        kr = torch.from_numpy(kbits.view(np.int16)).view(torch.bfloat16).double()
        oracle_k = ref.kB[0]                                   # [G][c L][64], oldest first
        c = oracle_k.shape[1] // L
        for i in range(c):
            j = t - c + 1 + i
            s = j % Wn
            got = kr[:, s * L:(s + 1) * L]
            want = oracle_k[:, i * L:(i + 1) * L]
            err = float((got - want).abs().max())
            assert err <= 2e-2 * float(want.abs().max()), (t, j, s, err)
            # and it is not any other chunk's keys
            for i2 in range(c):
                if i2 != i:
                    other = oracle_k[:, i2 * L:(i2 + 1) * L]
                    assert float((got - other).abs().max()) > 10 * err
    dec.close()
    Wt.close()


def test_api_errors():
    cfg = synth.PRESETS["tiny"]
    w = synth.make_weights(cfg)
    Wt = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    dec = fdp.Decoder(cfg, Wt)
    L = fdp.lib()
    lat = torch.zeros(16, 8, 8, device="cuda")
    pix = torch.zeros(3, 1, 64, 64, device="cuda")
    assert L.fd_decode_chunk(dec.handle, 0, pix.data_ptr(), 0) == 1
    assert L.fd_decode_chunk(dec.handle, lat.data_ptr() + 4, pix.data_ptr(), 0) == 1
    bad = fdp.make_config(cfg.replace(hidden=320, heads=5))
    assert L.fd_weights_blob_elems(bad) == 0
    other = cfg.replace(window=3)
    with pytest.raises(fdp.FdError) as e:
        fdp.Decoder(other, Wt)
    assert e.value.code == 2
    # a weights object with live handles cannot be destroyed
    assert L.fd_weights_destroy(Wt.handle) == 5
    dec.decode_chunk(lat, pix)
    assert dec.sync_status() == 0 and dec.chunk_index == 1
    dec.close()
    Wt.close()


@pytest.mark.slow
@pytest.mark.parametrize("name,chunks", [("480p", 5), ("720p", 1)])
def test_decode_full_size(name, chunks):
    """The benchmark's own configurations at full size and depth, first chunks (at 480p the
    full W = 4 window plus the first eviction; at 720p chunk 0, every block at 3600 tokens)."""
    cfg = synth.PRESETS[name]
    w, z = synth.make_weights(cfg), synth.make_latents(cfg, chunks=chunks)
    ref = oracle.StreamingDecoder(cfg, w)
    want = [ref.decode_chunk(z[t]) for t in range(chunks)]
    got = gpu_stream(cfg, w, z, chunks=chunks)
    compare(cfg, got, want, name)


@pytest.mark.slow
@pytest.mark.parametrize("name", ["720p_d3", "720p_wide_d3"])
def test_decode_full_token_count_reduced_depth(name):
    """The 720p token count (3600 tokens, 14400 refined rows) through whole streams at
    reduced depth (2 backbone + 1 refinement blocks): 720p_d3 decodes 5 chunks, so both W = 4
    rings fill and evict at 720p; 720p_wide_d3 is the wide model's shape (D = 1536, 24 heads on
    3 KV groups, W = 8, AR(1) latents), 2 chunks. Every chunk against the oracle, uint8 codes."""
    cfg = synth.PRESETS[name]
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    want = oracle.decode_stream(cfg, w, z)
    got = gpu_stream(cfg, w, z)
    compare(cfg, got, want, name)


@pytest.mark.parametrize("name", ["small", "small_f1", "small_u8"])
def test_decode_chunk_host_matches_oracle(name):
    """fd_decode_chunk_host (pinned host latents in, pinned host pixels out, copies on the
    stream; the end-to-end benchmark's call for several streams per GPU) against the oracle,
    chunk by chunk, and bit for bit equal to the device-buffer call. small_f1 checks the
    one-frame first chunk of the causal frame count (its copy-back is one frame)."""
    cfg = synth.PRESETS[name]
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    want = oracle.decode_stream(cfg, w, z)
    dev_out = gpu_stream(cfg, w, z)
    Wt = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    dec = fdp.Decoder(cfg, Wt)
    stream = torch.cuda.Stream()
    dt = torch.uint8 if cfg.out_u8 else torch.float32
    got = []
    for t in range(cfg.chunks):
        frames = 1 if (t == 0 and getattr(cfg, "first_chunk_frames", 0) == 1) else cfg.r_t
        lat = torch.from_numpy(np.ascontiguousarray(z[t])).pin_memory()
        pix = torch.full((cfg.out_channels, frames, cfg.out_h, cfg.out_w), 7, dtype=dt).pin_memory()
        dec.decode_chunk_host(lat, pix, stream)
        stream.synchronize()
        got.append(pix.clone())
    assert dec.sync_status() == fdp.FD_OK
    dec.close()
    Wt.close()
    compare(cfg, got, want, name + " host buffers")
    for t in range(cfg.chunks):
        assert torch.equal(got[t], dev_out[t]), t


@pytest.mark.parametrize("name", ["small", "small_f1", "small_u8"])
def test_decode_sequence_host_equals_device_decodes(name):
    """fd_decode_sequence_host (the overlapped host-buffer call the end-to-end benchmark times:
    chunk t decodes while chunk t+1's latent goes in and chunk t-1's pixels come out on the
    library's copy stream, two device buffers of each) gives the pixels of fd_decode_chunk bit
    for bit. The stream goes in two calls (chunks 0..2, then the rest: the second call continues
    the first's chunk counter and reuses its buffers), then again after fd_reset in one call.
    The pixel buffers start filled with 7s, so a copy that was missed or came from the wrong
    buffer shows."""
    cfg = synth.PRESETS[name]
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    dev_out = gpu_stream(cfg, w, z)
    Wt = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    dec = fdp.Decoder(cfg, Wt)
    stream = torch.cuda.Stream()
    dt = torch.uint8 if cfg.out_u8 else torch.float32
    lat = [torch.from_numpy(np.ascontiguousarray(z[t])).pin_memory() for t in range(cfg.chunks)]

    def pixels():
        out = []
        for t in range(cfg.chunks):
            frames = 1 if (t == 0 and getattr(cfg, "first_chunk_frames", 0) == 1) else cfg.r_t
            out.append(torch.full((cfg.out_channels, frames, cfg.out_h, cfg.out_w), 7,
                                  dtype=dt).pin_memory())
        return out

    first = pixels()
    dec.decode_sequence_host(lat[:3], first[:3], stream)
    dec.decode_sequence_host(lat[3:], first[3:], stream)
    stream.synchronize()
    assert dec.sync_status() == fdp.FD_OK and dec.chunk_index == cfg.chunks
    dec.reset()
    again = pixels()
    dec.decode_sequence_host(lat, again, stream)
    stream.synchronize()
    assert dec.sync_status() == fdp.FD_OK
    dec.close()
    Wt.close()
    for t in range(cfg.chunks):
        assert torch.equal(first[t], dev_out[t]), t
        assert torch.equal(again[t], dev_out[t]), t


def test_window_relative_rope_mode():
    """rope_mode = window (the temporal RoPE index counted from the window's first frame, Sec.
    4.3) against the oracle's window-relative decode, which keeps un-rotated keys and re-rotates
    the whole window every chunk; the library's pixels are bit-identical to its absolute mode
    (only index differences enter a score)."""
    for name in ("small", "tiny_rt"):
        cfg = synth.PRESETS[name]
        w, z = synth.make_weights(cfg), synth.make_latents(cfg)
        want = oracle.decode_stream(cfg, w, z, rope_mode="window")
        win = gpu_stream(cfg.replace(rope_mode="window"), w, z)
        compare(cfg, win, want, name + " window-relative RoPE")
        absolute = gpu_stream(cfg, w, z)
        for a, b in zip(win, absolute):
            assert torch.equal(a, b)


def test_bounded_wait_gives_up_and_the_handle_recovers():
    """Failure detection on the GPU without a fault: a kernel waits, through the bounded
    mbarrier wait every decode kernel uses, on a barrier nothing arrives at, with a 1 ms limit.
    The wait gives up and the kernel returns; the host sees FD_ERR_DEVICE_TIMEOUT from
    fd_sync_status within a fraction of a second, decodes are refused with FD_ERR_STATE until
    fd_reset, and after the reset the same context decodes the stream exactly as before."""
    import time
    cfg = synth.PRESETS["small"]
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    want = oracle.decode_stream(cfg, w, z)
    Wt = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    dec = fdp.Decoder(cfg, Wt)
    shape = (cfg.out_channels, cfg.r_t, cfg.out_h, cfg.out_w)
    dec.decode_chunk(dev(z[0]), torch.empty(shape, device="cuda"))
    assert dec.sync_status() == fdp.FD_OK
    t0 = time.perf_counter()
    dec.debug_wait_timeout(1000)
    status = dec.sync_status()
    elapsed = time.perf_counter() - t0
    assert status == 6, fdp.STATUS.get(status)          # FD_ERR_DEVICE_TIMEOUT
    assert elapsed < 1.0, elapsed                        # the 1 ms wait ended by itself
    with pytest.raises(fdp.FdError) as e:
        dec.decode_chunk(dev(z[1]), torch.empty(shape, device="cuda"))
    assert e.value.code == 5                             # FD_ERR_STATE until fd_reset
    L = fdp.lib()
    assert L.fd_debug_wait_timeout(dec.handle, 0, None) == 1
    assert L.fd_debug_wait_timeout(dec.handle, 100001, None) == 1
    dec.reset()
    got = []
    for t in range(cfg.chunks):
        pix = torch.empty(shape, device="cuda")
        dec.decode_chunk(dev(z[t]), pix)
        got.append(pix)
    torch.cuda.synchronize()
    assert dec.sync_status() == fdp.FD_OK
    compare(cfg, [g.cpu() for g in got], want, "small after a device timeout and fd_reset")
    dec.close()
    Wt.close()


@pytest.mark.slow
def test_decode_wide_model_structure():
    """The 720p wide model (D = 1536, 24 heads / 3 KV groups, 32 + 2 blocks, W = 8, AR(1)
    latents, uint8 pixels) on a 130-token frame, 10 chunks: the 8-chunk window fills, then
    evicts twice. Its full-size stream is too large for the fp64 oracle; every shape that
    differs from this case (token count) is covered at full size by the kernel tests and the
    480p / 720p decodes. The oracle's own bf16 / fp16 operand-rounding noise on this case is
    mean-abs 1.45e-3, so the configurations' bar (2e-3) applies."""
    cfg = synth.PRESETS["wide_small"]
    w, z = synth.make_weights(cfg), synth.make_latents(cfg)
    want = oracle.decode_stream(cfg, w, z)
    got = gpu_stream(cfg, w, z)
    compare(cfg, got, want, "wide_small")


@pytest.mark.slow
def test_decode_xl_layout():
    """The paper's XL layout at 480p (48-channel latents, patch 1, D = 1536, gated MLP, W = 2:
    chunk 2 evicts chunk 0) against the fp64 oracle. The bar is the one that the oracle itself
    needs once its matrix operands are rounded to bf16 / fp16, which is checked first."""
    cfg, chunks = synth.PRESETS["xl_480p"], 3
    w, z = synth.make_weights(cfg), synth.make_latents(cfg, chunks=chunks)
    ref = oracle.StreamingDecoder(cfg, w)
    want = [ref.decode_chunk(z[t]) for t in range(chunks)]
    with oracle.operand_rounding():  # chunk 0 fixes the derivation of the bar
        want_r = [oracle.StreamingDecoder(cfg, w).decode_chunk(z[0])]
    compare(cfg, want_r, want[:1], "xl_480p operand-rounded oracle vs fp64", XL_MAX_ABS,
            XL_MEAN_ABS)
    assert float((want_r[0] - want[0]).abs().mean()) > MEAN_ABS
    got = gpu_stream(cfg, w, z, chunks=chunks)
    compare(cfg, got, want, "xl_480p vs fp64", XL_MAX_ABS, XL_MEAN_ABS)


@pytest.mark.slow
def test_decode_fp8_mlp_full_size():
    """FP8 MLPs (Sec. 4.6) at 480p against the oracle's FP8 option (same e4m3 codes of the
    weights, same static power-of-two scales). Quantising activations to e4m3 turns a tiny
    difference in a value into a whole code step wherever it straddles a rounding boundary,
    and 26 blocks compound that: the fp64 oracle itself moves by mean-abs about 1e-2 once its
    matrix operands are rounded to bf16 / fp16 (checked first; the bf16 path moves by 8e-4).
    So the GPU is held to the noise of that computation: no farther from the fp64 FP8 oracle
    than 1.5x the operand-rounded oracle is, and the FP8 output must differ from the bf16 one."""
    cfg, chunks = synth.PRESETS["480p_fp8"], 2
    w, z = synth.make_weights(cfg), synth.make_latents(cfg, chunks=chunks)
    want = oracle.decode_stream(cfg, w, z)
    with oracle.operand_rounding():  # the noise of chunk 0 sets the bar of both chunks
        want_r = oracle.StreamingDecoder(cfg, w).decode_chunk(z[0])
    noise = pixel_errors(want_r, want[0])
    print("480p_fp8 operand-rounded oracle vs fp64 (chunk 0):", noise)
    assert noise[1] < 2e-2 and noise[0] < 0.15
    got = gpu_stream(cfg, w, z, chunks=chunks)
    for t, (g, o) in enumerate(zip(got, want)):
        mx, mean = pixel_errors(g, o)
        print(f"480p_fp8 chunk {t}: max-abs {mx:.3e} mean-abs {mean:.3e}")
        assert mean <= 1.5 * noise[1] and mx <= 1.5 * noise[0] + 2e-2, t
    bf = gpu_stream(synth.PRESETS["480p"], w, z, chunks=1)
    assert float((f64(bf[0]) - f64(got[0])).abs().mean()) > MEAN_ABS


@pytest.mark.slow
def test_decode_xl_fp8_mlp():
    """The XL layout with FP8 gated MLPs (the paper's lossy setting, Sec. 4.6) at 480p, held
    like the 480p FP8 case to 1.5x the operand-rounded oracle's own movement, which the test
    measures first (2 chunks; W = 2, so chunk 1 sees chunk 0)."""
    cfg, chunks = synth.PRESETS["xl_480p_fp8"], 2
    w, z = synth.make_weights(cfg), synth.make_latents(cfg, chunks=chunks)
    want = oracle.decode_stream(cfg, w, z)
    with oracle.operand_rounding():  # the noise of chunk 0 sets the bar of both chunks
        want_r = oracle.StreamingDecoder(cfg, w).decode_chunk(z[0])
    noise = pixel_errors(want_r, want[0])
    print("xl_480p_fp8 operand-rounded oracle vs fp64 (chunk 0):", noise)
    got = gpu_stream(cfg, w, z, chunks=chunks)
    for t, (g, o) in enumerate(zip(got, want)):
        mx, mean = pixel_errors(g, o)
        print(f"xl_480p_fp8 chunk {t}: max-abs {mx:.3e} mean-abs {mean:.3e}")
        assert mean <= 1.5 * noise[1] and mx <= 1.5 * noise[0] + 2e-2, t
