"""Batched decode (fd_batch_create / fd_decode_batch): several independent streams of one
weights object decoded with stacked GEMMs. Each stream's pixels must match the oracle's decode
of that stream alone, with streams joining the batch at different chunk indices (so one call
holds streams at different t, and the set of handles changes between calls)."""
import pytest
import torch

import oracle
import synth
from helpers import dev, pixel_errors
from test_gpu_decode import MAX_ABS, MEAN_ABS, compare

pytestmark = pytest.mark.gpu

fdp = pytest.importorskip("paper_2607_14898_gb300.flashdec")


@pytest.fixture(scope="module", autouse=True)
def _setup(torch_threads):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    fdp.lib()


def pixel_buffer(cfg, t):
    f1 = t == 0 and getattr(cfg, "first_chunk_frames", 0) == 1
    frames = 1 if f1 else cfg.r_t
    dt = torch.uint8 if cfg.out_u8 else torch.float32
    return torch.empty((cfg.out_channels, frames, cfg.out_h, cfg.out_w), dtype=dt, device="cuda")


def batch_streams(cfg, w, zs, starts, chunks, max_streams=None):
    """Decode stream s (latents zs[s]) from call starts[s] on, all through one batch object;
    returns each stream's pixels per chunk."""
    W = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    decs = [fdp.Decoder(cfg, W) for _ in zs]
    B = fdp.Batch(cfg, W, max_streams or len(zs))
    got = [[] for _ in zs]
    for k in range(max(starts) + chunks):
        live = [s for s in range(len(zs)) if starts[s] <= k < starts[s] + chunks]
        ts = [k - starts[s] for s in live]
        lat = [dev(zs[s][t]) for s, t in zip(live, ts)]
        pix = [pixel_buffer(cfg, t) for t in ts]
        B.decode([decs[s] for s in live], lat, pix)
        for s, p in zip(live, pix):
            got[s].append(p)
    torch.cuda.synchronize()
    for d in decs:
        assert d.sync_status() == fdp.FD_OK
        assert d.chunk_index == chunks
    out = [[p.cpu() for p in g] for g in got]
    B.close()
    for d in decs:
        d.close()
    W.close()
    return out


# small: L = 130 tokens, padded to 256 rows per frame (a ragged 2-token tail per 128-row tile
# pair); tiny_rt: L = 64 with r_t = 2; the gated, FP8, uint8 and one-frame-first-chunk options
@pytest.mark.parametrize("name", ["small", "tiny_rt", "tiny_gated", "small_fp8", "small_u8",
                                  "small_f1", "tiny_gated_fp8"])
def test_batch_decode_matches_oracle(name):
    cfg = synth.PRESETS[name]
    w = synth.make_weights(cfg)
    zs = [synth.make_latents(cfg, seed=s) for s in range(3)]
    starts = [0, 1, 2]
    got = batch_streams(cfg, w, zs, starts, cfg.chunks)
    for s, z in enumerate(zs):
        want = oracle.decode_stream(cfg, w, z)
        compare(cfg, got[s], want, f"{name} stream {s}")


def test_batch_of_one_and_changing_membership():
    """A batch object sized for 4 used with 1, 2 and 3 streams in turn (a stream leaves and
    another joins): every stream still matches its own oracle decode."""
    cfg = synth.PRESETS["tiny_rt"]
    w = synth.make_weights(cfg)
    zs = [synth.make_latents(cfg, seed=10 + s) for s in range(3)]
    got = batch_streams(cfg, w, zs, [0, 2, 1], cfg.chunks, max_streams=4)
    for s, z in enumerate(zs):
        compare(cfg, got[s], oracle.decode_stream(cfg, w, z), f"stream {s}")


def test_batch_replaced_handle_gets_its_own_rings():
    """A handle destroyed and replaced by a new one (whose address the allocator may well
    reuse) in the same batch slot: the batch must rebuild its per-stream tables, so the new
    stream writes and reads its own rings and matches its own oracle decode."""
    cfg = synth.PRESETS["tiny_rt"]
    w = synth.make_weights(cfg)
    W = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    B = fdp.Batch(cfg, W, 2)
    za, zb, zc = (synth.make_latents(cfg, seed=s) for s in (20, 21, 22))
    a, b = fdp.Decoder(cfg, W), fdp.Decoder(cfg, W)
    got_a, got_c = [], []
    for t in range(2):
        pa, pb = pixel_buffer(cfg, t), pixel_buffer(cfg, t)
        B.decode([a, b], [dev(za[t]), dev(zb[t])], [pa, pb])
        got_a.append(pa)
    torch.cuda.synchronize()
    b.close()
    c = fdp.Decoder(cfg, W)
    for t in range(cfg.chunks):
        if t + 2 < cfg.chunks:
            pa, pc = pixel_buffer(cfg, t + 2), pixel_buffer(cfg, t)
            B.decode([a, c], [dev(za[t + 2]), dev(zc[t])], [pa, pc])
            got_a.append(pa)
        else:
            pc = pixel_buffer(cfg, t)
            B.decode([c], [dev(zc[t])], [pc])
        got_c.append(pc)
    torch.cuda.synchronize()
    assert a.sync_status() == fdp.FD_OK and c.sync_status() == fdp.FD_OK
    compare(cfg, [p.cpu() for p in got_a], oracle.decode_stream(cfg, w, za), "kept stream")
    compare(cfg, [p.cpu() for p in got_c], oracle.decode_stream(cfg, w, zc), "new stream")
    B.close()
    a.close()
    c.close()
    W.close()


def test_batch_api_errors():
    cfg = synth.PRESETS["tiny"]
    w = synth.make_weights(cfg)
    W = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    W2 = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    a, b, c = fdp.Decoder(cfg, W), fdp.Decoder(cfg, W), fdp.Decoder(cfg, W2)
    B = fdp.Batch(cfg, W, 2)
    lat = [torch.zeros(16, 8, 8, device="cuda") for _ in range(3)]
    pix = [torch.zeros(3, 1, 64, 64, device="cuda") for _ in range(3)]
    with pytest.raises(fdp.FdError) as e:
        B.decode([a, b, c], lat, pix)  # more than max_streams
    assert e.value.code == 1
    with pytest.raises(fdp.FdError) as e:
        B.decode([a, a], lat[:2], pix[:2])  # the same handle twice
    assert e.value.code == 1
    with pytest.raises(fdp.FdError) as e:
        B.decode([a, c], lat[:2], pix[:2])  # another weights object
    assert e.value.code == 2
    with pytest.raises(fdp.FdError) as e:
        fdp.Batch(cfg.replace(window=3), W, 2)
    assert e.value.code == 2
    assert a.chunk_index == 0 and b.chunk_index == 0  # nothing was enqueued
    assert fdp.lib().fd_weights_destroy(W.handle) == 5  # the batch is a user of W
    B.decode([b, a], lat[:2], pix[:2])
    torch.cuda.synchronize()
    assert a.sync_status() == 0 and a.chunk_index == 1 and b.chunk_index == 1
    B.close()
    for d in (a, b, c):
        d.close()
    W.close()
    W2.close()


@pytest.mark.slow
def test_batch_decode_480p():
    """Two 480p streams (L = 1560 tokens, padded to 1664 rows per frame) one chunk apart,
    through the batched path, against the oracle."""
    cfg, chunks = synth.PRESETS["480p"], 2
    w = synth.make_weights(cfg)
    zs = [synth.make_latents(cfg, chunks=chunks, seed=s) for s in range(2)]
    got = batch_streams(cfg, w, zs, [0, 1], chunks)
    for s, z in enumerate(zs):
        want = oracle.decode_stream(cfg, w, z)
        for t, (g, o) in enumerate(zip(got[s], want)):
            mx, mean = pixel_errors(g, o)
            print(f"480p batch stream {s} chunk {t}: max-abs {mx:.3e} mean-abs {mean:.3e}")
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (s, t)


@pytest.mark.slow
def test_batch_of_eight_480p_streams():
    """Eight 480p streams in one batch (13,312 stacked backbone rows, 53,248 refinement rows:
    the products run on CTA pairs). The last stream against the oracle; every stream within the
    same bar of its own single-stream decode (the two computations round differently, in
    attention's key-range splits and the tile shapes, and 26 blocks carry that to about the
    size of the bf16 noise itself: measured max-abs 5e-3, mean-abs 6e-4; a stream mixed up
    with another, or a misplaced cache row, is off by orders of magnitude more)."""
    cfg, chunks, S = synth.PRESETS["480p"], 2, 8
    w = synth.make_weights(cfg)
    zs = [synth.make_latents(cfg, chunks=chunks, seed=s) for s in range(S)]
    got = batch_streams(cfg, w, zs, [0] * S, chunks)
    want = oracle.decode_stream(cfg, w, zs[S - 1])
    for t in range(chunks):
        mx, mean = pixel_errors(got[S - 1][t], want[t])
        print(f"480p x8 batch stream {S - 1} chunk {t}: max-abs {mx:.3e} mean-abs {mean:.3e}")
        assert mx <= MAX_ABS and mean <= MEAN_ABS
    W = fdp.Weights(cfg, fdp.pack_blob(cfg, w))
    for s in range(S):
        dec = fdp.Decoder(cfg, W)
        for t in range(chunks):
            pix = pixel_buffer(cfg, t)
            dec.decode_chunk(dev(zs[s][t]), pix)
            mx, mean = pixel_errors(got[s][t], pix.cpu())
            print(f"480p x8 batch stream {s} chunk {t} vs single: max-abs {mx:.3e} "
                  f"mean-abs {mean:.3e}")
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (s, t)
        dec.close()
    W.close()
