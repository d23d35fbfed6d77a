"""The C-ABI library builds, loads, and exports every symbol its headers declare; host-only
calls (sizes, validation, status strings) work without a GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
fdp = pytest.importorskip("paper_2607_14898_gb300.flashdec")


def declared_functions():
    names = []
    for h in ("flashdec.h", "flashdec_ops.h"):
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names += re.findall(r"\b(fd_\w+)\s*\(", src)
    return sorted(set(names))


def test_library_exports_every_declared_symbol():
    L = fdp.lib()
    names = declared_functions()
    assert len(names) >= 20
    for n in names:
        assert hasattr(L, n), n
    assert set(names) == set(fdp._SIGS), "binding signatures cover the header exactly"


def test_blob_layout_matches_seeded_layout_and_binding_order():
    L = fdp.lib()
    for name, cfg in synth.PRESETS.items():
        c = fdp.make_config(cfg)
        want = sum(int(np.prod(s)) for _, s, _ in synth.weight_layout(cfg))
        assert L.fd_weights_blob_elems(ctypes.byref(c)) == want, name
        assert [n for n, _, _ in synth.weight_layout(cfg)] == fdp.weight_names(cfg)


def test_blob_bytes_is_what_weights_create_expects():
    """fd_weights_blob_bytes = elements x element size of the blob dtype (fp32 4, bf16 2);
    any other dtype or an invalid configuration gives 0."""
    L = fdp.lib()
    for name in ("tiny", "480p", "xl_480p"):
        c = fdp.make_config(synth.PRESETS[name])
        n = L.fd_weights_blob_elems(ctypes.byref(c))
        assert n > 0
        assert L.fd_weights_blob_bytes(ctypes.byref(c), fdp.DTYPE_F32) == 4 * n
        assert L.fd_weights_blob_bytes(ctypes.byref(c), fdp.DTYPE_BF16) == 2 * n
        assert L.fd_weights_blob_bytes(ctypes.byref(c), fdp.DTYPE_U8) == 0
        assert L.fd_weights_blob_bytes(ctypes.byref(c), 7) == 0
    bad = fdp.make_config(synth.PRESETS["small"].replace(heads=3))
    assert L.fd_weights_blob_bytes(ctypes.byref(bad), fdp.DTYPE_F32) == 0
    assert L.fd_weights_blob_bytes(None, fdp.DTYPE_F32) == 0


def test_rope_mode_is_checked():
    """fd_config.rope_mode takes FD_ROPE_ABS (0) or FD_ROPE_WINDOW_REL (1); other values make
    the configuration invalid. The mode does not change the blob."""
    L = fdp.lib()
    cfg = synth.PRESETS["small"]
    n = L.fd_weights_blob_elems(ctypes.byref(fdp.make_config(cfg)))
    win = fdp.make_config(cfg.replace(rope_mode="window"))
    assert win.rope_mode == 1
    assert L.fd_weights_blob_elems(ctypes.byref(win)) == n
    for v in (2, -1):
        c = fdp.make_config(cfg)
        c.rope_mode = v
        assert L.fd_weights_blob_elems(ctypes.byref(c)) == 0


def test_sizes_follow_the_compression_factors():
    L = fdp.lib()
    c = fdp.make_config(synth.PRESETS["480p"])
    assert L.fd_pixels_bytes(ctypes.byref(c)) == 3 * 4 * 480 * 832 * 4
    assert L.fd_latent_bytes(ctypes.byref(c)) == 16 * 60 * 104 * 4
    c = fdp.make_config(synth.PRESETS["720p"])
    assert L.fd_pixels_bytes(ctypes.byref(c)) == 3 * 4 * 720 * 1280


def test_state_size_is_header_plus_every_ring():
    """Saved streaming state: a header (magic, version, t, payload size, the config) and, per
    layer, K [G][pitch][64] bf16 and V^T [G][64][pitch] fp16 with pitch = round_up(W rows, 128)
    (rows = L backbone, r_t L refinement)."""
    L = fdp.lib()
    cfg = synth.PRESETS["480p"]
    c = fdp.make_config(cfg)
    up = lambda x: -(-x // 128) * 128
    ring = lambda rows: cfg.kv_groups * up(cfg.window * rows) * 64 * 2
    payload = 2 * (cfg.n_blocks * ring(cfg.tokens) + cfg.n_refine * ring(cfg.r_t * cfg.tokens))
    header = -(-(8 + 3 * 8 + ctypes.sizeof(fdp.fd_config)) // 8) * 8  # 8-byte aligned struct
    assert L.fd_state_bytes(ctypes.byref(c)) == header + payload
    bad = fdp.make_config(synth.PRESETS["small"].replace(heads=3))
    assert L.fd_state_bytes(ctypes.byref(bad)) == 0
    buf = ctypes.create_string_buffer(16)
    assert L.fd_save_state(None, buf, 16, None) == 1
    assert L.fd_load_state(None, buf, 16, None) == 1


@pytest.mark.parametrize("field,value", [("hidden", 320), ("heads", 3), ("kv_groups", 3),
                                         ("patch", 3), ("window", 0), ("r_t", 0),
                                         ("n_blocks", 0), ("latent_channels", 1),
                                         # beyond the upper bounds (no int overflow inside)
                                         ("heads", 1 << 26), ("mlp_ratio", 1 << 20),
                                         ("vae_spatial", 1 << 12), ("r_t", 1 << 20),
                                         ("out_channels", 1 << 16)])
def test_invalid_configs_rejected(field, value):
    L = fdp.lib()
    cfg = synth.PRESETS["small"].replace(**{field: value})
    assert L.fd_weights_blob_elems(ctypes.byref(fdp.make_config(cfg))) == 0


def test_status_strings_and_null_arguments():
    L = fdp.lib()
    for code in range(8):
        assert L.fd_status_str(code)
    assert L.fd_weights_blob_elems(None) == 0
    assert L.fd_decode_chunk(None, None, None, None) == 1
    assert L.fd_decode_sequence_host(None, 1, None, None, None) == 1
    assert L.fd_reset(None) == 1 and L.fd_destroy(None) == 1
    out = ctypes.c_void_p()
    c = fdp.make_config(synth.PRESETS["tiny"])
    assert L.fd_weights_create(ctypes.byref(c), None, 0, 0, ctypes.byref(out)) == 1


def test_cost_model_matches_the_oracle_flop_count():
    """The closed-form work per chunk equals the multiply-adds the oracle performs (its matmuls
    count 2*M*N*K), chunk by chunk through warm-up and steady state."""
    import oracle
    from paper_2607_14898_gb300 import costs
    for name in ("small", "tiny_gated"):
        cfg = synth.PRESETS[name]
        w, z = synth.make_weights(cfg), synth.make_latents(cfg)
        dec = oracle.StreamingDecoder(cfg, w)
        for t in range(cfg.chunks):
            oracle.reset_flops()
            dec.decode_chunk(z[t])
            f = costs.chunk_flops(cfg, t)
            attn = f["attn_backbone"] + f["attn_refine"]
            assert oracle.FLOPS["attn"] == attn, (name, t)
            assert oracle.FLOPS["gemm"] == sum(f.values()) - attn, (name, t)
    # Sec. 3.3: attention cost linear in W and N, quadratic in L_frm
    big = synth.PRESETS["480p"]
    a = costs.chunk_flops(big, 10)["attn_backbone"]
    assert a == 24 * 4 * 1560 * (4 * 1560) * 64 * 16


def test_binding_refuses_buffers_the_library_would_overrun():
    """The C ABI takes raw pointers; the binding's stream-level calls check place, type,
    layout and size of every buffer first (here: the host-buffer rules, checkable without a
    GPU)."""
    import numpy as np
    import torch
    chk = fdp.check_buffer
    chk(np.zeros(16, np.float32), "x", 64, "float32", False)
    chk(torch.zeros(4, 4), "x", 64, "float32", False)
    chk(torch.zeros(64, dtype=torch.uint8), "x", 64, "uint8", False)
    bad = [
        (np.zeros(15, np.float32), "float32", False),          # too small
        (np.zeros(17, np.float32), "float32", False),          # too large
        (np.zeros(16, np.float64)[::2].copy(), "float32", False),  # wrong type
        (np.zeros((4, 8), np.float32)[:, ::2], "float32", False),  # not contiguous
        (torch.zeros(8, 4).t(), "float32", False),              # not contiguous
        (torch.zeros(16, dtype=torch.float64), "float32", False),
        (np.zeros(16, np.float32), "float32", True),            # host array for a device call
        (torch.zeros(16), "float32", True),                     # host tensor for a device call
        ([0.0] * 16, "float32", False),                         # not a buffer
    ]
    for x, dt, on_dev in bad:
        with pytest.raises((TypeError, ValueError)):
            chk(x, "x", 64, dt, on_dev)


def test_empty_inputs_are_refused_before_any_launch():
    """Zero-sized problems are argument errors, returned before the library touches the
    device (so this runs without a GPU); an empty list of streams is a no-op."""
    import ctypes
    L = fdp.lib()
    assert L.fd_op_linear(0, 0, 128, 64, 0, 0, 0, 0, 0, 0, 0, 0) == 1      # M = 0
    assert L.fd_op_linear(0, 128, 0, 64, 0, 0, 0, 0, 0, 0, 0, 0) == 1      # N = 0
    assert L.fd_op_linear(0, 128, 128, 0, 0, 0, 0, 0, 0, 0, 0, 0) == 1     # K = 0
    assert L.fd_op_attention(0, 4, 2, 0, 0, 0, 128, 1, 0, 0, 0, 0, 0) == 1  # no queries
    assert L.fd_op_attention(128, 4, 2, 0, 0, 0, 128, 0, 0, 0, 0, 0, 0) == 1  # no keys
    assert L.fd_op_attention_static(0, 4, 2, 0, 0, 0, 128, 1, 0, 0, 0, 0) == 1
    assert L.fd_op_rmsnorm(0, 0, 0, 128, 1e-6, 0, 0) == 1
    assert L.fd_op_kv_append(0, 0, 2, 0, 2, 0, 128, 0, 0, 0) == 1
    assert L.fd_op_unshuffle(0, 0, 8, 8, 1, 0, 0) == 1
    assert L.fd_op_pixel_head(0, 0, 8, 8, 3, 8, 0, 0, 0) == 1
    assert L.fd_decode_chunks(None, 0, None, None, None) == 1       # no handle array at all
    assert L.fd_decode_chunks((ctypes.c_void_p * 1)(), 0, None, None, None) == 0  # no streams


def test_library_is_rebuilt_when_a_source_or_header_changes():
    """build() recompiles when any kernel source or header is newer than the library, so a
    stale libflashdec.so is never loaded (checked on the mtimes, without compiling)."""
    import os
    from paper_2607_14898_gb300 import build as b
    fdp.lib()                                   # built and current
    assert b.up_to_date()
    hdr = os.path.join(b.INCLUDE, "flashdec.h")
    st = os.stat(hdr)
    try:
        os.utime(hdr, (st.st_atime, os.path.getmtime(b.LIB) + 10))
        assert not b.up_to_date()
    finally:
        os.utime(hdr, (st.st_atime, st.st_mtime))
    assert b.up_to_date()
