"""Python binding of libflashdec.so (ctypes): argument marshalling only.

Every step of the decode path runs in the library's CUDA kernels; this module only converts
Python / torch arguments into the C ABI of include/flashdec.h and include/flashdec_ops.h.
There is no fallback: if the library is missing or the device is not an sm_103 GPU, calls
raise.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

_LIB = None

FD_OK = 0
STATUS = {0: "FD_OK", 1: "FD_ERR_INVALID_ARG", 2: "FD_ERR_CONFIG", 3: "FD_ERR_OOM",
          4: "FD_ERR_CUDA", 5: "FD_ERR_STATE", 6: "FD_ERR_DEVICE_TIMEOUT",
          7: "FD_ERR_UNSUPPORTED"}
DTYPE_F32, DTYPE_BF16, DTYPE_U8 = 0, 1, 2
# fd_rope_mode, keyed like the oracle's rope_mode argument
ROPE_MODES = {"abs": 0, "window": 1}
EPI_F32, EPI_RESID, EPI_GELU, EPI_TUP, EPI_SWIGLU = 0, 1, 2, 3, 4
# fd_kernel_kind order
KERNEL_KINDS = ["unshuffle", "embed", "rmsnorm", "qkv", "attn_backbone", "attn_refine", "out",
                "mlp1", "mlp2", "tup", "head1", "head2", "pixel", "advance", "rope"]
# kernel kinds of the training step (enum fd_train_kind)
TRAIN_KINDS = ["linear", "dgrad", "wgrad", "attn_gemm", "softmax", "transpose", "norm",
               "pointwise"]


class FdError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {STATUS.get(code, code)}")
        self.code = code


class fd_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "latent_channels", "latent_h", "latent_w", "patch", "hidden", "heads", "kv_groups",
        "mlp_ratio", "n_blocks", "n_refine", "window", "r_t", "vae_spatial", "out_channels",
        "out_dtype", "mlp_gated")] + [("norm_eps", ctypes.c_float), ("rope_base", ctypes.c_float),
                                      ("qk_norm", ctypes.c_int32), ("mlp_fp8", ctypes.c_int32),
                                      ("first_chunk_frames", ctypes.c_int32),
                                      ("rope_mode", ctypes.c_int32)]


_P = ctypes.c_void_p
_I = ctypes.c_int
_F = ctypes.c_float
_SIGS = {
    "fd_status_str": (ctypes.c_char_p, [_I]),
    "fd_weights_blob_elems": (ctypes.c_size_t, [ctypes.POINTER(fd_config)]),
    "fd_weights_blob_bytes": (ctypes.c_size_t, [ctypes.POINTER(fd_config), _I]),
    "fd_latent_bytes": (ctypes.c_size_t, [ctypes.POINTER(fd_config)]),
    "fd_pixels_bytes": (ctypes.c_size_t, [ctypes.POINTER(fd_config)]),
    "fd_handle_device_bytes": (ctypes.c_size_t, [ctypes.POINTER(fd_config)]),
    "fd_weights_create": (_I, [ctypes.POINTER(fd_config), _P, ctypes.c_size_t, _I,
                               ctypes.POINTER(_P)]),
    "fd_weights_destroy": (_I, [_P]),
    "fd_create": (_I, [ctypes.POINTER(fd_config), _P, ctypes.POINTER(_P)]),
    "fd_decode_chunk": (_I, [_P, _P, _P, _P]),
    "fd_decode_chunks": (_I, [ctypes.POINTER(_P), _I, ctypes.POINTER(_P), ctypes.POINTER(_P),
                              _P]),
    "fd_decode_chunk_host": (_I, [_P, _P, _P, _P]),
    "fd_decode_sequence_host": (_I, [_P, _I, _P, _P, _P]),
    "fd_batch_create": (_I, [ctypes.POINTER(fd_config), _P, _I, ctypes.POINTER(_P)]),
    "fd_decode_batch": (_I, [_P, ctypes.POINTER(_P), _I, ctypes.POINTER(_P),
                             ctypes.POINTER(_P), _P]),
    "fd_batch_destroy": (_I, [_P]),
    "fd_reset": (_I, [_P]),
    "fd_profile_enable": (_I, [_P, _I]),
    "fd_profile_collect": (_I, [_P, ctypes.POINTER(ctypes.c_int64),
                                ctypes.POINTER(ctypes.c_double)]),
    "fd_launch_count": (ctypes.c_int64, [_P]),
    "fd_destroy": (_I, [_P]),
    "fd_chunk_index": (ctypes.c_int64, [_P]),
    "fd_sync_status": (_I, [_P]),
    "fd_debug_read_ring": (_I, [_P, _I, _I, _P, ctypes.c_size_t]),
    "fd_debug_wait_timeout": (_I, [_P, ctypes.c_uint, _P]),
    "fd_train_grad_elems": (ctypes.c_size_t, [ctypes.POINTER(fd_config)]),
    "fd_op_linear_pixel": (_I, [_I, _I, _P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P]),
    "fd_op_rmsnorm_bwd": (_I, [_P, _P, _P, _I, _I, _F, _P, _P, _P, _P]),
    "fd_op_scores_bwd": (_I, [_I, _I, _P, _P, _P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _P]),
    "fd_op_gelu_bwd": (_I, [_P, _P, ctypes.c_int64, _P, _P, _P]),
    "fd_op_l1_pixel_bwd": (_I, [_P, _P, _I, _I, _I, _I, _I, _P, _P, _P, _P]),
    "fd_train_create": (_I, [ctypes.POINTER(fd_config), _P, _I, ctypes.POINTER(_P)]),
    "fd_train_step": (_I, [_P, _P, _P, _P, _P, _P]),
    "fd_train_status": (_I, [_P, _P]),
    "fd_train_profile_enable": (_I, [_P, _I]),
    "fd_train_profile_collect": (_I, [_P, ctypes.POINTER(ctypes.c_int64),
                                      ctypes.POINTER(ctypes.c_double)]),
    "fd_train_destroy": (_I, [_P]),
    "fd_state_bytes": (ctypes.c_size_t, [ctypes.POINTER(fd_config)]),
    "fd_save_state": (_I, [_P, _P, ctypes.c_size_t, _P]),
    "fd_load_state": (_I, [_P, _P, ctypes.c_size_t, _P]),
    "fd_op_linear": (_I, [_I, _I, _I, _I, _P, _P, _P, _P, _I, _I, _P, _P]),
    "fd_op_linear_tiled": (_I, [_I, _I, _I, _I, _P, _P, _P, _P, _I, _I, _I, _P, _P]),
    "fd_op_rope_table": (_I, [_I, _I, _F, _P, _P]),
    "fd_op_qkv": (_I, [_I, _I, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _I, _F, _F,
                       _P, _P, _P, _P, _I, _I, _P, _P]),
    "fd_attention_workspace_bytes": (ctypes.c_size_t, [_I, _I, _I, _I, _I]),
    "fd_op_attention": (_I, [_I, _I, _I, _P, _P, _P, _I, _I, _P, _I, _P, _P, _P]),
    "fd_op_attention_static": (_I, [_I, _I, _I, _P, _P, _P, _I, _I, _P, _I, _P, _P]),
    "fd_op_kv_append": (_I, [_P, _P, _I, _I, _I, _I, _I, _P, _P, _P]),
    "fd_op_rmsnorm": (_I, [_P, _P, _I, _I, _F, _P, _P]),
    "fd_op_rmsnorm_e4m3": (_I, [_P, _P, _I, _I, _F, _F, _P, _P]),
    "fd_op_linear_e4m3": (_I, [_I, _I, _I, _I, _P, _P, _P, _P, _P, _F, _I, _P, _P]),
    "fd_op_unshuffle": (_I, [_P, _I, _I, _I, _I, _P, _P]),
    "fd_op_pixel_head": (_I, [_P, _I, _I, _I, _I, _I, _I, _P, _P]),
}


def lib(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load libflashdec.so (building it in-tree first if needed)."""
    global _LIB
    if _LIB is None:
        path = _build.LIB
        if build_if_missing:
            path = _build.build()
        if not os.path.exists(path):
            raise RuntimeError(f"libflashdec.so not built ({path}); run __graft_entry__.build()")
        L = ctypes.CDLL(path)
        for name, (res, args) in _SIGS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _LIB = L
    return _LIB


def _check(code: int, what: str) -> None:
    if code != FD_OK:
        raise FdError(code, what)


def make_config(cfg) -> fd_config:
    """fd_config from any object with the decoder's shape attributes (e.g. synth.FDConfig)."""
    c = fd_config()
    for n in ("latent_channels", "latent_h", "latent_w", "patch", "hidden", "heads",
              "kv_groups", "mlp_ratio", "n_blocks", "n_refine", "window", "r_t", "vae_spatial",
              "out_channels"):
        setattr(c, n, int(getattr(cfg, n)))
    c.out_dtype = DTYPE_U8 if getattr(cfg, "out_u8", False) else DTYPE_F32
    c.mlp_gated = 1 if cfg.mlp_gated else 0
    c.qk_norm = 1 if cfg.qk_norm else 0
    c.mlp_fp8 = 1 if getattr(cfg, "mlp_fp8", False) else 0
    c.first_chunk_frames = int(getattr(cfg, "first_chunk_frames", 0))
    c.rope_mode = ROPE_MODES[getattr(cfg, "rope_mode", "abs")]
    c.norm_eps = float(cfg.norm_eps)
    c.rope_base = float(cfg.rope_base)
    return c


def weight_names(cfg) -> list[str]:
    """Tensor names in weight-blob order (the order documented in include/flashdec.h)."""
    second = "qnorm.g" if getattr(cfg, "qk_norm", False) else "vnorm.g"
    blk = ["norm1.g", "qkv.w", "qkv.b", "knorm.g", second, "out.w", "out.b", "norm2.g",
           "mlp1.w", "mlp1.b", "mlp2.w", "mlp2.b"]
    names = ["embed.w", "embed.b"]
    names += [f"blocks.{b}.{n}" for b in range(cfg.n_blocks) for n in blk]
    names += ["normf.g", "tup.w", "tup.b"]
    names += [f"refine.{b}.{n}" for b in range(cfg.n_refine) for n in blk]
    names += ["normh.g", "head1.w", "head1.b", "head2.w", "head2.b"]
    return names


def pack_blob(cfg, weights: dict) -> np.ndarray:
    """Concatenate a name -> array dict into one fp32 blob in blob order."""
    return np.concatenate([np.asarray(weights[n], dtype=np.float32).ravel()
                           for n in weight_names(cfg)])


def _stream_ptr(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return int(getattr(stream, "cuda_stream", stream))


def _ptr(x) -> int:
    if x is None:
        return 0
    if isinstance(x, np.ndarray):
        return int(x.ctypes.data)
    return int(x.data_ptr()) if hasattr(x, "data_ptr") else int(x)


def check_buffer(x, what: str, nbytes: int, dtype: str, on_device: bool,
                 device: int | None = None) -> None:
    """Refuse a buffer that the library would overrun or misread. The C ABI receives raw
    pointers and cannot see sizes, so the binding checks, for the stream-level calls, that each
    buffer is where the call expects it (CUDA device / host), contiguous, of the element type
    (dtype "float32" or "uint8") and of exactly nbytes bytes."""
    import torch
    if isinstance(x, np.ndarray):
        if on_device:
            raise TypeError(f"{what}: a CUDA tensor is required, not a numpy array")
        if x.dtype != np.dtype(dtype) or not x.flags.c_contiguous:
            raise TypeError(f"{what}: a C-contiguous {dtype} array is required")
        size = x.nbytes
    elif isinstance(x, torch.Tensor):
        if x.is_cuda != on_device:
            raise TypeError(f"{what}: a {'CUDA' if on_device else 'host'} tensor is required")
        if on_device and device is not None and x.device.index != device:
            raise ValueError(f"{what}: on cuda:{x.device.index}, the decoder is on cuda:{device}")
        if x.dtype != getattr(torch, dtype) or not x.is_contiguous():
            raise TypeError(f"{what}: a contiguous {dtype} tensor is required")
        size = x.numel() * x.element_size()
    else:
        raise TypeError(f"{what}: a torch tensor{'' if on_device else ' or numpy array'} "
                        "is required")
    if size != nbytes:
        raise ValueError(f"{what}: {size} bytes, the call reads or writes {nbytes}")


class Weights:
    """Device copy of the decoder weights (fd_weights_create); shareable by several Decoders."""

    def __init__(self, cfg, blob: np.ndarray):
        L = lib()
        self.cfg = make_config(cfg)
        blob = np.ascontiguousarray(blob)
        dt = DTYPE_F32 if blob.dtype == np.float32 else DTYPE_BF16
        if blob.dtype not in (np.float32, np.uint16):
            raise TypeError("blob must be fp32, or bf16 bits as uint16")
        out = _P()
        _check(L.fd_weights_create(ctypes.byref(self.cfg), blob.ctypes.data, blob.nbytes, dt,
                                   ctypes.byref(out)), "fd_weights_create")
        self.handle = out

    def close(self) -> None:
        if getattr(self, "handle", None):
            _check(lib().fd_weights_destroy(self.handle), "fd_weights_destroy")
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Decoder:
    """One decoder stream (fd_create): rolling caches + chunk counter."""

    def __init__(self, cfg, weights: Weights):
        L = lib()
        self.cfg = make_config(cfg)
        self.weights = weights
        out = _P()
        _check(L.fd_create(ctypes.byref(self.cfg), weights.handle, ctypes.byref(out)),
               "fd_create")
        self.handle = out
        import torch
        self.device = torch.cuda.current_device()
        self._latent_bytes = L.fd_latent_bytes(ctypes.byref(self.cfg))
        self._pixels_bytes = L.fd_pixels_bytes(ctypes.byref(self.cfg))

    def _check_buffers(self, latent, pixels, on_device: bool) -> None:
        """The latent of one chunk and the pixels of the next chunk this decoder emits (one
        frame instead of r_t for chunk 0 under the causal frame count)."""
        pix = self._pixels_bytes
        if self.cfg.first_chunk_frames == 1 and self.chunk_index == 0:
            pix //= self.cfg.r_t
        dev = self.device if on_device else None
        check_buffer(latent, "latent", self._latent_bytes, "float32", on_device, dev)
        check_buffer(pixels, "pixels", pix,
                     "uint8" if self.cfg.out_dtype == DTYPE_U8 else "float32", on_device, dev)

    @property
    def pixels_bytes(self) -> int:
        return lib().fd_pixels_bytes(ctypes.byref(self.cfg))

    @property
    def latent_bytes(self) -> int:
        return lib().fd_latent_bytes(ctypes.byref(self.cfg))

    def decode_chunk(self, latent, pixels, stream=None) -> None:
        self._check_buffers(latent, pixels, True)
        _check(lib().fd_decode_chunk(self.handle, _ptr(latent), _ptr(pixels),
                                     _stream_ptr(stream)), "fd_decode_chunk")

    def decode_chunk_host(self, latent_host, pixels_host, stream=None) -> None:
        """Decode from / to host buffers (numpy arrays or pinned torch tensors)."""
        self._check_buffers(latent_host, pixels_host, False)
        lp = latent_host.ctypes.data if isinstance(latent_host, np.ndarray) else _ptr(latent_host)
        pp = pixels_host.ctypes.data if isinstance(pixels_host, np.ndarray) else _ptr(pixels_host)
        _check(lib().fd_decode_chunk_host(self.handle, lp, pp, _stream_ptr(stream)),
               "fd_decode_chunk_host")

    def decode_sequence_host(self, latents_host, pixels_host, stream=None) -> None:
        """Decode len(latents_host) consecutive chunks from / to host buffers (pinned torch
        tensors or numpy arrays), the copies overlapped with the decoding
        (fd_decode_sequence_host)."""
        n = len(latents_host)
        if len(pixels_host) != n:
            raise ValueError("one pixel buffer per latent")
        t0 = self.chunk_index
        dt = "uint8" if self.cfg.out_dtype == DTYPE_U8 else "float32"
        lps, pps = [], []
        for i, (z, p) in enumerate(zip(latents_host, pixels_host)):
            pix = self._pixels_bytes
            if self.cfg.first_chunk_frames == 1 and t0 + i == 0:
                pix //= self.cfg.r_t
            check_buffer(z, "latent", self._latent_bytes, "float32", False, None)
            check_buffer(p, "pixels", pix, dt, False, None)
            lps.append(z.ctypes.data if isinstance(z, np.ndarray) else _ptr(z))
            pps.append(p.ctypes.data if isinstance(p, np.ndarray) else _ptr(p))
        ls = (_P * max(n, 1))(*lps)
        ps = (_P * max(n, 1))(*pps)
        _check(lib().fd_decode_sequence_host(self.handle, n, ls, ps, _stream_ptr(stream)),
               "fd_decode_sequence_host")

    def reset(self) -> None:
        _check(lib().fd_reset(self.handle), "fd_reset")

    def profile(self, enable: bool) -> None:
        _check(lib().fd_profile_enable(self.handle, 1 if enable else 0), "fd_profile_enable")

    def profile_collect(self) -> dict:
        """{kind name: (launches, device ms)} since the last collect."""
        n = len(KERNEL_KINDS)
        launches = (ctypes.c_int64 * n)()
        ms = (ctypes.c_double * n)()
        _check(lib().fd_profile_collect(self.handle, launches, ms), "fd_profile_collect")
        return {k: (int(launches[i]), float(ms[i])) for i, k in enumerate(KERNEL_KINDS)}

    @property
    def launch_count(self) -> int:
        return lib().fd_launch_count(self.handle)

    def sync_status(self) -> int:
        return lib().fd_sync_status(self.handle)

    @property
    def chunk_index(self) -> int:
        return lib().fd_chunk_index(self.handle)

    def read_ring(self, which: int, layer: int, groups: int, window: int, rows: int):
        """(K, V) of one layer's ring as bf16 bit arrays [G][W*rows][64]."""
        n = groups * window * rows * 64
        buf = np.zeros(2 * n, dtype=np.uint16)
        _check(lib().fd_debug_read_ring(self.handle, which, layer, buf.ctypes.data, buf.nbytes),
               "fd_debug_read_ring")
        return (buf[:n].reshape(groups, window * rows, 64), buf[n:].reshape(groups, window * rows, 64))

    def debug_wait_timeout(self, limit_us: int, stream=None) -> None:
        """Enqueue the failure-path check: a bounded wait that runs out after limit_us."""
        _check(lib().fd_debug_wait_timeout(self.handle, int(limit_us), _stream_ptr(stream)),
               "fd_debug_wait_timeout")

    def state_bytes(self) -> int:
        return lib().fd_state_bytes(ctypes.byref(self.cfg))

    def save_state(self, buf, stream=None) -> None:
        """Copy the streaming state (chunk index, rolling caches) into buf (host memory of
        state_bytes() bytes: a numpy uint8 array or a pinned torch tensor), ordered on stream."""
        _check(lib().fd_save_state(self.handle, _ptr(buf), self.state_bytes(),
                                   _stream_ptr(stream)), "fd_save_state")

    def load_state(self, buf, stream=None) -> None:
        """Restore a state saved by a decoder of the same configuration."""
        _check(lib().fd_load_state(self.handle, _ptr(buf), self.state_bytes(),
                                   _stream_ptr(stream)), "fd_load_state")

    def close(self) -> None:
        if getattr(self, "handle", None):
            _check(lib().fd_destroy(self.handle), "fd_destroy")
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Trainer:
    """Streaming training step over clips of `chunks` latent frames (fd_train_create)."""

    def __init__(self, cfg, weights: Weights, chunks: int):
        L = lib()
        self.cfg = make_config(cfg)
        self.weights = weights
        self.chunks = int(chunks)
        out = _P()
        _check(L.fd_train_create(ctypes.byref(self.cfg), weights.handle, self.chunks,
                                 ctypes.byref(out)), "fd_train_create")
        self.handle = out
        import torch
        self.device = torch.cuda.current_device()
        self.grad_elems = L.fd_train_grad_elems(ctypes.byref(self.cfg))
        self._latent_bytes = self.chunks * L.fd_latent_bytes(ctypes.byref(self.cfg))
        self._target_bytes = self.chunks * L.fd_pixels_bytes(ctypes.byref(self.cfg))

    def step(self, latents, targets, loss, grads, stream=None) -> None:
        """latents fp32 [T][C'][H'][W'], targets fp32 [T][C][r_t][H][W], loss fp32 [1], grads
        fp32 [grad_elems], all on the trainer's device."""
        dev = self.device
        check_buffer(latents, "latents", self._latent_bytes, "float32", True, dev)
        check_buffer(targets, "targets", self._target_bytes * (4 if self.cfg.out_dtype ==
                                                                DTYPE_U8 else 1),
                     "float32", True, dev)
        check_buffer(loss, "loss", 4, "float32", True, dev)
        check_buffer(grads, "grads", 4 * self.grad_elems, "float32", True, dev)
        _check(lib().fd_train_step(self.handle, _ptr(latents), _ptr(targets), _ptr(loss),
                                   _ptr(grads), _stream_ptr(stream)), "fd_train_step")

    def status(self, stream=None) -> int:
        return lib().fd_train_status(self.handle, _stream_ptr(stream))

    def profile(self, enable: bool) -> None:
        _check(lib().fd_train_profile_enable(self.handle, 1 if enable else 0),
               "fd_train_profile_enable")

    def profile_collect(self) -> dict:
        """{kind name: (launches, device ms)} of the steps since the last collect."""
        n = len(TRAIN_KINDS)
        launches = (ctypes.c_int64 * n)()
        ms = (ctypes.c_double * n)()
        _check(lib().fd_train_profile_collect(self.handle, launches, ms),
               "fd_train_profile_collect")
        return {k: (int(launches[i]), float(ms[i])) for i, k in enumerate(TRAIN_KINDS)}

    def close(self) -> None:
        if getattr(self, "handle", None):
            _check(lib().fd_train_destroy(self.handle), "fd_train_destroy")
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def decode_chunks(decoders, latents, pixels, stream=None) -> None:
    n = len(decoders)
    if len(latents) != n or len(pixels) != n:
        raise ValueError("one latent and one pixel buffer per decoder")
    for d, z, p in zip(decoders, latents, pixels):
        d._check_buffers(z, p, True)
    hs = (_P * n)(*[d.handle for d in decoders])
    ls = (_P * n)(*[_ptr(x) for x in latents])
    ps = (_P * n)(*[_ptr(x) for x in pixels])
    _check(lib().fd_decode_chunks(hs, n, ls, ps, _stream_ptr(stream)), "fd_decode_chunks")


class Batch:
    """Stacked decode of up to max_streams decoders of one weights object (fd_batch_create):
    the GEMMs of a chunk run once on all streams' rows."""

    def __init__(self, cfg, weights: Weights, max_streams: int):
        self.cfg = make_config(cfg)
        self.weights = weights
        out = _P()
        _check(lib().fd_batch_create(ctypes.byref(self.cfg), weights.handle, int(max_streams),
                                     ctypes.byref(out)), "fd_batch_create")
        self.handle = out

    def decode(self, decoders, latents, pixels, stream=None) -> None:
        """One chunk for each decoder (fd_decode_batch)."""
        n = len(decoders)
        if len(latents) != n or len(pixels) != n:
            raise ValueError("one latent and one pixel buffer per decoder")
        for d, z, p in zip(decoders, latents, pixels):
            d._check_buffers(z, p, True)
        hs = (_P * n)(*[d.handle for d in decoders])
        ls = (_P * n)(*[_ptr(x) for x in latents])
        ps = (_P * n)(*[_ptr(x) for x in pixels])
        _check(lib().fd_decode_batch(self.handle, hs, n, ls, ps, _stream_ptr(stream)),
               "fd_decode_batch")

    def close(self) -> None:
        if getattr(self, "handle", None):
            _check(lib().fd_batch_destroy(self.handle), "fd_batch_destroy")
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# ------------------------------------------------------------------ kernel-level entry points
def op_linear(epi, A, W, bias, out, tup_hidden=0, bn=0, err=None, stream=None, pair=None
              ) -> None:
    """pair: None (fd_op_linear), or 0 / 1 / 2 (library choice / single CTAs / CTA pairs)."""
    M, K = A.shape
    N = W.shape[0]
    if pair is None:
        _check(lib().fd_op_linear(epi, M, N, K, _ptr(A), _ptr(W), _ptr(bias), _ptr(out),
                                  tup_hidden, bn, _ptr(err), _stream_ptr(stream)), "fd_op_linear")
    else:
        _check(lib().fd_op_linear_tiled(epi, M, N, K, _ptr(A), _ptr(W), _ptr(bias), _ptr(out),
                                        tup_hidden, bn, pair, _ptr(err), _stream_ptr(stream)),
               "fd_op_linear_tiled")


def op_rope_table(t, frames_per_chunk, rope_base, table, stream=None) -> None:
    _check(lib().fd_op_rope_table(t, frames_per_chunk, rope_base, _ptr(table),
                                  _stream_ptr(stream)), "fd_op_rope_table")


def op_qkv(A, Wqkv, bqkv, knorm_g, norm2_g, heads, groups, tokens, grid_w, frames_per_chunk,
           window, t, eps, rope_base, rope_t, q_out, k_ring, vt_ring, ring_pitch, bn=0, err=None,
           stream=None, qk_norm=False) -> None:
    """norm2_g: V's gain (KV-norm) or, with qk_norm, Q's gain."""
    M, K = A.shape
    _check(lib().fd_op_qkv(M, K, _ptr(A), _ptr(Wqkv), _ptr(bqkv), _ptr(knorm_g), _ptr(norm2_g),
                           1 if qk_norm else 0,
                           heads, groups, tokens, grid_w, frames_per_chunk, window, t, eps,
                           rope_base, _ptr(rope_t), _ptr(q_out), _ptr(k_ring), _ptr(vt_ring),
                           ring_pitch, bn, _ptr(err), _stream_ptr(stream)), "fd_op_qkv")


def attention_workspace_bytes(Lq, heads, groups, n_keys, parts=0) -> int:
    return lib().fd_attention_workspace_bytes(Lq, heads, groups, n_keys, parts)


def op_attention(q, k_ring, vt_ring, heads, groups, ring_pitch, n_keys, out, parts=0,
                 workspace=None, err=None, stream=None) -> None:
    """fd_op_attention; parts = CTAs of the persistent launch (0: one per SM)."""
    Lq = q.shape[0]
    _check(lib().fd_op_attention(Lq, heads, groups, _ptr(q), _ptr(k_ring), _ptr(vt_ring),
                                 ring_pitch, n_keys, _ptr(out), parts, _ptr(workspace),
                                 _ptr(err), _stream_ptr(stream)), "fd_op_attention")


def op_attention_static(q, k_ring, vt_ring, heads, groups, ring_pitch, n_keys, out, parts=0,
                        err=None, stream=None) -> None:
    """fd_op_attention with its workspace in the library's static device memory."""
    Lq = q.shape[0]
    _check(lib().fd_op_attention_static(Lq, heads, groups, _ptr(q), _ptr(k_ring), _ptr(vt_ring),
                                        ring_pitch, n_keys, _ptr(out), parts, _ptr(err),
                                        _stream_ptr(stream)), "fd_op_attention_static")


def op_kv_append(k, v, window, t, ring_pitch, k_ring, vt_ring, stream=None) -> None:
    G, rows, _ = k.shape
    _check(lib().fd_op_kv_append(_ptr(k), _ptr(v), G, rows, window, t, ring_pitch, _ptr(k_ring),
                                 _ptr(vt_ring), _stream_ptr(stream)), "fd_op_kv_append")


def op_rmsnorm(h, g, eps, u, stream=None) -> None:
    M, D = h.shape
    _check(lib().fd_op_rmsnorm(_ptr(h), _ptr(g), M, D, eps, _ptr(u), _stream_ptr(stream)),
           "fd_op_rmsnorm")


def op_rmsnorm_e4m3(h, g, eps, out_scale, u, stream=None) -> None:
    """u (uint8 tensor holding e4m3 codes) = e4m3(RMSNorm(h) g out_scale)."""
    M, D = h.shape
    _check(lib().fd_op_rmsnorm_e4m3(_ptr(h), _ptr(g), M, D, eps, out_scale, _ptr(u),
                                    _stream_ptr(stream)), "fd_op_rmsnorm_e4m3")


def op_linear_e4m3(epi, A, W, col_scale, bias, out, out_scale=1.0, bn=0, err=None,
                   stream=None) -> None:
    """FP8 linear: A [M][K], W [N][K] e4m3 codes (uint8 tensors), fp32 col_scale / bias."""
    M, K = A.shape
    N = W.shape[0]
    _check(lib().fd_op_linear_e4m3(epi, M, N, K, _ptr(A), _ptr(W), _ptr(col_scale), _ptr(bias),
                                   _ptr(out), out_scale, bn, _ptr(err), _stream_ptr(stream)),
           "fd_op_linear_e4m3")


def op_unshuffle(z, p, x0, stream=None) -> None:
    C, H, W = z.shape
    _check(lib().fd_op_unshuffle(_ptr(z), C, H, W, p, _ptr(x0), _stream_ptr(stream)),
           "fd_op_unshuffle")


def op_pixel_head(F, frames, grid_h, grid_w, channels, rs, out_dtype, pixels, stream=None) -> None:
    _check(lib().fd_op_pixel_head(_ptr(F), frames, grid_h, grid_w, channels, rs, out_dtype,
                                  _ptr(pixels), _stream_ptr(stream)), "fd_op_pixel_head")


def op_linear_pixel(A, W, bias, frames, grid_h, grid_w, channels, rs, out_dtype, pixels,
                    err=None, stream=None) -> None:
    """Head layer 2 with the pixel shuffle in its epilogue (fd_op_linear_pixel)."""
    M, K = A.shape
    _check(lib().fd_op_linear_pixel(M, K, _ptr(A), _ptr(W), _ptr(bias), frames, grid_h, grid_w,
                                    channels, rs, out_dtype, _ptr(pixels), _ptr(err),
                                    _stream_ptr(stream)), "fd_op_linear_pixel")


def op_scores_bwd(Q, dO, K, V, lse, delta, Pc, Lp, L, dS, dST, PT, err=None,
                  stream=None) -> None:
    """The attention's scores backward in one launch (fd_op_scores_bwd)."""
    M, N = Q.shape[0], K.shape[0]
    _check(lib().fd_op_scores_bwd(M, N, _ptr(Q), _ptr(dO), _ptr(K), _ptr(V), _ptr(lse),
                                  _ptr(delta), Pc, Lp, L, _ptr(dS), _ptr(dST), _ptr(PT), _ptr(err),
                                  _stream_ptr(stream)), "fd_op_scores_bwd")


def op_rmsnorm_bwd(x, g, dy, eps, dx, dg, stream=None) -> None:
    M, D = x.shape
    import torch
    work = torch.empty(M, D, dtype=torch.float32, device=x.device)
    _check(lib().fd_op_rmsnorm_bwd(_ptr(x), _ptr(g), _ptr(dy), M, D, eps, _ptr(dx), _ptr(dg),
                                   _ptr(work), _stream_ptr(stream)), "fd_op_rmsnorm_bwd")


def op_gelu_bwd(z, da, dz, dz_bf16, stream=None) -> None:
    _check(lib().fd_op_gelu_bwd(_ptr(z), _ptr(da), z.numel(), _ptr(dz), _ptr(dz_bf16),
                                _stream_ptr(stream)), "fd_op_gelu_bwd")


def op_l1_pixel_bwd(F, target, frames, grid_h, grid_w, channels, rs, dF, loss,
                    stream=None) -> None:
    import torch
    work = torch.empty((F.numel() + 255) // 256, dtype=torch.float32, device=F.device)
    _check(lib().fd_op_l1_pixel_bwd(_ptr(F), _ptr(target), frames, grid_h, grid_w, channels, rs,
                                    _ptr(dF), _ptr(loss), _ptr(work), _stream_ptr(stream)),
           "fd_op_l1_pixel_bwd")
