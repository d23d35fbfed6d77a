"""CPU oracle for the FlashDecoder streaming decode and its training step (test
infrastructure only; the training step is the submodule ``oracle.training``).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference arm
may import this package. The CUDA library and its Python binding never do.
"""
from .flashdecoder import (  # noqa: F401
    FLOPS, StreamingDecoder, attention, chunk_mask, decode_full_masked, decode_stream, gelu,
    kv_cache_elems, linear, pixel_shuffle, pixel_unshuffle, quantize_u8, reset_flops,
    e4m3, fp8_mlp_scales, fp8_weight, operand_rounding, pow2_ceil, rms_norm, rope, rope_bands,
    silu,
)
