"""GB300 (sm_103a) FlashDecoder streaming decoder: C-ABI library + thin Python binding."""
from . import flashdec  # noqa: F401
from .flashdec import Decoder, Weights, decode_chunks, lib, make_config, pack_blob  # noqa: F401
