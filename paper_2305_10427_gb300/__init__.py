"""GB300-native parallel (Jacobi / GS-Jacobi) decoding for encoder-decoder translation models.

The compute lives in ``libpd.so`` (CUDA for sm_103a, C ABI in ``include/pd.h``); this package
is its Python binding.  Build the library with ``__graft_entry__.build()`` (or
``paper_2305_10427_gb300.build.build()``).
"""
from ._binding import (Config, DecodeResult, Decoder, PdError, METHODS, EXPORTED, LIB_PATH,
                       load_library, weights_nbytes)

__all__ = ["Config", "DecodeResult", "Decoder", "PdError", "METHODS", "EXPORTED", "LIB_PATH",
           "load_library", "weights_nbytes"]
