"""GB300-native Gated VLA-Cache step: a C-ABI CUDA library (libvlac.so,
declared in include/vlac.h) and its Python binding."""
from .build import build
from .vlac import (BF16, F32, MARGIN_LOGIT, MARGIN_PROB, MARGIN_VOCAB, REDUCE_DEFAULT, REDUCE_MEAN, REDUCE_MIN,
                   Cache, Context, VlacError, lib)

__all__ = ["build", "lib", "Context", "Cache", "VlacError", "F32", "BF16", "MARGIN_PROB", "MARGIN_LOGIT", "MARGIN_VOCAB",
           "REDUCE_DEFAULT", "REDUCE_MEAN", "REDUCE_MIN"]
