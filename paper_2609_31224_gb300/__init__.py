"""GB300 (sm_103a) library for acoustic-to-text KV eviction and retained-cache
GQA attention ("Acoustic-to-Text KV Compression for Full-Duplex Speech
Models", Sec. 3.1 and Sec. 3.3).

The compute path is the CUDA library ``libkvc.so`` (C interface in
``include/kvc.h``); this package is its thin Python binding.
"""
from ._lib import (KVC_ACOUSTIC, KVC_ASR_DELIM, KVC_BF16, KVC_F32, KVC_TEXT, KVC_TRANSCRIPT,
                   KVC_UNIT_BEGIN, Config, KVCache, KvcError, load_library, query_sizes)

__all__ = ["KVCache", "KvcError", "Config", "load_library", "query_sizes", "KVC_F32", "KVC_BF16",
           "KVC_ACOUSTIC", "KVC_ASR_DELIM", "KVC_TRANSCRIPT", "KVC_TEXT", "KVC_UNIT_BEGIN"]
