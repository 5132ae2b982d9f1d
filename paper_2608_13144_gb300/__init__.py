"""GB300-native certified cache lookup of LipCache (arxiv 2608.13144).

The compute path is liblipcache.so (hand-written CUDA for sm_103a behind the
C ABI in include/lipcache.h); this package only loads it and marshals
arguments.
"""
from ._lib import LipCacheError, load  # noqa: F401


def __getattr__(name):
    if name == "LipCache":
        from .lipcache import LipCache
        return LipCache
    raise AttributeError(name)
