"""GB300 (sm_103a) decode path of codec-token speech synthesis with multi-token
prediction heads and Viterbi-based selection (arXiv 2410.13839, Sec. III).

The computation lives in libmtp.so (C ABI: include/mtp.h, sources in csrc/);
`paper_2410_13839_gb300.mtp` is its Python binding.  `build.build()` compiles
the library in-tree for sm_103a.
"""
import importlib

__all__ = ["build", "mtp"]


def __getattr__(name):
    if name in __all__:
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
