"""GB300-native hot path of fully quantized training (arXiv 2010.14298).

The CUDA library (``_lib/libfqt.so``, C ABI in ``include/fqt.h``) quantizes
the output gradient of a linear / im2col-conv layer with PTQ, PSQ or BHQ and
runs the two low-bit contractions grad_X and grad_W.  ``fqt`` is the thin
ctypes binding; importing this package loads nothing until it is used.
"""
__all__ = ["fqt", "workloads"]


def __getattr__(name):
    if name in ("fqt", "workloads"):
        import importlib
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
