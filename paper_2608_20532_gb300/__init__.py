"""GF(2) encoder learning on one GB300: batched streaming Gaussian elimination,
affine-map extraction and batched encoding with a span check.

The compute path is ``libf2gpu.so`` (hand-written CUDA for sm_103a, C ABI in
``include/f2gpu.h``); ``binding`` marshals torch device tensors into it.
``workloads`` synthesises the seeded benchmark inputs.  Importing the package
loads nothing; the library is loaded on first use and its absence is an error.
"""

__all__ = ["binding", "workloads", "build"]


def __getattr__(name):
    if name in __all__:
        import importlib

        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
