"""GB300-native heterogeneous data-parallel SGD step (arXiv 2110.08941).

The product is libhs.so (C ABI in include/hs.h, CUDA kernels for sm_103a under csrc/).
``paper_2110_08941_gb300.binding`` is its Python binding; every name of the binding is
also reachable from the package itself (``paper_2110_08941_gb300.hs_step`` and so on).
The binding loads the library on first use and raises ImportError if it was not built;
``python -m paper_2110_08941_gb300.build`` builds it without loading it.
"""
import importlib as _importlib


def __getattr__(name):
    if name.startswith("__"):
        raise AttributeError(name)
    if name in ("build", "binding"):
        return _importlib.import_module(f"{__name__}.{name}")
    binding = _importlib.import_module(__name__ + ".binding")
    return getattr(binding, name)
