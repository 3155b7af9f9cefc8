"""GB300 (sm_103a) implementation of VarRate's KV-codec hot path (arXiv 2607.15498).

The compute lives in the CUDA library ``libvarrate.so`` behind the C ABI of include/varrate.h;
``paper_2607_15498_gb300.varrate`` is its thin Python binding and ``build`` compiles it.
"""
from . import varrate  # noqa: F401

__all__ = ["varrate"]
