"""libstagefrontier: frontier accounting over per-(step, rank, stage) telemetry on GB300.

The compute path is the CUDA library ``libstagefrontier.so`` (C ABI in
``include/stagefrontier.h``); ``paper_2606_06751_gb300.stagefrontier`` is its
thin Python binding and ``paper_2606_06751_gb300.build`` compiles it.
"""


def load():
    """Import the binding (raises ImportError if the library is not built)."""
    from . import stagefrontier
    return stagefrontier
