"""GB300-native multipoint post-training quantization (arXiv 2002.09049).

The compute path lives in the C-ABI library ``libmpq.so`` (hand-written CUDA for sm_103a, built
from ``csrc/``); ``binding`` marshals torch tensors into its entry points.  There is no CPU
fallback: calling an entry point without the compiled library raises.
"""
from . import workloads, overhead  # noqa: F401

__all__ = ["workloads", "overhead"]


def __getattr__(name):
    # the binding loads the CUDA library lazily, on first use
    if name in ("binding",) or name.startswith("mpq_"):
        from . import binding
        return binding if name == "binding" else getattr(binding, name)
    raise AttributeError(name)
