"""GB300-native PARD speculative decode step (arXiv 2504.18583).

The hot path -- parallel draft with mask tokens, target verification,
greedy / speculative-sampling acceptance, KV commit and rollback -- lives in
``libpard.so`` (hand-written CUDA for sm_103a behind a C ABI declared in
``include/pard.h``).  ``pard`` is its Python binding.
"""
from ._build import build, LIB  # noqa: F401


def load():
    """Import the binding (raises if libpard.so has not been built)."""
    from . import pard
    pard.lib()
    return pard
