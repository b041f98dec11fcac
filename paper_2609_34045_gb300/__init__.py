"""GB300-native (sm_103a) stage-decode engine for Kafila's hot path.

The decode-time forward pass of one pipeline stage (decoder blocks [l0, l1), plus the head's
embedding gather, final RMSNorm, lm_head and greedy argmax) in hand-written CUDA behind the C
ABI of ``include/kafila_stage.h``.  ``stage`` is the Python binding of that ABI (argument
marshalling only), ``workload`` the seeded synthetic inputs, ``build`` the nvcc build step.
"""
from . import workload  # noqa: F401


def build() -> str:
    """Compile ``libkafila_stage.so`` for sm_103a (in-tree); returns its path."""
    from .build import build as _build
    return _build()
