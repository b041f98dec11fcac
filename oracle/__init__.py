"""CPU oracle for the Kafila stage-decode step.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU
baseline / reference arm may import it.  The product path (``paper_2609_34045_gb300``) never
imports, links or runs anything here and fails loudly when its CUDA library is missing.

The oracle is a plain, slow, fp64 numpy restatement of one decode step of a pipeline stage
(a contiguous range of decoder blocks, plus the head's embedding, final norm, unembedding
and greedy sampler), written from the paper (Kafila, sections III and V-A) and from the
textbook definitions of its parts.  It shares no code with the CUDA path.
"""
from .stage import *  # noqa: F401,F403
