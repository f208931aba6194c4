"""GB300-native (sm_103a) implementation of the SMem reader hot path
(arXiv 2609.32395): block-local causal self-attention plus block-causal
cross-attention over a block-paged bf16 memory cache, served as one-block
prefill and batched decode through a C ABI (include/smem.h).

``paper_2609_32395_gb300.smem`` is the thin Python binding of that ABI.
"""
from . import smem  # noqa: F401
from .smem import SmemCache, SmemConfig, SmemError, make_config  # noqa: F401

__all__ = ["smem", "SmemCache", "SmemConfig", "SmemError", "make_config"]
