"""padoc_attn: ancestor-masked attention for PaDoc's layout-grounded parallel decoding on GB300.

``padoc_attn`` is the ctypes binding of the C ABI in include/padoc_attn.h; ``inputs`` draws the
seeded synthetic workloads; ``engine`` strings the calls of one decode step or one packed prefill
together for callers that hold torch tensors. The CUDA library is built in-tree by ``build``.
"""
from . import padoc_attn  # noqa: F401

__all__ = ["padoc_attn"]
