"""GB300-native streaming frame-chunk attention (3D RoPE, rolling KV cache,
block-causal flash attention) behind a C ABI (``include/frt.h``).

Importing the package loads nothing native; ``paper_2607_18171_gb300.frt``
loads ``libfrt.so`` on first use and raises if it is missing.
"""
__all__ = ["synth"]
