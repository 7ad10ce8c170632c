"""SWAN decode hot path on GB300 (sm_103a): compress-on-append, decode
attention on the packed sparse KV cache, rotate-back.

The CUDA library (``libswan.so``) is loaded by :mod:`paper_2511_18936_gb300.swan`
on first use; importing this package alone loads nothing.
"""
__all__ = ["synth", "swan"]
