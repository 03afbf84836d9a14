"""GB300 (sm_103a) chunk-wise causal attention for streaming video DiTs.

The compute path is the C-ABI library ``libfastvr_attn.so`` built from
``csrc/``; ``fastvr`` is its thin Python binding.  Importing this package does
not load the library; ``fastvr`` does, and fails loudly when it is missing.
"""
__all__ = ["fastvr", "workloads"]
