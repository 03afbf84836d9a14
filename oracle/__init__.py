"""CPU oracle for chunk-wise causal attention -- TEST INFRASTRUCTURE ONLY.

Plain float64 NumPy written from Sec. 3.1 and Eq. 1 of the FastVR paper.  Only
tests/, the smoke check and the benchmark's CPU-baseline leg (and its reference
arm) may import it; the library never does, and the two share no code.
"""
from . import attention, kv_cache  # noqa: F401
