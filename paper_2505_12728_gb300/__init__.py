"""GB300-native (sm_103a) verification step of SpecFLASH speculative decoding.

The package holds the CUDA kernels and C-ABI library (``csrc/``), the ctypes
binding (``specflash_verify``) and the seeded synthetic workloads
(``workloads``).  Importing the package loads nothing; the binding loads the
compiled library on first use and raises if it is missing.
"""
__all__ = ["workloads", "specflash_verify"]
