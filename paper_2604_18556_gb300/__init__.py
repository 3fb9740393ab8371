"""GB300-native (sm_103a) GSQ relaxed-scalar-quantizer step.

The compute path is the C-ABI library `libgsq.so` (CUDA kernels under csrc/),
reached through the thin ctypes binding in `gsq.py`.  Importing this package
loads nothing; `from paper_2604_18556_gb300 import gsq` loads the library.
"""
