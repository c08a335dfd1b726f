"""GB300-native verifier hot path of VideoSpeculateRAG (libfvrag).

The compute path is ``libfvrag.so`` (hand-written sm_103a CUDA behind a C ABI,
declared in ``include/fvrag.h``); ``paper_2601_01513_gb300.fvrag`` is the thin
ctypes binding.  Importing this package loads nothing: the binding loads the
library on first use and raises if it is missing.
"""
