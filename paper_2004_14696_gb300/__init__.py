"""GB300-native hot path of Dynamic Backup Workers (arXiv 2004.14696).

The compute lives in ``libdbw.so`` (hand-written CUDA for sm_103a behind a C ABI,
declared in ``include/dbw.h``); ``dbw`` is the thin ctypes binding with the same
entry-point names.  ``inputs`` and ``workloads`` produce seeded synthetic inputs.
"""
