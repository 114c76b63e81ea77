"""CAST per-block anchor/skip step on one GB300: routing, routed anchor attention and
Phase-Aware Reconstruction as hand-written sm_103a kernels behind a C ABI (include/cast.h).

`paper_2609_34144_gb300.native` is the ctypes binding of the built library
(paper_2609_34144_gb300/_lib/libcast.so); importing it fails loudly when the library is
missing.
"""
