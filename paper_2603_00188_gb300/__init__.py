"""ST-Lite KV-cache compression pass for GB300 (sm_103a).

``paper_2603_00188_gb300.stlite`` binds the C-ABI library ``libstlite.so``
(hand-written CUDA kernels); ``paper_2603_00188_gb300.synth`` draws seeded
synthetic GUI-trajectory caches.  Importing the package itself loads nothing.
"""
__all__ = ["stlite", "synth", "build"]
