"""NetKV decode-instance scoring on GB300 (sm_103a).

The package is the C-ABI library ``libnetkv.so`` (CUDA kernels under ``csrc/``,
declared in ``include/netkv.h``), its Python binding ``netkv`` and the one-step
pipeline ``pipeline.Scorer``.  Build the library with ``build.build()``.
"""
