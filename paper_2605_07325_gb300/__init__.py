"""CSR incremental-prefill attention over a paged GQA KV cache, for GB300 (sm_103a).

The compute path is the C-ABI library ``libcsr.so`` (hand-written CUDA kernels)
behind the thin ctypes binding in :mod:`paper_2605_07325_gb300.csr`.  Importing
this package does not load the library; ``from paper_2605_07325_gb300 import csr``
does, and fails loudly when it has not been built.
"""
__all__ = ["csr", "synth", "costmodel"]
