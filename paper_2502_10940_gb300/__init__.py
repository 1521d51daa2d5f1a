"""CoLA auto-encoder layer (h = B sigma(A x), arXiv 2502.10940) on GB300.

The compute path is the C-ABI library ``libcola.so`` (hand-written sm_103a
kernels); ``paper_2502_10940_gb300.cola`` is its thin ctypes binding.  The
package imports nothing eagerly, so the pure-host modules (``inputs``,
``workloads``) stay importable without a GPU.
"""
__all__ = ["cola", "inputs", "workloads", "build"]
