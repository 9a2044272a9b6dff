"""Bucket-Level MOO resolve on GB300 (sm_103a).

Python binding of the C ABI declared in ``include/bkmoo.h``.  The CUDA library
is loaded on first use (``paper_2606_05613_gb300.native``); importing the
package itself loads nothing, so the synthetic-input module
(``paper_2606_05613_gb300.inputs``) is usable without a GPU.
"""
__version__ = "0.1.0"
