"""GB300 (sm_103a) token selection for LiteVLM (arXiv 2506.07416).

The compute path is the C-ABI library ``liblitevlm_select.so`` (CUDA kernels
under ``csrc/``); ``select`` is its thin ctypes binding. Importing this package
loads nothing: ``from paper_2506_07416_gb300 import select`` does.
"""
__all__ = ["inputs", "select"]
