"""MoE-ViE fine-grained MoE FFN layer forward for GB300 (sm_103a).

The computation lives in ``libmoevie.so`` (CUDA kernels behind the C ABI of
``include/moevie.h``).  ``paper_2608_17402_gb300.moevie`` is the thin ctypes
binding with the same entry-point names; import it explicitly.  Importing this
package itself loads nothing.
"""
__all__ = ["moevie"]
