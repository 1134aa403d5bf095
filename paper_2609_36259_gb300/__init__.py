"""CyFA (Cyclic Flow Attention) core operator for GB300 (sm_103a).

The compute lives in ``libcyfa.so`` (hand-written CUDA, C ABI of ``include/cyfa.h``);
``paper_2609_36259_gb300.cyfa`` is the thin Python binding over it.  Importing this package
loads nothing; the library is loaded on first use of the binding and its absence is an
error, never a fallback.
"""
__all__ = ['cyfa', 'synth', 'build_lib']
