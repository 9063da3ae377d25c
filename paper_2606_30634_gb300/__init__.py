"""GB300 (sm_103a) implementation of the one-step-delayed AdamW step with
Error Feedback (arXiv 2606.30634): a C-ABI library (include/dpo.h) of
hand-written CUDA kernels, with a thin Python binding in ``dpo``.

Submodules load their native libraries on first use; importing the package
itself loads nothing.
"""
__all__ = ["dpo", "synth", "build"]
