"""Seer (arXiv 2607.14557) hot path on one GB300: a C-ABI library of
hand-written sm_103a kernels (``libseer.so``, see ``include/seer.h``), its
ctypes binding (:mod:`.seer`) and a one-GPU denoising-step driver
(:mod:`.driver`)."""

__all__ = ["seer", "driver", "build"]
