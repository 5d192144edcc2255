"""GB300 (sm_103a) implementation of the ResNet-18 training step of the hybrid
dual-batch / cyclic-progressive learning scheme (arXiv 2509.26092).

Submodules are imported lazily: ``synth`` (seeded synthetic inputs) needs no
GPU, while ``dbl`` (the ctypes binding of ``libdbl.so``) and ``resnet18`` (the
two-stream training-step driver) need the compiled CUDA library.
"""
__all__ = ["synth", "dbl", "resnet18"]
