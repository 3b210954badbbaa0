"""GB300 (sm_103a) implementation of the PalQuant parallel low-precision convolution layer.

PalQuant (Hu et al., arXiv 2208.01944) expands a layer's channels G times, splits them into
G groups, quantises each group's activations and weights to B bits and runs a B-bit group
convolution (Sec. 4.1); a cyclic permutation moves every group's output to the next group
(Sec. 4.2, Eq. 6-8).  The compute path is the C-ABI library ``libpalquant.so`` built from
``csrc/`` (hand-written CUDA for sm_103a); :mod:`.binding` is its thin ctypes binding.

Importing the package loads nothing; ``binding`` loads the shared library on first use and
raises if it has not been built.
"""
__all__ = ["binding", "synth", "workloads"]


def __getattr__(name):
    if name in __all__:
        import importlib

        return importlib.import_module("." + name, __name__)
    raise AttributeError(name)
