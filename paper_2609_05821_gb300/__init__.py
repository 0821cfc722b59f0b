"""GB300-native Conduit scoring pass and budgeted selective refresh.

Submodules: ``conduit`` (binding of the libconduit C ABI, loads the CUDA
library), ``pipeline`` (the whole refresh step over one batch), ``synth``
(seeded synthetic workloads) and ``_build`` (nvcc build of the library).
Importing the package itself loads nothing.
"""

__all__ = ["conduit", "pipeline", "synth"]
