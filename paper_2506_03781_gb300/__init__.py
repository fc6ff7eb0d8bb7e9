"""GB300-native UniQuan_F weight quantizer (arXiv 2506.03781).

The compute path is a C-ABI shared library of hand-written sm_103a CUDA
kernels (``csrc/``, declared in ``include/uq_api.h``); ``api`` is a thin
ctypes binding with the same entry-point names.  Importing the package loads
nothing: the library is opened on first use by ``api`` and a missing library
raises instead of falling back to any other implementation.
"""

__version__ = "0.1.0"
