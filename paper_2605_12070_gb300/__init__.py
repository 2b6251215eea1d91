"""GB300-native decoupled off-policy correction (arXiv 2605.12070).

The compute lives in ``libocc.so`` (CUDA for sm_103a, C ABI in include/occ.h);
``occ`` is its ctypes binding for torch tensors and ``workloads`` holds the
seeded synthetic input generators.  Importing the package loads nothing: the
library is opened on the first call.
"""

__all__ = ["occ", "workloads"]
