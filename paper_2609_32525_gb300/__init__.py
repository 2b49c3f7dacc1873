"""GB300-native slice -> token mix -> deslice library (Transolver coupling).

The compute lives in the C-ABI shared library built from csrc/ (declared in
include/flashslice.h); `flashslice` is its thin Python binding (argument
marshalling only).  `workloads` holds the seeded synthetic inputs.
Importing the package does not load the library; importing `flashslice` does,
and fails loudly if it has not been built.
"""
