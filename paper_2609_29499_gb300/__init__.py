"""GB300-native implementation of TASP's compiled sparse execution path.

``csrc/`` holds the CUDA kernels (sm_103a), the host mask compiler and the
runtime behind the C ABI declared in ``include/tasp.h``; ``tasp`` is the thin
ctypes binding; ``build`` compiles ``libtasp.so`` in-tree.
"""
