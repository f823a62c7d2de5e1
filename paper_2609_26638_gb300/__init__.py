"""GB300-native greedy self-speculative draft/verify decoding (libgs + thin binding).

The compute lives in ``libgs.so`` (CUDA for sm_103a, C ABI in include/gs.h).
``paper_2609_26638_gb300.gs`` is the ctypes binding; ``runtime.Engine`` holds
the torch-owned device buffers.  Submodules are imported on use so that the
build step can run without the library.
"""
