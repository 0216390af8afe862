"""GB300-native Early-Bird (EB) decoding step for diffusion LLMs.

The compute path is libebd.so (C ABI, include/ebd.h); `_ebd` is its ctypes
binding and `runtime` holds the PyTorch plumbing (device buffers, streams)
used by the tests and the benchmark.  Importing the package does not load
the library; `_ebd.load()` does, and fails loudly if it is missing.
"""
__all__ = ["_ebd", "build", "runtime"]
