"""GB300-native block-restricted bidirectional selective scan (BDLM Mamba-H).

The computation lives in the CUDA library ``lib/libbdscan.so`` (sources in
``csrc/``, C ABI in ``include/bdscan.h``). ``binding`` is its ctypes binding
(same function names as the C ABI), ``layer`` keeps device tensors and
workspaces for repeated calls, and ``inputs`` draws the seeded synthetic
workloads. Loading is lazy: importing the package does not touch the GPU,
and any call raises if the CUDA library cannot be loaded.
"""

from . import binding, inputs  # noqa: F401

__all__ = ["binding", "inputs"]
