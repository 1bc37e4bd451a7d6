"""qx: exact integer GEMM substrate for GB300 (sm_103a).

The compute path lives in the CUDA library ``libqx.so`` built from ``csrc/``;
``paper_2606_09905_gb300.qx`` is the ctypes binding over its C ABI
(``include/qx.h``).  Importing this package loads nothing: the library is
opened on first use and a missing or unbuilt library is an error, never a
fallback.
"""

__all__ = ["qx", "inputs"]
