"""Prefix-cached paged attention for GB300 (sm_103a).

The CUDA library ``libpkv.so`` (built from ``csrc/``) exports a C ABI
(``include/pkv.h``); :mod:`paper_2605_11232_gb300.pkv` is a thin ctypes binding
with the same names.  :mod:`paper_2605_11232_gb300.workloads` generates the
seeded synthetic inputs.  Importing the package does not load the library.
"""

__all__ = ["pkv", "workloads"]
