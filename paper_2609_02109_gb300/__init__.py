"""GB300-native MeanField joint-configuration scorer (arXiv 2609.02109).

The compute path is the C-ABI library built from ``csrc/`` (see
``include/mf.h``); ``paper_2609_02109_gb300.mf`` is its thin ctypes binding.
``paper_2609_02109_gb300.workload`` draws seeded synthetic inputs.  Importing
the package itself loads nothing.
"""
__all__ = ["mf", "workload"]
