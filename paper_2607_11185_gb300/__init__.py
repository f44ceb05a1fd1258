"""GB300-native Visual Context Segmentation hot path.

``paper_2607_11185_gb300.vcs`` is the thin ctypes binding over ``libvcs.so``
(the C-ABI declared in ``include/vcs.h``).  ``workloads`` draws the seeded
synthetic inputs.  Importing this package loads nothing; importing ``vcs``
loads the shared library and fails loudly if it has not been built.
"""
