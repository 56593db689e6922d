"""GB300 (sm_103a) library for the per-chunk revisit-consistency attention path.

The C ABI lives in include/crc.h and libcrc.so (built in-tree by
`paper_2607_21848_gb300.build`); `paper_2607_21848_gb300.api` is the Python
binding with the same entry-point names.  Importing this package loads nothing;
the library is loaded on first use and a missing library raises.
"""

__all__ = ["api", "build"]
