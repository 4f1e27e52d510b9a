"""GB300-native DriveCache hot path: C-ABI library libdrivecache.so
(include/drivecache.h) plus a thin ctypes binding.

    from paper_2608_16354_gb300 import binding as dc
    dc.plan(...), dc.Model(...), dc.denoise(...)

The library must be built first (``python -m paper_2608_16354_gb300._build``
or ``__graft_entry__.build()``); there is no CPU fallback.
"""
