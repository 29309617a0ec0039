"""X-Cache chunk step on one GB300 (sm_103a).

The compute path is the CUDA library ``libxcache.so`` (C ABI in
``include/xcache.h`` / ``include/xcache_ops.h``); ``xcache`` is its ctypes
binding and ``rollout`` the AR inference driver over it.  Importing the
binding without the built library raises: there is no fallback path.
Build with ``python -m paper_2604_20289_gb300.build``.
"""
