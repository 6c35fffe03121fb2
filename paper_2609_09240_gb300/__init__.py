"""GB300-native packed ternary (W1.58A16) linear layer.

The compute path is the CUDA library ``libtq.so`` (built from ``csrc/`` for
sm_103a) behind the C ABI of ``include/tq.h``; ``tq`` is a thin ctypes
binding with the same entry-point names.  Importing this package loads
nothing; ``tq.lib()`` loads the library and raises if it is missing.
"""
