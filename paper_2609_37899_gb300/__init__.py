"""GB300-native SPSA training step for SOMA byte-LSTM experts.

The compute path lives in ``libsoma.so`` (hand-written CUDA for sm_103a behind
a C ABI, declared in ``include/soma_api.h``); ``api`` is its thin ctypes
binding.  Importing this package loads nothing: ``api`` loads the library on
first use and raises if it is missing.
"""
__all__ = ["api", "inputs"]
