"""GB300-native layer-wise KV-cache eviction (SnapKV / H2O / StreamingLLM routes).

The compute path is the C-ABI library ``lib/libkvev.so`` (hand-written CUDA for
sm_103a); :mod:`.kvev` is its thin ctypes binding.  Importing the package does
not load the library; the binding loads it on first use and raises if it is
missing.
"""
__all__ = ["kvev", "inputs"]
