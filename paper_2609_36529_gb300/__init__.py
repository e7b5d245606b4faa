"""GB300-native triadic linear attention (chunkwise forward/backward and decode).

The compute path is the CUDA library ``libtla.so`` built from ``csrc/``;
``paper_2609_36529_gb300.tla`` is its thin ctypes binding.  Importing this
package does not load the library; the binding loads it on first use and
raises if it is missing.
"""
__all__ = ["inputs", "tla"]
