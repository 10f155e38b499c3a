"""GB300-native byte-exact KV-state graft and GQA decode attention.

The compute path is libkvg.so (hand-written CUDA for sm_103a behind the C ABI
in include/kvg.h); ``paper_2607_14431_gb300.kvg`` is its ctypes binding and
``paper_2607_14431_gb300.build`` compiles it in-tree.
"""
__all__ = ["kvg", "build"]
