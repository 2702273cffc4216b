"""GB300 (sm_103a) library for the tensor-parallel shard of a Llama-style decoder layer.

The compute path is the CUDA library libvoltron.so (C ABI in include/voltron.h); `vt` is its thin
ctypes binding with the same function names, and `stack` wires a model, a partition and a KV cache
together from per-layer weight arrays.
"""
from . import vt  # noqa: F401

__all__ = ["vt"]
