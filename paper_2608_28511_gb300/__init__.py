"""GB300-native (sm_103a) dropless routed MoE layer: C-ABI library + binding.

``abi`` is the ctypes binding of ``include/moe.h`` (one function per entry
point); ``layer.MoeLayer`` owns the device buffers of one layer step and calls
the entry points in order.  The library ``libmoe.so`` is built in-tree by
``_build.build()`` (``__graft_entry__.build()`` at the repository root).
"""
from . import abi  # noqa: F401

__all__ = ["abi"]
