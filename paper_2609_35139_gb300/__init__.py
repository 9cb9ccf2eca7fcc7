"""GB300-native (sm_103a) CacheRepair online repair path.

The compute lives in libcacherepair.so (csrc/, C ABI in include/cr.h); this
package is its build script and a ctypes binding with the same names.
"""
from . import build, cr  # noqa: F401
from .session import (RepairSession, RepairPipeline, pack_host_weights, host_to_device,  # noqa: F401
                      dims_from)

__all__ = ["build", "cr", "RepairSession", "RepairPipeline", "pack_host_weights", "host_to_device",
           "dims_from"]
