"""GB300-native (sm_103a) CacheRepair online repair path.

The compute lives in libcacherepair.so (csrc/, C ABI in include/cr.h); this
package is its build script and a ctypes binding with the same names.
"""
from . import build, cr  # noqa: F401
from .session import (RepairSession, RepairPipeline, TrainSession, pack_host_weights,  # noqa: F401
                      host_to_device, dims_from, trained_tensor_names)

__all__ = ["build", "cr", "RepairSession", "RepairPipeline", "TrainSession", "pack_host_weights",
           "host_to_device", "dims_from", "trained_tensor_names"]
