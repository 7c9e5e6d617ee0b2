"""GB300 (sm_103a) DVI: self-speculative decode step and online drafter update.

The compute path is libdvi.so (csrc/, C-ABI in include/dvi.h); `dvi` is its
ctypes binding and `build` compiles it in-tree with nvcc.
"""
from .dvi import (DVIEngine, DeviceWeights, DVIError, lib, update_config, LIB_PATH, EXPORTS,  # noqa: F401
                  DVI_F32, DVI_BF16)
