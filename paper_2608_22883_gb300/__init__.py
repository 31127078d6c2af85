"""GB300-native FOVEA visual-evidence path (memory build, retrieve, fuse).

The work runs in libfovea.so (CUDA kernels for sm_103a behind the C ABI in
include/fovea.h); ``fovea`` is its thin Python binding.
"""

from . import fovea  # noqa: F401
from .fovea import (  # noqa: F401
    BF16, FP32, FoveaError, Memory, Params, build_memory, new_workspace, retrieve_fuse,
    step, sync_errors, timing_enable, timing_read, workspace_size,
)
