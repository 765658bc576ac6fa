"""LoCA forward-only adaptation hot path on one GB300 (sm_103a).

The CUDA library ``libloca.so`` (``csrc/``, C ABI in ``include/loca.h``) holds the kernels;
``paper_2608_03020_gb300.loca`` is its Python binding.  Build with ``_build.build()``.
"""

from . import loca  # noqa: F401
from .loca import (  # noqa: F401
    LOCA_BF16,
    LOCA_F32,
    LocaError,
    Pass,
    loca_accumulate,
    loca_calib_fit,
    loca_device_status,
    loca_error,
    loca_ridge_solve,
    loca_targets,
    loca_version,
)
