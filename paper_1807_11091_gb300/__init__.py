"""GB300-native (sm_103a) structured-pruned CONV forward (StructADMM, arXiv 1807.11091).

The compute path lives in the CUDA library libsadmm (csrc/, C ABI in
include/sadmm.h); ``sadmm`` is its ctypes binding.
"""
from . import build
from .sadmm import (  # noqa: F401
    SADMM_BF16, SADMM_FP32, SADMM_COL_NONE, SADMM_COL_SHAPE, SADMM_COL_CHANNEL,
    SadmmError, PrunedConv, project_groups, load, make_desc,
)
