"""GB300-native foreground-only block-sparse attention (UltraTex hot path).

The compute lives in libultratex.so (hand-written sm_103a CUDA behind the C ABI
of include/ultratex.h); this package holds its ctypes binding, the build step
and the end-to-end path that chains the five entry points.
"""
from .ultratex import (  # noqa: F401
    UT_BF16, UT_F32, UT_BG_FILL, UT_BG_KEEP, UT_BG_ZERO, UT_MASK_BITMAP, UT_MASK_TOPK, UtError, attn_shape,
    check_status, lib, status_word, ut_block_mask, ut_bsattn_bwd, ut_bsattn_fwd, ut_fg_compact, ut_fg_scatter,
    ut_topk_count,
)
