"""GB300-native delta-merge library: the element-wise TopKMask / TA / TIES /
ISO-retention pass over whole parameter sets, as hand-written CUDA for
sm_103a behind the C ABI in include/iso.h.  This package is the thin PyTorch
binding; see ``api`` for the entry points."""
from ._abi import IsoError, LIB_PATH  # noqa: F401
from .api import (FrameStats, frame_merge, frame_merge_factors, frame_workspace_size,  # noqa: F401
                  gemm_tf32, opt_step, opt_workspace_size, thin_svd)
from .api import (HostUpdate, Stats, Workspace, compact_candidates, force_two_pass, iso_delta, iso_merge,  # noqa: F401
                  iso_num_units, iso_topk_mask, iso_update, iso_update_host_staging_size,
                  iso_update_noalloc, iso_workspace_size, launch_count, range_hist, range_mask,
                  split_unit_topk, merge_cfg, profile_enable, profile_read, profile_reset, topk_cfg)
