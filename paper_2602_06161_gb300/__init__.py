"""COVER override attention + seed scoring on one GB300 (sm_103a).

The compute path is libcover.so (hand-written CUDA, C ABI in include/cover.h);
this package only loads it and marshals torch tensors into it.
"""
from .api import (  # noqa: F401
    cover_attn_fwd, cover_attn_fwd_f32, cover_attn_fwd_prefix, cover_attn_fwd_prefix_f32, cover_seed_route, cover_score_fwd, cover_score_fwd_noalloc,
    cover_score_workspace_bytes, cover_score_decide_fwd, cover_seed_select_fwd, cover_attn_mass_fwd,
    cover_attn_mass_workspace_bytes, COVER_DECIDE_ALL, COVER_DECIDE_UPDATE, cover_seed_kv_gather, cover_seed_kv_override, cover_decide_workspace_bytes, decide_workspace,
    score_workspace, cover_device_status, cover_status_str, cover_debug_umma_tile, cover_debug_wait_timeout,
)
from ._lib import CoverError, load as load_library  # noqa: F401
