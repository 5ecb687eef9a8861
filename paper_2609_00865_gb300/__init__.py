"""libmw Python binding: view-consistent scoring of compressed rollouts on GB300.

The compute path lives in ``libmw.so`` (hand-written CUDA for sm_103a behind
the C ABI of ``include/mw.h``); this package only marshals arguments. Import
fails loudly on first use when the library has not been built.
"""

from ._lib import (  # noqa: F401
    MW_BF16,
    MW_F32,
    MWError,
    TILE,
    Visibility,
    VisLayout,
    build_visibility,
    diverging_rows,
    exported_names,
    flatten_record,
    forward_kl_bwd,
    forward_kl_fwd,
    kernel_launches,
    logdiff,
    logical_positions,
    logprob_loss_bwd,
    logprob_loss_fwd,
    masked_attn_bwd,
    masked_attn_fwd,
    masked_attn_rope_bwd,
    masked_attn_rope_fwd,
    mw_build_visibility,
    mw_build_visibility_noalloc,
    mw_logprob_check_status,
    mw_logprob_loss_bwd,
    mw_logprob_loss_fwd,
    mw_logprob_loss_fwd_kl,
    mw_logprob_ws,
    mw_masked_attn_bwd,
    mw_masked_attn_bwd_ws,
    mw_logical_positions,
    mw_masked_attn_fwd,
    mw_masked_attn_rope_bwd,
    mw_masked_attn_rope_fwd,
    mw_masked_attn_rope_ws,
    mw_selftest_wait_timeout,
    mw_visibility_layout,
    rope_n_pos,
    rope_rows,
    rope_table,
)
