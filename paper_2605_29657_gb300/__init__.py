"""OccamToken prune path for GB300 (sm_103a).

Register-anchored relative evidence testing over visual tokens: Stage-I
[CLS]/mutual scores, the per-segment register threshold, Stage-II text scores,
the per-sample register threshold, and order-preserving compaction of the
kept rows -- all in the CUDA kernels of liboccam.so, reached through its C ABI
(include/occam.h). This package is the thin Python binding of that ABI.
"""

from ._lib import (  # noqa: F401
    OCCAM_REF_SAMPLE,
    OCCAM_REF_SEGMENT,
    OCCAM_ROUTE_AUTO,
    OCCAM_ROUTE_NARROW,
    OCCAM_ROUTE_TWOPASS,
    OCCAM_RULE_BUDGET,
    OCCAM_RULE_MEAN,
    OCCAM_RULE_REGISTER,
    OCCAM_STAGE1_CLS,
    OCCAM_STAGE1_MUTUAL,
    BatchLayout,
    OccamError,
    PruneCall,
    alloc_workspace,
    library,
    occam_budget_keep,
    occam_calibrate_lambda2,
    occam_compact,
    occam_compact_noalloc,
    occam_construct_registers,
    occam_get_status,
    occam_last_call_kernels,
    occam_mean_reference,
    occam_pool_scores,
    occam_selftest_wait,
    occam_set_stage2_route,
    occam_prune,
    occam_score_stage1,
    occam_score_stage2,
    occam_threshold,
    occam_version,
    occam_workspace_size,
)
