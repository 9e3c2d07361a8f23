"""GB300-native projected-gradient attribution (Bergson's TrackStar-style path).

The compute lives in ``libbergson.so`` (CUDA for sm_103a) behind the C ABI of
``include/bergson.h``; ``binding`` exposes the same entry points to Python.
"""
from .binding import (  # noqa: F401
    bergson_store_load, bergson_store_save,
    BERGSON_LAYER_BIAS,
    BERGSON_FISHER_INV, BERGSON_FISHER_INV_SQRT, bergson_fisher_fit, bergson_fisher_fit_workspace,
    bergson_fisher_preconditioner, bergson_fisher_preconditioner_workspace,
    bergson_fisher_preconditioner_tol,
    bergson_precondition_rows,
    BERGSON_AGG_MEAN, BERGSON_AGG_SUM, bergson_aggregate_rows, bergson_aggregate_rows_workspace,
    BERGSON_EALIGN, BERGSON_ECUDA, BERGSON_EDEVICE_TIMEOUT, BERGSON_EINVAL, BERGSON_EUNSUPPORTED,
    BERGSON_EMOMENT,
    BERGSON_EWORKSPACE, BERGSON_OK, BERGSON_PROJ_GAUSSIAN, BERGSON_PROJ_IDENTITY,
    BERGSON_PROJ_RADEMACHER, BERGSON_PROJ_UNIFORM, BergsonError,
    EXPORTED, LIB_PATH, Layer, bergson_build_store, bergson_debug_inject_status,
    bergson_build_store_blocks, bergson_score_topk_update, bergson_score_topk_update_workspace,
    bergson_score_topk_host, bergson_score_topk_host_workspace,
    bergson_debug_attr_once,
    bergson_debug_project_plan, bergson_debug_score_plan, bergson_debug_xgemm_plan,
    bergson_debug_wait_probe, bergson_last_error, bergson_module_seeds, bergson_project_grads,
    bergson_project_grads_noalloc, bergson_project_grads_workspace, bergson_projection_matrix, bergson_score_topk,
    bergson_score_bottomk,
    bergson_score_topk_workspace, bergson_score_grads, bergson_score_grads_workspace,
    bergson_sync_status, bergson_token_scores, bergson_token_scores_workspace, bergson_version, bergson_layer, lib,
    workspace_tensor,
)
