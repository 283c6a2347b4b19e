"""GB300 (sm_103a) speculative-step attention of BudgetDraft (arXiv 2606.00144).

The hot path (KV-budget selection, gamma drafter decode passes over the sparse view, the
verifier's causal block pass, the log-sum-exp merge and the greedy acceptance) lives in
libbudgetdraft.so (hand-written CUDA, C ABI in include/budgetdraft.h).  This package holds
its build step, a thin ctypes binding, a step runner, a pipelined host-buffer driver and the
seeded synthetic workloads.
"""

from .binding import (  # noqa: F401
    BD_DRAFT_VIEW_READY,
    BD_SELECT_WINDOW_READY,
    BD_DTYPE_BF16,
    BD_DTYPE_F32,
    BD_OP_DRAFT,
    BD_OP_SELECT,
    BD_OP_VERIFY,
    BdShape,
    BudgetDraftError,
    Workspace,
    bd_accept,
    bd_advance,
    bd_argmax,
    bd_check_wait_timeout,
    bd_combine,
    bd_draft_attn,
    bd_draft_attn_static,
    bd_draft_static_status,
    bd_select_budget,
    bd_strerror,
    bd_verify_attn,
    bd_workspace_size,
    bd_workspace_status,
    bd_write_block_rows,
    library,
    make_shape,
    shape_of,
)
from .build import LIB_PATH, build  # noqa: F401
from .hostio import HostStepIO  # noqa: F401
from .step import SpecStep  # noqa: F401
