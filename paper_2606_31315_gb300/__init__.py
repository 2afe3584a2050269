"""GB300 (sm_103a) block-verify hot path of BlockPilot (arxiv 2606.31315).

The computation lives in ``libblockpilot.so`` (hand-written CUDA behind the C ABI of
``include/blockpilot.h``); this package only builds it and marshals torch tensors into
it.  Importing the package does not load the library; the first call does, and raises
if the library is missing -- there is no CPU fallback.
"""
from ._binding import (  # noqa: F401
    BF16,
    F32,
    MASK_BIDIR,
    MASK_CAUSAL,
    BlockPilotError,
    block_attention,
    block_attention_paged,
    block_attention_workspace_size,
    get_status,
    kv_append,
    library_path,
    load,
    policy_select,
    policy_select_workspace_size,
    spec_accept,
    spec_accept_workspace_size,
    tau_select,
    tau_select_workspace_size,
    verify_commit,
    verify_epilogue,
    verify_epilogue_workspace_size,
    workspace,
)
from ._build import build  # noqa: F401
