"""REFLEX per-forward MoE hot path on one GB300 (sm_103a).

C ABI: include/reflex.h, implemented in csrc/ and built into
_build/libreflex.so by `python -m paper_2608_01784_gb300.build`.
`_binding` mirrors the C entry points one to one; `api` adds device-buffer
conveniences; `workloads` draws the seeded synthetic inputs.  There is no
CPU fallback: loading fails loudly when the library is missing.
"""
from ._binding import (  # noqa: F401
    REFLEX_DTYPE_BF16, REFLEX_DTYPE_F32, REFLEX_FLAG_RENORM_TOPK,
    REFLEX_FLAG_RESIDUAL,
    REFLEX_FLAG_SIMT_EXPERTS, REFLEX_OK, REFLEX_STAGE_COMBINE,
    REFLEX_STAGE_DISPATCH, REFLEX_STAGE_EXPERT_DOWN, REFLEX_STAGE_EXPERT_UP,
    REFLEX_STAGE_ROUTE,
    ReflexError, load, make_params, reflex_abi_version, reflex_allocate,
    reflex_default_params, reflex_moe_forward, reflex_moe_status,
    reflex_moe_workspace_size, reflex_read_status,
    reflex_selftest_wait_timeout, reflex_status_string)
