"""GB300-native tq2_0_fx4 (Tied Trit-Planes, arXiv 2608.08910) integer dot
pass and routed-expert MoE kernels, behind the C ABI of libtqfx4.

The public calls have the names of include/tqfx4.h and live in `binding`;
`ops` holds tensor-allocating conveniences built on them; `inputs` holds the
seeded synthetic input generators.
"""
from .binding import (  # noqa: F401
    TQFX4_BLOCK_BYTES, TQFX4_PATH_AUTO, TQFX4_PATH_DECODE, TQFX4_PATH_PREFILL, TQFX4_QK, TQFX4_ROWS,
    TQFX4_SRC_F32_RTN, TQFX4_SRC_F32_TIED, TQFX4_SRC_TRITS, TQFX4_STATUS_BYTES, TqfxError, c_experts, c_router, lib,
    tqfx4_basic_workspace_bytes, tqfx4_check, tqfx4_gemv, tqfx4_last_error, tqfx4_matrix_bytes,
    tqfx4_moe_ffn, tqfx4_moe_grouped, tqfx4_moe_stage_count, tqfx4_moe_stage_name,
    tqfx4_moe_workspace_bytes, tqfx4_moe_workspace_views, tqfx4_pack, tqfx4_quantize_act, tqfx4_moe_route,
    tqfx4_moe_experts)
