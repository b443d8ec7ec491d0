"""The five workloads the benchmark and the parity tests run, by name.

Shapes follow the paper's MoE expert matrices (256 routed experts, hidden
4096, expert-intermediate 2048, top-8; Sec. 1 and Sec. 2.1 give 256 experts
per stack and sizes consistent with 4096 x 2048 projections).
"""
from dataclasses import dataclass


@dataclass(frozen=True)
class Workload:
    name: str
    kind: str          # "gemv" | "ffn" | "moe" | "grouped"
    hidden: int = 4096
    inter: int = 2048
    n_experts: int = 256
    top_k: int = 8
    tokens: int = 1
    zipf: float = 0.0  # router bias -zipf * ln(rank); 0 = unbiased
    n: int = 0         # gemv only
    k: int = 0         # gemv only
    path: int = 0      # grouped: 0 auto, 1 decode, 2 prefill


GEMV_1024 = Workload("gemv_1024x1024", "gemv", n=1024, k=1024)
EXPERT_FFN = Workload("expert_ffn_4096x2048_b1", "ffn", n_experts=1, top_k=1)
MOE_DECODE_1 = Workload("moe_decode_t1_e256_k8", "moe")
MOE_DECODE_64 = Workload("moe_grouped_decode_t64_e256_k8_zipf1.1", "grouped", tokens=64,
                         zipf=1.1, path=1)
MOE_PREFILL_2048 = Workload("moe_prefill_t2048_e256_k8", "grouped", tokens=2048, path=2)

ALL = [GEMV_1024, EXPERT_FFN, MOE_DECODE_1, MOE_DECODE_64, MOE_PREFILL_2048]
BY_NAME = {w.name: w for w in ALL}
