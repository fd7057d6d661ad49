"""CPU oracle (test infrastructure only; never imported by the product path)."""
from .llama import (OracleModel, apply_rope, bf16_bits_to_f64, causal_gqa_attention, greedy,
                    rmsnorm, rope_cos_sin, round_bf16, run_workload, silu, softmax)

__all__ = ["OracleModel", "apply_rope", "bf16_bits_to_f64", "causal_gqa_attention", "greedy",
           "rmsnorm", "rope_cos_sin", "round_bf16", "run_workload", "silu", "softmax"]
