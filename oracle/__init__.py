"""CPU oracle of the Forcing-KV hot path (test infrastructure only).

Imported by the test suite, the smoke check and the benchmark's CPU-baseline
leg; never by the library.  See `oracle.forcing_kv` for the definitions.
"""
from .forcing_kv import *  # noqa: F401,F403
from .forcing_kv import (ForcingKVOracle, FrameRoles, attention_fp64, bottom_k, classify_head,
                         attention_fp8, attention_fp8_qk, P_SCALE_EXP, cosine_fp64, e4m3_round, head_attention_mass,
                         q_row_exponent, quantize_q_rows, rule_value, splitmix64,
                         dynamic_key_tokens, fixed_point, fmaf_bf16, frame_roles, keep_count,
                         score_from_sums, segment_range, segment_score_contract,
                         segment_sums_contract, static_key_tokens, token_dots_contract)
