"""Seeded synthetic workloads for the KVpop decode path.

This package only draws numbers and names workload shapes.  It holds none of
the method's arithmetic (no scoring, eviction or attention), so both the CUDA
path's tests/benchmark and the fp64 oracle can take their inputs from it.
"""
from .configs import CONFIGS, WorkloadConfig, get_config  # noqa: F401
from .gen import (  # noqa: F401
    normal_values,
    kv_tokens,
    q_tokens,
    decode_inputs,
    scorer_weights,
    prompt_lengths,
    outlier_channels,
    uniform_scores,
    stack_weights,
    prompt_hidden,
    decode_hidden,
    mlstm_weights,
)
