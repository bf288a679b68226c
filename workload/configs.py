"""Named synthetic workloads shaped like the paper's Qwen3-4B / Qwen3-8B runs.

Head layout 32 query heads / 8 KV heads / head_dim 128 is the Qwen3 attention
layout of the paper's base models (Sec. 4); 75% and 88% KV compression are the
paper's two operating points (Table 1).  The paper's datasets (AIME, HMMT, ...)
are not used: every tensor is drawn by ``workload.gen`` from a seed.

Budget notation (Eq. 1, ``B = s + w + k``): ``delay_D`` is the protected window
``w``; ``budget_B`` counts the sink slots plus the long-range top-k slots
(``s + k``); the window's D entries are held separately.
"""
from dataclasses import dataclass, field, replace
from typing import Optional


@dataclass(frozen=True)
class WorkloadConfig:
    name: str
    batch: int
    n_kv_heads: int
    q_per_kv: int
    head_dim: int
    kv_dtype: str            # "f32" or "bf16"
    prompt_len: int          # fixed prompt length; ignored when ragged
    budget_B: int
    delay_D: int
    decode_steps: int
    scorer_hidden: int
    n_sink: int = 0
    n_outlier: int = 0       # key channels scaled by `outlier_scale`
    outlier_scale: float = 10.0
    ragged: Optional[tuple] = None   # (lo, hi) inclusive range of prompt lengths
    n_layers: int = 1
    hidden: int = 0          # model width for the projection stack (layers > 1)
    seed: int = 0
    scorer_act: str = "gelu"  # hidden activation of the stateless scorer: gelu / silu / identity
    scorer_kv_only: bool = False  # scorer input [k; v] instead of [k; v; qbar]
    log_gamma: float = 0.0   # per-head log decay (0 = no decay)
    description: str = field(default="", compare=False)

    @property
    def n_q_heads(self) -> int:
        return self.n_kv_heads * self.q_per_kv

    @property
    def esz(self) -> int:
        return 4 if self.kv_dtype == "f32" else 2

    @property
    def scorer_in(self) -> int:
        return (2 if self.scorer_kv_only else 3) * self.head_dim

    def with_(self, **kw) -> "WorkloadConfig":
        return replace(self, **kw)


CONFIGS = {
    "tiny": WorkloadConfig(
        name="tiny", batch=1, n_kv_heads=2, q_per_kv=2, head_dim=64, kv_dtype="f32",
        prompt_len=128, budget_B=64, delay_D=4, decode_steps=512, scorer_hidden=32,
        description="1 layer, b1, 2 KV x 2 q heads, d64, fp32, P=128 -> B=64, D=4, 512 steps"),
    "q4b": WorkloadConfig(
        name="q4b", batch=8, n_kv_heads=8, q_per_kv=4, head_dim=128, kv_dtype="bf16",
        prompt_len=4096, budget_B=3072, delay_D=16, decode_steps=8192, scorer_hidden=256,
        n_outlier=4,
        description="Qwen3-4B-shaped layer, b8, 32q/8kv, d128, bf16, P=4096, B=3072, D=16"),
    "q8b_stack": WorkloadConfig(
        name="q8b_stack", batch=32, n_kv_heads=8, q_per_kv=4, head_dim=128, kv_dtype="bf16",
        prompt_len=32768, budget_B=8192, delay_D=16, decode_steps=1024, scorer_hidden=256,
        n_layers=36, hidden=4096,
        description="Qwen3-8B-shaped 36-layer stack, b32, hidden 4096, P=32768, B=8192, D=16"),
    "cr8x": WorkloadConfig(
        name="cr8x", batch=64, n_kv_heads=8, q_per_kv=4, head_dim=128, kv_dtype="bf16",
        prompt_len=32768, budget_B=4096, delay_D=16, decode_steps=2048, scorer_hidden=256,
        n_outlier=4,
        description="8x compression, b64, 32q/8kv, d128, bf16, P=32768, B=4096, D=16"),
    "ragged": WorkloadConfig(
        name="ragged", batch=128, n_kv_heads=8, q_per_kv=4, head_dim=128, kv_dtype="bf16",
        prompt_len=65536, budget_B=8192, delay_D=32, decode_steps=512, scorer_hidden=256,
        ragged=(1024, 65536),
        description="ragged b128, P_b ~ U[1024, 65536], B=8192, D=32, 512 steps"),
}


def get_config(name: str, **overrides) -> WorkloadConfig:
    cfg = CONFIGS[name]
    return cfg.with_(**overrides) if overrides else cfg
