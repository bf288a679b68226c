"""Drive the fp64 oracle over one (sequence, KV head) of a named workload.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).  Inputs come from the
seeded generator in ``workload``; nothing here reads CUDA-path output.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Callable, Optional

import numpy as np

from workload import gen
from .kvpop_oracle import HeadCache, OracleParams, prefill_head


def _f64(t):
    return t.to(dtype=__import__("torch").float64).numpy()


@dataclass
class PairTrace:
    b: int
    h: int
    prompt_len: int
    slots: list = field(default_factory=list)       # per step: kept slot or -1
    evicted: list = field(default_factory=list)     # per step: evicted position or -1
    scores: list = field(default_factory=list)      # per step: fp32 raw score (NaN if none)
    outputs: list = field(default_factory=list)     # per step: [G][d] fp64
    cache: Optional[HeadCache] = None


def head_params(cfg, weights, h: int) -> OracleParams:
    W1, b1, w2, b2, lg = weights
    return OracleParams.for_head(W1.numpy(), b1.numpy(), w2.numpy(), b2.numpy(), lg.numpy(),
                                 h, cfg.budget_B, cfg.delay_D, cfg.n_sink, cfg.scorer_act)


def prefill_pair(cfg, weights, b: int, h: int, prompt_len: int,
                 prefill_override: Optional[np.ndarray] = None, layer: int = 0) -> HeadCache:
    G = cfg.q_per_kv
    K = _f64(gen.kv_tokens(cfg, "k", b, 1, 0, prompt_len, heads=[h], layer=layer))[0, 0]
    V = _f64(gen.kv_tokens(cfg, "v", b, 1, 0, prompt_len, heads=[h], layer=layer))[0, 0]
    Q = _f64(gen.q_tokens(cfg, b, 1, 0, prompt_len, heads=range(h * G, (h + 1) * G), layer=layer))[0]
    return prefill_head(head_params(cfg, weights, h), Q, K, V, cfg.head_dim, G, prefill_override)


def prefill_pair_mlstm(cfg, mw, b: int, h: int, prompt_len: int,
                       prefill_override: Optional[np.ndarray] = None):
    from .mlstm import MlstmParams, prefill_mlstm
    G = cfg.q_per_kv
    K = _f64(gen.kv_tokens(cfg, "k", b, 1, 0, prompt_len, heads=[h]))[0, 0]
    V = _f64(gen.kv_tokens(cfg, "v", b, 1, 0, prompt_len, heads=[h]))[0, 0]
    Q = _f64(gen.q_tokens(cfg, b, 1, 0, prompt_len, heads=range(h * G, (h + 1) * G)))[0]
    lg = float(np.float32(mw["log_gamma"][h])) if "log_gamma" in mw else 0.0
    op = OracleParams(np.zeros((3 * cfg.head_dim, 1)), np.zeros(1), np.zeros(1), 0.0,
                      cfg.budget_B, cfg.delay_D, cfg.n_sink, lg)
    mp = MlstmParams.for_head({k: v.numpy() for k, v in mw.items()}, h)
    return prefill_mlstm(op, mp, Q, K, V, cfg.head_dim, G, prefill_override)


def run_pair(cfg, weights, b: int, h: int, prompt_len: int, n_steps: int,
             prefill_override: Optional[np.ndarray] = None,
             step_override: Optional[Callable[[int], float]] = None,
             attend: bool = True, layer: int = 0, keep_cache: bool = False,
             mlstm: Optional[dict] = None) -> PairTrace:
    """Prefill (b, h) with its prompt, then run ``n_steps`` decode steps.

    With ``mlstm`` (weights from ``workload.gen.mlstm_weights``) the scorer is the
    stateful mLSTM instead of the MLP in ``weights``."""
    G = cfg.q_per_kv
    if mlstm is not None:
        cache = prefill_pair_mlstm(cfg, mlstm, b, h, prompt_len, prefill_override)
    else:
        cache = prefill_pair(cfg, weights, b, h, prompt_len, prefill_override, layer)
    tr = PairTrace(b, h, prompt_len)
    if n_steps:
        q, k, v = gen.decode_inputs(cfg, [prompt_len], 0, n_steps, layer=layer, b0=b)
        q = _f64(q[:, 0, h * G:(h + 1) * G])
        k = _f64(k[:, 0, h])
        v = _f64(v[:, 0, h])
        for j in range(n_steps):
            ov = None if step_override is None else step_override(j)
            slot, ev, r = cache.append(q[j], k[j], v[j], ov)
            tr.slots.append(slot)
            tr.evicted.append(ev)
            tr.scores.append(r)
            if attend:
                out, _, _ = cache.attend(q[j])
                tr.outputs.append(out)
    if keep_cache:
        tr.cache = cache
    return tr
