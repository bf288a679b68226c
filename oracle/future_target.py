"""fp64 oracle of the future-attention target (Sec. 3.4, App. D.1-D.3, App. F.1-F.2).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

For one KV head h with G query heads, prompt/training length S, window w:

* dense causal logits l(d, t) = q_d^(g) . k_t / sqrt(d_k) and normaliser
  LSE_d = log sum_{t' <= d} exp(l(d, t'))                            (App. D.1)
* future mass of key t: mbar_t^(g) = sum_{d = t+w}^{S-1} p_{d->t}
  with p_{d->t} = exp(l(d, t) - LSE_d)                                 (App. D.1)
  Written as a log-sum-exp over future queries for a fixed key, this is what
  the transposed attention pass returns (App. D.2); with the sparse
  normaliser of the running top-k mask in place of LSE_d it becomes the
  approximate target of App. D.3.
* count N_t = max(1, S - (t + w)), clipped to L + 1 with a finite lookahead
  L, in which case only d <= t + w + L are summed (App. F.2).
* target per KV head (Eq. 2 with m = mbar / N_t, or without the count):
  max aggregation  r = log(eps + max_g m^(g))                         (App. F.1)
  mean aggregation r = log(eps + mean_g m^(g))                        (App. F.1)
  Reading: Eq. 2 places eps next to the count-normalised mass m, while App.
  F.2 subtracts log N_t after adding eps to the raw mass; the main-text form
  is used here (the two differ only in how eps is scaled).

``future_log_mass`` follows the definition (probabilities first, then the sum
over the future queries); nothing is blocked or reordered.
"""
from __future__ import annotations

import numpy as np


def causal_logits(Qg: np.ndarray, K: np.ndarray) -> np.ndarray:
    """l[d, t] for t <= d, -inf above the diagonal.  ``Qg [S][d_k]``, ``K [S][d_k]``."""
    S, dk = K.shape
    l = (np.asarray(Qg, dtype=np.float64) @ np.asarray(K, dtype=np.float64).T) / np.sqrt(dk)
    l[np.triu_indices(S, 1)] = -np.inf
    return l


def dense_causal_lse(Qg: np.ndarray, K: np.ndarray) -> np.ndarray:
    """LSE_d of Eq. (dense LSE), natural log, for d = 0 .. S-1."""
    l = causal_logits(Qg, K)
    mx = l.max(axis=1, keepdims=True)
    return (mx + np.log(np.exp(l - mx).sum(axis=1, keepdims=True)))[:, 0]


def future_log_mass(Qg: np.ndarray, K: np.ndarray, lse: np.ndarray, w: int,
                    lookahead: int = 0) -> np.ndarray:
    """log mbar_t for t = 0 .. S-1 given per-query normalisers ``lse[d]`` (dense or sparse).

    -inf where no query d satisfies t + w <= d <= S - 1 (and d <= t + w + lookahead)."""
    l = causal_logits(Qg, K)
    S = l.shape[0]
    p = np.exp(l - np.asarray(lse, dtype=np.float64)[:, None])      # p[d, t]
    out = np.full(S, -np.inf)
    for t in range(S):
        hi = S - 1 if lookahead <= 0 else min(S - 1, t + w + lookahead)
        if t + w <= hi:
            out[t] = np.log(p[t + w: hi + 1, t].sum())
    return out


def future_count(S: int, w: int, lookahead: int = 0) -> np.ndarray:
    """N_t = max(1, S - (t + w)), clipped to lookahead + 1 when a lookahead is set."""
    n = np.maximum(1, S - (np.arange(S) + w))
    if lookahead > 0:
        n = np.minimum(n, lookahead + 1)
    return n.astype(np.float64)


def aggregate_target(logm: np.ndarray, S: int, w: int, eps: float, agg: str = "max",
                     count_norm: bool = True, lookahead: int = 0) -> np.ndarray:
    """r_t from per-group log masses ``logm [G][S]`` (Eq. 2 / App. F.1, F.2)."""
    m = np.exp(np.asarray(logm, dtype=np.float64))                  # mbar (0 where -inf)
    if count_norm:
        m = m / future_count(S, w, lookahead)[None, :]
    a = m.max(axis=0) if agg == "max" else m.mean(axis=0)
    return np.log(eps + a)
