"""fp64 CPU oracle of the KVpop decode step (one sequence, one KV head at a time).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline legs.  It shares no code with the CUDA library.

What it computes, step by step in the paper's terms (s sinks, protected window
w = D, long-range top-k, budget slots B = s + k; the window is held apart):

* Eligible set E(q) = {t | s <= t <= q - w}; the token t_new = q - w has just
  left the protected window (Sec. 3.1, Eq. 4).
* Delayed scoring: a token is scored only when it leaves the window, with the
  context gathered meanwhile (Sec. 3.3, its paragraph on stateful scorers;
  App. E.4).  The scorer is the stateless two-layer MLP of Sec. 3.3 / App. E.2
  applied to the input [k_u; v_u; qbar_u], where qbar_u averages the D queries
  u+1..u+D over the G query heads that share the KV head, with an exact-erf
  GELU hidden layer;
  or the paper's plain variant on [k_u; v_u] (W1 with 2d rows), with a SiLU or
  identity hidden layer.
* Static priority for decay step n = 1: rbar = r - u * log(gamma_h)
  (App. B.3); with log(gamma) = 0 it is the raw score.
* Running top-k under a fixed budget (Sec. 3.2, App. C.1 mask definition): a
  newly eligible token enters a free slot while fewer than B slots are used;
  afterwards it replaces the slot of lowest priority (ties -> lowest slot
  index) iff its priority is strictly larger, else it is dropped.  Because priorities are static and E(q) only
  grows, this keeps exactly the running top-k of App. C.1.
* Decode attends over the compact cache only: slots plus the w pending tokens
  (App. C, first paragraph), softmax(q k^T / sqrt(d)) v per query head.

Precision: all arithmetic is fp64 on exactly widened inputs.  Each score is
rounded to fp32 before any comparison (the paper ranks in fp32, App. F); NaN
becomes -inf and -0 becomes +0.  The decay product uses fp32 ops in the same
order as the CUDA path, because that value decides an integer (the kept slot).

Parity status: the attention, window and eviction logic are pinned by tests
(dense-attention reduction, brute-force top-k subsets, the App. C.1 mask
recomputed from scratch).  The scorer's exact form ([k; v; mean of the next D
queries], GELU, F hidden units) is a workload choice the paper does not print:
parity unpinned for that form against the paper; the oracle's scorer is pinned
only at hand-set weights and closed-form GELU values.
"""
from __future__ import annotations

from collections import deque
from dataclasses import dataclass
from typing import Optional

import numpy as np
from scipy.special import erf, expit

_SQRT1_2 = 1.0 / np.sqrt(2.0)


@dataclass
class OracleParams:
    """Per-KV-head scorer parameters and budget (fp64 copies of the given arrays)."""
    W1: np.ndarray          # [3d][F]   input order [k; v; qbar]
    b1: np.ndarray          # [F]
    w2: np.ndarray          # [F]
    b2: float
    budget_B: int
    delay_D: int
    n_sink: int = 0
    log_gamma: float = 0.0
    activation: str = "gelu"   # gelu / silu / identity

    @staticmethod
    def for_head(W1, b1, w2, b2, log_gamma, h, budget_B, delay_D, n_sink=0, activation="gelu"):
        as64 = lambda a: np.asarray(a, dtype=np.float64)
        return OracleParams(as64(W1[h]), as64(b1[h]), as64(w2[h]), float(as64(b2[h])),
                            int(budget_B), int(delay_D), int(n_sink), float(np.float32(log_gamma[h])),
                            activation)


def gelu_erf(z):
    """GELU(z) = z * Phi(z) = 0.5 z (1 + erf(z / sqrt 2))."""
    return 0.5 * z * (1.0 + erf(z * _SQRT1_2))


def silu(z):
    """SiLU(z) = z * sigmoid(z)."""
    return z * expit(z)


def scorer_mlp(x: np.ndarray, p: OracleParams) -> np.ndarray:
    """Two-layer headwise MLP score (Sec. 3.3, App. E.2): w2 . act(W1^T x + b1) + b2.

    ``x`` is ``[I]`` or ``[n][I]`` (I = rows of W1); returns fp64 scores.
    """
    z = x @ p.W1 + p.b1
    act = {"gelu": gelu_erf, "silu": silu, "identity": lambda y: y}[p.activation]
    return act(z) @ p.w2 + p.b2


def round_score(r64) -> np.float32:
    """fp32 rounding used for every ranking decision; NaN -> -inf, -0 -> +0."""
    r = np.float32(r64)
    if np.isnan(r):
        return np.float32(-np.inf)
    if r == 0:
        return np.float32(0.0)
    return r


def static_priority(r32: np.float32, u: int, log_gamma: float) -> np.float32:
    """rbar_u = r_u - u * log(gamma) (App. B.3, n = 1), evaluated in fp32 ops."""
    if log_gamma == 0.0:
        return r32
    prod = np.float32(np.float32(u) * np.float32(log_gamma))
    return round_score(np.float32(np.float32(r32) - prod))


class HeadCache:
    """State of one (sequence, KV head): B slots, the pending window, the length."""

    def __init__(self, p: OracleParams, head_dim: int, q_per_kv: int):
        self.p = p
        self.d = head_dim
        self.G = q_per_kv
        B = p.budget_B
        self.slot_k = np.zeros((B, head_dim))
        self.slot_v = np.zeros((B, head_dim))
        self.slot_prio = np.full(B, np.nan)
        self.slot_raw = np.full(B, np.nan)
        self.slot_pos = np.full(B, -1, dtype=np.int64)
        self.n_valid = 0
        self.pending = deque()      # (pos, k[d], v[d], qmean[d]) oldest first
        self.length = 0
        self.prefill_raw = np.zeros(0, dtype=np.float32)

    # ---- Sec. 3.3 delayed scorer input -------------------------------------------------
    def scorer_input(self, qmean_p: np.ndarray):
        """[k_u; v_u; qbar_u] for u = p - D, the token at the head of the window."""
        u, k_u, v_u, _ = self.pending[0]
        later = [e[3] for e in list(self.pending)[1:]]          # qmean(u+1 .. p-1)
        qbar = (np.sum(later, axis=0) if later else 0.0) + qmean_p
        qbar = qbar / self.p.delay_D
        if self.p.W1.shape[0] == 2 * self.d:          # the [k; v] scorer
            return u, np.concatenate([k_u, v_u])
        return u, np.concatenate([k_u, v_u, qbar])

    # ---- Sec. 3.2 / App. C.1 keep-or-drop under the budget ---------------------------
    def _place(self, u: int, k_u, v_u, r32: np.float32):
        p = self.p
        prio = static_priority(r32, u, p.log_gamma)
        if self.n_valid < p.budget_B:
            slot, evicted = self.n_valid, -1
            self.n_valid += 1
        else:
            cand = self.slot_prio[p.n_sink:p.budget_B]
            j = int(np.argmin(cand)) + p.n_sink          # first minimum = lowest slot
            if prio > self.slot_prio[j]:
                slot, evicted = j, int(self.slot_pos[j])
            else:
                return -1, -1, prio
        self.slot_k[slot] = k_u
        self.slot_v[slot] = v_u
        self.slot_prio[slot] = prio
        self.slot_raw[slot] = r32
        self.slot_pos[slot] = u
        return slot, evicted, prio

    def append(self, q: np.ndarray, k: np.ndarray, v: np.ndarray, override=None):
        """Ingest position p = length: score u = p - D, keep or drop it, push p.

        ``q`` is ``[G][d]``.  Returns ``(slot, evicted_pos, r32)``; slot = -1 when u
        was dropped or no token left the window, r32 = NaN when nothing was scored.
        """
        qmean_p = np.asarray(q, dtype=np.float64).mean(axis=0)
        k = np.asarray(k, dtype=np.float64)
        v = np.asarray(v, dtype=np.float64)
        out = (-1, -1, np.float32(np.nan))
        if self.length >= self.p.delay_D:
            u, x = self.scorer_input(qmean_p)
            r32 = round_score(scorer_mlp(x, self.p) if override is None else override)
            _, k_u, v_u, _ = self.pending[0]
            slot, evicted, _ = self._place(u, k_u, v_u, r32)
            out = (slot, evicted, r32)
            self.pending.popleft()
        self.pending.append((self.length, k, v, qmean_p))
        self.length += 1
        return out

    # ---- App. C: decode attends over the compact cache -------------------------------
    def keys_values(self):
        n = self.n_valid
        ks = [self.slot_k[:n]] + [e[1][None] for e in self.pending]
        vs = [self.slot_v[:n]] + [e[2][None] for e in self.pending]
        pos = list(self.slot_pos[:n]) + [e[0] for e in self.pending]
        return np.concatenate(ks), np.concatenate(vs), np.asarray(pos, dtype=np.int64)

    def attend(self, q: np.ndarray):
        K, V, pos = self.keys_values()
        out, probs = attend_head(np.asarray(q, dtype=np.float64), K, V)
        return out, probs, pos

    def kept_positions(self):
        return sorted(int(t) for t in self.slot_pos[: self.n_valid])


def attend_head(q: np.ndarray, K: np.ndarray, V: np.ndarray):
    """Per query head g: o_g = softmax(q_g K^T / sqrt(d)) V.  Returns (o [G][d], p [G][n])."""
    d = K.shape[1]
    logits = (q @ K.T) / np.sqrt(d)
    logits = logits - logits.max(axis=1, keepdims=True)
    e = np.exp(logits)
    probs = e / e.sum(axis=1, keepdims=True)
    return probs @ V, probs


def prefill_head(p: OracleParams, Q: np.ndarray, K: np.ndarray, V: np.ndarray,
                 head_dim: int, q_per_kv: int, override: Optional[np.ndarray] = None) -> HeadCache:
    """Compress a prompt of length P for one KV head.

    ``Q [G][P][d]``, ``K, V [P][d]``.  Scores every eligible u <= P-1-D with the
    delayed scorer, keeps the sinks u < s and the top (B - s) of the rest under
    (priority desc, position asc), stores them in ascending position order, and
    leaves the last min(P, D) tokens in the window.  ``override[u]`` replaces the
    scorer output for u.
    """
    c = HeadCache(p, head_dim, q_per_kv)
    P = K.shape[0]
    D, s, B = p.delay_D, p.n_sink, p.budget_B
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    qmean = Q.mean(axis=0) if P > 0 else np.zeros((0, head_dim))     # [P][d]
    n_elig = max(P - D, 0)
    raw = np.zeros(n_elig, dtype=np.float32)
    prio = np.zeros(n_elig, dtype=np.float32)
    if n_elig:
        if override is None:
            # qbar_u = (1/D) sum_{j=1..D} qmean(u + j), for all u at once
            qsum = np.zeros((n_elig, head_dim))
            for j in range(1, D + 1):
                qsum += qmean[j:j + n_elig]
            qbar = qsum / D
            X = np.concatenate([K[:n_elig], V[:n_elig], qbar], axis=1)
            if p.W1.shape[0] == 2 * head_dim:
                X = X[:, : 2 * head_dim]
            r64 = scorer_mlp(X, p)
        else:
            r64 = np.asarray(override[:n_elig], dtype=np.float64)
        for u in range(n_elig):
            raw[u] = round_score(r64[u])
            prio[u] = static_priority(raw[u], u, p.log_gamma)
    sinks = list(range(min(s, n_elig)))
    rest = sorted(range(len(sinks), n_elig), key=lambda u: (-float(prio[u]), u))
    kept = sorted(sinks + rest[: B - s])
    for slot, u in enumerate(kept):
        c.slot_k[slot] = K[u]
        c.slot_v[slot] = V[u]
        c.slot_prio[slot] = prio[u]
        c.slot_raw[slot] = raw[u]
        c.slot_pos[slot] = u
    c.n_valid = len(kept)
    c.prefill_raw = raw            # fp32 raw score of every eligible prompt token
    for t in range(max(0, P - D), P):
        c.pending.append((t, K[t].copy(), V[t].copy(), qmean[t].copy()))
    c.length = P
    return c


def prefill_head_streaming(p: OracleParams, Q, K, V, head_dim: int, q_per_kv: int,
                           override: Optional[np.ndarray] = None) -> HeadCache:
    """The same prompt ingested one token at a time with ``HeadCache.append``."""
    c = HeadCache(p, head_dim, q_per_kv)
    Q = np.asarray(Q, dtype=np.float64)
    D = p.delay_D
    for t in range(K.shape[0]):
        ov = None
        if override is not None and t >= D:
            ov = override[t - D]
        c.append(Q[:, t, :], K[t], V[t], ov)
    return c
