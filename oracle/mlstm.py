"""fp64 oracle of the stateful delayed mLSTM scorer (App. A, App. E.3, App. E.4).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Per KV head, with x_t = [k_t; v_t] (App. E.1):
    q~_t = phi(W_q x_t),  k~_t = phi(W_k x_t),  v~_t = W_v x_t         (W_* in R^{2d x d/2})
    phi(y) = [softmax(y); softmax(-y)]  (Hedgehog feature map, in R^d)
    i_t = exp(a_i),  f_t = sigmoid(a_f),  a_i = w_i . x_t + b_i,  a_f = w_f . x_t + b_f
    C_t = f_t C_{t-1} + i_t k~_t v~_t^T,   z_t = f_t z_{t-1} + i_t k~_t
At query position q the token u = q - w that has just left the window is read
with the state that has already absorbed every token up to q (delayed readout):
    h = (q~_u^T C_q) / (q~_u^T z_q),    r = a^T SiLU(h) + b.
The state is kept in the stabilised form of the mLSTM (a running log-scale m
with C, z divided by exp(m)); the readout ratio does not depend on it.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from .kvpop_oracle import HeadCache, OracleParams, round_score


def hedgehog(y: np.ndarray) -> np.ndarray:
    """[softmax(y); softmax(-y)] over the last axis."""
    def sm(x):
        e = np.exp(x - x.max(axis=-1, keepdims=True))
        return e / e.sum(axis=-1, keepdims=True)
    return np.concatenate([sm(y), sm(-y)], axis=-1)


def log_sigmoid(x):
    return -np.logaddexp(0.0, -x)


@dataclass
class MlstmParams:
    Wq: np.ndarray      # [2d][d/2]
    Wk: np.ndarray
    Wv: np.ndarray
    wi: np.ndarray      # [2d]
    wf: np.ndarray
    bi: float
    bf: float
    a: np.ndarray       # [d/2]
    b: float

    @staticmethod
    def for_head(w: dict, h: int):
        g = lambda k: np.asarray(w[k][h], dtype=np.float64)
        return MlstmParams(g("Wq"), g("Wk"), g("Wv"), g("wi"), g("wf"), float(g("bi")),
                           float(g("bf")), g("a"), float(g("b")))


class MlstmState:
    """Stabilised recurrent state (C, z, m) of one KV head."""

    def __init__(self, p: MlstmParams, d: int):
        self.p = p
        self.C = np.zeros((d, d // 2))
        self.z = np.zeros(d)
        self.m = -np.inf

    def features(self, x: np.ndarray):
        p = self.p
        return (hedgehog(x @ p.Wq), hedgehog(x @ p.Wk), x @ p.Wv,
                float(x @ p.wi + p.bi), float(x @ p.wf + p.bf))

    def update(self, x: np.ndarray):
        """Absorb token x = [k; v]."""
        _, kt, vt, ai, af = self.features(x)
        lf = log_sigmoid(af)
        m_new = max(lf + self.m, ai)
        fs = np.exp(lf + self.m - m_new) if np.isfinite(self.m) else 0.0
        is_ = np.exp(ai - m_new)
        self.C = fs * self.C + is_ * np.outer(kt, vt)
        self.z = fs * self.z + is_ * kt
        self.m = m_new

    def readout(self, x_u: np.ndarray):
        qt = hedgehog(x_u @ self.p.Wq)
        return (qt @ self.C) / (qt @ self.z)

    def score(self, x_u: np.ndarray) -> float:
        h = self.readout(x_u)
        silu = h / (1.0 + np.exp(-h))
        return float(self.p.a @ silu + self.p.b)


class MlstmHeadCache(HeadCache):
    """HeadCache whose delayed scorer is the mLSTM instead of the MLP."""

    def __init__(self, p: OracleParams, mp: MlstmParams, head_dim: int, q_per_kv: int):
        super().__init__(p, head_dim, q_per_kv)
        self.state = MlstmState(mp, head_dim)

    def append(self, q, k, v, override=None):
        qmean_p = np.asarray(q, dtype=np.float64).mean(axis=0)
        k = np.asarray(k, dtype=np.float64)
        v = np.asarray(v, dtype=np.float64)
        self.state.update(np.concatenate([k, v]))      # memory now holds tokens 0..p
        out = (-1, -1, np.float32(np.nan))
        if self.length >= self.p.delay_D:
            u, k_u, v_u, _ = self.pending[0]
            r = self.state.score(np.concatenate([k_u, v_u])) if override is None else override
            r32 = round_score(r)
            slot, evicted, _ = self._place(u, k_u, v_u, r32)
            out = (slot, evicted, r32)
            self.pending.popleft()
        self.pending.append((self.length, k, v, qmean_p))
        self.length += 1
        return out


def prefill_mlstm(p: OracleParams, mp: MlstmParams, Q, K, V, head_dim: int, q_per_kv: int,
                  override=None) -> MlstmHeadCache:
    """Prompt compression with the mLSTM scorer.

    The recurrent state absorbs the prompt token by token; after absorbing token t
    the token u = t - D is read out and scored (delayed readout).  Selection is the
    same as for the MLP scorer (``prefill_head``): sinks plus the top (B - s) by
    (priority desc, position asc).  ``override[u]`` replaces the score of u.
    """
    from .kvpop_oracle import prefill_head
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    P, D = K.shape[0], p.delay_D
    st = MlstmState(mp, head_dim)
    raw = []
    for t in range(P):
        st.update(np.concatenate([K[t], V[t]]))
        if t >= D:
            u = t - D
            raw.append(st.score(np.concatenate([K[u], V[u]])))
    if override is not None:
        raw = list(np.asarray(override[:len(raw)], dtype=np.float64))
    base = prefill_head(p, Q, K, V, head_dim, q_per_kv, override=np.asarray(raw, dtype=np.float64))
    c = MlstmHeadCache(p, mp, head_dim, q_per_kv)
    c.__dict__.update({k: v for k, v in base.__dict__.items()})
    c.state = st
    return c
