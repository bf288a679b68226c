"""fp64 oracle of the running top-k sparse attention over a prompt (App. C).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

For one (sequence, KV head) with L prompt tokens, s sinks, protected window w
and long-range budget k (the build's B = s + k, D = w):

* static ranks (App. C.1): sort the tokens once by static priority, higher
  first; rank(t) = 0 is the best.  Equal priorities are ordered by position,
  earlier first (the same order prompt compression keeps).
* cutoffs (App. C.2, Algorithm 2): scan q = 0 .. L-1; the token t = q - w
  becomes eligible when t >= s and its rank is inserted into a Fenwick tree
  over ranks; tau_q = FindByPrefixCount(T, k), the smallest rank whose prefix
  count reaches k, found by binary lifting.  Reading where the algorithm and
  the mask definition disagree: Algorithm 2 leaves tau_q = -1 while fewer than
  k tokens are eligible, which, read literally, keeps none of them; the mask
  definition keeps the top k of E(q), i.e. all of E(q) when |E(q)| < k, and
  the budget starts to evict only when more than s + w + k tokens exist.  So here
  tau_q = FindByPrefixCount(T, min(k, |E(q)|)), and -1 only when E(q) is empty.
* mask (Eq. in App. C.1): M[q, t] = t < s  or  q - t < w  or
  (s <= t <= q - w and rank(t) <= tau_q), for t <= q.
* masked causal attention: per query head g of the KV head,
  y[g, q] = sum_t softmax_t(M ? q.k_t / sqrt(d) : -inf) v_t, and the natural
  log-normaliser LSE[g, q] = log sum_{t: M[q,t]} exp(q.k_t / sqrt(d)).

Nothing here is blocked, fused or reordered beyond those definitions.
"""
from __future__ import annotations

import numpy as np

from .kvpop_oracle import round_score, static_priority


def static_ranks(prio: np.ndarray) -> np.ndarray:
    """rank[t] for fp32 priorities ``prio[L]`` (NaN -> -inf, -0 -> +0 first).

    Order: priority descending, then position ascending; a library sort serves
    as the sort step."""
    p = np.array([np.float64(round_score(x)) for x in np.asarray(prio, dtype=np.float32)])
    L = p.shape[0]
    order = np.lexsort((np.arange(L), -p))       # last key is primary
    rank = np.empty(L, dtype=np.int64)
    rank[order] = np.arange(L)
    return rank


class Fenwick:
    """Binary indexed tree of counts over ranks 0 .. n-1 (Fenwick 1994)."""

    def __init__(self, n: int):
        self.n = n
        self.tree = np.zeros(n + 1, dtype=np.int64)     # 1-based

    def insert(self, r: int):
        i = r + 1
        while i <= self.n:
            self.tree[i] += 1
            i += i & (-i)

    def prefix_count(self, r: int) -> int:
        """Number of inserted ranks <= r."""
        i, c = r + 1, 0
        while i > 0:
            c += int(self.tree[i])
            i -= i & (-i)
        return c

    def find_by_prefix_count(self, c: int) -> int:
        """Smallest rank r with prefix_count(r) >= c (binary lifting, 1 <= c <= inserted)."""
        pos, rem = 0, c
        step = 1
        while step * 2 <= self.n:
            step *= 2
        while step:
            nxt = pos + step
            if nxt <= self.n and self.tree[nxt] < rem:
                pos = nxt
                rem -= int(self.tree[nxt])
            step //= 2
        return pos          # 1-based prefix end `pos` holds < c, so rank pos (0-based) reaches c


def fenwick_cutoffs(rank: np.ndarray, s: int, w: int, k: int) -> np.ndarray:
    """tau_q for q = 0 .. L-1 (Algorithm 2, with the |E(q)| < k reading above)."""
    rank = np.asarray(rank, dtype=np.int64)
    L = rank.shape[0]
    T = Fenwick(L)
    tau = np.full(L, -1, dtype=np.int64)
    n_elig = 0
    for q in range(L):
        t = q - w
        if t >= s:
            T.insert(int(rank[t]))
            n_elig += 1
        if n_elig > 0 and k > 0:
            tau[q] = T.find_by_prefix_count(min(k, n_elig))
    return tau


def mask_row(q: int, rank: np.ndarray, tau: np.ndarray, s: int, w: int) -> np.ndarray:
    """Boolean M[q, 0..q] of the running top-k mask."""
    t = np.arange(q + 1)
    elig = (t >= s) & (t <= q - w)
    return (t < s) | (q - t < w) | (elig & (rank[: q + 1] <= tau[q]))


def masked_attention(Q: np.ndarray, K: np.ndarray, V: np.ndarray, rank: np.ndarray,
                     tau: np.ndarray, s: int, w: int):
    """``Q [G][L][d]``, ``K, V [L][d]`` -> (y [G][L][d], lse [G][L]) in fp64."""
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    G, L, d = Q.shape
    y = np.zeros((G, L, d))
    lse = np.zeros((G, L))
    for q in range(L):
        keys = np.nonzero(mask_row(q, rank, tau, s, w))[0]
        logits = (Q[:, q, :] @ K[keys].T) / np.sqrt(d)          # [G][n]
        mx = logits.max(axis=1, keepdims=True)
        e = np.exp(logits - mx)
        z = e.sum(axis=1, keepdims=True)
        y[:, q, :] = (e / z) @ V[keys]
        lse[:, q] = (mx + np.log(z))[:, 0]
    return y, lse


def prompt_priorities(raw: np.ndarray, L: int, delay_D: int, log_gamma: float) -> np.ndarray:
    """fp32 static priorities of every prompt position 0 .. L-1.

    Tokens u <= L-1-D carry the fp32 raw score ``raw[u]`` of the delayed scorer;
    the last D tokens have no score yet and get -inf (they are never eligible
    for a query inside the prompt)."""
    prio = np.full(L, -np.inf, dtype=np.float32)
    n = max(L - delay_D, 0)
    for u in range(n):
        prio[u] = static_priority(round_score(raw[u]), u, log_gamma)
    return prio


def prefill_outputs(cache, Q: np.ndarray, K: np.ndarray, V: np.ndarray):
    """Prompt outputs of one compressed (sequence, KV head).

    ``cache`` is the HeadCache that prompt compression produced (its
    ``prefill_raw`` holds the fp32 raw scores); returns (y, lse, rank, tau)."""
    p = cache.p
    L = K.shape[0]
    prio = prompt_priorities(cache.prefill_raw, L, p.delay_D, p.log_gamma)
    rank = static_ranks(prio)
    tau = fenwick_cutoffs(rank, p.n_sink, p.delay_D, p.budget_B - p.n_sink)
    y, lse = masked_attention(Q, K, V, rank, tau, p.n_sink, p.delay_D)
    return y, lse, rank, tau
