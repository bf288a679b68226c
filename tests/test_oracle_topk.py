"""Pins of the running top-k sparse-attention oracle (App. C).

The cutoff scan (Algorithm 2) is checked against a sort of E(q) at every q;
the Fenwick tree's binary lifting against a cumulative-sum search; ranks
against their pairwise definition; the mask against the App. C.1 definition
recomputed from priorities, against the fixed budget, and against the decode
oracle's cache after every step (the running top-k of App. C.1 equals
replace-the-min under static priorities); the attention against torch SDPA in
fp64 and logsumexp.
"""
import numpy as np
import pytest
import torch

from conftest import read_golden
from oracle import HeadCache, OracleParams, prefill_head
from oracle import running_topk as rt
from test_oracle_pins import mask_from_definition


def tie_heavy_prio(rng, L, levels=None):
    if levels is None:
        return rng.standard_normal(L).astype(np.float32)
    return rng.integers(0, levels, L).astype(np.float32)


def better(pa, ta, pb, tb):
    return pa > pb or (pa == pb and ta < tb)


# ---------------------------------------------------------------- Fenwick tree
@pytest.mark.parametrize("n", [1, 2, 7, 16, 33, 100])
def test_fenwick_find_matches_cumsum_search(n):
    rng = np.random.default_rng(n)
    T = rt.Fenwick(n)
    hist = np.zeros(n, dtype=np.int64)
    for _ in range(3 * n):
        r = int(rng.integers(0, n))
        T.insert(r)
        hist[r] += 1
        cs = np.cumsum(hist)
        for c in range(1, int(cs[-1]) + 1):
            assert T.find_by_prefix_count(c) == int(np.searchsorted(cs, c))
        j = int(rng.integers(0, n))
        assert T.prefix_count(j) == int(cs[j])


# ---------------------------------------------------------------- ranks
@pytest.mark.parametrize("levels", [None, 3, 1])
def test_static_ranks_pairwise_definition(levels):
    rng = np.random.default_rng(5)
    L = 57
    prio = tie_heavy_prio(rng, L, levels)
    prio[3] = np.nan          # canonicalised to -inf
    prio[4] = -0.0            # equal to +0
    prio[9] = 0.0
    rank = rt.static_ranks(prio)
    p = [(-np.inf if np.isnan(x) else float(x) + 0.0) for x in prio]
    for t in range(L):
        want = sum(better(p[u], u, p[t], t) for u in range(L))
        assert rank[t] == want
    assert sorted(rank) == list(range(L))


# ---------------------------------------------------------------- cutoffs
CASES = [(40, 0, 1, 5), (40, 2, 3, 4), (33, 1, 4, 100), (25, 0, 2, 1), (60, 3, 5, 7), (9, 4, 2, 3)]


@pytest.mark.parametrize("L,s,w,k", CASES)
@pytest.mark.parametrize("levels", [None, 2])
def test_cutoffs_equal_sorted_eligible_set(L, s, w, k, levels):
    rng = np.random.default_rng(L * 100 + k)
    rank = rt.static_ranks(tie_heavy_prio(rng, L, levels))
    tau = rt.fenwick_cutoffs(rank, s, w, k)
    for q in range(L):
        elig = [t for t in range(s, q - w + 1)]
        if not elig:
            assert tau[q] == -1
            continue
        ranks = sorted(int(rank[t]) for t in elig)
        assert tau[q] == ranks[min(k, len(ranks)) - 1], q


def test_cutoffs_nonincreasing_once_budget_binds():
    rng = np.random.default_rng(2)
    L, s, w, k = 200, 2, 4, 9
    tau = rt.fenwick_cutoffs(rt.static_ranks(tie_heavy_prio(rng, L)), s, w, k)
    full = s + w + k - 1            # first q with |E(q)| = k
    assert np.all(np.diff(tau[full:]) <= 0)


def test_hand_traced_cutoffs():
    rows = read_golden("running_topk_tiny.txt")
    L, s, w, k = (int(x) for x in rows[0])
    prio = np.array([float(x) for x in rows[1]], dtype=np.float32)
    rank = rt.static_ranks(prio)
    assert list(rank) == [int(x) for x in rows[2]]
    tau = rt.fenwick_cutoffs(rank, s, w, k)
    assert list(tau) == [int(x) for x in rows[3]]
    assert list(np.nonzero(rt.mask_row(L - 1, rank, tau, s, w))[0]) == [int(x) for x in rows[4]]


# ---------------------------------------------------------------- mask
@pytest.mark.parametrize("L,s,w,k", CASES)
@pytest.mark.parametrize("levels", [None, 3])
def test_mask_matches_definition_and_budget(L, s, w, k, levels):
    rng = np.random.default_rng(L + 7 * k)
    prio = tie_heavy_prio(rng, L, levels)
    rank = rt.static_ranks(prio)
    tau = rt.fenwick_cutoffs(rank, s, w, k)
    for q in range(L):
        row = rt.mask_row(q, rank, tau, s, w)
        assert np.array_equal(row, mask_from_definition(q, [float(x) for x in prio], s, w, k)), q
        assert row.sum() == min(q + 1, s + w + k)      # the fixed budget of Eq. 1


@pytest.mark.parametrize("B,D,s", [(4, 2, 0), (5, 3, 1), (3, 1, 2), (8, 4, 0)])
def test_mask_rows_equal_decode_cache(B, D, s):
    """After each decode step q the oracle cache holds exactly row q of the mask."""
    rng = np.random.default_rng(B * 10 + D)
    L = 70
    raw = rng.permutation(L).astype(np.float32) * 0.5 - 3.0   # distinct scores
    p = OracleParams(np.zeros((3, 1)), np.zeros(1), np.zeros(1), 0.0, B, D, s)
    c = HeadCache(p, 1, 1)
    prio = rt.prompt_priorities(raw, L + D, D, 0.0)[:L]
    rank = rt.static_ranks(prio)
    tau = rt.fenwick_cutoffs(rank, s, D, B - s)
    for q in range(L):
        c.append(np.zeros((1, 1)), np.zeros(1), np.zeros(1), raw[q - D] if q >= D else None)
        held = sorted(c.kept_positions() + [e[0] for e in c.pending])
        assert held == list(np.nonzero(rt.mask_row(q, rank, tau, s, D))[0]), q


# ---------------------------------------------------------------- attention
def sdpa_rows(Q, K, V, masks):
    """torch SDPA (fp64) per query row with a boolean key mask; returns y and logsumexp."""
    G, L, d = Q.shape
    y = np.zeros((G, L, d))
    lse = np.zeros((G, L))
    Kt, Vt = torch.from_numpy(K), torch.from_numpy(V)
    for q in range(L):
        m = torch.from_numpy(masks[q])
        qt = torch.from_numpy(Q[:, q, :])
        o = torch.nn.functional.scaled_dot_product_attention(
            qt[None, :, None, :], Kt[None, None].expand(1, G, -1, -1),
            Vt[None, None].expand(1, G, -1, -1),
            attn_mask=m[None, None, None, :].expand(1, G, 1, -1))
        y[:, q, :] = o[0, :, 0, :].numpy()
        logits = (qt @ Kt.T) / np.sqrt(d)
        lse[:, q] = torch.logsumexp(logits.masked_fill(~m[None, :], -np.inf), dim=1).numpy()
    return y, lse


def test_budget_covering_prompt_is_dense_causal():
    rng = np.random.default_rng(3)
    G, L, d, s, w = 2, 24, 8, 1, 3
    Q, K, V = rng.standard_normal((G, L, d)), rng.standard_normal((L, d)), rng.standard_normal((L, d))
    rank = rt.static_ranks(tie_heavy_prio(rng, L))
    tau = rt.fenwick_cutoffs(rank, s, w, L)
    y, lse = rt.masked_attention(Q, K, V, rank, tau, s, w)
    o = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(Q)[None], torch.from_numpy(K)[None, None].expand(1, G, -1, -1),
        torch.from_numpy(V)[None, None].expand(1, G, -1, -1), is_causal=True)[0].numpy()
    assert np.abs(y - o).max() < 1e-12
    logits = np.einsum("gqd,td->gqt", Q, K) / np.sqrt(d)
    logits[:, np.triu_indices(L, 1)[0], np.triu_indices(L, 1)[1]] = -np.inf
    ref = torch.logsumexp(torch.from_numpy(logits), dim=2).numpy()
    assert np.abs(lse - ref).max() < 1e-12


@pytest.mark.parametrize("levels", [None, 2])
def test_sparse_attention_matches_sdpa_with_defined_mask(levels):
    rng = np.random.default_rng(17)
    G, L, d, s, w, k = 4, 48, 16, 2, 3, 6
    Q, K, V = rng.standard_normal((G, L, d)), rng.standard_normal((L, d)), rng.standard_normal((L, d))
    prio = tie_heavy_prio(rng, L, levels)
    rank = rt.static_ranks(prio)
    tau = rt.fenwick_cutoffs(rank, s, w, k)
    y, lse = rt.masked_attention(Q, K, V, rank, tau, s, w)
    masks = [np.concatenate([mask_from_definition(q, [float(x) for x in prio], s, w, k),
                             np.zeros(L - q - 1, dtype=bool)]) for q in range(L)]
    y2, lse2 = sdpa_rows(Q, K, V, masks)
    assert np.abs(y - y2).max() < 1e-12
    assert np.abs(lse - lse2).max() < 1e-12


def test_last_prompt_row_equals_compressed_cache_attention():
    """y at q = P-1 is decode attention over the cache prompt compression builds."""
    rng = np.random.default_rng(23)
    G, P, d, B, D, s = 2, 40, 8, 6, 3, 1
    Q, K, V = rng.standard_normal((G, P, d)), rng.standard_normal((P, d)), rng.standard_normal((P, d))
    raw = rng.standard_normal(P).astype(np.float32)
    p = OracleParams(np.zeros((3 * d, 1)), np.zeros(1), np.zeros(1), 0.0, B, D, s, -0.01)
    cache = prefill_head(p, Q, K, V, d, G, override=raw)
    y, lse, rank, tau = rt.prefill_outputs(cache, Q, K, V)
    out, _, pos = cache.attend(Q[:, P - 1, :])
    assert sorted(pos) == list(np.nonzero(rt.mask_row(P - 1, rank, tau, s, D))[0])
    assert np.abs(y[:, P - 1, :] - out).max() < 1e-12


# ---------------------------------------------------------------- planted mistakes
def test_topk_pins_catch_planted_mistakes(monkeypatch):
    rng = np.random.default_rng(0)
    L, s, w, k = 30, 1, 2, 4
    prio = tie_heavy_prio(rng, L, 3)
    rank = rt.static_ranks(prio)

    def cutoffs_ok():
        tau = rt.fenwick_cutoffs(rank, s, w, k)
        for q in range(L):
            elig = sorted(int(rank[t]) for t in range(s, q - w + 1))
            want = elig[min(k, len(elig)) - 1] if elig else -1
            if tau[q] != want:
                return False
        return True

    def mask_ok():
        tau = rt.fenwick_cutoffs(rank, s, w, k)
        return all(np.array_equal(rt.mask_row(q, rank, tau, s, w),
                                  mask_from_definition(q, [float(x) for x in prio], s, w, k))
                   for q in range(L))

    assert cutoffs_ok() and mask_ok()
    # 1. binary lifting returning the last rank below the count
    orig = rt.Fenwick.find_by_prefix_count
    monkeypatch.setattr(rt.Fenwick, "find_by_prefix_count", lambda self, c: orig(self, c) - 1)
    assert not cutoffs_ok()
    monkeypatch.setattr(rt.Fenwick, "find_by_prefix_count", orig)
    # 2. the literal tau = -1 while fewer than k are eligible
    orig_cut = rt.fenwick_cutoffs

    def literal(rank_, s_, w_, k_):
        tau = orig_cut(rank_, s_, w_, k_)
        for q in range(len(rank_)):
            if max(0, q - w_ - s_ + 1) < k_:
                tau[q] = -1
        return tau
    monkeypatch.setattr(rt, "fenwick_cutoffs", literal)
    assert not mask_ok()
    monkeypatch.setattr(rt, "fenwick_cutoffs", orig_cut)
    # 3. ties ranked latest-first
    orig_rank = rt.static_ranks

    def late_first(p):
        pp = np.asarray(p, dtype=np.float64)
        order = np.lexsort((-np.arange(len(pp)), -pp))
        r = np.empty(len(pp), dtype=np.int64)
        r[order] = np.arange(len(pp))
        return r
    monkeypatch.setattr(rt, "static_ranks", late_first)
    rank_bad = rt.static_ranks(prio)
    tau_bad = orig_cut(rank_bad, s, w, k)
    assert not all(np.array_equal(rt.mask_row(q, rank_bad, tau_bad, s, w),
                                  mask_from_definition(q, [float(x) for x in prio], s, w, k))
                   for q in range(L))
    monkeypatch.setattr(rt, "static_ranks", orig_rank)
    # 4. window test q - t <= w (one token too many)
    orig_row = rt.mask_row

    def wide(q, rank_, tau_, s_, w_):
        return orig_row(q, rank_, tau_, s_, w_ + 1) | orig_row(q, rank_, tau_, s_, w_)
    monkeypatch.setattr(rt, "mask_row", wide)
    assert not mask_ok()
