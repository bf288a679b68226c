"""Pins of the future-attention target oracle (App. D, App. F.1-F.2).

Checked against: torch's softmax / logsumexp in fp64 (the App. D.1 identity
and the transposed-attention form of App. D.2), the closed form with all
logits equal (p_{d->t} = 1/(d+1), so the future mass is a difference of
harmonic numbers), the mass-conservation identity over all keys, the
sparse/dense normaliser relation of App. D.3 and hand-counted N_t.
"""
import numpy as np
import pytest
import torch

from oracle import future_target as ft
from oracle import running_topk as rt


def rand_qk(seed, S, dk, G=1):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((G, S, dk)), rng.standard_normal((S, dk))


def harmonic(n):
    return np.concatenate([[0.0], np.cumsum(1.0 / np.arange(1, n + 1))])


@pytest.mark.parametrize("S,w", [(20, 1), (33, 4), (16, 16), (9, 12)])
def test_dense_identity_against_library_softmax(S, w):
    Q, K = rand_qk(S + w, S, 8)
    lse = ft.dense_causal_lse(Q[0], K)
    logits = torch.from_numpy(Q[0] @ K.T / np.sqrt(8)).masked_fill(
        torch.triu(torch.ones(S, S, dtype=torch.bool), 1), -np.inf)
    assert np.abs(lse - torch.logsumexp(logits, 1).numpy()).max() < 1e-12
    P = torch.softmax(logits, dim=1).numpy()            # P[d, t]
    want = np.array([np.log(P[t + w:, t].sum()) if t + w < S else -np.inf for t in range(S)])
    got = ft.future_log_mass(Q[0], K, lse, w)
    fin = np.isfinite(want)
    assert np.array_equal(fin, np.isfinite(got))
    assert not fin.any() or np.abs(got[fin] - want[fin]).max() < 1e-12


def test_transposed_pass_form():
    """App. D.2: swap roles, subtract LSE_d as a score modifier, mask d >= t + w, take the LSE."""
    S, w, dk = 40, 3, 16
    Q, K = rand_qk(1, S, dk)
    lse = ft.dense_causal_lse(Q[0], K)
    qt, kt = torch.from_numpy(K), torch.from_numpy(Q[0])                  # q'_t = k_t, k'_d = q_d
    scores = qt @ kt.T / np.sqrt(dk) - torch.from_numpy(lse)[None, :]     # [t][d]
    d_idx, t_idx = torch.arange(S)[None, :], torch.arange(S)[:, None]
    scores = scores.masked_fill(d_idx < t_idx + w, -np.inf)
    want = torch.logsumexp(scores, dim=1).numpy()
    got = ft.future_log_mass(Q[0], K, lse, w)
    fin = np.isfinite(want)
    assert np.array_equal(fin, np.isfinite(got))
    assert np.abs(got[fin] - want[fin]).max() < 1e-12


@pytest.mark.parametrize("S,w,L", [(30, 1, 0), (30, 5, 0), (25, 2, 4), (25, 2, 100)])
def test_equal_logits_closed_form(S, w, L):
    """K = 0 gives p_{d->t} = 1/(d+1): mbar_t = H_{hi+1} - H_{t+w} (harmonic numbers)."""
    Q, _ = rand_qk(2, S, 4)
    K = np.zeros((S, 4))
    lse = ft.dense_causal_lse(Q[0], K)
    got = ft.future_log_mass(Q[0], K, lse, w, lookahead=L)
    Hn = harmonic(S + 1)
    for t in range(S):
        hi = S - 1 if L <= 0 else min(S - 1, t + w + L)
        if t + w > hi:
            assert got[t] == -np.inf
        else:
            assert abs(got[t] - np.log(Hn[hi + 1] - Hn[t + w])) < 1e-12


@pytest.mark.parametrize("w", [1, 3])
def test_mass_conservation(w):
    """sum_t mbar_t = sum_d (1 - mass of d's window), since each query row sums to one."""
    S = 50
    Q, K = rand_qk(3, S, 8)
    lse = ft.dense_causal_lse(Q[0], K)
    mb = np.exp(ft.future_log_mass(Q[0], K, lse, w))
    logits = torch.from_numpy(Q[0] @ K.T / np.sqrt(8)).masked_fill(
        torch.triu(torch.ones(S, S, dtype=torch.bool), 1), -np.inf)
    P = torch.softmax(logits, 1).numpy()
    win = sum(P[d, max(0, d - w + 1): d + 1].sum() for d in range(S))
    assert abs(mb.sum() - (S - win)) < 1e-10


def test_sparse_normaliser_variant():
    """App. D.3: the sparse LSE never exceeds the dense one, so its target is never smaller;
    with a budget covering the sequence the two coincide."""
    S, s, w, k, dk, G = 60, 1, 4, 10, 8, 2
    Q, K = rand_qk(4, S, dk, G)
    V = np.zeros((S, dk))
    rng = np.random.default_rng(4)
    rank = rt.static_ranks(rng.standard_normal(S).astype(np.float32))
    for kk, same in ((k, False), (S, True)):
        tau = rt.fenwick_cutoffs(rank, s, w, kk)
        _, lse_sp = rt.masked_attention(Q, K, V, rank, tau, s, w)
        for g in range(G):
            dense = ft.dense_causal_lse(Q[g], K)
            assert np.all(lse_sp[g] <= dense + 1e-12)
            a = ft.future_log_mass(Q[g], K, lse_sp[g], w)
            b = ft.future_log_mass(Q[g], K, dense, w)
            fin = np.isfinite(b)
            if same:
                assert np.abs(a[fin] - b[fin]).max() < 1e-12
            else:
                assert np.all(a[fin] >= b[fin] - 1e-12)


def test_counts_by_hand():
    assert list(ft.future_count(10, 3)) == [7, 6, 5, 4, 3, 2, 1, 1, 1, 1]
    assert list(ft.future_count(10, 3, lookahead=2)) == [3, 3, 3, 3, 3, 2, 1, 1, 1, 1]


def test_aggregation_variants():
    S, w, eps = 12, 2, 1e-6
    with np.errstate(divide="ignore"):
        logm = np.log(np.array([[0.5, 0.2, 0.0, 0.3] * 3, [0.1, 0.4, 0.0, 0.3] * 3]))
    N = ft.future_count(S, w)
    r_max = ft.aggregate_target(logm, S, w, eps, "max")
    r_mean = ft.aggregate_target(logm, S, w, eps, "mean")
    m = np.exp(logm) / N
    assert np.allclose(r_max, np.log(eps + np.maximum(m[0], m[1])), rtol=0, atol=1e-14)
    assert np.allclose(r_mean, np.log(eps + 0.5 * (m[0] + m[1])), rtol=0, atol=1e-14)
    assert r_max[2] == np.log(eps)                          # no mass from any head
    raw = ft.aggregate_target(logm, S, w, eps, "max", count_norm=False)
    assert np.allclose(raw, np.log(eps + np.maximum(np.exp(logm[0]), np.exp(logm[1]))), atol=1e-14)


def test_target_pins_catch_planted_mistakes(monkeypatch):
    S, w = 30, 2
    Q, K = rand_qk(5, S, 4)
    K0 = np.zeros((S, 4))
    Hn = harmonic(S + 1)

    def closed_form_ok():
        got = ft.future_log_mass(Q[0], K0, ft.dense_causal_lse(Q[0], K0), w)
        return all(abs(got[t] - np.log(Hn[S] - Hn[t + w])) < 1e-12 for t in range(S - w))

    assert closed_form_ok()
    orig = ft.future_log_mass
    # 1. window off by one (d > t + w)
    monkeypatch.setattr(ft, "future_log_mass", lambda Qg, K_, lse, w_, lookahead=0: orig(Qg, K_, lse, w_ + 1, lookahead))
    assert not closed_form_ok()
    # 2. the normaliser dropped from the score modifier
    monkeypatch.setattr(ft, "future_log_mass", lambda Qg, K_, lse, w_, lookahead=0: orig(Qg, K_, np.zeros_like(lse), w_, lookahead))
    assert not closed_form_ok()
    monkeypatch.setattr(ft, "future_log_mass", orig)
    # 3. aggregation by sum instead of max
    orig_agg = ft.aggregate_target
    monkeypatch.setattr(ft, "aggregate_target", lambda lm, S_, w_, e, agg="max", **kw:
                        np.log(e + (np.exp(lm) / ft.future_count(S_, w_)[None]).sum(0)))
    logm = np.log(np.full((2, S), 0.25))
    m = 0.25 / ft.future_count(S, w)
    assert not np.allclose(ft.aggregate_target(logm, S, w, 1e-6, "max"), np.log(1e-6 + m))
    monkeypatch.setattr(ft, "aggregate_target", orig_agg)
