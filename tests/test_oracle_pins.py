"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these checks re-types the oracle's own formulas: they compare it with
library routines (torch SDPA in fp64, scipy's normal CDF tables), with brute
force over all subsets, with the App. C.1 mask recomputed from its definition,
and with hand-traced fixtures under tests/golden/.
"""
import itertools

import numpy as np
import pytest
import torch

from conftest import read_golden
from oracle import (HeadCache, OracleParams, gelu_erf, prefill_head,
                    prefill_head_streaming, round_score, scorer_mlp)
from oracle import kvpop_oracle as ok


def make_params(rng, d, F, B, D, s=0, log_gamma=0.0, scale=1.0):
    W1 = rng.standard_normal((3 * d, F)) * scale / np.sqrt(3 * d)
    b1 = rng.standard_normal(F) * 0.1
    w2 = rng.standard_normal(F) / np.sqrt(F)
    return OracleParams(W1, b1, w2, 0.05, B, D, s, log_gamma)


def random_stream(rng, n, G, d):
    return (rng.standard_normal((n, G, d)), rng.standard_normal((n, d)),
            rng.standard_normal((n, d)))


# ---------------------------------------------------------------- reference pieces
def sdpa_masked(q, K, V, mask):
    """Library attention (torch SDPA, fp64) of one query row per head over keys with a mask."""
    qt = torch.from_numpy(q)[None, :, None, :]                      # [1][G][1][d]
    kt = torch.from_numpy(K)[None, None].expand(1, q.shape[0], -1, -1)
    vt = torch.from_numpy(V)[None, None].expand(1, q.shape[0], -1, -1)
    m = torch.from_numpy(mask)[None, None, None, :].expand(1, q.shape[0], 1, -1)
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=m)
    return o[0, :, 0, :].numpy()


def mask_from_definition(q_pos, prio, s, w, k):
    """App. C.1: M_{q,t} = [t < s] or [q - t < w] or ([t in E(q)] and rank(t) <= tau_q).

    E(q) = {t : s <= t <= q - w} (Eq. 4).  The top-k of E(q) is taken by sorting
    the static priorities (App. B.3) descending, earlier position first on ties;
    when |E(q)| < k every eligible token is kept.
    """
    n = q_pos + 1
    mask = np.zeros(n, dtype=bool)
    for t in range(n):
        if t < s or q_pos - t < w:
            mask[t] = True
    elig = [t for t in range(s, q_pos - w + 1)]
    ranked = sorted(elig, key=lambda t: (-prio[t], t))
    for t in ranked[:k]:
        mask[t] = True
    return mask


# ---------------------------------------------------------------- GELU / scorer
def test_gelu_matches_normal_cdf_table():
    for z, phi in read_golden("normal_cdf.txt"):
        z, phi = float(z), float(phi)
        assert abs(gelu_erf(z) - z * phi) < 1e-15 * max(1.0, abs(z))


def test_gelu_limits():
    assert gelu_erf(0.0) == 0.0
    assert abs(gelu_erf(40.0) - 40.0) < 1e-12
    assert abs(gelu_erf(-40.0)) < 1e-12


def test_scorer_input_order_and_handset_weights():
    """A one-hot W1 routes a single input coordinate into one hidden unit."""
    d, F = 4, 3
    W1 = np.zeros((3 * d, F))
    W1[1, 0] = 1.0           # k[1]
    W1[d + 2, 1] = 1.0       # v[2]
    W1[2 * d + 3, 2] = 1.0   # qbar[3]
    p = OracleParams(W1, np.zeros(F), np.array([1.0, 10.0, 100.0]), 0.5, 4, 1)
    k = np.array([0.0, 1.0, 0.0, 0.0])
    v = np.array([0.0, 0.0, -1.0, 0.0])
    qb = np.array([0.0, 0.0, 0.0, 2.0])
    x = np.concatenate([k, v, qb])
    phi = {float(a): float(b) for a, b in read_golden("normal_cdf.txt")}
    # GELU(z) = z Phi(z) at z = 1, -1, 2 from the table
    expect = 1.0 * (1.0 * phi[1.0]) + 10.0 * (-1.0 * phi[-1.0]) + 100.0 * (2.0 * phi[2.0]) + 0.5
    assert abs(scorer_mlp(x, p) - expect) < 1e-12


def test_qbar_is_mean_of_next_D_queries_over_group():
    """qbar_u averages queries u+1..u+D over the G heads (delayed scoring, Sec. 3.3)."""
    d, G, D = 3, 2, 4
    p = OracleParams(np.zeros((3 * d, 1)), np.zeros(1), np.zeros(1), 0.0, 8, D)
    c = HeadCache(p, d, G)
    seen = []
    for t in range(12):
        q = np.stack([np.full(d, t + 0.1 * g) for g in range(G)])   # mean over g: t + 0.05
        if t >= D:
            u, x = c.scorer_input(q.mean(axis=0))
            seen.append((u, x[2 * d:]))
        c.append(q, np.full(d, float(t)), np.full(d, -float(t)))
    for u, qbar in seen:
        # closed form: (1/D) sum_{j=1..D} (u + j + 0.05) = u + (D + 1)/2 + 0.05
        assert np.allclose(qbar, u + (D + 1) / 2 + 0.05, atol=1e-12)


def test_round_score_canonical():
    assert round_score(np.nan) == -np.inf
    assert np.signbit(round_score(-0.0)) == False  # noqa: E712
    assert round_score(1.0 / 3.0) == np.float32(1.0 / 3.0)


# ---------------------------------------------------------------- attention reductions
def dense_equivalence_error(seed=0, d=8, G=2, D=3, P=10, steps=12):
    rng = np.random.default_rng(seed)
    p = make_params(rng, d, 5, P + steps + 4, D)      # B >= context: nothing is evicted
    Q, K, V = random_stream(rng, P + steps, G, d)
    c = prefill_head(p, Q[:P].transpose(1, 0, 2), K[:P], V[:P], d, G)
    err = 0.0
    for j in range(steps):
        t = P + j
        c.append(Q[t], K[t], V[t])
        out, probs, pos = c.attend(Q[t])
        ref = sdpa_masked(Q[t], K[:t + 1], V[:t + 1], np.ones(t + 1, dtype=bool))
        # the compact cache holds positions in slot/window order; compare as sets of keys
        assert sorted(pos.tolist()) == list(range(t + 1))
        err = max(err, float(np.abs(out - ref).max()))
    return err


def test_budget_covering_context_is_dense_causal_attention():
    assert dense_equivalence_error() < 1e-12


def test_attention_rows_sum_to_one():
    rng = np.random.default_rng(3)
    d, G = 16, 4
    p = make_params(rng, d, 8, 6, 2)
    Q, K, V = random_stream(rng, 40, G, d)
    c = HeadCache(p, d, G)
    for t in range(40):
        c.append(Q[t], K[t], V[t])
        _, probs, _ = c.attend(Q[t])
        assert np.all(probs >= 0)
        assert np.abs(probs.sum(axis=1) - 1.0).max() < 1e-12


def mask_equivalence_error(seed=1, d=8, G=2, B=5, D=3, s=0, log_gamma=0.0, n=40):
    """Oracle decode output vs dense attention under the App. C.1 mask built from scratch."""
    rng = np.random.default_rng(seed)
    p = make_params(rng, d, 6, B, D, s, log_gamma)
    Q, K, V = random_stream(rng, n, G, d)
    raw = rng.standard_normal(n).astype(np.float32)
    c = HeadCache(p, d, G)
    err = 0.0
    for t in range(n):
        ov = raw[t - D] if t >= D else None
        c.append(Q[t], K[t], V[t], ov)
        out, _, _ = c.attend(Q[t])
        prio = [float(raw[u]) - u * np.float32(log_gamma) for u in range(n)]
        mask = mask_from_definition(t, prio, s, D, B - s)
        ref = sdpa_masked(Q[t], K[:t + 1], V[:t + 1], mask)
        err = max(err, float(np.abs(out - ref).max()))
    return err


@pytest.mark.parametrize("B,D,s,lg", [(5, 3, 0, 0.0), (4, 1, 0, 0.0), (6, 2, 2, 0.0),
                                      (5, 3, 1, -0.05), (1, 1, 0, 0.0), (3, 4, 0, -0.3)])
def test_decode_equals_running_topk_mask(B, D, s, lg):
    assert mask_equivalence_error(seed=B * 7 + D, B=B, D=D, s=s, log_gamma=lg) < 1e-12


# ---------------------------------------------------------------- selection: brute force
def all_subset_best(elig, prio, k):
    """The k-subset of `elig` with the largest priority sum (unique for distinct priorities)."""
    if len(elig) <= k:
        return set(elig)
    best, best_sum = None, -np.inf
    for comb in itertools.combinations(elig, k):
        ssum = sum(prio[t] for t in comb)
        if ssum > best_sum:
            best, best_sum = set(comb), ssum
    return best


@pytest.mark.parametrize("seed", range(12))
def test_kept_set_is_topB_by_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    P = int(rng.integers(2, 17))
    B = int(rng.integers(1, 5))
    D = int(rng.integers(1, 4))
    d, G = 4, 2
    p = make_params(rng, d, 3, B, D)
    Q, K, V = random_stream(rng, P, G, d)
    raw = rng.permutation(P).astype(np.float32) * 0.5 - 3.0       # distinct scores
    c = HeadCache(p, d, G)
    for t in range(P):
        c.append(Q[t], K[t], V[t], raw[t - D] if t >= D else None)
        elig = list(range(0, t - D + 1))
        assert set(c.kept_positions()) == all_subset_best(elig, raw, B)
        pend = [e[0] for e in c.pending]
        assert pend == list(range(max(0, t - D + 1), t + 1))       # the D pending tokens
    cp = prefill_head(p, Q.transpose(1, 0, 2), K, V, d, G, override=raw)
    assert cp.kept_positions() == c.kept_positions()
    assert [e[0] for e in cp.pending] == [e[0] for e in c.pending]


def test_prefill_equals_streaming_with_scorer():
    rng = np.random.default_rng(7)
    d, G, B, D, P = 8, 2, 6, 3, 30
    p = make_params(rng, d, 7, B, D)
    Q, K, V = random_stream(rng, P, G, d)
    a = prefill_head(p, Q.transpose(1, 0, 2), K, V, d, G)
    b = prefill_head_streaming(p, Q.transpose(1, 0, 2), K, V, d, G)
    assert a.kept_positions() == b.kept_positions()
    assert sorted(a.slot_prio[:a.n_valid]) == sorted(b.slot_prio[:b.n_valid])


def test_all_equal_scores_keep_earliest():
    """With one score value, (score desc, pos asc) and the strict-beat rule both keep the first B."""
    rng = np.random.default_rng(8)
    d, G, B, D, P = 4, 1, 3, 2, 12
    p = make_params(rng, d, 2, B, D)
    Q, K, V = random_stream(rng, P, G, d)
    ov = np.full(P, 0.25, dtype=np.float32)
    a = prefill_head(p, Q.transpose(1, 0, 2), K, V, d, G, ov)
    b = prefill_head_streaming(p, Q.transpose(1, 0, 2), K, V, d, G, ov)
    assert a.kept_positions() == b.kept_positions() == [0, 1, 2]


def test_ties_keep_equal_score_multiset():
    rng = np.random.default_rng(9)
    d, G, B, D, P = 4, 1, 4, 2, 40
    p = make_params(rng, d, 2, B, D)
    Q, K, V = random_stream(rng, P, G, d)
    ov = (rng.integers(0, 4, P) * 0.5).astype(np.float32)
    a = prefill_head(p, Q.transpose(1, 0, 2), K, V, d, G, ov)
    b = prefill_head_streaming(p, Q.transpose(1, 0, 2), K, V, d, G, ov)
    assert sorted(a.slot_prio[:B]) == sorted(b.slot_prio[:B])


# ---------------------------------------------------------------- hand-traced fixtures
@pytest.mark.parametrize("name", ["eviction_trace_basic.txt", "eviction_trace_sink.txt"])
def test_hand_traced_eviction(name):
    rows = read_golden(name)
    B, D, s = (int(x) for x in rows[0])
    steps = [r for r in rows[1:-1]]
    final = [int(x) for x in rows[-1]]
    d, G = 2, 1
    p = OracleParams(np.zeros((3 * d, 1)), np.zeros(1), np.zeros(1), 0.0, B, D, s)
    c = HeadCache(p, d, G)
    scores = {int(r[1]): float(r[2]) for r in steps}
    expect = {int(r[0]): (int(r[3]), int(r[4])) for r in steps}
    last = max(expect)
    for t in range(last + 1):
        u = t - D
        slot, ev, _ = c.append(np.zeros((G, d)), np.full(d, t), np.full(d, -t),
                               scores.get(u) if u >= 0 else None)
        if t in expect:
            assert (slot, ev) == expect[t], f"p={t}"
    assert [int(x) for x in c.slot_pos[:c.n_valid]] == final


# ---------------------------------------------------------------- decay (App. B.3)
def test_static_priority_matches_effective_score_ranking():
    """Ranking by r + (q - t) log(gamma) at each q equals ranking by r - t log(gamma) (n = 1)."""
    rng = np.random.default_rng(11)
    n, B, D, lg = 60, 5, 2, -0.2
    raw = (rng.permutation(n) * 0.37).astype(np.float32)
    p = OracleParams(np.zeros((3, 1)), np.zeros(1), np.zeros(1), 0.0, B, D, 0, lg)
    c = HeadCache(p, 1, 1)
    for t in range(n):
        c.append(np.zeros((1, 1)), np.zeros(1), np.zeros(1), raw[t - D] if t >= D else None)
        elig = list(range(0, t - D + 1))
        eff = {u: float(raw[u]) + (t - u) * lg for u in elig}       # Eq. 5 form, q = t
        top = sorted(elig, key=lambda u: (-eff[u], u))[:B]
        assert set(c.kept_positions()) == set(top)


def test_nan_scores_never_displace():
    p = OracleParams(np.zeros((3, 1)), np.zeros(1), np.zeros(1), 0.0, 2, 1)
    c = HeadCache(p, 1, 1)
    seq = [1.0, 2.0, np.nan, np.nan, 3.0]
    for t in range(len(seq) + 1):
        c.append(np.zeros((1, 1)), np.zeros(1), np.zeros(1), seq[t - 1] if t >= 1 else None)
    assert c.kept_positions() == [1, 4]


# ---------------------------------------------------------------- planted mistakes
def test_pins_catch_planted_mistakes(monkeypatch):
    """Each plausible oracle mistake, planted on the CPU, fails at least one pin."""
    # 1. attention without the 1/sqrt(d) scale
    orig = ok.attend_head

    def no_scale(q, K, V):
        logits = q @ K.T
        e = np.exp(logits - logits.max(axis=1, keepdims=True))
        pr = e / e.sum(axis=1, keepdims=True)
        return pr @ V, pr
    monkeypatch.setattr(ok, "attend_head", no_scale)
    assert dense_equivalence_error() > 1e-6
    monkeypatch.setattr(ok, "attend_head", orig)

    # 2. window one token too short (u = p - D + 1 scored and moved early)
    orig_append = HeadCache.append

    def short_window(self, q, k, v, override=None):
        self.p.delay_D -= 1
        try:
            if self.p.delay_D < 1:
                self.p.delay_D = 1
            return orig_append(self, q, k, v, override)
        finally:
            self.p.delay_D += 1
    monkeypatch.setattr(HeadCache, "append", short_window)
    assert mask_equivalence_error(B=5, D=3) > 1e-6
    monkeypatch.setattr(HeadCache, "append", orig_append)

    # 3. ties evicting the highest slot instead of the lowest
    orig_place = HeadCache._place

    def tie_high(self, u, k_u, v_u, r32):
        if self.n_valid < self.p.budget_B:
            return orig_place(self, u, k_u, v_u, r32)
        cand = self.slot_prio[self.p.n_sink:]
        j = len(cand) - 1 - int(np.argmin(cand[::-1])) + self.p.n_sink
        if r32 > self.slot_prio[j]:
            ev = int(self.slot_pos[j])
            self.slot_prio[j] = r32
            self.slot_pos[j] = u
            return j, ev, r32
        return -1, -1, r32
    monkeypatch.setattr(HeadCache, "_place", tie_high)
    with pytest.raises(AssertionError):
        test_hand_traced_eviction("eviction_trace_basic.txt")
    monkeypatch.setattr(HeadCache, "_place", orig_place)

    # 4. tanh-approximate GELU
    monkeypatch.setattr(ok, "gelu_erf",
                        lambda z: 0.5 * z * (1 + np.tanh(np.sqrt(2 / np.pi) * (z + 0.044715 * z ** 3))))
    with pytest.raises(AssertionError):
        for z, phi in read_golden("normal_cdf.txt"):
            assert abs(ok.gelu_erf(float(z)) - float(z) * float(phi)) < 1e-12


# ---------------------------------------------------------------- plain [k; v] scorer variants
def test_silu_textbook_values():
    """SiLU(z) = z * sigmoid(z); sigmoid(1) = 0.7310585786300049, sigmoid(2) = 0.8807970779778823."""
    z = np.array([0.0, 1.0, 2.0, -1.0, -2.0, 60.0, -60.0])
    want = [0.0, 0.7310585786300049, 2 * 0.8807970779778823, -(1 - 0.7310585786300049),
            -2 * (1 - 0.8807970779778823), 60.0, 0.0]
    got = ok.silu(z)
    assert np.allclose(got, want, rtol=1e-14, atol=1e-24)


@pytest.mark.parametrize("act", ["silu", "identity"])
def test_kv_only_scorer_handset_weights(act):
    """Input [k; v] (no query mean): W1 rows 0..d-1 read k, d..2d-1 read v."""
    d, F, D = 2, 2, 2
    W1 = np.zeros((2 * d, F))
    W1[0, 0] = 1.0          # unit 0 <- k[0]
    W1[d + 1, 1] = -2.0     # unit 1 <- -2 v[1]
    b1 = np.array([0.5, 0.0])
    w2 = np.array([1.0, 3.0])
    p = OracleParams(W1, b1, w2, 0.25, 4, D, 0, 0.0, act)
    c = HeadCache(p, d, 1)
    k0, v0 = np.array([1.5, 9.0]), np.array([7.0, -0.75])
    c.append(np.full((1, d), 100.0), k0, v0)
    c.append(np.full((1, d), 100.0), np.zeros(d), np.zeros(d))
    u, x = c.scorer_input(np.full(d, 100.0))
    assert u == 0 and np.array_equal(x, np.concatenate([k0, v0]))
    z0, z1 = 1.5 + 0.5, -2.0 * -0.75
    f = ok.silu if act == "silu" else (lambda y: y)
    want = 1.0 * f(z0) + 3.0 * f(z1) + 0.25
    assert abs(float(ok.scorer_mlp(x, p)) - want) < 1e-14
