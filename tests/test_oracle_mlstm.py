"""Pins of the mLSTM scorer oracle (App. A, App. E.3-E.4) against closed forms:
the gated recurrence unrolled as an explicit sum, its reduction to linear
attention, Hedgehog feature invariants and the delayed-readout index."""
import numpy as np
import pytest

from oracle.kvpop_oracle import OracleParams
from oracle.mlstm import (MlstmHeadCache, MlstmParams, MlstmState, hedgehog, log_sigmoid,
                          prefill_mlstm)


def rand_params(rng, d, bf=1.0, scale=1.0):
    n2, h = 2 * d, d // 2
    g = lambda *s: rng.standard_normal(s) * scale / np.sqrt(s[0])
    return MlstmParams(g(n2, h), g(n2, h), g(n2, h), g(n2), g(n2), 0.1, bf, g(h), 0.05)


def test_hedgehog_invariants():
    rng = np.random.default_rng(0)
    y = rng.standard_normal((5, 8)) * 3
    f = hedgehog(y)
    assert f.shape == (5, 16)
    assert np.all(f > 0)
    assert np.allclose(f[:, :8].sum(axis=1), 1.0) and np.allclose(f[:, 8:].sum(axis=1), 1.0)
    assert np.allclose(hedgehog(np.zeros(8)), 1.0 / 8)
    # the negative half is the positive half of -y
    assert np.allclose(f[:, 8:], hedgehog(-y)[:, :8])


def unrolled_readout(p: MlstmParams, xs, x_u):
    """h from C_T = sum_t (prod_{s>t} f_s) i_t k~_t v~_t^T, no recurrence, no stabiliser."""
    sig = lambda a: 1.0 / (1.0 + np.exp(-a))
    T = len(xs)
    f = np.array([sig(x @ p.wf + p.bf) for x in xs])
    i = np.array([np.exp(x @ p.wi + p.bi) for x in xs])
    C = 0.0
    z = 0.0
    for t in range(T):
        w = np.prod(f[t + 1:]) * i[t]
        C = C + w * np.outer(hedgehog(xs[t] @ p.Wk), xs[t] @ p.Wv)
        z = z + w * hedgehog(xs[t] @ p.Wk)
    q = hedgehog(x_u @ p.Wq)
    return (q @ C) / (q @ z)


@pytest.mark.parametrize("seed", range(4))
def test_stabilised_recurrence_equals_unrolled_sum(seed):
    rng = np.random.default_rng(seed)
    d = 8
    p = rand_params(rng, d, bf=rng.normal())
    xs = rng.standard_normal((30, 2 * d)) * 2
    st = MlstmState(p, d)
    for t, x in enumerate(xs):
        st.update(x)
        if t >= 3:
            x_u = xs[t - 3]
            h_rec = st.readout(x_u)
            h_ref = unrolled_readout(p, xs[:t + 1], x_u)
            assert np.allclose(h_rec, h_ref, rtol=1e-10, atol=1e-12)


def test_unit_gates_reduce_to_linear_attention():
    """f = 1, i = 1: h = sum_t (q~ . k~_t) v~_t / sum_t (q~ . k~_t) (App. A linear attention)."""
    rng = np.random.default_rng(5)
    d = 8
    p = rand_params(rng, d)
    p.wi[:] = 0.0
    p.bi = 0.0
    p.wf[:] = 0.0
    p.bf = 80.0                       # sigmoid(80) = 1 in fp64
    xs = rng.standard_normal((12, 2 * d))
    st = MlstmState(p, d)
    for x in xs:
        st.update(x)
    x_u = xs[4]
    q = hedgehog(x_u @ p.Wq)
    w = np.array([q @ hedgehog(x @ p.Wk) for x in xs])
    ref = (w[:, None] * np.stack([x @ p.Wv for x in xs])).sum(0) / w.sum()
    assert np.allclose(st.readout(x_u), ref, rtol=1e-12)


def test_delayed_readout_sees_tokens_up_to_the_current_position():
    """With uniform features and unit gates, h[0] is the mean of v~_t[0] = t over t = 0..p."""
    d, D = 4, 3
    n2, h = 2 * d, d // 2
    mp = MlstmParams(np.zeros((n2, h)), np.zeros((n2, h)), np.zeros((n2, h)), np.zeros(n2),
                     np.zeros(n2), 0.0, 80.0, np.array([1.0, 0.0]), 0.0)
    mp.Wv[0, 0] = 1.0                 # v~_t[0] = k_t[0]
    op = OracleParams(np.zeros((3 * d, 1)), np.zeros(1), np.zeros(1), 0.0, 100, D)
    c = MlstmHeadCache(op, mp, d, 1)
    for t in range(12):
        k = np.zeros(d)
        k[0] = t
        _, _, r = c.append(np.zeros((1, d)), k, np.zeros(d))
        if t >= D:
            hval = t / 2.0                            # mean of 0..t
            silu = hval / (1.0 + np.exp(-hval))       # a = e_0, b = 0
            assert abs(float(r) - np.float32(silu)) < 1e-6


def test_log_sigmoid_matches_definition():
    for x in (-30.0, -1.0, 0.0, 2.5, 40.0):
        assert abs(log_sigmoid(x) - np.log(1.0 / (1.0 + np.exp(-x)))) < 1e-12


def test_mlstm_prefill_equals_streaming():
    rng = np.random.default_rng(9)
    d, G, B, D, P = 8, 2, 5, 3, 40
    mp = rand_params(rng, d)
    op = OracleParams(np.zeros((3 * d, 1)), np.zeros(1), np.zeros(1), 0.0, B, D)
    Q = rng.standard_normal((G, P, d))
    K = rng.standard_normal((P, d))
    V = rng.standard_normal((P, d))
    a = prefill_mlstm(op, mp, Q, K, V, d, G)
    s = MlstmHeadCache(op, mp, d, G)
    for t in range(P):
        s.append(Q[:, t], K[t], V[t])
    assert a.kept_positions() == s.kept_positions()
    assert np.allclose(a.state.C, s.state.C) and np.allclose(a.state.z, s.state.z)
