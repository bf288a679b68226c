"""The seeded input recipe (workload/gen.py), checked on the CPU: the counter hash
against a scalar restatement of PCG-RXS-M-XS (Jarzynski & Olano, JCGT 2020), the
discretised N(0, 1) table and its moments, prompt and decode tokens drawn from one
stream per (sequence, head), the outlier key channels, the ragged prompt lengths
and the Xavier-normal scorer weights.  The generator holds none of the method's
arithmetic; these tests pin only what the input recipe states."""
import numpy as np
import pytest
import torch
from scipy.special import ndtri

from workload import gen, get_config

M32 = 0xFFFFFFFF


def pcg_scalar(v: int) -> int:
    """PCG-RXS-M-XS, 32-bit state and output, from its published definition."""
    state = (v * 747796405 + 2891336453) % (1 << 32)
    word = (((state >> ((state >> 28) + 4)) ^ state) * 277803737) % (1 << 32)
    return (word >> 22) ^ word


def test_vectorised_hash_equals_the_scalar_definition():
    rng = np.random.default_rng(5)
    xs = np.concatenate([np.arange(64), rng.integers(0, 1 << 32, 4096), [M32, M32 - 1, 1 << 31]])
    got = gen._pcg(torch.tensor(xs, dtype=torch.int64)).numpy()
    want = np.array([pcg_scalar(int(x)) for x in xs], dtype=np.int64)
    assert np.array_equal(got, want)
    assert all(gen._pcg_int(int(x)) == pcg_scalar(int(x)) for x in xs[:256])


def test_normal_table_is_the_midpoint_quantiles():
    t = gen._table_cpu().numpy().astype(np.float64)
    mid = (np.arange(65536) + 0.5) / 65536.0
    assert np.array_equal(t, ndtri(mid).astype(np.float32).astype(np.float64))
    assert np.all(np.diff(t) > 0) and abs(t[0] + t[-1]) < 1e-6      # sorted, symmetric
    assert 4.2 < t[-1] < 4.4                                          # tails cut near 4.3 sigma


def test_normal_values_have_unit_moments_and_are_reproducible():
    flat = torch.arange(1 << 20, dtype=torch.int64)
    v = gen.normal_values(0, gen.STREAM_K, flat).double()
    assert abs(v.mean().item()) < 5e-3 and abs(v.std().item() - 1.0) < 5e-3
    assert torch.equal(gen.normal_values(0, gen.STREAM_K, flat[:1000]),
                       gen.normal_values(0, gen.STREAM_K, flat[:1000]))
    # streams and seeds are independent index spaces
    w = gen.normal_values(0, gen.STREAM_V, flat).double()
    u = gen.normal_values(1, gen.STREAM_K, flat).double()
    assert abs(float((v * w).mean())) < 5e-3 and abs(float((v * u).mean())) < 5e-3


def test_prompt_and_decode_tokens_are_one_stream():
    cfg = get_config("q4b", batch=3, prompt_len=40)
    L = [40, 17, 33]
    q, k, v = gen.decode_inputs(cfg, L, 2, 3)
    G = cfg.q_per_kv
    for b in range(3):
        for j in range(3):
            p = L[b] + 2 + j
            kt = gen.kv_tokens(cfg, "k", b, 1, p, 1)[0, :, 0]
            vt = gen.kv_tokens(cfg, "v", b, 1, p, 1)[0, :, 0]
            qt = gen.q_tokens(cfg, b, 1, p, 1)[0, :, 0]
            assert torch.equal(k[j, b], kt) and torch.equal(v[j, b], vt) and torch.equal(q[j, b], qt)
    assert q.shape == (3, 3, cfg.n_kv_heads * G, cfg.head_dim)


def test_outlier_key_channels_are_scaled_on_every_head():
    cfg = get_config("cr8x", batch=1)
    ch = gen.outlier_channels(cfg)
    assert len(ch) == cfg.n_outlier == 4 and ch == sorted(set(ch))
    assert all(0 <= c < cfg.head_dim for c in ch)
    K = gen.kv_tokens(cfg, "k", 0, 1, 0, 2048).float()[0]          # [H][t][d]
    V = gen.kv_tokens(cfg, "v", 0, 1, 0, 2048).float()[0]
    rest = [c for c in range(cfg.head_dim) if c not in ch]
    for h in (0, cfg.n_kv_heads - 1):
        sd = K[h].std(dim=0)
        assert torch.all((sd[ch] > 9.0) & (sd[ch] < 11.0))
        assert torch.all((sd[rest] > 0.9) & (sd[rest] < 1.1))
    assert float(V.std(dim=1).max()) < 1.1                          # values carry no outliers
    assert gen.outlier_channels(get_config("q8b_stack")) == []


def test_ragged_lengths_are_seeded_and_in_range():
    cfg = get_config("ragged")
    L = gen.prompt_lengths(cfg)
    assert L == gen.prompt_lengths(cfg) and len(L) == cfg.batch
    assert min(L) >= 1024 and max(L) <= 65536 and len(set(L)) > cfg.batch // 2
    assert gen.prompt_lengths(get_config("cr8x")) == [32768] * 64


@pytest.mark.parametrize("name", ["tiny", "cr8x"])
def test_scorer_weights_are_xavier_normal_with_zero_biases(name):
    cfg = get_config(name)
    W1, b1, w2, b2, lg = gen.scorer_weights(cfg)
    H, I, F = cfg.n_kv_heads, cfg.scorer_in, cfg.scorer_hidden
    assert W1.shape == (H, I, F) and w2.shape == (H, F) and b1.shape == (H, F) and b2.shape == (H,)
    assert abs(W1.double().std().item() / np.sqrt(2.0 / (I + F)) - 1.0) < 0.05
    assert not torch.any(b1) and not torch.any(b2)
    assert torch.all(lg == cfg.log_gamma)
    W1b = gen.scorer_weights(cfg)[0]
    assert torch.equal(W1, W1b)
