"""GPU parity of the stateful delayed mLSTM scorer (App. A, E.3, E.4) against the
fp64 oracle: bit-exact evictions with injected scores, per-token scores of the
GPU recurrence against the oracle's, and checkpoint/resume of the state."""
import numpy as np
import pytest
import torch

from gpu_harness import (TOL, compare, gpu_decode, gpu_prefill, injected_decode_scores,
                         injected_prefill_scores, make_cache, oracle_pairs)
from workload import gen, get_config

pytestmark = pytest.mark.gpu

CASES = [
    ("tiny", dict(prompt_len=100, budget_B=24, decode_steps=80)),
    ("q4b", dict(batch=2, prompt_len=400, budget_B=96, decode_steps=80)),
    ("q4b", dict(batch=2, prompt_len=300, budget_B=64, decode_steps=60, n_sink=2, log_gamma=-0.003)),
]


def all_pairs(cfg):
    return [(b, h) for b in range(cfg.batch) for h in range(cfg.n_kv_heads)]


@pytest.mark.parametrize("name,over", CASES)
def test_mlstm_injected_scores_bitexact(cuda_device, name, over):
    cfg = get_config(name, **over)
    mw = gen.mlstm_weights(cfg)
    L = gen.prompt_lengths(cfg)
    pairs = all_pairs(cfg)
    pov = injected_prefill_scores(cfg, max(L), "cpu")
    dov = injected_decode_scores(cfg, cfg.decode_steps, "cpu")
    cache = make_cache(cfg, None, mlstm=mw)
    gpu_prefill(cache, cfg, L, cuda_device, override=pov.to(cuda_device))
    g = gpu_decode(cache, cfg, L, cfg.decode_steps, cuda_device, override=dov.to(cuda_device))
    ref = oracle_pairs(cfg, None, L, cfg.decode_steps, pairs, prefill_override=pov,
                       decode_override=dov, mlstm=mw)
    err = compare(cfg, g, ref, pairs)
    print(f"mlstm {name} {over}: max-abs attention error {err:.3e}")
    assert err <= TOL[cfg.kv_dtype]
    cache.free()


@pytest.mark.parametrize("name,over", CASES[:2])
def test_mlstm_scores_match_oracle_recurrence(cuda_device, name, over):
    cfg = get_config(name, **over)
    mw = gen.mlstm_weights(cfg)
    L = gen.prompt_lengths(cfg)
    pairs = all_pairs(cfg)
    steps = cfg.decode_steps
    cache = make_cache(cfg, None, mlstm=mw)
    gpu_prefill(cache, cfg, L, cuda_device)
    pre = oracle_pairs(cfg, None, L, 0, pairs, mlstm=mw)
    agree, worst = [], 0.0
    for (b, h), tr in zip(pairs, pre):
        pos, sc = cache.pair_state(b, h)
        o = set(tr.cache.kept_positions())
        agree.append(len(o & set(pos)) / max(1, len(o)))
        raw = tr.cache.prefill_raw
        for p_, s_ in zip(pos, sc):
            worst = max(worst, abs(s_ - float(raw[p_])) / (1.0 + abs(float(raw[p_]))))
    g = gpu_decode(cache, cfg, L, steps, cuda_device)
    ref = oracle_pairs(cfg, None, L, steps, pairs, mlstm=mw, attend=False)
    n_same = 0
    for (b, h), tr in zip(pairs, ref):
        want = np.asarray(tr.scores, dtype=np.float64)
        got = g.scores[:, b, h].astype(np.float64)
        worst = max(worst, float(np.max(np.abs(got - want) / (1.0 + np.abs(want)))))
        ev = g.evict[:, b, h]
        n_same += int(((ev[:, 0] == np.asarray(tr.slots)) & (ev[:, 1] == np.asarray(tr.evicted))).sum())
    print(f"mlstm {name}: worst relative score error {worst:.2e}; prefill kept-set agreement "
          f"{np.mean(agree):.4f}; decode eviction agreement {n_same / (steps * len(pairs)):.4f}")
    assert worst <= 1e-4
    cache.free()


def test_mlstm_checkpoint_resume_is_bit_identical(cuda_device):
    cfg = get_config("q4b", batch=2, prompt_len=300, budget_B=64, decode_steps=40)
    mw = gen.mlstm_weights(cfg)
    L = gen.prompt_lengths(cfg)
    a = make_cache(cfg, None, mlstm=mw)
    gpu_prefill(a, cfg, L, cuda_device)
    gpu_decode(a, cfg, L, 20, cuda_device)
    blob = a.export_state()
    b = make_cache(cfg, None, mlstm=mw)
    b.import_state(blob)
    ga = gpu_decode(a, cfg, L, 20, cuda_device, step0=20)
    gb = gpu_decode(b, cfg, L, 20, cuda_device, step0=20)
    assert np.array_equal(ga.evict, gb.evict)
    assert np.array_equal(ga.scores, gb.scores)
    assert np.array_equal(ga.outputs, gb.outputs)
    a.free()
    b.free()


def test_mlstm_full_size_sampled(cuda_device):
    """cr8x shape (P 32768, B 4096, D 16) with the mLSTM scorer, on sampled pairs the
    oracle computes in full: bit-exact evictions and attention with injected scores,
    then the GPU recurrence's own scores against the oracle's."""
    cfg = get_config("cr8x", batch=8)
    mw = gen.mlstm_weights(cfg)
    L = gen.prompt_lengths(cfg)
    steps = 24
    sample = [(0, 0), (5, 3), (7, 7)]
    pov = injected_prefill_scores(cfg, max(L), "cpu")
    dov = injected_decode_scores(cfg, steps, "cpu")
    cache = make_cache(cfg, None, mlstm=mw)
    gpu_prefill(cache, cfg, L, cuda_device, override=pov.to(cuda_device))
    g = gpu_decode(cache, cfg, L, steps, cuda_device, override=dov.to(cuda_device), sample=sample)
    ref = oracle_pairs(cfg, None, L, steps, sample, prefill_override=pov, decode_override=dov,
                       mlstm=mw)
    err = compare(cfg, g, ref, sample)
    print(f"mlstm cr8x injected: max-abs attention error {err:.3e}")
    assert err <= TOL[cfg.kv_dtype]
    cache.free()
    # own scores: the recurrence over the whole 32768-token prompt, then decode
    cache = make_cache(cfg, None, mlstm=mw)
    gpu_prefill(cache, cfg, L, cuda_device)
    g = gpu_decode(cache, cfg, L, steps, cuda_device, sample=sample)
    ref = oracle_pairs(cfg, None, L, steps, sample, mlstm=mw, attend=False)
    worst = 0.0
    for (b, h), tr in zip(sample, ref):
        want = np.asarray(tr.scores, dtype=np.float64)
        got = g.scores[:, b, h].astype(np.float64)
        worst = max(worst, float(np.max(np.abs(got - want) / (1.0 + np.abs(want)))))
        ev = g.evict[:, b, h]
        same = (ev[:, 0] == np.asarray(tr.slots)) & (ev[:, 1] == np.asarray(tr.evicted))
        print(f"mlstm cr8x {(b, h)}: decode eviction agreement {same.mean():.4f}")
    print(f"mlstm cr8x: worst relative decode score error {worst:.2e}")
    assert worst <= 1e-4
    cache.free()
