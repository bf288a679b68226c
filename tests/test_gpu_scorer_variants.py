"""GPU parity of the plain stateless scorer variants (Sec. 3.3): the MLP on [k; v]
with a SiLU or identity hidden layer, and SiLU on [k; v; qbar].  The GPU
scorer's values against the oracle's (relative 2e-5), evictions bit-exact when
both consume the oracle's scores, attention within the dtype tolerance; both
ingest kernels (plain and cluster) and the prompt scorer are exercised."""
import numpy as np
import pytest
import torch

from gpu_harness import TOL, compare, gpu_decode, gpu_prefill, make_cache, oracle_pairs
from workload import gen, get_config

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,over", [
    ("tiny", dict(scorer_act="silu", scorer_kv_only=True, decode_steps=200)),
    ("tiny", dict(scorer_act="identity", scorer_kv_only=True, decode_steps=120)),
    ("tiny", dict(scorer_act="silu", decode_steps=120)),
    ("q4b", dict(scorer_act="silu", scorer_kv_only=True, batch=16, prompt_len=600, budget_B=256,
                 decode_steps=64)),
])
def test_scorer_variant_against_oracle(cuda_device, name, over):
    cfg = get_config(name).with_(**over)
    w = gen.scorer_weights(cfg)
    assert w[0].shape[1] == cfg.scorer_in
    L = gen.prompt_lengths(cfg)
    steps = cfg.decode_steps
    pairs = [(b, h) for b in range(cfg.batch) for h in range(cfg.n_kv_heads)]
    if cfg.batch > 2:
        pairs = [(0, 0), (cfg.batch - 1, cfg.n_kv_heads - 1), (5, 3)]
    ref = oracle_pairs(cfg, w, L, steps, pairs)
    # own scores: per-token values
    cache = make_cache(cfg, w)
    gpu_prefill(cache, cfg, L, cuda_device)
    g = gpu_decode(cache, cfg, L, steps, cuda_device, sample=pairs)
    for (b, h), tr in zip(pairs, ref):
        want = np.asarray(tr.scores, dtype=np.float64)
        got = g.scores[:, b, h].astype(np.float64)
        ok = np.isnan(want) == np.isnan(got)
        assert ok.all()
        m = ~np.isnan(want)
        assert np.all(np.abs(got[m] - want[m]) <= 2e-5 * (1.0 + np.abs(want[m]))), (b, h)
        raw = tr.cache.prefill_raw
        pos, sc = cache.pair_state(b, h)
    cache.free()
    # the oracle's scores injected: bit-exact evictions
    Pmax = max(L)
    pov = torch.zeros((cfg.batch, cfg.n_kv_heads, Pmax), dtype=torch.float32)
    dov = torch.zeros((steps, cfg.batch, cfg.n_kv_heads), dtype=torch.float32)
    pre = oracle_pairs(cfg, w, L, 0, pairs)
    for (b, h), tr, tp in zip(pairs, ref, pre):
        raw = tp.cache.prefill_raw
        pov[b, h, :raw.size] = torch.from_numpy(raw)
        dov[:, b, h] = torch.tensor(np.asarray(tr.scores, dtype=np.float32))
    cache = make_cache(cfg, w)
    gpu_prefill(cache, cfg, L, cuda_device, override=pov.to(cuda_device))
    g = gpu_decode(cache, cfg, L, steps, cuda_device, override=dov.to(cuda_device), sample=pairs)
    err = 0.0
    for i, ((b, h), tr) in enumerate(zip(pairs, ref)):
        sub = type(g)(g.evict, g.scores, g.outputs[:, i:i + 1])
        err = max(err, compare(cfg, sub, [tr], [(b, h)]))
    print(f"{name} {over}: max-abs attention error {err:.2e}")
    assert err <= TOL[cfg.kv_dtype]
    cache.free()
