"""The largest configuration the C ABI accepts: 12288 (sequence, KV head) pairs, the
limit set by the decode attention's tile schedule in shared memory.  With injected
scores, evictions must match the oracle bit for bit and attention within the bf16
tolerance on sampled pairs (first, last and one in between), after a prompt that
already overflows the budget.  One pair more is rejected by kvpop_init_cache (a
host-side check, tests/test_abi_host.py).

This file is named to be collected after the other parity tests (only the
allocation-free attention's test comes later), so a run that stops at the first
failure has run them before this large case."""
import pytest

from gpu_harness import (TOL, compare, gpu_decode, gpu_prefill, injected_decode_scores,
                         injected_prefill_scores, make_cache, oracle_pairs)
from workload import gen, get_config

pytestmark = pytest.mark.gpu

MAX_PAIRS = 12288


def test_largest_accepted_pair_count(cuda_device):
    cfg = get_config("q4b", batch=MAX_PAIRS // 8, prompt_len=24, budget_B=16, delay_D=4,
                     decode_steps=6)
    assert cfg.batch * cfg.n_kv_heads == MAX_PAIRS
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    steps = cfg.decode_steps
    sample = [(0, 0), (cfg.batch // 2, 3), (cfg.batch - 1, cfg.n_kv_heads - 1)]
    pov = injected_prefill_scores(cfg, max(L), cuda_device)
    dov = injected_decode_scores(cfg, steps, cuda_device)
    cache = make_cache(cfg, w)
    gpu_prefill(cache, cfg, L, cuda_device, override=pov)
    g = gpu_decode(cache, cfg, L, steps, cuda_device, override=dov, sample=sample)
    ref = oracle_pairs(cfg, w, L, steps, sample, prefill_override=pov.cpu(),
                       decode_override=dov.cpu())
    err = 0.0
    for i, ((b, h), tr) in enumerate(zip(sample, ref)):
        pos, _ = cache.pair_state(b, h)
        assert len(pos) == min(cfg.budget_B, max(0, L[b] + steps - cfg.delay_D))
        sub = type(g)(g.evict, g.scores, g.outputs[:, i:i + 1])
        err = max(err, compare(cfg, sub, [tr], [(b, h)]))
    print(f"{MAX_PAIRS} pairs: sampled max-abs attention error {err:.3e}")
    assert err <= TOL[cfg.kv_dtype]
    cache.free()
