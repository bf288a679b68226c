"""kvpop_attend_noalloc: decode attention whose split-K scratch is a fixed array
inside the library, for callers that may not allocate device memory while they
decode (a serving loop with a device-memory plan fixed up front, or a plugin
that may only use the buffers its host framework hands it).

Its output is compared with the fp64 oracle's decode attention on sampled
(sequence, KV head) pairs, on two calls in a row (the calls share the array),
within the attention tolerance of every other parity test; after each call
kvpop_standalone_status, which reads the device error word the call records
into, must report no expired wait.

This file is named to be collected last, so a run that stops at the first
failure has run every other test before it."""
import numpy as np
import pytest
import torch

from gpu_harness import (TOL, gpu_prefill, injected_decode_scores, injected_prefill_scores,
                         make_cache, oracle_pairs)
from workload import gen, get_config

pytestmark = pytest.mark.gpu

STATE_FIELDS = ("slotK", "slotV", "ringK", "ringV", "nvalid", "len")
N_CALLS = 2


def caller_buffers(cache, device):
    """Device copies, owned by the caller, of the cache state the entry point reads."""
    from paper_2607_05061_gb300 import kvpop
    st = kvpop.parse_state(cache.export_state(), cache.cfg)
    return {k: torch.from_numpy(np.array(st[k], copy=True)).to(device) for k in STATE_FIELDS}


def sampled_pairs(cfg, n=4):
    total = cfg.batch * cfg.n_kv_heads
    idx = sorted({(i * total) // n + (i % cfg.n_kv_heads) for i in range(n)})
    return [(i // cfg.n_kv_heads, i % cfg.n_kv_heads) for i in idx if i < total]


@pytest.mark.parametrize("name,over", [
    ("tiny", {}),
    ("q4b", dict(batch=4, prompt_len=2000, budget_B=512)),
    ("cr8x", dict(batch=8, prompt_len=6000)),
])
def test_noalloc_attention_matches_oracle(cuda_device, name, over):
    from paper_2607_05061_gb300 import kvpop
    cfg = get_config(name, **over)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    pairs = sampled_pairs(cfg)
    # injected scores make both sides keep the same tokens by construction
    pov = injected_prefill_scores(cfg, max(L), "cpu")
    dov = injected_decode_scores(cfg, N_CALLS, "cpu")
    cache = make_cache(cfg, w)
    gpu_prefill(cache, cfg, L, cuda_device, override=pov.to(cuda_device))
    # the oracle computes the sampled pairs from the same seeds and scores
    traces = oracle_pairs(cfg, w, L, N_CALLS, pairs, prefill_override=pov, decode_override=dov)
    dov_d = dov.to(cuda_device)
    q, k, v = gen.decode_inputs(cfg, L, 0, N_CALLS, device=cuda_device)
    shape = (cfg.batch, cfg.n_q_heads, cfg.head_dim)
    G = cfg.q_per_kv
    stream = torch.cuda.current_stream().cuda_stream
    assert kvpop.kvpop_standalone_status(stream) == 0, kvpop.kvpop_last_error()
    for j in range(N_CALLS):                 # two calls in a row share the scratch array
        ei = torch.empty((cfg.batch, cfg.n_kv_heads, 2), dtype=torch.int32, device=cuda_device)
        cache.ingest(q[j], k[j], v[j], override=dov_d[j], evict_info=ei)
        buf = caller_buffers(cache, cuda_device)
        out = torch.full(shape, float("nan"), dtype=torch.float32, device=cuda_device)
        rc = kvpop.kvpop_attend_noalloc(
            buf["slotK"].data_ptr(), buf["slotV"].data_ptr(), buf["ringK"].data_ptr(),
            buf["ringV"].data_ptr(), buf["nvalid"].data_ptr(), buf["len"].data_ptr(),
            q[j].data_ptr(), out.data_ptr(), cfg.batch, cfg.n_kv_heads, cfg.q_per_kv,
            cfg.head_dim, cfg.budget_B, cfg.delay_D, kvpop.dtype_code(cfg.kv_dtype), stream)
        assert rc == 0, kvpop.kvpop_last_error()
        assert kvpop.kvpop_standalone_status(stream) == 0, kvpop.kvpop_last_error()
        o = out.cpu().numpy().reshape(cfg.batch, cfg.n_kv_heads, G, cfg.head_dim)
        ei = ei.cpu().numpy()
        err = 0.0
        for (bb, hh), tr in zip(pairs, traces):
            # the kept set the caller's buffers hold is the oracle's (same decisions)
            assert tuple(ei[bb, hh]) == (tr.slots[j], tr.evicted[j]), (bb, hh, j)
            err = max(err, float(np.abs(o[bb, hh] - tr.outputs[j]).max()))
        assert np.isfinite(o).all()
        print(f"{name} call {j}: max-abs error to the fp64 oracle {err:.3e} on {len(pairs)} pairs")
        assert err <= TOL[cfg.kv_dtype]
    cache.check()
    cache.free()


def test_noalloc_rejects_oversize(cuda_device):
    from paper_2607_05061_gb300 import kvpop
    x = torch.zeros(64, dtype=torch.float32, device=cuda_device)
    p = x.data_ptr()
    stream = torch.cuda.current_stream().cuda_stream
    rc = kvpop.kvpop_attend_noalloc(p, p, p, p, p, p, p, p, 4096, 8, 4, 128, 64, 16,
                                    kvpop.KVPOP_BF16, stream)
    assert rc == 1
    assert b"12288" in kvpop.kvpop_last_error()
