"""kvpop_attend_noalloc: decode attention whose split-K scratch is a fixed array
inside the library, for callers that may not allocate device memory while they
decode.  Its output must match kvpop_decode_attend's on the same cache state,
within the tolerance of the other attention tests, on two calls in a row.

This file is named to be collected last, so a run that stops at the first
failure has run every other test before it."""
import numpy as np
import pytest
import torch

from gpu_harness import TOL, gpu_prefill, make_cache
from workload import gen, get_config

pytestmark = pytest.mark.gpu

STATE_FIELDS = ("slotK", "slotV", "ringK", "ringV", "nvalid", "len")


def caller_buffers(cache, device):
    """Device copies, owned by the caller, of the cache state the entry point reads."""
    from paper_2607_05061_gb300 import kvpop
    st = kvpop.parse_state(cache.export_state(), cache.cfg)
    return {k: torch.from_numpy(np.ascontiguousarray(st[k])).to(device) for k in STATE_FIELDS}


@pytest.mark.parametrize("name,over", [
    ("tiny", {}),
    ("q4b", dict(batch=4, prompt_len=2000, budget_B=512)),
    ("cr8x", dict(batch=8, prompt_len=6000)),
])
def test_noalloc_attention_matches_decode_attend(cuda_device, name, over):
    from paper_2607_05061_gb300 import kvpop
    cfg = get_config(name, **over)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    cache = make_cache(cfg, w)
    gpu_prefill(cache, cfg, L, cuda_device)
    q, k, v = gen.decode_inputs(cfg, L, 0, 2, device=cuda_device)
    shape = (cfg.batch, cfg.n_q_heads, cfg.head_dim)
    stream = torch.cuda.current_stream().cuda_stream
    for j in range(2):                      # two calls in a row share the scratch array
        cache.ingest(q[j], k[j], v[j])
        ref = torch.empty(shape, dtype=torch.float32, device=cuda_device)
        cache.attend(q[j], ref)
        buf = caller_buffers(cache, cuda_device)
        out = torch.full(shape, float("nan"), dtype=torch.float32, device=cuda_device)
        rc = kvpop.kvpop_attend_noalloc(
            buf["slotK"].data_ptr(), buf["slotV"].data_ptr(), buf["ringK"].data_ptr(),
            buf["ringV"].data_ptr(), buf["nvalid"].data_ptr(), buf["len"].data_ptr(),
            q[j].data_ptr(), out.data_ptr(), cfg.batch, cfg.n_kv_heads, cfg.q_per_kv,
            cfg.head_dim, cfg.budget_B, cfg.delay_D, kvpop.dtype_code(cfg.kv_dtype), stream)
        assert rc == 0, kvpop.kvpop_last_error()
        torch.cuda.synchronize()
        err = (out - ref).abs().max().item()
        print(f"{name} call {j}: max-abs difference to kvpop_decode_attend {err:.3e}")
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
