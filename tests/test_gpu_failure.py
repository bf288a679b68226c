"""Failure detection on the GPU without a GPU fault.

* A bounded device wait that runs out is reported, and the context stays usable:
  with the testing hook kvpop_debug_skip_attention_copies on, the tensor-core
  decode attention's copy thread issues nothing, so every consumer's first
  mbarrier wait expires after the kernels' wait limit, records a timeout and
  skips its work.  kvpop_check must then return KVPOP_ERR_DEVICE_CHECK; with the
  hook off the same cache keeps decoding and still matches the fp64 oracle
  (evictions bit-exact, attention within the bf16 tolerance).
* The device-check build (index checks that record an error instead of
  trapping) runs the small parity cases in a child process and must pass them
  with no check recorded.
"""
import os
import subprocess
import sys

import pytest
import torch

from gpu_harness import (TOL, compare, gpu_decode, gpu_prefill, injected_decode_scores,
                         injected_prefill_scores, make_cache, oracle_pairs)
from workload import gen, get_config

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
KVPOP_ERR_DEVICE_CHECK = 6


def test_expired_wait_is_reported_and_the_cache_keeps_working(cuda_device):
    from paper_2607_05061_gb300 import kvpop
    cfg = get_config("q4b", batch=2, prompt_len=600, budget_B=256, decode_steps=12)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    steps = cfg.decode_steps
    pov = injected_prefill_scores(cfg, max(L), "cpu")
    dov = injected_decode_scores(cfg, steps + 1, "cpu")
    cache = make_cache(cfg, w)
    gpu_prefill(cache, cfg, L, cuda_device, override=pov.to(cuda_device))
    assert cache.check() is None
    q, k, v = gen.decode_inputs(cfg, L, 0, 1, device=cuda_device)
    # the state the attention reads is the same before and after the failed launch:
    # run the failing attention on step 0's state, then step 0 again for real
    blob = cache.export_state()
    cache.ingest(q[0], k[0], v[0], override=dov[0].to(cuda_device))
    out = torch.zeros((cfg.batch, cfg.n_q_heads, cfg.head_dim), device=cuda_device)
    stream = torch.cuda.current_stream().cuda_stream
    kvpop.kvpop_debug_skip_attention_copies(1)
    try:
        cache.attend(q[0], out)
    finally:
        kvpop.kvpop_debug_skip_attention_copies(0)
    rc = kvpop.kvpop_check(cache.handle, stream)
    assert rc == KVPOP_ERR_DEVICE_CHECK, kvpop.STATUS.get(rc, rc)
    assert kvpop.kvpop_check(cache.handle, stream) == 0          # the record was cleared
    # the context and the cache are usable: restore the pre-step state and decode
    cache.import_state(blob)
    pairs = [(b, h) for b in range(cfg.batch) for h in range(cfg.n_kv_heads)]
    g = gpu_decode(cache, cfg, L, steps, cuda_device, override=dov[:steps].to(cuda_device))
    ref = oracle_pairs(cfg, w, L, steps, pairs, prefill_override=pov, decode_override=dov[:steps])
    err = compare(cfg, g, ref, pairs)
    print(f"after the expired wait: max-abs attention error {err:.3e}")
    assert err <= TOL[cfg.kv_dtype]
    cache.free()


def test_parity_cases_under_the_device_check_build(cuda_device):
    from paper_2607_05061_gb300 import build
    build.build(checked=True)
    env = dict(os.environ, KVPOP_DEVICE_CHECKS="1")
    cmd = [sys.executable, "-m", "pytest", "-x", "-q", "-m", "gpu", "-p", "no:cacheprovider",
           "tests/test_gpu_parity.py", "tests/test_gpu_prompt.py", "tests/test_gpu_mlstm.py",
           "-k", "tiny or injected or planted or checkpoint or bitexact or matches_oracle"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    tail = r.stdout[-3000:] + r.stderr[-2000:]
    print(tail)
    assert r.returncode == 0, tail
    assert " passed" in r.stdout
