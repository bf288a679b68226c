"""Shared helpers of the GPU parity tests: drive the CUDA library through the
C ABI (via the ctypes binding) on inputs from the seeded generator, and drive
the fp64 oracle on the same inputs."""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional, Sequence

import numpy as np
import torch

from workload import gen

TOL = {"f32": 1e-5, "bf16": 2e-2}      # attention max-abs tolerance per K/V dtype
STREAM_PREFILL_OV, STREAM_DECODE_OV = 30, 31


def make_cache(cfg, weights, mlstm=None, step=None):
    """A cache for `cfg`; step="fused" / "split" forces the one-kernel / two-kernel
    kvpop_decode_step (default: the library's choice by the size of a step)."""
    import os
    from paper_2607_05061_gb300 import kvpop
    if step is not None:
        saved = {k: os.environ.pop(k, None) for k in ("KVPOP_FUSED_STEP", "KVPOP_SPLIT_STEP")}
        os.environ["KVPOP_FUSED_STEP" if step == "fused" else "KVPOP_SPLIT_STEP"] = "1"
        try:
            return make_cache(cfg, weights, mlstm)
        finally:
            for k in ("KVPOP_FUSED_STEP", "KVPOP_SPLIT_STEP"):
                os.environ.pop(k, None)
                if saved[k] is not None:
                    os.environ[k] = saved[k]
    if mlstm is not None:
        return kvpop.KVpopCache(cfg.batch, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim, cfg.budget_B,
                                cfg.delay_D, cfg.scorer_hidden, cfg.kv_dtype, n_sink=cfg.n_sink,
                                mlstm=mlstm)
    W1, b1, w2, b2, lg = weights
    return kvpop.KVpopCache(cfg.batch, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim, cfg.budget_B,
                            cfg.delay_D, cfg.scorer_hidden, cfg.kv_dtype, W1, b1, w2, b2,
                            log_gamma=(lg if cfg.log_gamma != 0.0 else None), n_sink=cfg.n_sink,
                            activation=cfg.scorer_act, kv_only=cfg.scorer_kv_only)


def injected_prefill_scores(cfg, Pmax, device, levels=None):
    return gen.uniform_scores(cfg.seed, STREAM_PREFILL_OV, (cfg.batch, cfg.n_kv_heads, Pmax),
                              device=device, levels=levels)


def injected_decode_scores(cfg, nsteps, device, levels=None):
    return gen.uniform_scores(cfg.seed, STREAM_DECODE_OV, (nsteps, cfg.batch, cfg.n_kv_heads),
                              device=device, levels=levels)


def gpu_prefill(cache, cfg, lengths, device, override=None, group=8, layer=0):
    for b0 in range(0, cfg.batch, group):
        nb = min(group, cfg.batch - b0)
        L = list(lengths[b0:b0 + nb])
        Pm = max(L) if L else 0
        if Pm == 0:
            cache.prefill(None, None, None, L, first_seq=b0)
            continue
        Q = gen.q_tokens(cfg, b0, nb, 0, Pm, device=device, layer=layer)
        K = gen.kv_tokens(cfg, "k", b0, nb, 0, Pm, device=device, layer=layer)
        V = gen.kv_tokens(cfg, "v", b0, nb, 0, Pm, device=device, layer=layer)
        ov = None
        if override is not None:
            ov = override[b0:b0 + nb, :, :Pm].contiguous()
        cache.prefill(Q, K, V, L, first_seq=b0, override=ov)
        del Q, K, V, ov


@dataclass
class GpuTrace:
    evict: np.ndarray        # [steps][b][H][2]
    scores: np.ndarray       # [steps][b][H]
    outputs: np.ndarray      # [steps][n_pairs_sampled][G][d]


def gpu_decode(cache, cfg, lengths, nsteps, device, override=None,
               sample: Optional[Sequence] = None, step0: int = 0, split: bool = False) -> GpuTrace:
    """Run ``nsteps`` decode steps; keep outputs of the sampled (b, h) pairs (all if None).

    Each step is one kvpop_decode_step call (one kernel where the cache supports it), or
    with ``split`` a kvpop_decode_ingest and a kvpop_decode_attend call."""
    b, H, G, d = cfg.batch, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim
    q, k, v = gen.decode_inputs(cfg, lengths, step0, nsteps, device=device)
    out = torch.empty((b, H * G, d), dtype=torch.float32, device=device)
    ei = torch.empty((nsteps, b, H, 2), dtype=torch.int32, device=device)
    sc = torch.empty((nsteps, b, H), dtype=torch.float32, device=device)
    pairs = [(bb, hh) for bb in range(b) for hh in range(H)] if sample is None else list(sample)
    sel = torch.tensor([bb * H + hh for bb, hh in pairs], dtype=torch.int64, device=device)
    outs = torch.empty((nsteps, len(pairs), G, d), dtype=torch.float32, device=device)
    for j in range(nsteps):
        ov = None if override is None else override[j]
        if split:
            cache.ingest(q[j], k[j], v[j], override=ov, evict_info=ei[j], score_out=sc[j])
            cache.attend(q[j], out)
        else:
            cache.step(q[j], k[j], v[j], out, override=ov, evict_info=ei[j], score_out=sc[j])
        outs[j] = out.view(b * H, G, d).index_select(0, sel)
    torch.cuda.synchronize()
    cache.check()
    return GpuTrace(ei.cpu().numpy(), sc.cpu().numpy(), outs.cpu().numpy())


def oracle_pairs(cfg, weights, lengths, nsteps, pairs, prefill_override=None, decode_override=None,
                 attend=True, mlstm=None):
    """Oracle traces for the listed (b, h) pairs (injected scores given as CPU tensors)."""
    from oracle.run import run_pair
    traces = []
    for bb, hh in pairs:
        P = lengths[bb]
        pov = None if prefill_override is None else prefill_override[bb, hh, :P].numpy()
        dov = None
        if decode_override is not None:
            col = decode_override[:, bb, hh].numpy()
            dov = (lambda c: (lambda j: float(c[j])))(col)
        traces.append(run_pair(cfg, weights, bb, hh, P, nsteps, prefill_override=pov,
                               step_override=dov, attend=attend, keep_cache=True, mlstm=mlstm))
    return traces


def compare(cfg, gpu: GpuTrace, traces, pairs, check_evict=True):
    """Bit-exact evictions (when asked) and max-abs attention error; returns the error."""
    err = 0.0
    for i, ((bb, hh), tr) in enumerate(zip(pairs, traces)):
        n = len(tr.slots)
        if check_evict:
            got = gpu.evict[:n, bb, hh]
            want = np.stack([np.asarray(tr.slots), np.asarray(tr.evicted)], axis=1)
            bad = np.nonzero((got != want).any(axis=1))[0]
            assert bad.size == 0, (f"pair {(bb, hh)}: first eviction mismatch at step {bad[0]}: "
                                   f"gpu {got[bad[0]]} oracle {want[bad[0]]}")
        if tr.outputs:
            o = np.stack(tr.outputs)
            err = max(err, float(np.abs(gpu.outputs[:n, i] - o).max()))
    return err
