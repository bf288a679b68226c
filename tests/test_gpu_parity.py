"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on the
same seeded inputs.

* Evictions (slot, evicted position) must match bit for bit when both sides
  consume the same scores (the oracle's own fp32 scores, or injected ones).
* Attention outputs must match within max-abs 1e-5 (fp32 K/V) or 2e-2 (bf16).
* The GPU scorer is compared with the oracle's scorer value by value, and the
  end-to-end eviction agreement with the GPU's own scores is reported.
"""
import numpy as np
import pytest
import torch

from gpu_harness import (TOL, compare, gpu_decode, gpu_prefill, injected_decode_scores,
                         injected_prefill_scores, make_cache, oracle_pairs)
from workload import gen, get_config

pytestmark = pytest.mark.gpu


def all_pairs(cfg):
    return [(b, h) for b in range(cfg.batch) for h in range(cfg.n_kv_heads)]


# ---------------------------------------------------------------- tiny config, full
def test_tiny_bitexact_with_oracle_scores(cuda_device):
    cfg = get_config("tiny")
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    pairs = all_pairs(cfg)
    steps = cfg.decode_steps
    ref = oracle_pairs(cfg, w, L, steps, pairs)             # oracle with its own scorer
    Pmax = max(L)
    pov = torch.zeros((cfg.batch, cfg.n_kv_heads, Pmax), dtype=torch.float32)
    dov = torch.zeros((steps, cfg.batch, cfg.n_kv_heads), dtype=torch.float32)
    for (b, h), tr in zip(pairs, ref):
        raw = tr.cache.prefill_raw
        pov[b, h, :raw.size] = torch.from_numpy(raw)
        dov[:, b, h] = torch.tensor(np.asarray(tr.scores, dtype=np.float32))
    cache = make_cache(cfg, w)
    gpu_prefill(cache, cfg, L, cuda_device, override=pov.to(cuda_device))
    pre = oracle_pairs(cfg, w, L, 0, pairs, prefill_override=pov)
    for (b, h), t in zip(pairs, pre):
        pos, _ = cache.pair_state(b, h)
        assert pos == t.cache.kept_positions()
    g = gpu_decode(cache, cfg, L, steps, cuda_device, override=dov.to(cuda_device))
    err = compare(cfg, g, ref, pairs)
    print(f"tiny: max-abs attention error {err:.3e} over {steps} steps")
    assert err <= TOL["f32"]
    cache.free()


def test_tiny_gpu_scorer_against_oracle(cuda_device):
    cfg = get_config("tiny")
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    pairs = all_pairs(cfg)
    steps = cfg.decode_steps
    ref = oracle_pairs(cfg, w, L, steps, pairs)
    pre = oracle_pairs(cfg, w, L, 0, pairs)                   # oracle state right after prefill
    cache = make_cache(cfg, w)
    gpu_prefill(cache, cfg, L, cuda_device)
    # prefill: kept set agreement and per-slot priorities of the common slots
    agree = []
    for (b, h), tr in zip(pairs, pre):
        pos, sc = cache.pair_state(b, h)
        o = set(tr.cache.kept_positions())
        agree.append(len(o & set(pos)) / max(1, len(o)))
        raw = tr.cache.prefill_raw
        for p_, s_ in zip(pos, sc):
            assert abs(s_ - float(raw[p_])) <= 2e-5 * (1.0 + abs(float(raw[p_])))
    g = gpu_decode(cache, cfg, L, steps, cuda_device)
    n_same, n_all = 0, 0
    for (b, h), tr in zip(pairs, ref):
        want = np.asarray(tr.scores, dtype=np.float64)
        got = g.scores[:, b, h].astype(np.float64)
        assert np.all(np.abs(got - want) <= 2e-5 * (1.0 + np.abs(want))), "scorer mismatch"
        ev = g.evict[:, b, h]
        n_same += int(((ev[:, 0] == np.asarray(tr.slots)) & (ev[:, 1] == np.asarray(tr.evicted))).sum())
        n_all += steps
    print(f"tiny: prefill kept-set agreement {np.mean(agree):.4f}; "
          f"decode eviction agreement with GPU scores {n_same / n_all:.4f}")
    assert np.mean(agree) >= 0.99
    cache.free()


# ---------------------------------------------------------------- reduced bf16, all pairs
SMALL = dict(batch=2, prompt_len=600, budget_B=256, decode_steps=200)


@pytest.mark.parametrize("name,over", [
    ("q4b", SMALL),
    ("q4b", dict(SMALL, n_sink=3)),
    ("q4b", dict(SMALL, log_gamma=-0.002)),
    ("q4b", dict(SMALL, budget_B=1, delay_D=1, prompt_len=40, decode_steps=60)),
    ("q4b", dict(SMALL, budget_B=900, prompt_len=300, decode_steps=100)),       # B >= context: dense
    ("q4b", dict(SMALL, prompt_len=5, decode_steps=80)),                       # P < D
    ("q4b", dict(SMALL, prompt_len=0, decode_steps=70)),                       # no prompt
    ("q4b", dict(SMALL, q_per_kv=1, head_dim=64)),
    ("q4b", dict(SMALL, q_per_kv=2)),
    ("tiny", dict(batch=3, head_dim=128, q_per_kv=4, prompt_len=200, budget_B=40, delay_D=7,
                  decode_steps=120)),
    ("tiny", dict(q_per_kv=1, prompt_len=90, budget_B=16, delay_D=2, decode_steps=90)),
])
@pytest.mark.parametrize("path", ["fused", "split"])
def test_injected_scores_bitexact(cuda_device, name, over, path):
    """Every case on both kvpop_decode_step paths (one kernel where the shape allows it:
    bf16, d = 128; the fp32 and d = 64 cases run the two-kernel path either way)."""
    cfg = get_config(name, **over)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    pairs = all_pairs(cfg)
    steps = cfg.decode_steps
    Pmax = max(1, max(L))
    pov = injected_prefill_scores(cfg, Pmax, "cpu")
    dov = injected_decode_scores(cfg, steps, "cpu")
    cache = make_cache(cfg, w, step=path)
    gpu_prefill(cache, cfg, L, cuda_device, override=pov.to(cuda_device))
    g = gpu_decode(cache, cfg, L, steps, cuda_device, override=dov.to(cuda_device))
    ref = oracle_pairs(cfg, w, L, steps, pairs, prefill_override=pov, decode_override=dov)
    err = compare(cfg, g, ref, pairs)
    print(f"{name} {over} {path} (one kernel: {cache.fused_step}): max-abs attention error {err:.3e}")
    assert err <= TOL[cfg.kv_dtype]
    cache.free()


def test_fused_step_selected(cuda_device):
    """kvpop_decode_step is one kernel for bf16, d = 128, F = 256 when a step streams at
    least 600 MB of K/V (cr8x: 1.08 GB) or when asked; two kernels for a small stream
    (q4b: 0.10 GB), d = 64, fp32, or when asked."""
    def fused(name, step=None, **over):
        cfg = get_config(name, **over)
        c = make_cache(cfg, gen.scorer_weights(cfg), step=step)
        f = c.fused_step
        c.free()
        return f
    assert fused("cr8x", prompt_len=64)
    assert not fused("q4b")
    assert fused("q4b", step="fused", **SMALL)
    assert not fused("q4b", step="fused", **dict(SMALL, q_per_kv=1, head_dim=64))
    assert not fused("tiny", step="fused")
    assert not fused("cr8x", step="split", prompt_len=64)


@pytest.mark.parametrize("name,over", [
    ("q4b", SMALL),
    ("q4b", dict(SMALL, prompt_len=5, decode_steps=80, n_sink=2)),
])
def test_split_step_bitexact(cuda_device, name, over):
    """The two-call path (kvpop_decode_ingest + kvpop_decode_attend) on a cache whose
    kvpop_decode_step is one kernel: the same oracle bar."""
    cfg = get_config(name, **over)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    pairs = all_pairs(cfg)
    steps = cfg.decode_steps
    pov = injected_prefill_scores(cfg, max(1, max(L)), "cpu")
    dov = injected_decode_scores(cfg, steps, "cpu")
    cache = make_cache(cfg, w, step="fused")
    gpu_prefill(cache, cfg, L, cuda_device, override=pov.to(cuda_device))
    g = gpu_decode(cache, cfg, L, steps, cuda_device, override=dov.to(cuda_device), split=True)
    ref = oracle_pairs(cfg, w, L, steps, pairs, prefill_override=pov, decode_override=dov)
    assert compare(cfg, g, ref, pairs) <= TOL[cfg.kv_dtype]
    cache.free()


def test_fused_partial_scorer_group(cuda_device):
    """20 sequences: two scorer units per KV head, the second with 4 of 16 rows."""
    cfg = get_config("q4b", batch=20, prompt_len=400, budget_B=128, decode_steps=64)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    pairs = all_pairs(cfg)
    steps = cfg.decode_steps
    pov = injected_prefill_scores(cfg, max(L), "cpu")
    dov = injected_decode_scores(cfg, steps, "cpu")
    cache = make_cache(cfg, w, step="fused")
    assert cache.fused_step
    gpu_prefill(cache, cfg, L, cuda_device, override=pov.to(cuda_device))
    g = gpu_decode(cache, cfg, L, steps, cuda_device, override=dov.to(cuda_device))
    ref = oracle_pairs(cfg, w, L, steps, pairs, prefill_override=pov, decode_override=dov)
    err = compare(cfg, g, ref, pairs)
    print(f"q4b b20: max-abs attention error {err:.3e}")
    assert err <= TOL["bf16"]
    cache.free()


def test_fused_and_split_own_scores(cuda_device):
    """Each path scoring on its own: the fused scorer against the oracle's scores (rel
    2e-5, the fp32-accurate bound of every scorer check), and both paths' outputs within
    the bf16 tolerance of each other."""
    cfg = get_config("q4b", batch=18, prompt_len=700, budget_B=256, decode_steps=48)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    steps = cfg.decode_steps
    a = make_cache(cfg, w, step="fused")
    b = make_cache(cfg, w, step="split")
    assert a.fused_step and not b.fused_step
    gpu_prefill(a, cfg, L, cuda_device)
    gpu_prefill(b, cfg, L, cuda_device)
    ga = gpu_decode(a, cfg, L, steps, cuda_device)
    gb = gpu_decode(b, cfg, L, steps, cuda_device)
    sample = [(0, 0), (17, 7)]
    ref = oracle_pairs(cfg, w, L, steps, sample, attend=False)
    for (bb, hh), tr in zip(sample, ref):
        want = np.asarray(tr.scores, dtype=np.float64)
        got = ga.scores[:, bb, hh].astype(np.float64)
        rel = np.abs(got - want) / (1.0 + np.abs(want))
        assert np.all(rel <= 2e-5), f"fused scorer {(bb, hh)}: {np.nanmax(rel):.2e}"
    eq = (ga.evict == gb.evict).all(axis=-1)              # [steps][b][H]
    same = eq.mean()
    # outputs compared up to a pair's first differing decision (a near-tie decided the
    # other way by the last bit of a score changes the kept set from then on)
    diff = 0.0
    for bb in range(cfg.batch):
        for hh in range(cfg.n_kv_heads):
            bad = np.nonzero(~eq[:, bb, hh])[0]
            n = int(bad[0]) if bad.size else steps
            if n:
                i = bb * cfg.n_kv_heads + hh
                diff = max(diff, float(np.abs(ga.outputs[:n, i] - gb.outputs[:n, i]).max()))
    print(f"fused vs split, own scores: decisions equal {same:.4f}, max-abs output difference {diff:.2e}")
    assert diff <= TOL["bf16"]
    a.free()
    b.free()


def test_planted_ties_bitexact(cuda_device):
    """Scores drawn from 3 levels: argmin ties (lowest slot) and strict-beat drops."""
    cfg = get_config("q4b", batch=2, prompt_len=300, budget_B=64, decode_steps=150)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    pairs = all_pairs(cfg)
    pov = injected_prefill_scores(cfg, max(L), "cpu", levels=3)
    dov = injected_decode_scores(cfg, cfg.decode_steps, "cpu", levels=3)
    cache = make_cache(cfg, w)
    gpu_prefill(cache, cfg, L, cuda_device, override=pov.to(cuda_device))
    g = gpu_decode(cache, cfg, L, cfg.decode_steps, cuda_device, override=dov.to(cuda_device))
    ref = oracle_pairs(cfg, w, L, cfg.decode_steps, pairs, prefill_override=pov, decode_override=dov)
    assert compare(cfg, g, ref, pairs) <= TOL["bf16"]
    cache.free()


# ---------------------------------------------------------------- full sizes, sampled pairs
@pytest.mark.parametrize("name,steps,sample", [
    ("q4b", 256, [(0, 0), (3, 5), (7, 7)]),
    ("cr8x", 48, [(0, 0), (63, 7)]),
    ("ragged", 24, None),
    ("q8b_stack", 24, [(0, 0), (31, 7)]),    # one layer of the 8B stack: b32, P=32768, B=8192
])
def test_full_size_sampled(cuda_device, name, steps, sample):
    cfg = get_config(name, n_layers=1)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    if sample is None:   # shortest and longest sequence, and one below the budget
        order = sorted(range(cfg.batch), key=lambda b: L[b])
        below = [b for b in order if L[b] - cfg.delay_D < cfg.budget_B]
        sample = [(order[0], 1), (order[-1], 6)] + ([(below[-1], 3)] if below else [])
    Pmax = max(L)
    pov = injected_prefill_scores(cfg, Pmax, cuda_device)
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
    print(f"{name}: sampled max-abs attention error {err:.3e}")
    assert err <= TOL[cfg.kv_dtype]
    cache.free()


@pytest.mark.parametrize("path", ["fused", "split"])
def test_full_size_gpu_scorer(cuda_device, path):
    """cr8x shape, GPU scorer (of either kvpop_decode_step path): per-token scores vs the
    oracle scorer on sampled pairs."""
    cfg = get_config("cr8x", batch=8)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    steps = 32
    sample = [(0, 0), (5, 3)]
    cache = make_cache(cfg, w, step=path)
    gpu_prefill(cache, cfg, L, cuda_device)
    g = gpu_decode(cache, cfg, L, steps, cuda_device, sample=sample)
    ref = oracle_pairs(cfg, w, L, steps, sample, attend=False)
    for (b, h), tr in zip(sample, ref):
        want = np.asarray(tr.scores, dtype=np.float64)
        got = g.scores[:, b, h].astype(np.float64)
        # the same fp32-accurate bound as the other scorer checks (3xTF32 hidden slice)
        rel = np.abs(got - want) / (1.0 + np.abs(want))
        print(f"cr8x GPU scorer {(b, h)}: max relative score error {np.nanmax(rel):.2e}")
        assert np.all(rel <= 2e-5)
        pos, sc = cache.pair_state(b, h)
        o = set(tr.cache.kept_positions())
        # end-to-end decisions with each side's own scores: reported, not gated
        ev = g.evict[:, b, h]
        same = (ev[:, 0] == np.asarray(tr.slots)) & (ev[:, 1] == np.asarray(tr.evicted))
        print(f"cr8x GPU scorer {(b, h)}: final kept-set agreement "
              f"{len(o & set(pos)) / len(o):.4f}; decode eviction agreement {same.mean():.4f}")
    cache.free()


# ---------------------------------------------------------------- API behaviour
def test_checkpoint_resume_is_bit_identical(cuda_device):
    cfg = get_config("q4b", batch=2, prompt_len=500, budget_B=128, decode_steps=60)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    a = make_cache(cfg, w)
    gpu_prefill(a, cfg, L, cuda_device)
    gpu_decode(a, cfg, L, 30, cuda_device)
    blob = a.export_state()
    b = make_cache(cfg, w)
    b.import_state(blob)
    ga = gpu_decode(a, cfg, L, 30, cuda_device, step0=30)
    gb = gpu_decode(b, cfg, L, 30, cuda_device, step0=30)
    assert np.array_equal(ga.evict, gb.evict)
    assert np.array_equal(ga.outputs, gb.outputs)
    assert a.lengths() == [x + 60 for x in L]
    a.free()
    b.free()


@pytest.mark.parametrize("inputs,pinned_out,step", [
    ("pinned", True, None), ("packed", False, None), ("packed", True, None),
    ("pageable", True, None), ("packed_pageable", False, None),
    ("packed", True, "fused"), ("pageable", False, "fused")])
def test_host_buffer_step_matches_device_step(cuda_device, inputs, pinned_out, step):
    """kvpop_decode_step_host equals the device step bit for bit, on the two-kernel and
    the one-kernel path: pinned inputs (separate, or q | k | v in one buffer) read in
    place by the kernels, pageable inputs copied in (three copies, or one when packed);
    output written by the attention into pinned host memory or copied back from device
    staging (pageable output)."""
    cfg = get_config("q4b", batch=2, prompt_len=300, budget_B=64, decode_steps=20)
    w = gen.scorer_weights(cfg)
    L = gen.prompt_lengths(cfg)
    a, b = make_cache(cfg, w, step=step), make_cache(cfg, w, step=step)
    assert a.fused_step == (step == "fused")
    gpu_prefill(a, cfg, L, cuda_device)
    gpu_prefill(b, cfg, L, cuda_device)
    q, k, v = gen.decode_inputs(cfg, L, 0, 20, device="cpu")
    out_d = torch.empty((cfg.batch, cfg.n_q_heads, cfg.head_dim), device=cuda_device)
    out_h = torch.empty((cfg.batch, cfg.n_q_heads, cfg.head_dim))
    out_h = out_h.pin_memory() if pinned_out else out_h
    qb, kb = q[0].numel() * q.element_size(), k[0].numel() * k.element_size()
    buf = torch.empty(qb + 2 * kb, dtype=torch.uint8)
    buf = buf if inputs == "packed_pageable" else buf.pin_memory()
    for j in range(20):
        a.step(q[j].to(cuda_device), k[j].to(cuda_device), v[j].to(cuda_device), out_d)
        if inputs.startswith("packed"):
            hq = buf[:qb].view(q.dtype).view(q[j].shape)
            hk = buf[qb:qb + kb].view(k.dtype).view(k[j].shape)
            hv = buf[qb + kb:].view(v.dtype).view(v[j].shape)
            hq.copy_(q[j]); hk.copy_(k[j]); hv.copy_(v[j])
            b.step_host(hq, hk, hv, out_h)
        elif inputs == "pinned":
            b.step_host(q[j].pin_memory(), k[j].pin_memory(), v[j].pin_memory(), out_h)
        else:
            b.step_host(q[j].clone(), k[j].clone(), v[j].clone(), out_h)
        torch.cuda.synchronize()
        assert torch.equal(out_d.cpu(), out_h)
    a.free()
    b.free()


def test_alloc_failure_is_reported_and_recoverable(cuda_device):
    from paper_2607_05061_gb300 import kvpop
    cfg = get_config("tiny")
    w = gen.scorer_weights(cfg)
    for n in (1, 3, 7, 12):
        kvpop.kvpop_debug_fail_alloc_after(n)
        with pytest.raises(kvpop.KVpopError) as ei:
            make_cache(cfg, w)
        assert ei.value.status == 3
    kvpop.kvpop_debug_fail_alloc_after(0)
    c = make_cache(cfg, w)
    c.check()
    c.free()


def test_misaligned_and_bad_arguments(cuda_device):
    from paper_2607_05061_gb300 import kvpop
    cfg = get_config("q4b", batch=1, prompt_len=64, budget_B=32)
    c = make_cache(cfg, gen.scorer_weights(cfg))
    buf = torch.zeros(4096, dtype=torch.bfloat16, device=cuda_device)
    out = torch.zeros(4096, dtype=torch.float32, device=cuda_device)
    with pytest.raises(kvpop.KVpopError) as ei:
        c.ingest(buf.data_ptr() + 2, buf, buf)
    assert ei.value.status == 2
    with pytest.raises(kvpop.KVpopError) as ei:
        c.attend(buf, out.data_ptr() + 4)
    assert ei.value.status == 2
    Qp = torch.zeros((2, 32, 16, 128), dtype=torch.bfloat16, device=cuda_device)
    Kp = torch.zeros((2, 8, 16, 128), dtype=torch.bfloat16, device=cuda_device)
    with pytest.raises(kvpop.KVpopError) as ei:
        c.prefill(Qp, Kp, Kp, [10, 10])             # two sequences in a batch of one
    assert ei.value.status == 1
    with pytest.raises(kvpop.KVpopError) as ei:
        c.prefill(Qp[:1], Kp[:1], Kp[:1], [17])     # prompt longer than Pmax
    assert ei.value.status == 1
    c.check()
    c.free()


@pytest.mark.parametrize("F,act,kv_only,G,dt,D", [(256, "gelu", False, 4, "bf16", 16),
                                                 (128, "gelu", False, 4, "bf16", 16),
                                                 (256, "silu", True, 4, "bf16", 16),
                                                 (128, "identity", False, 2, "f32", 5),
                                                 (256, "gelu", False, 1, "bf16", 33)])
def test_prefill_scores_against_oracle(cuda_device, F, act, kv_only, G, dt, D):
    """Prompt scorer (3xTF32 tensor-core GEMM for F = 128 / 256): stored priorities of
    the kept slots equal the oracle's fp32 scores within 2e-5 relative, and the kept
    sets agree."""
    cfg = get_config("q4b", batch=2, prompt_len=700, budget_B=200, scorer_hidden=F,
                     scorer_act=act, scorer_kv_only=kv_only, log_gamma=-1e-3, q_per_kv=G,
                     kv_dtype=dt, delay_D=D)
    w = gen.scorer_weights(cfg)
    L = [700, 437]
    cache = make_cache(cfg, w)
    gpu_prefill(cache, cfg, L, cuda_device)
    pairs = all_pairs(cfg)
    pre = oracle_pairs(cfg, w, L, 0, pairs)
    agree = []
    for (b, h), tr in zip(pairs, pre):
        pos, sc = cache.pair_state(b, h)
        o = set(tr.cache.kept_positions())
        agree.append(len(o & set(pos)) / max(1, len(o)))
        prio = {int(p): float(v) for p, v in zip(tr.cache.slot_pos[:tr.cache.n_valid],
                                                  tr.cache.slot_prio[:tr.cache.n_valid])}
        for p_, s_ in zip(pos, sc):
            if p_ in prio:
                assert abs(s_ - prio[p_]) <= 2e-5 * (1.0 + abs(prio[p_])), (b, h, p_)
    print(f"prefill scorer F={F} {act} kv_only={kv_only} G={G} {dt} D={D}: "
          f"kept-set agreement {np.mean(agree):.4f}")
    assert np.mean(agree) >= 0.99
    cache.free()
