#!/usr/bin/env python
"""Decode throughput of the KVpop hot path on GB300.

One "step" = one decode step of the whole batch through the C ABI: ingest the
new token, delayed scorer on the token leaving the window, keep-or-drop
eviction, scatter (kvpop_decode_ingest) and GQA decode attention over the
compressed cache (kvpop_decode_attend).  Prefill is done once, untimed.

Prints one JSON line.  ``--impl reference`` times the fp64 CPU oracle instead
(the reference arm: the paper publishes no code and no decode throughput).

``--workload prompt`` measures the prompt path instead (one step = one
kvpop_prefill_attend call over a group of sequences: scoring, compression,
static ranks, running top-k cutoffs and masked attention with outputs), and
``--workload target`` the training target (one step = kvpop_future_target over
the group, fed with the prompt pass's sparse normalisers).  Both print their
own JSON line; the dominant kernel is tensor-bound.
Under torchrun (N > 1) every rank runs an independent replica of the workload
(the path has no cross-sequence exchange); value = all ranks' tokens / max time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode tokens/sec at 1 GB300 (batch x steps) and achieved HBM GB/s"
DEFAULT_CONFIG = "cr8x"
CSRC = os.path.join(ROOT, "paper_2607_05061_gb300", "csrc")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "attend_kernel_traffic.txt")
FALLBACK_HBM_GBS = 6800.0


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2048)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["kvpop", "reference"], default="kvpop")
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--batch", type=int, default=None,
                    help="override the workload's batch (small profiling cases)")
    ap.add_argument("--prompt-len", type=int, default=None,
                    help="override the workload's prompt length (small profiling cases)")
    ap.add_argument("--scorer", choices=["mlp", "mlstm"], default="mlp",
                    help="delayed MLP scorer (the workload's) or the stateful mLSTM scorer")
    ap.add_argument("--e2e-steps", type=int, default=256)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-steps", type=int, default=96)
    ap.add_argument("--workload", choices=["decode", "prompt", "target"], default="decode",
                    help="decode steps (default), the prompt path with outputs, or the target pass")
    ap.add_argument("--group", type=int, default=8, help="sequences per prompt/target step")
    return ap.parse_args(argv)


# ------------------------------------------------------------------ distributed plumbing
def dist_info():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


def dist_init(world, backend):
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        dist.init_process_group(backend=backend)
    return dist


def reduce_max_sum(local_max: float, local_sum: float, world: int, device=None):
    """(max over ranks of local_max, sum over ranks of local_sum)."""
    if world <= 1:
        return local_max, local_sum
    import torch
    import torch.distributed as dist
    t = torch.tensor([local_max], dtype=torch.float64, device=device)
    s = torch.tensor([local_sum], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(s, op=dist.ReduceOp.SUM)
    return float(t.item()), float(s.item())


# ------------------------------------------------------------------ workload arithmetic
def kv_stream_bytes(cfg, lengths, step: int) -> int:
    """Algorithmic K/V bytes one attention launch reads at decode step `step` (0-based).

    Per (sequence, KV head): (used slots + window entries) * 2 (K and V) * d * esz,
    with len = P + step + 1 after the step's token is ingested.
    """
    tot = 0
    for P in lengths:
        ln = P + step + 1
        keys = min(cfg.budget_B, max(0, ln - cfg.delay_D)) + min(ln, cfg.delay_D)
        tot += keys
    return tot * cfg.n_kv_heads * 2 * cfg.head_dim * cfg.esz


L2_BYTES = 129e6           # GB300 L2 (126 MiB)
FLUSH_BYTES = 512 << 20    # written between timed steps whose inputs fit in twice the L2
ATTN_POST_LAUNCHES = 32    # event-timed attention launches after the timed region


def flushes_l2(bytes_per_step: float) -> bool:
    """Whether a step's inputs are too small to push the last step's data out of L2."""
    return bytes_per_step < 2 * L2_BYTES


def decode_dtype(cfg) -> str:
    """The arithmetic of the decode path: bf16 K/V products on tensor cores with fp32
    accumulation (P rounded to bf16 for the PV product), or fp32 throughout."""
    return "bf16 (fp32 accumulate)" if cfg.kv_dtype == "bf16" else "f32"


def scorer_description(cfg, scorer: str) -> str:
    if scorer == "mlstm":
        return (f"stateful delayed mLSTM (Hedgehog, C {cfg.head_dim}x{cfg.head_dim // 2} per "
                f"head) fp32")
    return f"MLP {cfg.scorer_in}->{cfg.scorer_hidden} GELU->1 fp32"


def decode_config(cfg, scorer: str, bytes_per_step: float, world: int) -> dict:
    """The `config` object of the decode line; both arms print the same one."""
    if flushes_l2(bytes_per_step):
        l2 = (f"inputs smaller than twice L2 ({bytes_per_step / 1e9:.3f} GB K/V read per step): "
              f"a {FLUSH_BYTES >> 20} MiB buffer is written before every timed step, and each "
              f"step is timed on its own with CUDA events, the flush outside them")
    else:
        l2 = f"inputs larger than L2: {bytes_per_step / 1e9:.3f} GB K/V read per step"
    return {"workload": f"{cfg.name}: {cfg.description}", "batch": cfg.batch,
            "kv_heads": cfg.n_kv_heads, "q_per_kv": cfg.q_per_kv, "head_dim": cfg.head_dim,
            "prompt_len": "ragged U[%d,%d]" % cfg.ragged if cfg.ragged else cfg.prompt_len,
            "budget_B": cfg.budget_B, "delay_D": cfg.delay_D, "kv_dtype": cfg.kv_dtype,
            "scorer": scorer_description(cfg, scorer), "l2": l2,
            "parallelism": "replicas" if world > 1 else "single GPU"}


def mean_stream_bytes(cfg, lengths, step0: int, n: int) -> float:
    return statistics.mean(kv_stream_bytes(cfg, lengths, step0 + i) for i in range(n))


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return float(j["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def committed_traffic(config_name: str, path: str = TRAFFIC_FILE, sequences: int = 0):
    """DRAM bytes per launch from a committed ncu summary, if it matches the source.

    With ``sequences`` the captured figure is scaled from the capture's sequence count."""
    if not os.path.exists(path):
        return None
    kv = {}
    with open(path) as f:
        for line in f:
            parts = line.split()
            if len(parts) >= 2 and not line.startswith("#"):
                kv[parts[0]] = parts[1:] if parts[0] == "source_files" else parts[1]
    h = hashlib.sha256()
    for rel in kv.get("source_files", []):
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    sha = h.hexdigest()
    if kv.get("source_sha256") != sha or kv.get("config") != config_name:
        return None
    try:
        v = float(kv["dram_bytes_per_launch"])
        if sequences:
            v *= sequences / float(kv["capture_sequences"])
        return int(v)
    except (KeyError, ValueError, ZeroDivisionError):
        return None


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples taken while the timed region runs."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-f", self.path], stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                cols = [c.strip() for c in line.split(",")]
                if len(cols) >= 9:
                    rows.append(cols)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


# ------------------------------------------------------------------ oracle (CPU) legs
def _oracle_pair_job(args):
    """Prefill one (sequence, KV head) in the oracle (untimed), then time n decode steps.

    Returns (seconds, kept positions after the prefill, per-step (slot, evicted
    position) decisions) -- the decisions feed the eviction-agreement report."""
    cfg_name, b, h, n_steps, scorer = args
    import torch
    torch.set_num_threads(1)
    from oracle.run import prefill_pair, prefill_pair_mlstm
    from workload import gen, get_config
    cfg = get_config(cfg_name)
    L = gen.prompt_lengths(cfg)
    if scorer == "mlstm":
        cache = prefill_pair_mlstm(cfg, gen.mlstm_weights(cfg), b, h, L[b])
    else:
        cache = prefill_pair(cfg, gen.scorer_weights(cfg), b, h, L[b])
    kept = cache.kept_positions()
    G = cfg.q_per_kv
    q, k, v = gen.decode_inputs(cfg, [L[b]], 0, n_steps, b0=b)
    q = q[:, 0, h * G:(h + 1) * G].double().numpy()
    k = k[:, 0, h].double().numpy()
    v = v[:, 0, h].double().numpy()
    decisions = []
    t0 = time.perf_counter()
    for j in range(n_steps):
        slot, ev, _ = cache.append(q[j], k[j], v[j])
        cache.attend(q[j])
        decisions.append((int(slot), int(ev)))
    return time.perf_counter() - t0, kept, decisions


def sample_pairs(cfg, n):
    total = cfg.batch * cfg.n_kv_heads
    idx = sorted({(i * total) // n for i in range(n)})
    return [(i // cfg.n_kv_heads, i % cfg.n_kv_heads) for i in idx]


def baseline_pairs(cfg):
    """The (sequence, KV head) pairs the CPU baseline runs: one per host core, at most 16."""
    return sample_pairs(cfg, max(1, min(os.cpu_count() or 1, 16)))


def cpu_baseline(cfg, n_steps: int, scorer: str = "mlp"):
    """fp64 oracle decode throughput on this host's cores (spawned pool, one pair per core).

    Returns (the cpu_baseline object, per-pair (kept positions, decisions))."""
    import multiprocessing as mp
    pairs = baseline_pairs(cfg)
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[var] = "1"
    ctx = mp.get_context("spawn")
    with ctx.Pool(len(pairs)) as pool:
        res = pool.map(_oracle_pair_job, [(cfg.name, b, h, n_steps, scorer) for b, h in pairs])
    times = [r[0] for r in res]
    per_pair_step = statistics.mean(times) / n_steps            # seconds per (pair, step)
    step_time = cfg.batch * cfg.n_kv_heads * per_pair_step / len(pairs)
    rec = {"value": cfg.batch / step_time, "unit": "tokens/s", "cores": len(pairs), "kind": "oracle",
           "sample": (f"{len(pairs)} of {cfg.batch * cfg.n_kv_heads} (sequence, KV head) pairs, "
                      f"{n_steps} decode steps each after an untimed oracle prefill, one pair per "
                      f"core in parallel; whole-batch step time extrapolated as pairs/cores x "
                      f"mean pair-step time")}
    return rec, {pr: (r[1], r[2]) for pr, r in zip(pairs, res)}


def agreement(gpu_kept: dict, gpu_decisions, oracle: dict) -> dict:
    """End-to-end eviction agreement, each side with its own scores.

    ``gpu_decisions[j][b][h]`` = (slot, evicted position) at decode step j;
    ``oracle[(b, h)]`` = (kept positions after prefill, per-step decisions)."""
    n = eq = kept_eq = 0
    first = None
    for (b, h), (kept, dec) in sorted(oracle.items()):
        kept_eq += int(sorted(gpu_kept[(b, h)]) == list(kept))
        for j, d in enumerate(dec):
            g = tuple(int(x) for x in gpu_decisions[j][b][h])
            n += 1
            if g == tuple(d):
                eq += 1
            elif first is None:
                first = {"pair": [b, h], "step": j, "gpu": list(g), "oracle": list(d)}
    return {"decode_decisions_equal": eq / n if n else None, "decisions": n,
            "prefill_kept_sets_equal": kept_eq / len(oracle) if oracle else None,
            "pairs": len(oracle), "steps": len(next(iter(oracle.values()))[1]) if oracle else 0,
            "first_mismatch": first,
            "how": ("each side scores with its own arithmetic (CUDA fp32 kernels; the fp64 oracle "
                    "rounded to fp32) from the same seeded prompt; a decision is the (slot, evicted "
                    "position) of one (sequence, KV head) at one decode step; kept sets compared "
                    "after the prompt compression")}


# ------------------------------------------------------------------ GPU arm
def run_kvpop(args):
    import torch
    rank, local_rank, world = dist_info()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    dist = dist_init(world, "nccl")

    from paper_2607_05061_gb300 import build as _build
    _build.build()
    from paper_2607_05061_gb300 import kvpop
    from workload import gen, get_config

    over = {}
    if args.batch:
        over["batch"] = args.batch
    if args.prompt_len:
        over["prompt_len"] = args.prompt_len
    cfg = get_config(args.config, **over)
    if cfg.n_layers != 1:
        return run_stack_bench(args, cfg, rank, local_rank, world, dev, dist)
    L = gen.prompt_lengths(cfg)
    if args.scorer == "mlstm":
        cache = kvpop.KVpopCache(cfg.batch, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim, cfg.budget_B,
                                 cfg.delay_D, cfg.scorer_hidden, cfg.kv_dtype, n_sink=cfg.n_sink,
                                 mlstm=gen.mlstm_weights(cfg))
    else:
        W1, b1, w2, b2, lg = gen.scorer_weights(cfg)
        cache = kvpop.KVpopCache(cfg.batch, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim, cfg.budget_B,
                                 cfg.delay_D, cfg.scorer_hidden, cfg.kv_dtype, W1, b1, w2, b2,
                                 n_sink=cfg.n_sink)

    def prefill_all():
        """Prompt compression of the whole batch, 16 sequences at a time (bounded buffers:
        about 6.5 GB of bf16 Q/K/V at 32768 tokens; 16 x 8 (sequence, head) pairs keep most
        SMs busy in the sequential parts of the mLSTM prefill)."""
        t = 0.0
        group = 16
        for b0 in range(0, cfg.batch, group):
            nb = min(group, cfg.batch - b0)
            Lg = L[b0:b0 + nb]
            Pm = max(Lg)
            Q = gen.q_tokens(cfg, b0, nb, 0, Pm, device=dev)
            K = gen.kv_tokens(cfg, "k", b0, nb, 0, Pm, device=dev)
            V = gen.kv_tokens(cfg, "v", b0, nb, 0, Pm, device=dev)
            torch.cuda.synchronize()
            tp = time.perf_counter()
            cache.prefill(Q, K, V, Lg, first_seq=b0)
            t += time.perf_counter() - tp
            del Q, K, V
        torch.cuda.synchronize()
        return t

    t_prefill = prefill_all()
    W, K = args.warmup, args.steps
    bytes_per_launch = mean_stream_bytes(cfg, L, W, K)
    flush = flushes_l2(bytes_per_launch)
    flush_buf = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev) if flush else None
    post = ATTN_POST_LAUNCHES
    q, k, v = gen.decode_inputs(cfg, L, 0, W + K + post + 2, device=dev)
    out = torch.empty((cfg.batch, cfg.n_q_heads, cfg.head_dim), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    fused = cache.fused_step           # one kernel per kvpop_decode_step
    for j in range(W):
        cache.step(q[j], k[j], v[j], out)
    torch.cuda.synchronize()

    def ev():
        return torch.cuda.Event(enable_timing=True)

    def capture(body):
        """One CUDA graph of the library calls `body` makes (nothing runs while capturing)."""
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            with torch.cuda.graph(g, stream=side):
                body()
        stream.wait_stream(side)
        return g

    # Inputs larger than L2: the K timed steps are replayed from one CUDA graph between
    # two events on the stream, so the device runs them back to back (in an eager loop
    # the first steps also wait for the host to enqueue them).  Inputs smaller than twice
    # L2: an eager loop writes the flush buffer before every step and brackets each step
    # with its own events; the flush gives the host time to enqueue the step.
    step_ev = [(ev(), ev()) for _ in range(K)] if flush else []
    t_start, t_end = ev(), ev()
    graph = None
    if not flush:
        def timed_body():
            for i in range(K):
                cache.step(q[W + i], k[W + i], v[W + i], out)
        graph = capture(timed_body)
    clocks = ClockSampler(local_rank)
    clocks.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_start.record(stream)
    if flush:
        for i in range(K):
            flush_buf.fill_(float(i))
            step_ev[i][0].record(stream)
            cache.step(q[W + i], k[W + i], v[W + i], out)
            step_ev[i][1].record(stream)
    else:
        graph.replay()
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    cache.check()
    if flush:
        step_ms_local = statistics.mean(a.elapsed_time(b) for a, b in step_ev)
    else:
        step_ms_local = t_start.elapsed_time(t_end) / K
    del graph
    # The dominant kernel's own duration: ATTN_POST_LAUNCHES further decode steps with
    # events around each launch of it -- the whole step where it is one kernel, else the
    # attention (events between the ingest and the attention stop the attention from
    # launching as a programmatic dependent of the ingest, which is why the timed steps
    # carry none); the first two, which wait for the host to enqueue them after the
    # synchronisation, are not counted.
    attn_ev = []
    for i in range(post + 2):
        j = W + K + i
        if not fused:
            cache.ingest(q[j], k[j], v[j])
        if flush:
            flush_buf.fill_(float(i))
        a, b = ev(), ev()
        a.record(stream)
        if fused:
            cache.step(q[j], k[j], v[j], out)
        else:
            cache.attend(q[j], out)
        b.record(stream)
        attn_ev.append((a, b))
    torch.cuda.synchronize()
    cache.check()
    attn_ms = statistics.mean(a.elapsed_time(b) for a, b in attn_ev[2:])
    attn_bytes = mean_stream_bytes(cfg, L, W + K + 2, post)
    if fused:
        attn_how = (f"CUDA events around each of {post} one-kernel decode steps after the timed "
                    f"region" + (", L2 flushed before each" if flush else ""))
    else:
        attn_how = (f"CUDA events around the attention in {post} decode steps after the timed "
                    f"region (the ingest between them untimed" +
                    (", L2 flushed before each)" if flush else ")"))

    # end to end through the C ABI on host buffers (pinned), copies inside the timed region
    E = max(1, args.e2e_steps)
    s0 = W + K + post + 2
    qa, ka, va = gen.decode_inputs(cfg, L, s0, E, device="cpu")
    # each step's q, k, v back to back in one pinned buffer (one host-to-device copy)
    qb, kb = qa[0].numel() * qa.element_size(), ka[0].numel() * ka.element_size()
    packed = torch.empty((E, qb + 2 * kb), dtype=torch.uint8).pin_memory()
    qh, kh, vh = [], [], []
    for i in range(E):
        for t, lo, n, lst in ((qa[i], 0, qb, qh), (ka[i], qb, kb, kh), (va[i], qb + kb, kb, vh)):
            view = packed[i, lo:lo + n].view(t.dtype).view(t.shape)
            view.copy_(t)
            lst.append(view)
    outh = torch.empty((cfg.batch, cfg.n_q_heads, cfg.head_dim), dtype=torch.float32).pin_memory()
    torch.cuda.synchronize()
    e2e_s = 0.0
    t0 = time.perf_counter()
    for i in range(E):
        if flush:                     # flush, wait, then time the step alone
            flush_buf.fill_(float(i))
            stream.synchronize()
            t0 = time.perf_counter()
        cache.step_host(qh[i], kh[i], vh[i], outh, stream=stream)
        stream.synchronize()          # the host reads each step's output
        if flush:
            e2e_s += time.perf_counter() - t0
    if not flush:
        e2e_s = time.perf_counter() - t0
    cache.check()
    h2d = qb + 2 * kb
    d2h = outh.numel() * 4

    # eviction agreement: the same prompts again, then the first decode steps with every
    # (slot, evicted position) recorded, for comparison with the oracle's own decisions
    agree_pairs = baseline_pairs(cfg) if (rank == 0 and not args.no_cpu_baseline) else []
    gpu_kept, gpu_dec = {}, None
    if agree_pairs:
        prefill_all()
        for b_, h_ in agree_pairs:
            pos, _ = cache.pair_state(b_, h_)
            gpu_kept[(b_, h_)] = [int(t) for t in pos]
        n_ag = args.cpu_steps
        qg, kg, vg = gen.decode_inputs(cfg, L, 0, n_ag, device=dev)
        eig = torch.empty((n_ag, cfg.batch, cfg.n_kv_heads, 2), dtype=torch.int32, device=dev)
        for j in range(n_ag):
            cache.ingest(qg[j], kg[j], vg[j], evict_info=eig[j])
        gpu_dec = eig.cpu().numpy()
        cache.check()
        del qg, kg, vg

    step_ms, _ = reduce_max_sum(step_ms_local, 0.0, world, dev)
    e2e_max, _ = reduce_max_sum(e2e_s / E * 1e3, 0.0, world, dev)
    tokens_per_step = cfg.batch * world
    value = tokens_per_step / (step_ms / 1e3)
    achieved = attn_bytes / (attn_ms / 1e3) / 1e9
    peak, peak_src = measured_peaks()
    rec = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": W, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": decode_dtype(cfg),
        "data": "synthetic (seeded counter-based generator)",
        "config": decode_config(cfg, args.scorer, bytes_per_launch, world),
        "steps_per_s": 1e3 / step_ms,
        "hbm_gbs_step": bytes_per_launch / (step_ms / 1e3) / 1e9,
        "prefill_s": t_prefill,
        "roofline": {"bound": "hbm", "kernel": ("attend_tc_kernel<fused step>" if fused else
                                                 "attend_tc_kernel" if cfg.kv_dtype == "bf16"
                                                 else "attend_kernel"),
                     "achieved": achieved, "peak": peak,
                     "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured"
                     else "fallback 6.8 TB/s", "unit": "GB/s", "frac": achieved / peak,
                     "frac_of_8tbs_nominal": achieved / 8000.0,
                     "traffic": None if over else committed_traffic(cfg.name),
                     "algorithmic_bytes_per_launch": attn_bytes, "ms_per_launch": attn_ms,
                     "ms_per_launch_how": attn_how},
        "e2e": {"value": tokens_per_step / (e2e_max / 1e3), "unit": "tokens/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": E,
                "how": "kvpop_decode_step_host on pinned host buffers: the step's kernels read q|k|v "
                       "and write out in place over NVLink-C2C; stream sync every step"
                       + ("; L2 flushed before each step, outside its timing" if flush else "")},
        "gpu_launches": K if fused else 2 * K,
        "clocks": clk,
    }
    cache.free()
    del q, k, v
    if rank == 0 and not args.no_cpu_baseline:
        rec["cpu_baseline"], oracle_dec = cpu_baseline(cfg, args.cpu_steps, args.scorer)
        rec["agreement"] = agreement(gpu_kept, gpu_dec, oracle_dec)
    if rank == 0:
        print(json.dumps(rec), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ------------------------------------------------------------------ GPU arm, layer stack
def run_stack_bench(args, cfg, rank, local_rank, world, dev, dist):
    """Decode steps of the Qwen3-8B-shaped stack: per layer Q/K/V projections (cuBLAS bf16),
    one KVpop cache step, output projection and residual; one step = all layers, replayed
    from a CUDA graph."""
    import torch
    from paper_2607_05061_gb300.stack import DecodeStack
    from workload import gen
    L = gen.prompt_lengths(cfg)
    layers = []
    for l in range(cfg.n_layers):
        w = gen.stack_weights(cfg, l, device=dev)
        for k in ("W1", "b1", "w2", "b2"):
            w[k] = w[k].cpu()
        layers.append(w)
    st = DecodeStack(layers, cfg.batch, cfg.hidden, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim,
                     cfg.budget_B, cfg.delay_D, cfg.scorer_hidden, n_sink=cfg.n_sink, device=dev)
    group = 4
    for l in range(cfg.n_layers):
        for b0 in range(0, cfg.batch, group):
            nb = min(group, cfg.batch - b0)
            X = gen.prompt_hidden(cfg, l, b0, nb, 0, max(L[b0:b0 + nb]), device=dev)
            st.prefill_layer(l, X, L[b0:b0 + nb], first_seq=b0)
            del X
    torch.cuda.synchronize()
    W, K = args.warmup, args.steps
    n_attn = 32                                   # eager steps timing each attention launch
    xs = gen.decode_hidden(cfg, L, 0, W + K + n_attn, device=dev)
    x_in = torch.empty((cfg.batch, cfg.hidden), dtype=torch.bfloat16, device=dev)
    x_out = torch.empty_like(x_in)
    st.capture(x_in, x_out)
    stream = torch.cuda.current_stream()
    for j in range(W):
        x_in.copy_(xs[j])
        st.graph.replay()
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local_rank)
    clocks.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_start.record(stream)
    for i in range(K):
        x_in.copy_(xs[W + i])
        st.graph.replay()
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    for c in st.caches:
        c.check()
    step_ms_local = t_start.elapsed_time(t_end) / K
    # durations of the dominant kernel: eager steps with events around every layer's
    # one-kernel decode step (or, on the two-kernel path, around its attention)
    fused = all(c.fused_step for c in st.caches)
    ev = []
    x = torch.empty_like(x_in)
    for i in range(n_attn):
        xcur = xs[W + K + i]
        for l, (Lw, cache) in enumerate(zip(st.layers, st.caches)):
            torch.matmul(xcur, Lw["Wq"], out=st.q)
            torch.matmul(xcur, Lw["Wk"], out=st.k)
            torch.matmul(xcur, Lw["Wv"], out=st.v)
            if not fused:
                cache.ingest(st.q, st.k, st.v)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            if fused:
                cache.step(st.q, st.k, st.v, st.o)
            else:
                cache.attend(st.q, st.o)
            e1.record(stream)
            ev.append((e0, e1))
            st.o_bf.copy_(st.o)
            torch.matmul(st.o_bf, Lw["Wo"], out=st.y)
            torch.add(xcur, st.y, out=x)
            xcur = x.clone()
    torch.cuda.synchronize()
    attn_ms = statistics.mean(a.elapsed_time(b) for a, b in ev)
    # end to end: host hidden state in (pinned), final hidden state out, per step
    E = max(1, min(args.e2e_steps, 64))
    xh = gen.decode_hidden(cfg, L, W + K + n_attn, E).pin_memory()
    oh = torch.empty((cfg.batch, cfg.hidden), dtype=torch.bfloat16).pin_memory()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for i in range(E):
        x_in.copy_(xh[i], non_blocking=True)
        st.graph.replay()
        oh.copy_(x_out, non_blocking=True)
        stream.synchronize()
    e2e_s = (time.perf_counter() - t0) / E
    step_ms, _ = reduce_max_sum(step_ms_local, 0.0, world, dev)
    e2e_ms, _ = reduce_max_sum(e2e_s * 1e3, 0.0, world, dev)
    tokens_per_step = cfg.batch * world
    bytes_per_launch = statistics.mean(kv_stream_bytes(cfg, L, W + K + i) for i in range(n_attn))
    proj_bytes = cfg.n_layers * 2 * (cfg.hidden * (cfg.n_q_heads + 2 * cfg.n_kv_heads) * cfg.head_dim
                                     + cfg.n_q_heads * cfg.head_dim * cfg.hidden)
    achieved = bytes_per_launch / (attn_ms / 1e3) / 1e9
    peak, peak_src = measured_peaks()
    rec = {
        "metric": METRIC, "value": tokens_per_step / (step_ms / 1e3), "unit": "tokens/s",
        "n_gpus": world, "steps": K, "warmup": W, "ms_per_step": step_ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": decode_dtype(cfg),
        "data": "synthetic (seeded counter-based generator)",
        "config": {"workload": f"{cfg.name}: {cfg.description}", "batch": cfg.batch,
                   "layers": cfg.n_layers, "hidden": cfg.hidden, "kv_heads": cfg.n_kv_heads,
                   "q_per_kv": cfg.q_per_kv, "head_dim": cfg.head_dim, "prompt_len": cfg.prompt_len,
                   "budget_B": cfg.budget_B, "delay_D": cfg.delay_D, "kv_dtype": cfg.kv_dtype,
                   "projections": "cuBLAS bf16 GEMMs (torch.matmul), fp32 accumulate",
                   "l2": f"inputs larger than L2: {cfg.n_layers * bytes_per_launch / 1e9:.2f} GB K/V "
                         f"+ {proj_bytes / 1e9:.2f} GB weights per step",
                   "graph": "one CUDA graph per step (all layers)",
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "steps_per_s": 1e3 / step_ms,
        "hbm_gbs_step": (cfg.n_layers * bytes_per_launch + proj_bytes) / (step_ms / 1e3) / 1e9,
        "roofline": {"bound": "hbm", "kernel": "attend_tc_kernel<fused step>" if fused else "attend_tc_kernel",
                     "achieved": achieved, "peak": peak,
                     "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)", "unit": "GB/s",
                     "frac": achieved / peak, "frac_of_8tbs_nominal": achieved / 8000.0,
                     "traffic": None, "algorithmic_bytes_per_launch": bytes_per_launch,
                     "ms_per_launch": attn_ms},
        "e2e": {"value": tokens_per_step / (e2e_ms / 1e3), "unit": "tokens/s",
                "h2d_bytes_per_step": cfg.batch * cfg.hidden * 2,
                "d2h_bytes_per_step": cfg.batch * cfg.hidden * 2, "steps": E,
                "how": "pinned hidden state in, graph replay, final hidden state out, sync per step"},
        "gpu_launches": K * cfg.n_layers * (1 if fused else 2),
        "clocks": clk,
        "cpu_baseline": None,
        "cpu_baseline_note": ("not run for the stack: the fp64 oracle would have to prefill 36 layers "
                              "of a 32768-token prompt (about 58 PFLOP of fp64 projections)"),
    }
    st.free()
    if rank == 0:
        print(json.dumps(rec), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ------------------------------------------------------------------ reference arm (oracle)
def run_reference(args):
    rank, _, world = dist_info()
    if rank != 0:
        return
    from oracle.run import prefill_pair, prefill_pair_mlstm
    from workload import gen, get_config
    cfg = get_config(args.config)
    if cfg.n_layers != 1:
        raise SystemExit("--impl reference times the oracle on single-layer workloads only")
    if args.scorer == "mlstm":
        mw = gen.mlstm_weights(cfg)
        prefill = lambda b, h, P: prefill_pair_mlstm(cfg, mw, b, h, P)
    else:
        w = gen.scorer_weights(cfg)
        prefill = lambda b, h, P: prefill_pair(cfg, w, b, h, P)
    L = gen.prompt_lengths(cfg)
    W, K = args.warmup, args.steps
    budget_s = 120.0
    pairs = sample_pairs(cfg, 64)
    caches, inputs = [], []
    G = cfg.q_per_kv
    t_setup = time.perf_counter()
    for b, h in pairs:
        caches.append(prefill(b, h, L[b]))
        q, k, v = gen.decode_inputs(cfg, [L[b]], 0, W + K, b0=b)
        inputs.append((q[:, 0, h * G:(h + 1) * G].double().numpy(), k[:, 0, h].double().numpy(),
                       v[:, 0, h].double().numpy()))
        # bound the sample so the whole run stays within the budget
        if len(caches) >= 1 and time.perf_counter() - t_setup > 60:
            break
    # calibrate: pairs per step so that (W + K) steps take about budget_s
    c0 = caches[0]
    t0 = time.perf_counter()
    qa, ka, va = inputs[0]
    c0.append(qa[0], ka[0], va[0])
    c0.attend(qa[0])
    t_pair = max(time.perf_counter() - t0, 1e-5)
    n_use = max(1, min(len(caches), int(budget_s / ((W + K) * t_pair))))
    ptr = [1 if i == 0 else 0 for i in range(len(caches))]
    times = []
    for s in range(W + K):
        t0 = time.perf_counter()
        for i in range(n_use):
            qa, ka, va = inputs[i]
            j = ptr[i]
            if j >= qa.shape[0]:
                continue
            caches[i].append(qa[j], ka[j], va[j])
            caches[i].attend(qa[j])
            ptr[i] += 1
        if s >= W:
            times.append(time.perf_counter() - t0)
    step_sample_s = sum(times) / len(times)
    step_s = step_sample_s * (cfg.batch * cfg.n_kv_heads) / n_use
    value = cfg.batch / step_s
    rec = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": W, "ms_per_step": step_s * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded counter-based generator)",
        "impl": "reference",
        "config": decode_config(cfg, args.scorer, mean_stream_bytes(cfg, L, W, K), world),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                         "sample": (f"each step = one decode step of {n_use} of "
                                    f"{cfg.batch * cfg.n_kv_heads} (sequence, KV head) pairs on one "
                                    f"core after an untimed oracle prefill; whole-batch step time "
                                    f"extrapolated by pairs")},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(rec), flush=True)


# ------------------------------------------------------------------ prompt path and target pass
def measured_tensor_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return float(json.load(f)["bf16_tflops"]), "measured (MEASURED_PEAKS.json bf16_tflops, burst)"
    return 1900.0, "fallback 1.9 PFLOP/s bf16 burst"


def prompt_attention_flops(cfg, lengths) -> float:
    """QK + PV flops of the masked prompt attention: 4 d G per retained (query, key)."""
    import numpy as np
    keep = cfg.budget_B + cfg.delay_D
    tot = sum(int(np.minimum(np.arange(1, P + 1), keep).sum()) for P in lengths)
    return 4.0 * cfg.head_dim * cfg.q_per_kv * cfg.n_kv_heads * tot


def target_flops(cfg, lengths) -> float:
    """QK flops of the transposed pass: 2 d G per (key t, future query d >= t + w)."""
    import numpy as np
    tot = 0
    for P in lengths:
        t = np.arange(P)
        tot += int(np.maximum(0, P - t - cfg.delay_D).sum())
    return 2.0 * cfg.head_dim * cfg.q_per_kv * cfg.n_kv_heads * tot


def _oracle_prompt_job(args):
    """Oracle time of one (sequence, KV head) prompt: scoring + compression, ranks and cutoffs
    in full, masked attention on `nq` evenly spaced queries (extrapolated to all P)."""
    cfg_name, b, h, nq, over = args
    import numpy as np
    import torch
    torch.set_num_threads(1)
    from oracle import running_topk as rt
    from oracle.run import prefill_pair, _f64
    from workload import gen, get_config
    cfg = get_config(cfg_name, **over)
    P = gen.prompt_lengths(cfg)[b]
    G = cfg.q_per_kv
    t0 = time.perf_counter()
    cache = prefill_pair(cfg, gen.scorer_weights(cfg), b, h, P)
    prio = rt.prompt_priorities(cache.prefill_raw, P, cfg.delay_D, cache.p.log_gamma)
    rank = rt.static_ranks(prio)
    tau = rt.fenwick_cutoffs(rank, cfg.n_sink, cfg.delay_D, cfg.budget_B - cfg.n_sink)
    t_fixed = time.perf_counter() - t0
    Q = _f64(gen.q_tokens(cfg, b, 1, 0, P, heads=range(h * G, (h + 1) * G)))[0]
    K = _f64(gen.kv_tokens(cfg, "k", b, 1, 0, P, heads=[h]))[0, 0]
    V = _f64(gen.kv_tokens(cfg, "v", b, 1, 0, P, heads=[h]))[0, 0]
    qs = np.linspace(0, P - 1, nq).astype(int)
    t0 = time.perf_counter()
    for q in qs:
        keys = np.nonzero(rt.mask_row(int(q), rank, tau, cfg.n_sink, cfg.delay_D))[0]
        lg = Q[:, q, :] @ K[keys].T / np.sqrt(cfg.head_dim)
        e = np.exp(lg - lg.max(axis=1, keepdims=True))
        _ = (e / e.sum(axis=1, keepdims=True)) @ V[keys]
    t_q = (time.perf_counter() - t0) / nq
    return t_fixed + P * t_q


def _oracle_target_job(args):
    """Oracle time of one (sequence, KV head) target: the future log mass of `nk` evenly
    spaced keys for every query head (extrapolated to all P keys)."""
    cfg_name, b, h, nk, over = args
    import numpy as np
    import torch
    torch.set_num_threads(1)
    from oracle.run import _f64
    from workload import gen, get_config
    cfg = get_config(cfg_name, **over)
    P = gen.prompt_lengths(cfg)[b]
    G, d, w = cfg.q_per_kv, cfg.head_dim, cfg.delay_D
    Q = _f64(gen.q_tokens(cfg, b, 1, 0, P, heads=range(h * G, (h + 1) * G)))[0]
    K = _f64(gen.kv_tokens(cfg, "k", b, 1, 0, P, heads=[h]))[0, 0]
    lse = np.zeros((G, P))            # normalisers are an input of the pass
    ts = np.linspace(0, P - 1, nk).astype(int)
    t0 = time.perf_counter()
    for t in ts:
        for g in range(G):
            if t + w <= P - 1:
                v = Q[g, t + w:] @ K[t] / np.sqrt(d) - lse[g, t + w:]
                _ = np.logaddexp.reduce(v)
    return (time.perf_counter() - t0) / nk * P


def cpu_prompt_baseline(cfg, over, group, kind):
    import multiprocessing as mp
    cores = max(1, min(os.cpu_count() or 1, 16))
    pairs = [(b % group, b % cfg.n_kv_heads) for b in range(cores)]
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[var] = "1"
    ctx = mp.get_context("spawn")
    job = _oracle_prompt_job if kind == "prompt" else _oracle_target_job
    n = 48 if kind == "prompt" else 64
    with ctx.Pool(len(pairs)) as pool:
        times = pool.map(job, [(cfg.name, b, h, n, over) for b, h in pairs])
    pair_s = statistics.mean(times)
    group_s = group * cfg.n_kv_heads * pair_s / len(pairs)
    what = ("scoring, compression, ranks and cutoffs in full plus masked attention of "
            f"{n} evenly spaced queries" if kind == "prompt" else
            f"future log mass of {n} evenly spaced keys for every query head")
    return {"value": group * cfg.prompt_len / group_s, "unit": "tokens/s", "cores": len(pairs),
            "kind": "oracle",
            "sample": (f"{len(pairs)} (sequence, KV head) pairs of the {group}-sequence group, one "
                       f"per core in parallel: {what}, extrapolated to the whole prompt and group")}


def prompt_metric(workload):
    """(metric, step description) of the prompt / target lines, shared by both arms."""
    if workload == "prompt":
        return ("prompt tokens/sec with outputs under the running top-k mask (1 GB300)",
                "kvpop_prefill_attend: delayed scorer on every prompt token, prompt compression, "
                "static ranks + running top-k cutoffs, masked causal attention with y and LSE")
    return ("future-target tokens/sec (transposed attention pass + aggregation, 1 GB300)",
            "kvpop_future_target with the prompt pass's sparse LSE: log future mass per key "
            "and query head, max aggregation, count normalisation")


def prompt_workload_config(cfg, n):
    P, H, G, d = cfg.prompt_len, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim
    return (f"{cfg.name} prompt group: {n} sequences x {P} tokens, {H} KV heads x {G} query heads, "
            f"d {d}, B {cfg.budget_B}, D {cfg.delay_D}")


def run_reference_prompt(args):
    """The oracle as the reference arm of --workload prompt / target: one (sequence, KV head)
    pair per step on one core, extrapolated to the whole group (rank 0 only)."""
    rank, _, world = dist_info()
    if rank != 0:
        return
    from workload import get_config
    over = {}
    if args.batch:
        over["batch"] = args.batch
    if args.prompt_len:
        over["prompt_len"] = args.prompt_len
    cfg = get_config(args.config, **over)
    if cfg.n_layers != 1 or cfg.ragged:
        raise SystemExit("--workload prompt/target runs fixed-length single-layer workloads")
    n = min(args.group, cfg.batch)
    W, K = args.warmup, args.steps
    job = _oracle_prompt_job if args.workload == "prompt" else _oracle_target_job
    nsample = 8 if args.workload == "prompt" else 16       # queries / keys timed per pair
    times = []
    for s in range(W + K):
        b, h = s % n, s % cfg.n_kv_heads
        t = job((cfg.name, b, h, nsample, over))          # extrapolated to the pair's P
        if s >= W:
            times.append(t)
    pair_s = statistics.mean(times)
    step_s = n * cfg.n_kv_heads * pair_s
    value = n * cfg.prompt_len / step_s
    metric, what = prompt_metric(args.workload)
    rec = {
        "metric": metric, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": W, "ms_per_step": step_s * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded counter-based generator)",
        "impl": "reference",
        "config": {"workload": prompt_workload_config(cfg, n), "step": what},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                         "sample": (f"each step = one (sequence, KV head) pair of the {n}-sequence "
                                    f"group on one core ({nsample} evenly spaced "
                                    f"{'queries' if args.workload == 'prompt' else 'keys'}, "
                                    f"extrapolated to the prompt), then to the whole group by pairs")},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(rec), flush=True)


def run_prompt_bench(args):
    import torch
    rank_, local_rank, world = dist_info()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    dist = dist_init(world, "nccl")
    from paper_2607_05061_gb300 import build as _build
    _build.build()
    from paper_2607_05061_gb300 import kvpop
    from workload import gen, get_config
    over = {}
    if args.batch:
        over["batch"] = args.batch
    if args.prompt_len:
        over["prompt_len"] = args.prompt_len
    cfg = get_config(args.config, **over)
    if cfg.n_layers != 1 or cfg.ragged:
        raise SystemExit("--workload prompt/target runs fixed-length single-layer workloads")
    n = min(args.group, cfg.batch)
    P, H, G, d = cfg.prompt_len, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim
    L = [P] * n
    W1, b1, w2, b2, lg = gen.scorer_weights(cfg)
    cache = kvpop.KVpopCache(cfg.batch, H, G, d, cfg.budget_B, cfg.delay_D, cfg.scorer_hidden,
                             cfg.kv_dtype, W1, b1, w2, b2, n_sink=cfg.n_sink)
    Q = gen.q_tokens(cfg, 0, n, 0, P, device=dev)
    K = gen.kv_tokens(cfg, "k", 0, n, 0, P, device=dev)
    V = gen.kv_tokens(cfg, "v", 0, n, 0, P, device=dev)
    Y = torch.empty((n, H * G, P, d), dtype=torch.float32, device=dev)
    lse = torch.empty((n, H * G, P), dtype=torch.float32, device=dev)
    rk = torch.empty((n, H, P), dtype=torch.int32, device=dev)
    tu = torch.empty((n, H, P), dtype=torch.int32, device=dev)
    od = torch.empty((n, H, P), dtype=torch.int32, device=dev)
    logm = torch.empty((n, H * G, P), dtype=torch.float32, device=dev)
    tgt = torch.empty((n, H, P), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    k_b = cfg.budget_B - cfg.n_sink

    def prompt_step():
        cache.prefill_attend(Q, K, V, L, Y, lse, rank=rk, tau=tu, order=od)

    def target_step():
        kvpop.future_target(Q, K, lse, cfg.delay_D, logm=logm, target=tgt)

    def kernel_only():
        if args.workload == "prompt":
            kvpop.prompt_attention(Q, K, V, rk, tu, cfg.n_sink, cfg.delay_D, k_b, Y=Y, lse=lse, order=od)
        else:
            kvpop.future_target(Q, K, lse, cfg.delay_D, logm=logm, want_target=False)

    step = prompt_step if args.workload == "prompt" else target_step
    prompt_step()                                  # the target pass consumes these normalisers
    W, Kn = max(3, args.warmup), args.steps
    for _ in range(W):
        step()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local_rank)
    clocks.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(Kn):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    step_ms, _ = reduce_max_sum(e0.elapsed_time(e1) / Kn, 0.0, world, dev)
    # dominant kernel alone (same stream, CUDA events)
    ks = []
    for _ in range(3):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        kernel_only()
        b.record(stream)
        torch.cuda.synchronize()
        ks.append(a.elapsed_time(b))
    k_ms = statistics.mean(ks)
    cache.check()
    flops = prompt_attention_flops(cfg, L) if args.workload == "prompt" else target_flops(cfg, L)
    peak, peak_src = measured_tensor_peak()
    achieved = flops / (k_ms / 1e3) / 1e12
    # end to end through the public API on pinned host buffers
    Qh, Kh, Vh = Q.cpu().pin_memory(), K.cpu().pin_memory(), V.cpu().pin_memory()
    if args.workload == "prompt":
        outs_h = [torch.empty_like(Y, device="cpu").pin_memory(), torch.empty_like(lse, device="cpu").pin_memory()]
        h2d = (Qh.numel() + Kh.numel() + Vh.numel()) * Qh.element_size()
    else:
        lse_h = lse.cpu().pin_memory()
        outs_h = [torch.empty_like(tgt, device="cpu").pin_memory()]
        h2d = (Qh.numel() + Kh.numel()) * Qh.element_size() + lse_h.numel() * 4
    d2h = sum(o.numel() * o.element_size() for o in outs_h)
    E = 2
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(E):
        Q.copy_(Qh, non_blocking=True)
        K.copy_(Kh, non_blocking=True)
        if args.workload == "prompt":
            V.copy_(Vh, non_blocking=True)
            prompt_step()
            outs_h[0].copy_(Y, non_blocking=True)
            outs_h[1].copy_(lse, non_blocking=True)
        else:
            lse.copy_(lse_h, non_blocking=True)
            target_step()
            outs_h[0].copy_(tgt, non_blocking=True)
        stream.synchronize()
    e2e_s = (time.perf_counter() - t0) / E
    tokens = n * P * world
    tfile = os.path.join(ROOT, "profiles", ("prompt_t5_kernel_traffic.txt" if args.workload == "prompt"
                                            else "target_t5_kernel_traffic.txt"))
    traffic = (committed_traffic(cfg.name, tfile, sequences=n)
               if (cfg.kv_dtype == "bf16" and d == 128 and not over) else None)
    metric, what = prompt_metric(args.workload)
    if args.workload == "prompt":
        kname = (("prompt_t5_kernel" if d == 128 and not os.environ.get("KVPOP_PROMPT_MMA_SYNC")
                  else "prompt_tc_kernel") if cfg.kv_dtype == "bf16" else "prompt_simt_kernel")
    else:
        kname = (("target_t5_kernel" if d == 128 and not os.environ.get("KVPOP_TARGET_MMA_SYNC")
                  else "target_tc_kernel") if cfg.kv_dtype == "bf16" else "target_simt_kernel")
    rec = {
        "metric": metric, "value": tokens / (step_ms / 1e3), "unit": "tokens/s", "n_gpus": world,
        "steps": Kn, "warmup": W, "ms_per_step": step_ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": cfg.kv_dtype,
        "data": "synthetic (seeded counter-based generator)",
        "config": {"workload": prompt_workload_config(cfg, n),
                   "step": what,
                   "l2": f"inputs larger than L2: Q/K/V {(Q.numel() + K.numel() + V.numel()) * 2 / 1e9:.2f} GB",
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "roofline": {"bound": "tensor", "kernel": kname, "achieved": achieved, "peak": peak,
                     "peak_source": peak_src, "unit": "TFLOP/s", "frac": achieved / peak,
                     "traffic": traffic, "algorithmic_flops_per_launch": flops, "ms_per_launch": k_ms},
        "e2e": {"value": tokens / e2e_s, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": E,
                "how": "pinned host inputs copied in, outputs copied out, inside the timed region"},
        "gpu_launches": Kn * (5 if args.workload == "prompt" else 2),
        "clocks": clk,
    }
    cache.free()
    if rank_ == 0 and not args.no_cpu_baseline:
        rec["cpu_baseline"] = cpu_prompt_baseline(cfg, over, n, args.workload)
    if rank_ == 0:
        print(json.dumps(rec), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse_args()
    if args.impl == "reference":
        if args.workload == "decode":
            run_reference(args)
        else:
            run_reference_prompt(args)
    elif args.workload != "decode":
        run_prompt_bench(args)
    else:
        run_kvpop(args)


if __name__ == "__main__":
    main()
