"""Host-side logic of bench.py: multi-rank aggregation (world size 2 over gloo on
CPU), the algorithmic byte count, sampling of oracle pairs, the committed
traffic figure, the prompt and target flop counts behind their roofline (against the
oracle's mask and a pair-by-pair count), and the reference arm's JSON line (the
oracle on host cores), alone and under torchrun with two ranks, where rank 0 alone
prints it."""
import os
import socket

import pytest
import torch.multiprocessing as mp

import bench
from workload import get_config


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    # rank r reports a step time of 1 + r ms and 100 * (r + 1) tokens
    mx, sm = bench.reduce_max_sum(1.0 + rank, 100.0 * (rank + 1), world, None)
    q.put((rank, mx, sm))
    dist.barrier()
    dist.destroy_process_group()


def test_reduce_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # max over ranks of the time, sum over ranks of the tokens, the same on every rank
    assert res == [(0, 2.0, 300.0), (1, 2.0, 300.0)]


def test_single_rank_reduce_is_identity():
    assert bench.reduce_max_sum(3.5, 7.0, 1) == (3.5, 7.0)


def test_kv_stream_bytes_counts_slots_and_window():
    cfg = get_config("cr8x")
    # steady state: every pair holds B slots + D window keys of 2 * d * 2 bytes
    full = cfg.batch * cfg.n_kv_heads * (cfg.budget_B + cfg.delay_D) * 2 * cfg.head_dim * 2
    assert bench.kv_stream_bytes(cfg, [cfg.prompt_len] * cfg.batch, 0) == full
    # a short sequence keeps all its eligible tokens
    tiny = get_config("tiny", budget_B=1000)
    P = 100
    expect = tiny.n_kv_heads * ((P + 1 - tiny.delay_D) + tiny.delay_D) * 2 * tiny.head_dim * 4
    assert bench.kv_stream_bytes(tiny, [P], 0) == expect


def test_sample_pairs_are_distinct_and_in_range():
    cfg = get_config("cr8x")
    pairs = bench.sample_pairs(cfg, 16)
    assert len(pairs) == len(set(pairs)) == 16
    assert all(0 <= b < cfg.batch and 0 <= h < cfg.n_kv_heads for b, h in pairs)


def test_committed_traffic_requires_matching_config():
    assert bench.committed_traffic("ragged") is None
    t = bench.committed_traffic("cr8x")
    assert t is None or t > 1_000_000_000


# ---------------------------------------------------------------- the reference arm's JSON line
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
REQUIRED = ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
            "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config")


def _json_lines(out):
    import json
    return [json.loads(l) for l in out.splitlines() if l.startswith("{")]


def _check_reference_line(rec, n_gpus, steps, warmup):
    for k in REQUIRED:
        assert k in rec, k
    assert rec["impl"] == "reference"
    assert rec["n_gpus"] == n_gpus and rec["steps"] == steps and rec["warmup"] == warmup
    assert rec["value"] > 0 and rec["unit"] == "tokens/s" and rec["higher_is_better"] is True
    assert rec["vs_baseline"] is None and rec["config"]["workload"].startswith("tiny")
    cb = rec["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and isinstance(cb["sample"], str)
    assert cb["value"] == rec["value"]
    e = rec["e2e"]
    assert e["value"] == rec["value"] and e["unit"] == rec["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


@pytest.mark.parametrize("workload", ["decode", "prompt", "target"])
def test_reference_arm_prints_one_contract_line(workload):
    import subprocess
    import sys
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", workload,
                        "--config", "tiny", "--steps", "2", "--warmup", "3"], cwd=ROOT,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    recs = _json_lines(r.stdout)
    assert len(recs) == 1
    _check_reference_line(recs[0], 1, 2, 3)
    # the same metric as the GPU arm of that workload
    want = bench.METRIC if workload == "decode" else bench.prompt_metric(workload)[0]
    assert recs[0]["metric"] == want
    if workload == "decode":
        # and the same config object the GPU arm prints for these steps
        from workload import gen
        cfg = get_config("tiny")
        L = gen.prompt_lengths(cfg)
        assert recs[0]["config"] == bench.decode_config(cfg, "mlp", bench.mean_stream_bytes(cfg, L, 3, 2), 1)


def test_reference_arm_under_torchrun_prints_once_from_rank0():
    import subprocess
    import sys
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), "bench.py",
           "--impl", "reference", "--config", "tiny", "--gpus", "2", "--steps", "1", "--warmup", "3"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600,
                       env=dict(os.environ, OMP_NUM_THREADS="1"))
    assert r.returncode == 0, r.stderr[-2000:]
    recs = _json_lines(r.stdout)
    assert len(recs) == 1
    _check_reference_line(recs[0], 2, 1, 3)


# ---------------------------------------------------------------- roofline arithmetic of the prompt paths
@pytest.mark.parametrize("P,B,D,s", [(60, 16, 4, 0), (97, 24, 7, 3), (10, 16, 4, 2)])
def test_prompt_flops_count_the_oracle_mask(P, B, D, s):
    """4 d G per retained (query, key) of the running top-k mask built by the oracle."""
    import numpy as np
    from oracle import running_topk as rt
    cfg = get_config("q4b", batch=1, prompt_len=P, budget_B=B, delay_D=D, n_sink=s)
    raw = np.random.default_rng(P).standard_normal(P).astype(np.float32)
    prio = rt.prompt_priorities(raw, P, D, 0.0)
    rank = rt.static_ranks(prio)
    tau = rt.fenwick_cutoffs(rank, s, D, B - s)
    kept = sum(int(rt.mask_row(q, rank, tau, s, D).sum()) for q in range(P))
    want = 4.0 * cfg.head_dim * cfg.q_per_kv * cfg.n_kv_heads * kept
    assert bench.prompt_attention_flops(cfg, [P]) == want


@pytest.mark.parametrize("P,D", [(50, 4), (7, 16), (33, 1)])
def test_target_flops_count_key_query_pairs(P, D):
    """2 d G per (key t, query d) with t + w <= d < P, counted one by one."""
    cfg = get_config("q4b", batch=1, prompt_len=P, delay_D=D)
    pairs = sum(1 for t in range(P) for d in range(P) if d >= t + D)
    want = 2.0 * cfg.head_dim * cfg.q_per_kv * cfg.n_kv_heads * pairs
    assert bench.target_flops(cfg, [P]) == want


# ---------------------------------------------------------------- decode line: L2 rule, dtype, agreement
def test_l2_flush_only_for_workloads_smaller_than_twice_l2():
    from workload import gen
    for name, want in (("q4b", True), ("cr8x", False), ("ragged", False), ("tiny", True)):
        cfg = get_config(name)
        L = gen.prompt_lengths(cfg)
        assert bench.flushes_l2(bench.kv_stream_bytes(cfg, L, 0)) is want, name
    assert bench.decode_dtype(get_config("cr8x")) == "bf16 (fp32 accumulate)"
    assert bench.decode_dtype(get_config("tiny")) == "f32"


def test_agreement_counts_decisions_and_kept_sets():
    gpu_dec = [[[(0, -1), (3, 7)]], [[(-1, -1), (2, 9)]]]          # [step][b][h]
    oracle = {(0, 0): ([1, 2], [(0, -1), (-1, -1)]),
              (0, 1): ([4, 5], [(3, 7), (2, 8)])}
    gpu_kept = {(0, 0): [2, 1], (0, 1): [4, 6]}
    a = bench.agreement(gpu_kept, gpu_dec, oracle)
    assert a["decisions"] == 4 and a["decode_decisions_equal"] == 0.75
    assert a["prefill_kept_sets_equal"] == 0.5 and a["pairs"] == 2 and a["steps"] == 2
    assert a["first_mismatch"] == {"pair": [0, 1], "step": 1, "gpu": [2, 9], "oracle": [2, 8]}


def test_oracle_pair_job_reports_the_oracle_decisions():
    from oracle.run import run_pair
    from workload import gen
    cfg = get_config("tiny")
    L = gen.prompt_lengths(cfg)
    t, kept, dec = bench._oracle_pair_job(("tiny", 0, 1, 12, "mlp"))
    tr = run_pair(cfg, gen.scorer_weights(cfg), 0, 1, L[0], 12, attend=False, keep_cache=True)
    assert t > 0
    assert dec == list(zip(tr.slots, tr.evicted))
    assert any(e >= 0 for _, e in dec)
    ref = run_pair(cfg, gen.scorer_weights(cfg), 0, 1, L[0], 0, keep_cache=True)
    assert kept == ref.cache.kept_positions()
