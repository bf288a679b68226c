"""GPU parity of the future-attention target (App. D, App. F.1-F.2) through the C ABI.

* Dense causal normalisers against the oracle's logsumexp.
* Transposed pass (log future mass per key and query head) and the aggregated
  per-KV-head target against the oracle, given the same fp32 normalisers:
  max-abs 1e-5 (fp32 inputs) or 1e-3 (bf16 inputs: fp32 sums of exact bf16
  products), with -inf (no future query) at exactly the same places.
* The approximate target of App. D.3 end to end: sparse normalisers from
  kvpop_prefill_attend, then the transposed pass, against the oracle chain.
* Full size (the cr8x prompt): normalisers at sampled queries and log masses of
  the last keys, whose future the oracle sums in full.
"""
import numpy as np
import pytest
import torch

from gpu_harness import make_cache
from oracle import future_target as ft
from oracle import running_topk as rt
from test_gpu_prompt import f64, oracle_pair_cache, run_prefill_attend
from workload import gen, get_config

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-5, "bf16": 1e-3}


def kv():
    from paper_2607_05061_gb300 import kvpop
    return kvpop


def small_case(dtype, d, G, lengths):
    cfg = get_config("tiny").with_(kv_dtype=dtype, head_dim=d, q_per_kv=G, n_kv_heads=2,
                                   batch=len(lengths))
    S = max(lengths)
    return cfg, gen.q_tokens(cfg, 0, len(lengths), 0, S), gen.kv_tokens(cfg, "k", 0, len(lengths), 0, S)


CASES = [("f32", 64, 2), ("f32", 128, 4), ("bf16", 128, 4), ("bf16", 64, 1)]


@pytest.mark.parametrize("dtype,d,G", CASES)
def test_causal_lse_matches_oracle(cuda_device, dtype, d, G):
    lengths = [300, 211]
    cfg, Q, K = small_case(dtype, d, G, lengths)
    L = torch.tensor(lengths, dtype=torch.int32, device=cuda_device)
    lse = kv().causal_lse(Q.to(cuda_device), K.to(cuda_device), lengths=L).cpu().numpy()
    err = 0.0
    for b, n in enumerate(lengths):
        for h in range(cfg.n_kv_heads):
            for g in range(G):
                want = ft.dense_causal_lse(f64(Q[b, h * G + g, :n]), f64(K[b, h, :n]))
                err = max(err, float(np.abs(lse[b, h * G + g, :n] - want).max()))
    print(f"causal lse {dtype} d{d} G{G}: max-abs {err:.2e}")
    assert err <= TOL[dtype]


@pytest.mark.parametrize("dtype,d,G", CASES)
@pytest.mark.parametrize("w,la", [(4, 0), (1, 7), (16, 0), (0, 0)])
def test_future_target_matches_oracle(cuda_device, dtype, d, G, w, la):
    lengths = [300, 211]
    cfg, Q, K = small_case(dtype, d, G, lengths)
    S, H = max(lengths), cfg.n_kv_heads
    lse = np.zeros((len(lengths), H * G, S), dtype=np.float32)
    for b, n in enumerate(lengths):
        for r in range(H * G):
            lse[b, r, :n] = ft.dense_causal_lse(f64(Q[b, r, :n]), f64(K[b, r // G, :n]))
    dev = cuda_device
    L = torch.tensor(lengths, dtype=torch.int32, device=dev)
    eps = 1e-6
    for agg, cn in (("max", True), ("mean", False)):
        logm, tgt = kv().future_target(Q.to(dev), K.to(dev), torch.from_numpy(lse).to(dev), w,
                                       lookahead=la, agg=agg, count_norm=cn, eps=eps, lengths=L)
        logm, tgt = logm.cpu().numpy(), tgt.cpu().numpy()
        em = et = 0.0
        for b, n in enumerate(lengths):
            for h in range(H):
                want = np.stack([ft.future_log_mass(f64(Q[b, h * G + g, :n]), f64(K[b, h, :n]),
                                                    lse[b, h * G + g, :n].astype(np.float64), w, la)
                                 for g in range(G)])
                got = logm[b, h * G:(h + 1) * G, :n]
                fin = np.isfinite(want)
                assert np.array_equal(fin, np.isfinite(got)), (b, h)
                if fin.any():
                    em = max(em, float(np.abs(got[fin] - want[fin]).max()))
                r = ft.aggregate_target(want, n, w, eps, agg, cn, la)
                et = max(et, float(np.abs(tgt[b, h, :n] - r).max()))
        print(f"future target {dtype} d{d} G{G} w{w} L{la} {agg}: log-mass {em:.2e}, target {et:.2e}")
        assert em <= TOL[dtype] and et <= TOL[dtype]


def test_sparse_normaliser_target_end_to_end(cuda_device):
    """App. D.3: the prompt path's sparse LSE feeds the transposed pass."""
    cfg = get_config("q4b").with_(batch=2, budget_B=128, delay_D=16, n_sink=3, log_gamma=-2e-3,
                                  prompt_len=700, scorer_hidden=32)
    lengths = [700, 513]
    w = gen.scorer_weights(cfg)
    ov = gen.uniform_scores(cfg.seed, 41, (cfg.batch, cfg.n_kv_heads, max(lengths)))
    cache = make_cache(cfg, w)
    Y, lse, rank, tau = run_prefill_attend(cache, cfg, lengths, cuda_device, ov.to(cuda_device))
    S, G, D = max(lengths), cfg.q_per_kv, cfg.delay_D
    Q = gen.q_tokens(cfg, 0, 2, 0, S, device=cuda_device)
    K = gen.kv_tokens(cfg, "k", 0, 2, 0, S, device=cuda_device)
    L = torch.tensor(lengths, dtype=torch.int32, device=cuda_device)
    logm, tgt = kv().future_target(Q, K, lse, D, lengths=L)
    logm, tgt = logm.cpu().numpy(), tgt.cpu().numpy()
    em = et = 0.0
    for b, P in enumerate(lengths):
        for h in range(cfg.n_kv_heads):
            c, Qo, Ko, Vo = oracle_pair_cache(cfg, w, b, h, P, ov)
            _, lse_o, _, _ = rt.prefill_outputs(c, Qo, Ko, Vo)
            want = np.stack([ft.future_log_mass(Qo[g], Ko, lse_o[g], D) for g in range(G)])
            fin = np.isfinite(want)
            got = logm[b, h * G:(h + 1) * G, :P]
            assert np.array_equal(fin, np.isfinite(got))
            em = max(em, float(np.abs(got[fin] - want[fin]).max()))
            et = max(et, float(np.abs(tgt[b, h, :P] - ft.aggregate_target(want, P, D, 1e-6)).max()))
    print(f"sparse-LSE target end to end: log-mass {em:.2e}, target {et:.2e}")
    assert em <= TOL["bf16"] and et <= TOL["bf16"]
    cache.free()


def test_future_target_full_size_sampled(cuda_device):
    cfg = get_config("cr8x")
    n, S, G, D, d = 8, cfg.prompt_len, cfg.q_per_kv, cfg.delay_D, cfg.head_dim
    dev = cuda_device
    Q = gen.q_tokens(cfg, 0, n, 0, S, device=dev)
    K = gen.kv_tokens(cfg, "k", 0, n, 0, S, device=dev)
    lse = kv().causal_lse(Q, K)
    logm, tgt = kv().future_target(Q, K, lse, D)
    torch.cuda.synchronize()
    rng = np.random.default_rng(3)
    tail = 300
    el = em = 0.0
    for b, h, g in ((0, 0, 0), (n - 1, cfg.n_kv_heads - 1, G - 1), (3, 5, 2)):
        r = h * G + g
        Qg, Kh = f64(Q[b, r]), f64(K[b, h])
        qs = sorted(set(list(rng.integers(0, S, 16)) + [0, S - 1]))
        for q in qs:
            x = Qg[q] @ Kh[: q + 1].T / np.sqrt(d)
            mx = x.max()
            el = max(el, abs(float(lse[b, r, q]) - (mx + np.log(np.exp(x - mx).sum()))))
        lse_tail = np.array([np.logaddexp.reduce(Qg[q] @ Kh[: q + 1].T / np.sqrt(d))
                             for q in range(S - tail, S)])
        for t in range(S - tail, S):
            if t + D > S - 1:
                assert float(logm[b, r, t]) == -np.inf
                continue
            ds = np.arange(t + D, S)
            v = Qg[ds] @ Kh[t] / np.sqrt(d) - lse_tail[ds - (S - tail)]
            em = max(em, abs(float(logm[b, r, t]) - np.logaddexp.reduce(v)))
        assert torch.isfinite(logm[b, r, : S - D]).all()
    print(f"cr8x full size: sampled lse {el:.2e}, tail log-mass {em:.2e}")
    assert el <= TOL["bf16"] and em <= TOL["bf16"]
