"""GPU parity of the running top-k prompt path (App. C) through the C ABI.

* Static ranks and cutoffs tau_q: bit-exact against the oracle (sort + Fenwick
  scan) on the same fp32 priorities, ties and NaN included.
* Prompt attention under the running top-k mask: y within the K/V dtype's
  max-abs tolerance (1e-5 fp32, 2e-2 bf16); the natural-log normaliser within
  1e-5 (fp32) or 1e-3 (bf16: the logits are fp32 sums of exact bf16 products).
* kvpop_prefill_attend: ranks/cutoffs/outputs against the oracle on injected
  scores, and, at any size, the retained set of the last prompt query equals the
  cache that prompt compression leaves (two independent kernels).
Full sizes (the q4b and cr8x prompts) are checked on sampled (sequence, head)
pairs and sampled queries, which the oracle computes one by one.
"""
import numpy as np
import pytest
import torch

from gpu_harness import make_cache
from oracle import prefill_head
from oracle import running_topk as rt
from oracle.run import head_params
from workload import gen, get_config

pytestmark = pytest.mark.gpu

Y_TOL = {"f32": 1e-5, "bf16": 2e-2}
LSE_TOL = {"f32": 1e-5, "bf16": 1e-3}
STREAM_PRIO = 40


def kv():
    from paper_2607_05061_gb300 import kvpop
    return kvpop


def f64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def plant_specials(prio: torch.Tensor):
    """NaN and -0 entries (canonicalised to -inf and +0 on both sides)."""
    flat = prio.view(-1)
    n = flat.numel()
    flat[n // 7] = float("nan")
    flat[n // 3] = -0.0
    flat[n // 3 + 1] = 0.0
    return prio


# ---------------------------------------------------------------- ranks and cutoffs
@pytest.mark.parametrize("s,w,k", [(0, 16, 100), (3, 5, 1), (2, 1, 5000), (0, 32, 700)])
@pytest.mark.parametrize("levels", [None, 3])
def test_topk_cutoff_bitexact(cuda_device, s, w, k, levels):
    S = 3000
    lengths = [3000, 2999, 1, 0, 1500, 2055]
    prio = plant_specials(gen.uniform_scores(7, STREAM_PRIO, (len(lengths), S), levels=levels))
    L = torch.tensor(lengths, dtype=torch.int32, device=cuda_device)
    order = torch.full((len(lengths), S), -7, dtype=torch.int32, device=cuda_device)
    rank, tau = kv().topk_cutoff(prio.to(cuda_device), s, w, k, lengths=L, order=order)
    rank, tau, order = rank.cpu().numpy(), tau.cpu().numpy(), order.cpu().numpy()
    for r, n in enumerate(lengths):
        want_rank = rt.static_ranks(prio[r, :n].numpy())
        want_tau = rt.fenwick_cutoffs(want_rank, s, w, k)
        assert np.array_equal(rank[r, :n], want_rank), f"row {r}: ranks differ"
        assert np.array_equal(tau[r, :n], want_tau), f"row {r}: cutoffs differ"
        assert np.all(rank[r, n:] == -1) and np.all(tau[r, n:] == -1)
        # order is the inverse permutation of the ranks; entries past the length untouched
        assert np.array_equal(order[r, want_rank], np.arange(n)), f"row {r}: order differs"
        assert np.all(order[r, n:] == -7)


def test_topk_cutoff_longest_rows(cuda_device):
    """Rows of 65536 tokens (the longest prompts of the ragged workload), B = 8192, D = 32."""
    S, s, w, k = 65536, 0, 32, 8192
    prio = gen.uniform_scores(8, STREAM_PRIO, (2, S))
    prio[1] = gen.uniform_scores(9, STREAM_PRIO, (S,), levels=50)
    rank, tau = kv().topk_cutoff(prio.to(cuda_device), s, w, k)
    for r in range(2):
        want_rank = rt.static_ranks(prio[r].numpy())
        assert np.array_equal(rank[r].cpu().numpy(), want_rank)
        assert np.array_equal(tau[r].cpu().numpy(), rt.fenwick_cutoffs(want_rank, s, w, k))


# ---------------------------------------------------------------- prompt attention
def attention_case(cfg, lengths, s, w, k, seed_prio, device):
    n, H = len(lengths), cfg.n_kv_heads
    S = max(lengths)
    Q = gen.q_tokens(cfg, 0, n, 0, S)
    K = gen.kv_tokens(cfg, "k", 0, n, 0, S)
    V = gen.kv_tokens(cfg, "v", 0, n, 0, S)
    prio = gen.uniform_scores(seed_prio, STREAM_PRIO, (n, H, S), levels=None)
    ranks = np.full((n, H, S), -1, dtype=np.int32)
    taus = np.full((n, H, S), -1, dtype=np.int32)
    for b in range(n):
        for h in range(H):
            r = rt.static_ranks(prio[b, h, :lengths[b]].numpy())
            ranks[b, h, :lengths[b]] = r
            taus[b, h, :lengths[b]] = rt.fenwick_cutoffs(r, s, w, k)
    return Q, K, V, ranks, taus


def inverse_ranks(ranks, lengths):
    """Positions by rank, built from the oracle's ranks (the order a rank walk reads)."""
    order = np.full(ranks.shape, -1, dtype=np.int32)
    for b, n in enumerate(lengths):
        for h in range(ranks.shape[1]):
            order[b, h, ranks[b, h, :n]] = np.arange(n, dtype=np.int32)
    return order


@pytest.mark.parametrize("dtype,d,G", [("f32", 64, 2), ("f32", 128, 4), ("bf16", 128, 4),
                                       ("bf16", 64, 2), ("bf16", 128, 1)])
@pytest.mark.parametrize("by_rank", [False, True])
def test_prompt_attention_matches_oracle(cuda_device, dtype, d, G, by_rank):
    """Masked attention against the oracle; with ``by_rank`` the key lists of the late
    tiles are built by walking the ranks up to the tile's largest cutoff."""
    cfg = get_config("tiny").with_(kv_dtype=dtype, head_dim=d, q_per_kv=G, n_kv_heads=2, batch=2)
    lengths = [300, 237]
    s, w, k = 2, 5, 40
    Q, K, V, ranks, taus = attention_case(cfg, lengths, s, w, k, 3, cuda_device)
    dev = cuda_device
    L = torch.tensor(lengths, dtype=torch.int32, device=dev)
    order = torch.from_numpy(inverse_ranks(ranks, lengths)).to(dev) if by_rank else None
    Y, lse = kv().prompt_attention(Q.to(dev), K.to(dev), V.to(dev), torch.from_numpy(ranks).to(dev),
                                   torch.from_numpy(taus).to(dev), s, w, k, lengths=L, order=order)
    Y, lse = Y.cpu().numpy(), lse.cpu().numpy()
    ey = el = 0.0
    for b, n in enumerate(lengths):
        for h in range(cfg.n_kv_heads):
            y, l = rt.masked_attention(f64(Q[b, h * G:(h + 1) * G, :n]), f64(K[b, h, :n]),
                                       f64(V[b, h, :n]), ranks[b, h, :n], taus[b, h, :n], s, w)
            ey = max(ey, float(np.abs(Y[b, h * G:(h + 1) * G, :n] - y).max()))
            el = max(el, float(np.abs(lse[b, h * G:(h + 1) * G, :n] - l).max()))
    print(f"prompt attention {dtype} d{d} G{G} by_rank={by_rank}: max-abs y {ey:.2e}, lse {el:.2e}")
    assert ey <= Y_TOL[dtype] and el <= LSE_TOL[dtype]


# ---------------------------------------------------------------- prefill with outputs
def run_prefill_attend(cache, cfg, lengths, device, override, b0=0, want=True):
    n = len(lengths)
    S = max(lengths)
    Q = gen.q_tokens(cfg, b0, n, 0, S, device=device)
    K = gen.kv_tokens(cfg, "k", b0, n, 0, S, device=device)
    V = gen.kv_tokens(cfg, "v", b0, n, 0, S, device=device)
    HG, H, d = cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim
    Y = torch.full((n, HG, S, d), float("nan"), dtype=torch.float32, device=device)
    lse = torch.empty((n, HG, S), dtype=torch.float32, device=device)
    rank = torch.empty((n, H, S), dtype=torch.int32, device=device)
    tau = torch.empty((n, H, S), dtype=torch.int32, device=device)
    order = torch.full((n, H, S), -7, dtype=torch.int32, device=device)
    ov = None if override is None else override[b0:b0 + n, :, :S].contiguous()
    cache.prefill_attend(Q, K, V, lengths, Y, lse, first_seq=b0, override=ov, rank=rank, tau=tau,
                         order=order)
    torch.cuda.synchronize()
    cache.check()
    rk, od = rank.cpu().numpy(), order.cpu().numpy()
    for b, P in enumerate(lengths):
        for h in range(H):
            assert np.array_equal(od[b, h, rk[b, h, :P]], np.arange(P)), (b, h)
            assert np.all(od[b, h, P:] == -7), (b, h)
    return Y, lse, rank, tau


def oracle_pair_cache(cfg, w, b, h, P, ov):
    G = cfg.q_per_kv
    K = f64(gen.kv_tokens(cfg, "k", b, 1, 0, P, heads=[h]))[0, 0]
    V = f64(gen.kv_tokens(cfg, "v", b, 1, 0, P, heads=[h]))[0, 0]
    Q = f64(gen.q_tokens(cfg, b, 1, 0, P, heads=range(h * G, (h + 1) * G)))[0]
    c = prefill_head(head_params(cfg, w, h), Q, K, V, cfg.head_dim, G,
                     None if ov is None else ov[b, h, :P].numpy())
    return c, Q, K, V


def check_last_query_is_cache(cache, cfg, lengths, rank, tau, b0=0, pairs=None):
    """Retained long-range set of q = P - 1 equals the compressed cache (any size)."""
    s, D = cfg.n_sink, cfg.delay_D
    rank, tau = rank.cpu().numpy(), tau.cpu().numpy()
    pairs = pairs or [(b, h) for b in range(len(lengths)) for h in range(cfg.n_kv_heads)]
    for b, h in pairs:
        P = lengths[b]
        if P == 0:
            continue
        pos, _ = cache.pair_state(b0 + b, h)
        t = np.arange(P)
        kept = (t < s) & (t <= P - 1 - D) | ((t >= s) & (t <= P - 1 - D) & (rank[b, h, :P] <= tau[b, h, P - 1]))
        assert sorted(pos) == list(np.nonzero(kept)[0]), (b, h)


@pytest.mark.parametrize("name", ["tiny", "mixed"])
def test_prefill_attend_full_parity(cuda_device, name):
    if name == "tiny":
        cfg = get_config("tiny")
        lengths = gen.prompt_lengths(cfg)
    else:   # bf16, sinks and decay, ragged prompts spanning several tiles
        cfg = get_config("q4b").with_(batch=2, budget_B=128, delay_D=16, n_sink=3, log_gamma=-2e-3,
                                      prompt_len=700, scorer_hidden=32)
        lengths = [700, 513]
    w = gen.scorer_weights(cfg)
    Pmax = max(lengths)
    ov = gen.uniform_scores(cfg.seed, 41, (cfg.batch, cfg.n_kv_heads, Pmax))
    cache = make_cache(cfg, w)
    Y, lse, rank, tau = run_prefill_attend(cache, cfg, lengths, cuda_device, ov.to(cuda_device))
    check_last_query_is_cache(cache, cfg, lengths, rank, tau)
    G = cfg.q_per_kv
    Yc, lc, rc, tc = Y.cpu().numpy(), lse.cpu().numpy(), rank.cpu().numpy(), tau.cpu().numpy()
    ey = el = 0.0
    for b, P in enumerate(lengths):
        for h in range(cfg.n_kv_heads):
            c, Q, K, V = oracle_pair_cache(cfg, w, b, h, P, ov)
            y, l, r, t = rt.prefill_outputs(c, Q, K, V)
            assert np.array_equal(rc[b, h, :P], r) and np.array_equal(tc[b, h, :P], t), (b, h)
            pos, _ = cache.pair_state(b, h)
            assert pos == c.kept_positions()
            ey = max(ey, float(np.abs(Yc[b, h * G:(h + 1) * G, :P] - y).max()))
            el = max(el, float(np.abs(lc[b, h * G:(h + 1) * G, :P] - l).max()))
    print(f"prefill_attend {name}: max-abs y {ey:.2e}, lse {el:.2e}")
    assert ey <= Y_TOL[cfg.kv_dtype] and el <= LSE_TOL[cfg.kv_dtype]
    cache.free()


def test_prefill_attend_own_scorer_matches_compression(cuda_device):
    """With the cache's own scorer, ranks/cutoffs agree with prompt compression's selection."""
    cfg = get_config("q4b").with_(batch=3, prompt_len=1500)
    lengths = [1500, 1200, 17]
    w = gen.scorer_weights(cfg)
    cache = make_cache(cfg, w)
    Y, lse, rank, tau = run_prefill_attend(cache, cfg, lengths, cuda_device, None)
    check_last_query_is_cache(cache, cfg, lengths, rank, tau)
    for b, P in enumerate(lengths):
        assert torch.isfinite(Y[b, :, :P]).all() and torch.isfinite(lse[b, :, :P]).all()
    # y and LSE against the oracle, which scores with its own fp64 scorer: each side
    # builds its mask from its own fp32 scores, so a near-tie may order two tokens
    # differently; compare the queries whose retained sets agree (nearly all) and
    # require that they are nearly all
    G = cfg.q_per_kv
    ey = el = 0.0
    n_q = n_same = 0
    for b, h in [(0, 2), (1, 7), (2, 0)]:
        P = lengths[b]
        c, Q, K, V = oracle_pair_cache(cfg, w, b, h, P, None)
        prio = rt.prompt_priorities(c.prefill_raw, P, cfg.delay_D, c.p.log_gamma)
        r = rt.static_ranks(prio)
        t = rt.fenwick_cutoffs(r, cfg.n_sink, cfg.delay_D, cfg.budget_B - cfg.n_sink)
        gr = rank[b, h, :P].cpu().numpy()
        gt = tau[b, h, :P].cpu().numpy()
        for q in sorted(set(np.linspace(0, P - 1, 40).astype(int).tolist())):
            n_q += 1
            m_o = rt.mask_row(q, r, t, cfg.n_sink, cfg.delay_D)
            if not np.array_equal(m_o, rt.mask_row(q, gr, gt, cfg.n_sink, cfg.delay_D)):
                continue
            n_same += 1
            keys = np.nonzero(m_o)[0]
            logits = (Q[:, q, :] @ K[keys].T) / np.sqrt(cfg.head_dim)
            mx = logits.max(axis=1, keepdims=True)
            e = np.exp(logits - mx)
            y = (e / e.sum(axis=1, keepdims=True)) @ V[keys]
            l = (mx + np.log(e.sum(axis=1, keepdims=True)))[:, 0]
            ey = max(ey, float(np.abs(f64(Y[b, h * G:(h + 1) * G, q]) - y).max()))
            el = max(el, float(np.abs(f64(lse[b, h * G:(h + 1) * G, q]) - l).max()))
    print(f"prefill_attend own scorer: {n_same}/{n_q} sampled queries with the same retained "
          f"set; max-abs y {ey:.2e}, lse {el:.2e}")
    assert n_same >= 0.95 * n_q
    assert ey <= Y_TOL[cfg.kv_dtype] and el <= LSE_TOL[cfg.kv_dtype]
    cache.free()


def test_prefill_attend_mlstm_dispatch(cuda_device):
    """The mLSTM cache runs the same prompt path (scores injected)."""
    cfg = get_config("tiny")
    lengths = gen.prompt_lengths(cfg)
    ov = gen.uniform_scores(cfg.seed, 41, (cfg.batch, cfg.n_kv_heads, max(lengths)))
    w = gen.scorer_weights(cfg)
    c1 = make_cache(cfg, None, mlstm=gen.mlstm_weights(cfg))
    c2 = make_cache(cfg, w)
    a = run_prefill_attend(c1, cfg, lengths, cuda_device, ov.to(cuda_device))
    b = run_prefill_attend(c2, cfg, lengths, cuda_device, ov.to(cuda_device))
    for x, y in zip(a, b):
        assert torch.equal(x, y)
    c1.free()
    c2.free()


# ---------------------------------------------------------------- full sizes, sampled
def sampled_outputs_check(cfg, w, ov, lengths, Y, lse, rank, tau, pairs, n_q, seed, b0=0):
    rng = np.random.default_rng(seed)
    G = cfg.q_per_kv
    ey = el = 0.0
    for b, h in pairs:
        P = lengths[b]
        c, Q, K, V = oracle_pair_cache(cfg, w, b0 + b, h, P, ov)
        prio = rt.prompt_priorities(c.prefill_raw, P, cfg.delay_D, c.p.log_gamma)
        r = rt.static_ranks(prio)
        t = rt.fenwick_cutoffs(r, cfg.n_sink, cfg.delay_D, cfg.budget_B - cfg.n_sink)
        assert np.array_equal(rank[b, h, :P].cpu().numpy(), r), (b, h)
        assert np.array_equal(tau[b, h, :P].cpu().numpy(), t), (b, h)
        qs = sorted(set([0, P - 1, min(P - 1, cfg.budget_B + cfg.delay_D)] +
                        list(rng.integers(0, P, n_q))))
        for q in qs:
            keys = np.nonzero(rt.mask_row(q, r, t, cfg.n_sink, cfg.delay_D))[0]
            logits = (Q[:, q, :] @ K[keys].T) / np.sqrt(cfg.head_dim)
            mx = logits.max(axis=1, keepdims=True)
            e = np.exp(logits - mx)
            y = (e / e.sum(axis=1, keepdims=True)) @ V[keys]
            l = (mx + np.log(e.sum(axis=1, keepdims=True)))[:, 0]
            ey = max(ey, float(np.abs(f64(Y[b, h * G:(h + 1) * G, q]) - y).max()))
            el = max(el, float(np.abs(f64(lse[b, h * G:(h + 1) * G, q]) - l).max()))
    return ey, el


@pytest.mark.parametrize("name,group", [("q4b", 8), ("cr8x", 8)])
def test_prefill_attend_full_size_sampled(cuda_device, name, group):
    cfg = get_config(name)
    w = gen.scorer_weights(cfg)
    lengths = gen.prompt_lengths(cfg)[:group]
    ov = gen.uniform_scores(cfg.seed, 41, (group, cfg.n_kv_heads, max(lengths)))
    cache = make_cache(cfg, w)
    Y, lse, rank, tau = run_prefill_attend(cache, cfg, lengths, cuda_device, ov.to(cuda_device))
    pairs = [(0, 0), (group - 1, cfg.n_kv_heads - 1), (3, 5)]
    check_last_query_is_cache(cache, cfg, lengths, rank, tau)
    ey, el = sampled_outputs_check(cfg, w, ov, lengths, Y, lse, rank, tau, pairs, 24, 5)
    print(f"prefill_attend {name}: sampled max-abs y {ey:.2e}, lse {el:.2e}")
    assert ey <= Y_TOL[cfg.kv_dtype] and el <= LSE_TOL[cfg.kv_dtype]
    cache.free()
