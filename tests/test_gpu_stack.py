"""GPU parity of the multi-layer decode stack (projections + KVpop layers)
against the fp64 oracle stack on a reduced Qwen3-8B-shaped configuration."""
import numpy as np
import pytest
import torch

from gpu_harness import TOL
from workload import gen, get_config

pytestmark = pytest.mark.gpu

SMALL_STACK = dict(batch=2, n_kv_heads=2, hidden=1024, prompt_len=300, budget_B=64,
                   decode_steps=40, n_layers=2)


def build_stack(cfg, device):
    from paper_2607_05061_gb300.stack import DecodeStack
    layers = []
    for l in range(cfg.n_layers):
        w = gen.stack_weights(cfg, l, device=device)
        for k in ("W1", "b1", "w2", "b2"):
            w[k] = w[k].cpu()
        layers.append(w)
    return DecodeStack(layers, cfg.batch, cfg.hidden, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim,
                       cfg.budget_B, cfg.delay_D, cfg.scorer_hidden, n_sink=cfg.n_sink, device=device)


def prefill_stack(st, cfg, L, device, overrides=None):
    for l in range(cfg.n_layers):
        X = gen.prompt_hidden(cfg, l, 0, cfg.batch, 0, max(L), device=device)
        ov = None if overrides is None else overrides[l].to(device)
        st.prefill_layer(l, X, L, override=ov)


@pytest.mark.parametrize("path", ["fused", "split"])
def test_stack_matches_oracle_stack(cuda_device, monkeypatch, path):
    """Both kvpop_decode_step paths (the full-size stack runs the one-kernel step)."""
    from oracle.stack import run_stack
    cfg = get_config("q8b_stack", **SMALL_STACK)
    L = gen.prompt_lengths(cfg)
    steps = cfg.decode_steps
    b, H, Hq, d = cfg.batch, cfg.n_kv_heads, cfg.n_q_heads, cfg.head_dim
    pov = [gen.uniform_scores(cfg.seed, 70 + l, (b, H, max(L))) for l in range(cfg.n_layers)]
    dov = [gen.uniform_scores(cfg.seed, 80 + l, (steps, b, H)) for l in range(cfg.n_layers)]
    monkeypatch.delenv("KVPOP_FUSED_STEP", raising=False)
    monkeypatch.delenv("KVPOP_SPLIT_STEP", raising=False)
    monkeypatch.setenv("KVPOP_FUSED_STEP" if path == "fused" else "KVPOP_SPLIT_STEP", "1")
    st = build_stack(cfg, cuda_device)
    monkeypatch.delenv("KVPOP_FUSED_STEP", raising=False)
    monkeypatch.delenv("KVPOP_SPLIT_STEP", raising=False)
    assert all(c.fused_step == (path == "fused") for c in st.caches)
    prefill_stack(st, cfg, L, cuda_device, pov)
    xs = gen.decode_hidden(cfg, L, 0, steps, device=cuda_device)
    outs = [torch.empty((b, Hq * d), device=cuda_device) for _ in range(cfg.n_layers)]
    eis = [torch.empty((b, H, 2), dtype=torch.int32, device=cuda_device) for _ in range(cfg.n_layers)]
    dov_d = [t.to(cuda_device) for t in dov]
    got_o = np.zeros((cfg.n_layers, steps, b, Hq * d))
    got_e = np.zeros((cfg.n_layers, steps, b, H, 2), dtype=np.int64)
    got_x = np.zeros((steps, b, cfg.hidden))
    x_out = torch.empty((b, cfg.hidden), dtype=torch.bfloat16, device=cuda_device)
    for j in range(steps):
        st.step(xs[j], x_out, overrides=[t[j] for t in dov_d], evict_info=eis, outputs=outs)
        for l in range(cfg.n_layers):
            got_o[l, j] = outs[l].cpu().numpy()
            got_e[l, j] = eis[l].cpu().numpy()
        got_x[j] = x_out.float().cpu().numpy()
    for c in st.caches:
        c.check()
    ref_o, ref_e, ref_x = run_stack(cfg, L, steps, pov, dov)
    for l in range(cfg.n_layers):
        assert np.array_equal(got_e[l], ref_e[l]), f"layer {l} evictions differ"
        err = np.abs(got_o[l] - np.stack(ref_o[l]).reshape(steps, b, Hq * d)).max()
        print(f"stack layer {l}: max-abs attention error {err:.3e}")
        assert err <= TOL["bf16"]
    xerr = np.abs(got_x - ref_x).max()
    print(f"stack final hidden state max-abs error {xerr:.3e}")
    # two bf16-rounded projections and residual sums per layer compound: looser bound
    assert xerr <= 5e-2
    st.free()


def test_stack_graph_replay_equals_eager(cuda_device):
    cfg = get_config("q8b_stack", **dict(SMALL_STACK, decode_steps=12))
    L = gen.prompt_lengths(cfg)
    a, g = build_stack(cfg, cuda_device), build_stack(cfg, cuda_device)
    prefill_stack(a, cfg, L, cuda_device)
    prefill_stack(g, cfg, L, cuda_device)
    xs = gen.decode_hidden(cfg, L, 0, cfg.decode_steps, device=cuda_device)
    x_in = torch.empty((cfg.batch, cfg.hidden), dtype=torch.bfloat16, device=cuda_device)
    x_out_g = torch.empty_like(x_in)
    x_out_a = torch.empty_like(x_in)
    g.capture(x_in, x_out_g)
    for j in range(cfg.decode_steps):
        a.step(xs[j], x_out_a)
        x_in.copy_(xs[j])
        g.graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(x_out_a, x_out_g), f"step {j}"
    assert a.caches[0].lengths() == g.caches[0].lengths()
    a.free()
    g.free()
