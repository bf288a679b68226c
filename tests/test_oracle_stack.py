"""Pins of the fp64 decode-stack oracle (``oracle/stack.py``).

The stack oracle is checked against things fixed outside it:

* its per-layer attention delegates to the single-head oracle on the right head
  slices (identity projections put each head's q / k / v in known columns of
  the hidden state; with W_o = 0 the residual stream passes through unchanged);
* with a budget that covers the whole context, KVpop keeps every token, so each
  layer is dense causal attention -- checked against torch's fp64
  scaled_dot_product_attention over the projected history -- and the layers
  chain through the residual update x + o W_o in model order, with the bf16
  storage points of a bf16 model;
* planted mistakes in the oracle (residual dropped, layers in the wrong order,
  the attention output used in W_o before its bf16 rounding, q left unrounded)
  each fail the dense pin.
"""
import numpy as np
import pytest
import torch

from oracle import OracleParams, prefill_head
from oracle import stack as ostack
from workload import gen, get_config

TINY_STACK = dict(batch=2, n_kv_heads=2, q_per_kv=2, head_dim=16, hidden=64, prompt_len=24,
                  delay_D=4, scorer_hidden=8, decode_steps=6, n_layers=2)


def bf16(a):
    return torch.as_tensor(a, dtype=torch.float64).to(torch.bfloat16).to(torch.float64)


def t64(a):
    return a.double() if isinstance(a, torch.Tensor) else torch.as_tensor(a, dtype=torch.float64)


def identity_weights(cfg):
    """Wq = I, Wk / Wv select the first / last H*d hidden columns, Wo = 0 (bf16-exact)."""
    hid, Hd = cfg.hidden, cfg.n_kv_heads * cfg.head_dim
    assert hid == cfg.n_q_heads * cfg.head_dim
    eye = np.eye(hid)
    L = gen.stack_weights(cfg, 0)
    return [dict(Wq=eye, Wk=eye[:, :Hd], Wv=eye[:, hid - Hd:], Wo=np.zeros((hid, hid)),
                 W1=L["W1"], b1=L["b1"], w2=L["w2"], b2=L["b2"])]


def test_stack_layer_is_the_head_oracle_on_its_head_slices():
    """One layer, identity projections, W_o = 0, a budget smaller than the context
    (evictions happen): every head's output and eviction equal a HeadCache driven
    directly on that head's columns, and the stack returns its input unchanged."""
    cfg = get_config("q8b_stack", **dict(TINY_STACK, n_layers=1, budget_B=6))
    b, H, G, d = cfg.batch, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim
    Hd = H * d
    L = gen.prompt_lengths(cfg)
    steps = cfg.decode_steps
    w = identity_weights(cfg)
    outs, evict, finals = ostack.run_stack(cfg, L, steps, weights=w)
    xs = gen.decode_hidden(cfg, L, 0, steps).double().numpy()
    assert np.array_equal(finals, xs)
    n_evicted = 0
    for bb in range(b):
        X = gen.prompt_hidden(cfg, 0, bb, 1, 0, L[bb])[0].double().numpy()      # [P][hid]
        for h in range(H):
            p = OracleParams.for_head(w[0]["W1"].numpy(), w[0]["b1"].numpy(), w[0]["w2"].numpy(),
                                      w[0]["b2"].numpy(), np.zeros(H), h, cfg.budget_B, cfg.delay_D)
            qcols = slice(h * G * d, (h + 1) * G * d)
            kcols = slice(h * d, (h + 1) * d)
            vcols = slice(cfg.hidden - Hd + h * d, cfg.hidden - Hd + (h + 1) * d)
            Q = X[:, qcols].reshape(L[bb], G, d).transpose(1, 0, 2)
            c = prefill_head(p, Q, X[:, kcols], X[:, vcols], d, G)
            for j in range(steps):
                x = xs[j, bb]
                slot, ev, _ = c.append(x[qcols].reshape(G, d), x[kcols], x[vcols])
                assert (slot, ev) == tuple(evict[0][j, bb, h])
                n_evicted += ev >= 0
                o, _, _ = c.attend(x[qcols].reshape(G, d))
                assert np.array_equal(outs[0][j][bb, h * G:(h + 1) * G], o)
    assert n_evicted > 0


def dense_stack_reference(cfg, L, steps, weights):
    """The stack with dense causal attention, evaluated with torch fp64 SDPA.

    Per layer: q, k, v = bf16(x W); o = SDPA(q, K_hist, V_hist) over the layer's
    projected prompt plus the decode tokens so far (GQA: query head h*G+g reads KV
    head h); x <- bf16(x + bf16(bf16(o) W_o)).  Returns (outputs [l][step][b][Hq][d],
    finals [step][b][hidden])."""
    b, H, G, d, hid = cfg.batch, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim, cfg.hidden
    Hq = H * G
    Wt = [{k: t64(w[k]) for k in ("Wq", "Wk", "Wv", "Wo")} for w in weights]
    hist = []                                   # hist[l][bb] = [K [H][t][d], V]
    for l in range(cfg.n_layers):
        row = []
        for bb in range(b):
            X = gen.prompt_hidden(cfg, l, bb, 1, 0, L[bb])[0].double()
            K = bf16(X @ Wt[l]["Wk"]).view(L[bb], H, d).transpose(0, 1)
            V = bf16(X @ Wt[l]["Wv"]).view(L[bb], H, d).transpose(0, 1)
            row.append([K, V])
        hist.append(row)
    xs = gen.decode_hidden(cfg, L, 0, steps).double()
    outs = np.zeros((cfg.n_layers, steps, b, Hq, d))
    finals = np.zeros((steps, b, hid))
    for j in range(steps):
        x = xs[j]
        for l in range(cfg.n_layers):
            q = bf16(x @ Wt[l]["Wq"]).view(b, Hq, d)
            k = bf16(x @ Wt[l]["Wk"]).view(b, H, d)
            v = bf16(x @ Wt[l]["Wv"]).view(b, H, d)
            o = torch.zeros(b, Hq, d, dtype=torch.float64)
            for bb in range(b):
                hist[l][bb][0] = torch.cat([hist[l][bb][0], k[bb][:, None]], dim=1)
                hist[l][bb][1] = torch.cat([hist[l][bb][1], v[bb][:, None]], dim=1)
                Kh = hist[l][bb][0].repeat_interleave(G, dim=0)            # [Hq][t][d]
                Vh = hist[l][bb][1].repeat_interleave(G, dim=0)
                o[bb] = torch.nn.functional.scaled_dot_product_attention(
                    q[bb][:, None], Kh, Vh)[:, 0]
            outs[l, j] = o.numpy()
            x = bf16(x + bf16(bf16(o.reshape(b, Hq * d)) @ Wt[l]["Wo"]))
        finals[j] = x.numpy()
    return outs, finals


def dense_pin(cfg, L, steps, weights):
    """(max |o - SDPA|, number of final hidden elements that differ) for the oracle."""
    o_ref, x_ref = dense_stack_reference(cfg, L, steps, weights)
    outs, evict, finals = ostack.run_stack(cfg, L, steps, weights=weights)
    o = np.stack([np.stack(outs[l]) for l in range(cfg.n_layers)])
    for e in evict:            # every token is kept: nothing is ever evicted or dropped
        assert (e[..., 1] == -1).all() and (e[..., 0] >= 0).all()
    return float(np.abs(o - o_ref).max()), int((finals != x_ref).sum())


def dense_case():
    steps = TINY_STACK["decode_steps"]
    cfg = get_config("q8b_stack", **dict(TINY_STACK, budget_B=TINY_STACK["prompt_len"] + steps))
    weights = [gen.stack_weights(cfg, l) for l in range(cfg.n_layers)]
    return cfg, gen.prompt_lengths(cfg), steps, weights


def test_budget_covering_context_is_a_dense_attention_stack():
    cfg, L, steps, weights = dense_case()
    oerr, xbad = dense_pin(cfg, L, steps, weights)
    assert oerr < 1e-12
    assert xbad == 0


def _planted_no_residual(x, o, Wo):
    return ostack.project(ostack._bf16(o), Wo)


def _planted_unrounded_o(x, o, Wo):
    return ostack._bf16(x + ostack.project(o, Wo))


@pytest.mark.parametrize("mistake", ["residual dropped", "layers reversed",
                                     "o unrounded before W_o", "projections unrounded"])
def test_dense_pin_catches_planted_mistakes(monkeypatch, mistake):
    cfg, L, steps, weights = dense_case()
    if mistake == "residual dropped":
        monkeypatch.setattr(ostack, "residual_update", _planted_no_residual)
    elif mistake == "layers reversed":
        orig = ostack.layer_weights
        monkeypatch.setattr(ostack, "layer_weights", lambda c, w: orig(c, w)[::-1])
    elif mistake == "o unrounded before W_o":
        monkeypatch.setattr(ostack, "residual_update", _planted_unrounded_o)
    else:
        monkeypatch.setattr(ostack, "project", lambda x, W: x @ W)
    oerr, xbad = dense_pin(cfg, L, steps, weights)
    assert oerr >= 1e-12 or xbad > 0, mistake
