"""fp64 oracle of the multi-layer decode stack (projections + KVpop layers).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

The stack is the workload's Qwen3-8B-shaped decode model, attention and
eviction only: per layer ``q, k, v = x W_{q,k,v}``, one KVpop cache step per KV
head (Sec. 3, App. C; ``HeadCache``), then the residual update
``x <- x + o W_o``; no norms and no MLP blocks.  The projections are plain
matrix products of the workload, not part of the paper's method.

Rounding points.  The workload is a bf16 model: its weights are bf16 and every
activation it materialises between two operations is a bf16 tensor -- the
projected q, k and v, the attention output that enters W_o, the projection
result y, and the residual stream x.  Each product and sum is evaluated here in
fp64 on those bf16 values and rounded to bf16 (round to nearest even) where the
model stores it; the KVpop layer itself runs in fp64 on the bf16 q, k, v like
every other oracle path.  Evaluating a product exactly and rounding once is the
definition of a correctly rounded bf16 result, so these points follow from the
model's storage type alone.

Each KV head of each layer is an independent ``HeadCache``.
"""
from __future__ import annotations

from typing import Optional, Sequence

import numpy as np
import torch

from workload import gen
from .kvpop_oracle import OracleParams, prefill_head


def _bf16(x: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.asarray(x, dtype=np.float64)).to(torch.bfloat16).to(torch.float64).numpy()


def _f64(t) -> np.ndarray:
    if isinstance(t, np.ndarray):
        return t.astype(np.float64)
    return t.to(torch.float64).numpy()


def project(x: np.ndarray, W: np.ndarray) -> np.ndarray:
    """A bf16 projection of bf16 activations: bf16(x W), the product exact in fp64."""
    return _bf16(x @ W)


def residual_update(x: np.ndarray, o: np.ndarray, Wo: np.ndarray) -> np.ndarray:
    """x_{l+1} = bf16(x_l + bf16(bf16(o_l) W_o)): the attention output is stored in
    bf16 before the output projection, the projection result is stored in bf16, and
    so is the residual sum."""
    y = project(_bf16(o), Wo)
    return _bf16(x + y)


def layer_weights(cfg, weights: Optional[Sequence[dict]]):
    """The layers in model order: ``weights[l]`` if given, else the seeded weights."""
    if weights is None:
        weights = [gen.stack_weights(cfg, l) for l in range(cfg.n_layers)]
    return list(weights)


def run_stack(cfg, lengths, n_steps, prefill_overrides=None, decode_overrides=None,
              weights: Optional[Sequence[dict]] = None):
    """Prefill every layer from its seeded prompt hidden states, then run ``n_steps``
    decode steps of the whole stack on the seeded decode hidden states.

    ``weights[l]`` (optional) holds ``Wq, Wk, Wv, Wo`` (bf16 values, torch or numpy)
    and the scorer arrays ``W1, b1, w2, b2``; by default they come from
    ``workload.gen.stack_weights``.  Returns ``(outputs, evict, finals)``:
    ``outputs[l][step]`` -> ``[b][Hq][d]`` fp64 attention output of layer l,
    ``evict[l]`` -> ``[steps][b][H][2]`` (slot, evicted position), ``finals``
    -> ``[steps][b][hidden]`` the stack's output hidden state.
    """
    b, H, G, d, hid = cfg.batch, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim, cfg.hidden
    Hq = H * G
    layers = layer_weights(cfg, weights)
    W = [{k: _f64(v) for k, v in L.items() if k in ("Wq", "Wk", "Wv", "Wo")} for L in layers]
    caches = []
    for l, L in enumerate(layers):
        row = []
        sc = {k: _f64(L[k]) for k in ("W1", "b1", "w2", "b2")}
        for bb in range(b):
            P = lengths[bb]
            X = _f64(gen.prompt_hidden(cfg, l, bb, 1, 0, P))[0]               # [P][hid]
            Q = project(X, W[l]["Wq"]).reshape(P, Hq, d).transpose(1, 0, 2)    # [Hq][P][d]
            K = project(X, W[l]["Wk"]).reshape(P, H, d).transpose(1, 0, 2)
            V = project(X, W[l]["Wv"]).reshape(P, H, d).transpose(1, 0, 2)
            heads = []
            for h in range(H):
                p = OracleParams.for_head(sc["W1"], sc["b1"], sc["w2"], sc["b2"],
                                          np.zeros(H, dtype=np.float32), h,
                                          cfg.budget_B, cfg.delay_D, cfg.n_sink)
                ov = None if prefill_overrides is None else _f64(prefill_overrides[l][bb, h, :P])
                heads.append(prefill_head(p, Q[h * G:(h + 1) * G], K[h], V[h], d, G, ov))
            row.append(heads)
        caches.append(row)
    xs = _f64(gen.decode_hidden(cfg, lengths, 0, n_steps))                      # [steps][b][hid]
    outputs = [[None] * n_steps for _ in range(len(layers))]
    evict = [np.zeros((n_steps, b, H, 2), dtype=np.int64) for _ in range(len(layers))]
    finals = np.zeros((n_steps, b, hid))
    for j in range(n_steps):
        x = xs[j]
        for l in range(len(layers)):
            q = project(x, W[l]["Wq"]).reshape(b, Hq, d)
            k = project(x, W[l]["Wk"]).reshape(b, H, d)
            v = project(x, W[l]["Wv"]).reshape(b, H, d)
            o = np.zeros((b, Hq, d))
            for bb in range(b):
                for h in range(H):
                    c = caches[l][bb][h]
                    ov = None if decode_overrides is None else float(decode_overrides[l][j, bb, h])
                    slot, ev, _ = c.append(q[bb, h * G:(h + 1) * G], k[bb, h], v[bb, h], ov)
                    evict[l][j, bb, h] = (slot, ev)
                    o[bb, h * G:(h + 1) * G], _, _ = c.attend(q[bb, h * G:(h + 1) * G])
            outputs[l][j] = o
            x = residual_update(x, o.reshape(b, Hq * d), W[l]["Wo"])
        finals[j] = x
    return outputs, evict, finals
