"""fp64 oracle of the multi-layer decode stack (projections + KVpop layers).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).  The projections are the
plain matrix products of the workload (not part of the paper's method); they
are evaluated in fp64 from the same bf16 weights and rounded to bf16 at the
same points as the CUDA stack (q, k, v; the attention output; the output
projection; the residual sum), so that the KVpop layers see matching inputs.
Each KV head of each layer is an independent ``HeadCache`` (Sec. 3, App. C).
"""
from __future__ import annotations

import numpy as np
import torch

from workload import gen
from .kvpop_oracle import OracleParams, prefill_head


def _bf16(x: np.ndarray) -> np.ndarray:
    return torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()


def _f64(t: torch.Tensor) -> np.ndarray:
    return t.to(torch.float64).numpy()


def run_stack(cfg, lengths, n_steps, prefill_overrides=None, decode_overrides=None):
    """Returns (outputs[l][step] -> [b][Hq][d], evict[l] -> [steps][b][H][2], final x [steps][b][hidden])."""
    b, H, G, d, hid = cfg.batch, cfg.n_kv_heads, cfg.q_per_kv, cfg.head_dim, cfg.hidden
    Hq = H * G
    layers = [gen.stack_weights(cfg, l) for l in range(cfg.n_layers)]
    W = [{k: _f64(v) for k, v in L.items() if k in ("Wq", "Wk", "Wv", "Wo")} for L in layers]
    caches = []
    for l, L in enumerate(layers):
        row = []
        for bb in range(b):
            P = lengths[bb]
            X = _f64(gen.prompt_hidden(cfg, l, bb, 1, 0, P))[0]               # [P][hid]
            Q = _bf16(X @ W[l]["Wq"]).reshape(P, Hq, d).transpose(1, 0, 2)     # [Hq][P][d]
            K = _bf16(X @ W[l]["Wk"]).reshape(P, H, d).transpose(1, 0, 2)
            V = _bf16(X @ W[l]["Wv"]).reshape(P, H, d).transpose(1, 0, 2)
            heads = []
            for h in range(H):
                p = OracleParams.for_head(L["W1"].numpy(), L["b1"].numpy(), L["w2"].numpy(),
                                          L["b2"].numpy(), np.zeros(H, dtype=np.float32), h,
                                          cfg.budget_B, cfg.delay_D, cfg.n_sink)
                ov = None if prefill_overrides is None else prefill_overrides[l][bb, h, :P].numpy()
                heads.append(prefill_head(p, Q[h * G:(h + 1) * G], K[h], V[h], d, G, ov))
            row.append(heads)
        caches.append(row)
    xs = _f64(gen.decode_hidden(cfg, lengths, 0, n_steps))                      # [steps][b][hid]
    outputs = [[None] * n_steps for _ in range(cfg.n_layers)]
    evict = [np.zeros((n_steps, b, H, 2), dtype=np.int64) for _ in range(cfg.n_layers)]
    finals = np.zeros((n_steps, b, hid))
    for j in range(n_steps):
        x = xs[j]
        for l in range(cfg.n_layers):
            q = _bf16(x @ W[l]["Wq"]).reshape(b, Hq, d)
            k = _bf16(x @ W[l]["Wk"]).reshape(b, H, d)
            v = _bf16(x @ W[l]["Wv"]).reshape(b, H, d)
            o = np.zeros((b, Hq, d))
            for bb in range(b):
                for h in range(H):
                    c = caches[l][bb][h]
                    ov = None if decode_overrides is None else float(decode_overrides[l][j, bb, h])
                    slot, ev, _ = c.append(q[bb, h * G:(h + 1) * G], k[bb, h], v[bb, h], ov)
                    evict[l][j, bb, h] = (slot, ev)
                    o[bb, h * G:(h + 1) * G], _, _ = c.attend(q[bb, h * G:(h + 1) * G])
            outputs[l][j] = o
            y = _bf16(_bf16(o.reshape(b, Hq * d)) @ W[l]["Wo"])
            x = _bf16(x + y)
        finals[j] = x
    return outputs, evict, finals
