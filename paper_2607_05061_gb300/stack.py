"""Multi-layer decode stack: per layer, Q/K/V projections, a KVpop cache step
through the C ABI, the output projection and the residual add.

This is the workload around the hot path for the Qwen3-8B-shaped stack
(hidden 4096, 32 query / 8 KV heads, d = 128): it reproduces the decode loop
of a dense-attention model whose attention layers are the KVpop caches, with no
norms and no MLP blocks.  The projections are plain bf16 GEMMs run by cuBLAS
(`torch.matmul`, fp32 accumulation); everything KVpop does per layer -- the
delayed scorer, the keep-or-drop decision, the scatter and the attention over
the compressed cache -- runs in `libkvpop.so`.

Rounding points (bf16): q, k, v after their projections; the attention output
before the output projection; the projection result; the residual sum.
"""
from __future__ import annotations

from typing import List, Optional, Sequence

import torch

from .kvpop import KVpopCache


class DecodeStack:
    def __init__(self, layers: Sequence[dict], batch: int, hidden: int, n_kv_heads: int,
                 q_per_kv: int, head_dim: int, budget_B: int, delay_D: int, scorer_hidden: int,
                 n_sink: int = 0, device="cuda"):
        """``layers[l]`` holds bf16 device weights ``Wq [hidden][Hq*d]``, ``Wk``, ``Wv``
        ``[hidden][H*d]``, ``Wo [Hq*d][hidden]`` and fp32 scorer arrays ``W1, b1, w2, b2``
        (optionally ``log_gamma``)."""
        self.layers = list(layers)
        self.b, self.hidden = batch, hidden
        self.H, self.G, self.d = n_kv_heads, q_per_kv, head_dim
        self.Hq = n_kv_heads * q_per_kv
        self.device = torch.device(device)
        self.caches: List[KVpopCache] = [
            KVpopCache(batch, n_kv_heads, q_per_kv, head_dim, budget_B, delay_D, scorer_hidden,
                       torch.bfloat16, L["W1"], L["b1"], L["w2"], L["b2"],
                       log_gamma=L.get("log_gamma"), n_sink=n_sink)
            for L in self.layers]
        dt = torch.bfloat16
        dev = self.device
        # per-step work buffers (static addresses: the step can be captured in a CUDA graph)
        self.q = torch.empty((batch, self.Hq * head_dim), dtype=dt, device=dev)
        self.k = torch.empty((batch, n_kv_heads * head_dim), dtype=dt, device=dev)
        self.v = torch.empty((batch, n_kv_heads * head_dim), dtype=dt, device=dev)
        self.o = torch.empty((batch, self.Hq * head_dim), dtype=torch.float32, device=dev)
        self.o_bf = torch.empty((batch, self.Hq * head_dim), dtype=dt, device=dev)
        self.y = torch.empty((batch, hidden), dtype=dt, device=dev)
        self.x = [torch.empty((batch, hidden), dtype=dt, device=dev) for _ in range(2)]
        self.graph = None

    # ------------------------------------------------------------------ prefill
    def prefill_layer(self, l: int, X: torch.Tensor, lengths: Sequence[int], first_seq: int = 0,
                      override=None):
        """Compress layer l's prompt for ``len(lengths)`` sequences from their hidden states
        ``X [n][Pmax][hidden]`` (bf16): Q/K/V = bf16(X W), reshaped head-major."""
        L = self.layers[l]
        n, Pm, _ = X.shape
        Xf = X.reshape(n * Pm, self.hidden)

        def proj(W, heads):
            t = torch.matmul(Xf, W).view(n, Pm, heads, self.d)
            return t.permute(0, 2, 1, 3).contiguous()
        Q = proj(L["Wq"], self.Hq)
        K = proj(L["Wk"], self.H)
        V = proj(L["Wv"], self.H)
        self.caches[l].prefill(Q, K, V, lengths, first_seq=first_seq, override=override)

    # ------------------------------------------------------------------ decode
    def _step_into(self, x_in: torch.Tensor, x_out: torch.Tensor, overrides=None,
                   evict_info=None, outputs=None):
        x = x_in
        for l, (L, cache) in enumerate(zip(self.layers, self.caches)):
            torch.matmul(x, L["Wq"], out=self.q)
            torch.matmul(x, L["Wk"], out=self.k)
            torch.matmul(x, L["Wv"], out=self.v)
            ov = None if overrides is None else overrides[l]
            ei = None if evict_info is None else evict_info[l]
            cache.step(self.q, self.k, self.v, self.o, override=ov, evict_info=ei)
            if outputs is not None:
                outputs[l].copy_(self.o)
            self.o_bf.copy_(self.o)
            torch.matmul(self.o_bf, L["Wo"], out=self.y)
            nxt = self.x[l % 2] if l + 1 < len(self.layers) else x_out
            torch.add(x, self.y, out=nxt)
            x = nxt
        return x_out

    def step(self, x_in: torch.Tensor, x_out: Optional[torch.Tensor] = None, overrides=None,
             evict_info=None, outputs=None) -> torch.Tensor:
        """One decode step of the whole stack on hidden states ``x_in [b][hidden]``."""
        if x_out is None:
            x_out = torch.empty_like(x_in)
        return self._step_into(x_in, x_out, overrides, evict_info, outputs)

    def capture(self, x_in: torch.Tensor, x_out: torch.Tensor):
        """Capture one step (all layers) into a CUDA graph on static ``x_in`` / ``x_out``."""
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(s):
            with torch.cuda.graph(g, stream=s):
                self._step_into(x_in, x_out)
        torch.cuda.current_stream().wait_stream(s)
        self.graph = g
        return g

    def free(self):
        for c in self.caches:
            c.free()
