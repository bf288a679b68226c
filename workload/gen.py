"""Counter-based, device-independent seeded generator for synthetic inputs.

Every value is a pure function of ``(seed, stream, flat index)``:

    h   = pcg(pcg(lo32(idx) ^ k1) ^ pcg(hi32(idx) ^ k2))      k1, k2 from (seed, stream)
    val = NORMAL_TABLE[h >> 16]

``pcg`` is the 32-bit PCG-RXS-M-XS hash of Jarzynski & Olano, "Hash Functions
for GPU Rendering" (JCGT 9(3), 2020).  It is evaluated with int64 torch ops
whose products stay below 2**63, so the CPU and CUDA evaluations give the same
bits.  ``NORMAL_TABLE`` holds the standard-normal quantiles at the 65536
midpoints ``(i + 0.5) / 65536``: a 16-bit discretised N(0, 1) with tails cut at
about 4.3 sigma.  Casting to bf16 is IEEE round-to-nearest-even on both
devices, so the CUDA path and the oracle see identical inputs without either
one producing the other's.

Token streams have one index space per (sequence, head): position ``t`` of
head ``h`` of sequence ``b`` has flat index ``((b * heads + h) * LP + t) * d + i``
with ``LP = 2**20`` positions.  Prompt and decode tokens are slices of the same
stream, so a decode step at position ``p`` takes the stream's token ``p``.
"""
from __future__ import annotations

import functools
from typing import Optional, Sequence

import numpy as np
import torch

M32 = 0xFFFFFFFF
LP = 1 << 20            # positions per (sequence, head) stream

STREAM_K, STREAM_V, STREAM_Q = 1, 2, 3
STREAM_W1, STREAM_W2 = 10, 11
STREAM_MLSTM = 12
STREAM_LEN, STREAM_OUTLIER = 20, 21
STREAM_HIDDEN, STREAM_WPROJ, STREAM_DECODE_HIDDEN = 40, 50, 60
LAYER_STRIDE = 1000     # stream offset between layers of a stack

_CHUNK = 1 << 24        # elements generated per torch pass


def _pcg_int(x: int) -> int:
    s = (x * 747796405 + 2891336453) & M32
    w = (((s >> ((s >> 28) + 4)) ^ s) * 277803737) & M32
    return (w >> 22) ^ w


def _pcg(x: torch.Tensor) -> torch.Tensor:
    s = (x * 747796405 + 2891336453) & M32
    w = ((torch.bitwise_right_shift(s, (s >> 28) + 4) ^ s) * 277803737) & M32
    return (w >> 22) ^ w


def _keys(seed: int, stream: int):
    k1 = _pcg_int((_pcg_int(seed & M32) ^ (stream * 0x9E3779B1)) & M32)
    k2 = _pcg_int(k1 ^ 0x85EBCA6B)
    return k1, k2


@functools.lru_cache(maxsize=None)
def _table_cpu() -> torch.Tensor:
    from scipy.special import ndtri
    mid = (np.arange(65536, dtype=np.float64) + 0.5) / 65536.0
    return torch.from_numpy(ndtri(mid).astype(np.float32))


_TABLES = {}


def _table(device) -> torch.Tensor:
    key = str(device)
    if key not in _TABLES:
        _TABLES[key] = _table_cpu().to(device)
    return _TABLES[key]


def _hash_flat(seed: int, stream: int, flat: torch.Tensor) -> torch.Tensor:
    k1, k2 = _keys(seed, stream)
    lo = flat & M32
    hi = flat >> 32
    return _pcg(_pcg(lo ^ k1) ^ _pcg(hi ^ k2))


def normal_values(seed: int, stream: int, flat: torch.Tensor) -> torch.Tensor:
    """fp32 N(0,1)-distributed values for int64 flat indices (any device)."""
    h = _hash_flat(seed, stream, flat)
    return _table(flat.device)[h >> 16]


def uniform_u32(seed: int, stream: int, flat: torch.Tensor) -> torch.Tensor:
    return _hash_flat(seed, stream, flat)


def _rows(seed, stream, row_offsets: torch.Tensor, row_len: int, out: torch.Tensor,
          scale: Optional[torch.Tensor] = None):
    """Fill ``out`` ([n_rows, row_len]) with values at flat = row_offsets[r] + j."""
    dev = out.device
    n = row_offsets.numel()
    rows_per = max(1, _CHUNK // row_len)
    col = torch.arange(row_len, dtype=torch.int64, device=dev)
    for r0 in range(0, n, rows_per):
        r1 = min(n, r0 + rows_per)
        flat = row_offsets[r0:r1, None] + col[None, :]
        v = normal_values(seed, stream, flat)
        if scale is not None:
            v = v * scale
        out[r0:r1] = v.to(out.dtype)
    return out


def torch_dtype(kv_dtype: str):
    return torch.float32 if kv_dtype == "f32" else torch.bfloat16


def outlier_channels(cfg) -> list:
    """Key channels scaled by ``cfg.outlier_scale`` (same for every head and layer)."""
    if cfg.n_outlier <= 0:
        return []
    k1, _ = _keys(cfg.seed, STREAM_OUTLIER)
    h = [_pcg_int(k1 ^ i) for i in range(cfg.head_dim)]
    order = sorted(range(cfg.head_dim), key=lambda i: (h[i], i))
    return sorted(order[: cfg.n_outlier])


def _key_scale(cfg, device):
    ch = outlier_channels(cfg)
    if not ch:
        return None
    s = torch.ones(cfg.head_dim, dtype=torch.float32, device=device)
    s[ch] = cfg.outlier_scale
    return s


def prompt_lengths(cfg) -> list:
    """Per-sequence prompt lengths (all ``cfg.prompt_len`` unless ragged)."""
    if cfg.ragged is None:
        return [cfg.prompt_len] * cfg.batch
    lo, hi = cfg.ragged
    k1, _ = _keys(cfg.seed, STREAM_LEN)
    return [lo + (_pcg_int(k1 ^ b) % (hi - lo + 1)) for b in range(cfg.batch)]


def _token_tensor(cfg, stream, n_heads_total, b0, nb, heads, t0, nt, device, layer, scale):
    d = cfg.head_dim
    heads = list(range(n_heads_total)) if heads is None else list(heads)
    out = torch.empty((nb, len(heads), nt, d), dtype=torch_dtype(cfg.kv_dtype), device=device)
    bs = torch.arange(b0, b0 + nb, dtype=torch.int64, device=device)
    hs = torch.tensor(heads, dtype=torch.int64, device=device)
    ts = torch.arange(t0, t0 + nt, dtype=torch.int64, device=device)
    st = stream + layer * LAYER_STRIDE
    view = out.view(nb, len(heads), nt * d)
    for bi in range(nb):
        for hi_, h in enumerate(heads):
            base = ((bs[bi] * n_heads_total + hs[hi_]) * LP + ts) * d
            _rows(cfg.seed, st, base, d, view[bi, hi_].view(nt, d), scale)
    return out


def kv_tokens(cfg, which: str, b0: int = 0, nb: Optional[int] = None, t0: int = 0,
              nt: int = 1, heads: Optional[Sequence[int]] = None, device="cpu",
              layer: int = 0) -> torch.Tensor:
    """K or V tokens ``[nb][len(heads)][nt][d]`` at positions t0..t0+nt-1."""
    nb = cfg.batch - b0 if nb is None else nb
    stream = STREAM_K if which == "k" else STREAM_V
    scale = _key_scale(cfg, device) if which == "k" else None
    return _token_tensor(cfg, stream, cfg.n_kv_heads, b0, nb, heads, t0, nt, device, layer, scale)


def q_tokens(cfg, b0: int = 0, nb: Optional[int] = None, t0: int = 0, nt: int = 1,
             heads: Optional[Sequence[int]] = None, device="cpu", layer: int = 0) -> torch.Tensor:
    """Query tokens ``[nb][len(heads)][nt][d]`` (query-head index space)."""
    nb = cfg.batch - b0 if nb is None else nb
    return _token_tensor(cfg, STREAM_Q, cfg.n_q_heads, b0, nb, heads, t0, nt, device, layer, None)


def decode_inputs(cfg, lengths: Sequence[int], step0: int, nsteps: int, device="cpu",
                  layer: int = 0, b0: int = 0):
    """Per-step decode inputs at positions ``lengths[b] + step``.

    Returns ``q [nsteps][nb][H*G][d]``, ``k, v [nsteps][nb][H][d]`` where nb = len(lengths)
    and sequence index ``b0 + i`` draws from its own stream.
    """
    d = cfg.head_dim
    nb = len(lengths)
    dt = torch_dtype(cfg.kv_dtype)
    L = torch.tensor(list(lengths), dtype=torch.int64, device=device)
    steps = torch.arange(step0, step0 + nsteps, dtype=torch.int64, device=device)
    bs = torch.arange(b0, b0 + nb, dtype=torch.int64, device=device)
    pos = L[None, :] + steps[:, None]                      # [nsteps][nb]
    out = []
    for stream, nh, scale in ((STREAM_Q, cfg.n_q_heads, None),
                              (STREAM_K, cfg.n_kv_heads, _key_scale(cfg, device)),
                              (STREAM_V, cfg.n_kv_heads, None)):
        hs = torch.arange(nh, dtype=torch.int64, device=device)
        base = ((bs[None, :, None] * nh + hs[None, None, :]) * LP + pos[:, :, None]) * d
        t = torch.empty((nsteps, nb, nh, d), dtype=dt, device=device)
        _rows(cfg.seed, stream + layer * LAYER_STRIDE, base.reshape(-1), d,
              t.view(-1, d), scale)
        out.append(t)
    return tuple(out)


def scorer_weights(cfg, layer: int = 0):
    """Random-init scorer MLP ``3d -> F (GELU) -> 1`` per KV head, fp32 (CPU tensors).

    Xavier-normal weights (std = sqrt(2 / (fan_in + fan_out))) and zero biases.
    Returns ``W1 [H][3d][F]``, ``b1 [H][F]``, ``w2 [H][F]``, ``b2 [H]``, ``log_gamma [H]``.
    """
    H, F, I = cfg.n_kv_heads, cfg.scorer_hidden, cfg.scorer_in
    st = layer * LAYER_STRIDE
    flat1 = torch.arange(H * I * F, dtype=torch.int64)
    W1 = normal_values(cfg.seed, STREAM_W1 + st, flat1).view(H, I, F) * np.float32(np.sqrt(2.0 / (I + F)))
    flat2 = torch.arange(H * F, dtype=torch.int64)
    w2 = normal_values(cfg.seed, STREAM_W2 + st, flat2).view(H, F) * np.float32(np.sqrt(2.0 / (F + 1)))
    b1 = torch.zeros(H, F, dtype=torch.float32)
    b2 = torch.zeros(H, dtype=torch.float32)
    lg = torch.full((H,), float(cfg.log_gamma), dtype=torch.float32)
    return W1.contiguous(), b1, w2.contiguous(), b2, lg


def uniform_scores(seed: int, stream: int, shape, device="cpu", levels: Optional[int] = None):
    """fp32 scores for injected-score tests.

    With ``levels`` the scores take only ``levels`` distinct values (to plant ties).
    """
    n = int(np.prod(shape))
    flat = torch.arange(n, dtype=torch.int64, device=device)
    if levels is None:
        v = normal_values(seed, stream, flat)
    else:
        v = (uniform_u32(seed, stream, flat) % levels).to(torch.float32) * 0.25 - 1.0
    return v.view(*shape)


# ---------------------------------------------------------------------- projection stack
def stack_weights(cfg, layer: int, device="cpu") -> dict:
    """bf16 projections of one layer, N(0, 1/hidden): ``Wq [hidden][Hq*d]``, ``Wk``, ``Wv``
    ``[hidden][H*d]``, ``Wo [Hq*d][hidden]``; plus that layer's fp32 scorer (CPU)."""
    hid, d = cfg.hidden, cfg.head_dim
    shapes = {"Wq": (hid, cfg.n_q_heads * d), "Wk": (hid, cfg.n_kv_heads * d),
              "Wv": (hid, cfg.n_kv_heads * d), "Wo": (cfg.n_q_heads * d, hid)}
    out = {}
    scale = torch.tensor(1.0 / np.sqrt(hid), dtype=torch.float32, device=device)
    for m, (name, shp) in enumerate(shapes.items()):
        n = shp[0] * shp[1]
        t = torch.empty((n,), dtype=torch.bfloat16, device=device)
        flat = torch.arange(n, dtype=torch.int64, device=device)
        for c0 in range(0, n, _CHUNK):
            c1 = min(n, c0 + _CHUNK)
            t[c0:c1] = (normal_values(cfg.seed, STREAM_WPROJ + m + layer * LAYER_STRIDE,
                                      flat[c0:c1]) * scale).to(torch.bfloat16)
        out[name] = t.view(*shp)
    W1, b1, w2, b2, lg = scorer_weights(cfg, layer)
    out.update(W1=W1, b1=b1, w2=w2, b2=b2)
    if cfg.log_gamma != 0.0:
        out["log_gamma"] = lg
    return out


def prompt_hidden(cfg, layer: int, b0: int, nb: int, t0: int, nt: int, device="cpu") -> torch.Tensor:
    """Prompt hidden states of one layer ``[nb][nt][hidden]`` bf16, N(0, 1)."""
    hid = cfg.hidden
    out = torch.empty((nb, nt, hid), dtype=torch.bfloat16, device=device)
    ts = torch.arange(t0, t0 + nt, dtype=torch.int64, device=device)
    for i in range(nb):
        base = ((b0 + i) * LP + ts) * hid
        _rows(cfg.seed, STREAM_HIDDEN + layer * LAYER_STRIDE, base, hid, out[i])
    return out


def decode_hidden(cfg, lengths: Sequence[int], step0: int, nsteps: int, device="cpu") -> torch.Tensor:
    """Input hidden state of every decode step ``[nsteps][b][hidden]`` bf16, N(0, 1)."""
    hid = cfg.hidden
    L = torch.tensor(list(lengths), dtype=torch.int64, device=device)
    steps = torch.arange(step0, step0 + nsteps, dtype=torch.int64, device=device)
    bs = torch.arange(len(lengths), dtype=torch.int64, device=device)
    base = ((bs[None, :] * LP + L[None, :] + steps[:, None]) * hid).reshape(-1)
    out = torch.empty((nsteps, len(lengths), hid), dtype=torch.bfloat16, device=device)
    _rows(cfg.seed, STREAM_DECODE_HIDDEN, base, hid, out.view(-1, hid))
    return out


def mlstm_weights(cfg, layer: int = 0) -> dict:
    """Random-init stateful mLSTM scorer per KV head (fp32, CPU tensors).

    Xavier-normal W_q, W_k, W_v [H][2d][d/2] and a [H][d/2]; gate weights
    w_i, w_f [H][2d] ~ N(0, 1/(2d)); b_i = 0 and b_f = 3 (a forget gate near 0.95,
    i.e. a memory of a few dozen tokens); b = 0.
    """
    H, d = cfg.n_kv_heads, cfg.head_dim
    n2, hh = 2 * d, d // 2
    st = STREAM_MLSTM + layer * LAYER_STRIDE
    out = {}
    off = 0

    def draw(shape, std):
        nonlocal off
        n = int(np.prod(shape))
        v = normal_values(cfg.seed, st, torch.arange(off, off + n, dtype=torch.int64))
        off += n
        return (v * np.float32(std)).view(*shape).contiguous()
    xav = np.sqrt(2.0 / (n2 + hh))
    out["Wq"] = draw((H, n2, hh), xav)
    out["Wk"] = draw((H, n2, hh), xav)
    out["Wv"] = draw((H, n2, hh), xav)
    out["wi"] = draw((H, n2), 1.0 / np.sqrt(n2))
    out["wf"] = draw((H, n2), 1.0 / np.sqrt(n2))
    out["a"] = draw((H, hh), np.sqrt(2.0 / (hh + 1)))
    out["bi"] = torch.zeros(H)
    out["bf"] = torch.full((H,), 3.0)
    out["b"] = torch.zeros(H)
    if cfg.log_gamma != 0.0:
        out["log_gamma"] = torch.full((H,), float(cfg.log_gamma))
    return out
