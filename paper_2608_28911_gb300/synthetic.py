"""Seeded synthetic inputs shaped like the paper's KV caches.

This module only draws random numbers; it holds none of SemKV's arithmetic, so
both the GPU library's tests/bench and the CPU oracle may consume what it makes.

The paper's workloads (LongBench prompts run through Llama-3.1-8B / Mistral-7B,
Sec. 4.1) are not available here; these tensors stand in for them with the real
KV shape (8 KV heads, head_dim 128, 32 query heads, Sec. 4.5) and:
  - K, V: fp16 N(0,1) with 4 outlier channels per (layer, KV head) scaled by 8;
  - q: fp16 N(0,1);
  - scores: float32(Zipf(1.1)) per (sequence, token): integer-valued with heavy
    ties, which exercises the tie rule of the top-r selection;
  - signs: +-1 per (layer, KV head, dim) for the TurboQuant-style rotation;
  - rotations: a Haar-random orthogonal Q per (layer, KV head) (QR of a Gaussian
    matrix with the signs of R's diagonal taken into Q), stored as fp16 of sqrt(128) Q.
Streams: numpy PCG64 seeded with seed*1000 + {0 K, 1 V, 2 q, 3 scores, 4 signs,
5 outlier channels, 6 rotations} + 10000*layer, so a many-layer cache is reproducible
layer by layer.
"""
from __future__ import annotations

import numpy as np

HEAD_DIM = 128
STREAM_K, STREAM_V, STREAM_Q, STREAM_SCORES, STREAM_SIGNS, STREAM_OUTLIERS, STREAM_ROT = range(7)


def _rng(seed: int, stream: int, layer: int = 0) -> np.random.Generator:
    return np.random.default_rng(seed * 1000 + stream + 10000 * layer)


def kv_layer(seed: int, layer: int, batch: int, kv_heads: int, T: int,
             outliers: int = 4, factor: float = 8.0):
    """K and V of one layer: float16 arrays [batch][kv_heads][T][128]."""
    ro = _rng(seed, STREAM_OUTLIERS, layer)
    chans = [ro.choice(HEAD_DIM, outliers, replace=False) for _ in range(kv_heads)]
    out = []
    for stream in (STREAM_K, STREAM_V):
        r = _rng(seed, stream, layer)
        x = r.standard_normal((batch, kv_heads, T, HEAD_DIM), dtype=np.float32)
        for h in range(kv_heads):
            x[:, h, :, chans[h]] *= factor
        out.append(x.astype(np.float16))
    return out[0], out[1]


def kv(seed: int, batch: int, layers: int, kv_heads: int, T: int, **kw):
    """K and V of every layer: float16 [batch][layers][kv_heads][T][128]."""
    ks, vs = zip(*(kv_layer(seed, l, batch, kv_heads, T, **kw) for l in range(layers)))
    return np.stack(ks, axis=1), np.stack(vs, axis=1)


def queries(seed: int, batch: int, q_heads: int, step: int = 0) -> np.ndarray:
    """Decode queries: float16 [batch][q_heads][128] ~ N(0,1)."""
    r = _rng(seed, STREAM_Q, step)
    return r.standard_normal((batch, q_heads, HEAD_DIM), dtype=np.float32).astype(np.float16)


def scores_zipf(seed: int, batch: int, T: int, a: float = 1.1, offset: int = 0) -> np.ndarray:
    """Importance scores float32 [batch][T] drawn from Zipf(a) (ties are common)."""
    r = _rng(seed, STREAM_SCORES, offset)
    return r.zipf(a, size=(batch, T)).astype(np.float32)


def scores_tiefree(seed: int, batch: int, T: int, a: float = 1.1) -> np.ndarray:
    """Zipf-shaped scores without ties: (pi_i + 1)^-a for a random permutation pi."""
    r = _rng(seed, STREAM_SCORES)
    out = np.empty((batch, T), np.float32)
    for b in range(batch):
        out[b] = (r.permutation(T) + 1.0) ** (-a)
    return out


def signs(seed: int, layers: int, kv_heads: int) -> np.ndarray:
    """+-1 int8 [layers][kv_heads][128] for the randomized Hadamard rotation."""
    r = _rng(seed, STREAM_SIGNS)
    return np.where(r.random((layers, kv_heads, HEAD_DIM)) < 0.5, -1, 1).astype(np.int8)


def rotations(seed: int, layers: int, kv_heads: int) -> np.ndarray:
    """fp16 bits [layers][kv_heads][128][128] of sqrt(128) Q, Q Haar-random orthogonal."""
    out = np.empty((layers, kv_heads, HEAD_DIM, HEAD_DIM), np.float16)
    for l in range(layers):
        r = _rng(seed, STREAM_ROT, l)
        for h in range(kv_heads):
            q, rr = np.linalg.qr(r.standard_normal((HEAD_DIM, HEAD_DIM)))
            q = q * np.where(np.diag(rr) < 0, -1.0, 1.0)[None, :]
            out[l, h] = (np.sqrt(HEAD_DIM) * q).astype(np.float16)
    return out.view(np.uint16)


def f16_bits(a: np.ndarray) -> np.ndarray:
    """View a float16 array as its uint16 bit patterns."""
    return np.ascontiguousarray(a, dtype=np.float16).view(np.uint16)


def kv_layer_device(seed: int, layer: int, batch: int, kv_heads: int, T: int, device,
                    outliers: int = 4, factor: float = 8.0):
    """Like kv_layer, drawn on the GPU (torch's seeded CUDA generator) for caches too
    large to draw on the host; outlier channels come from the same numpy stream.
    Returns float16 torch tensors [batch][kv_heads][T][128] on `device`."""
    import torch
    ro = _rng(seed, STREAM_OUTLIERS, layer)
    chans = [ro.choice(HEAD_DIM, outliers, replace=False) for _ in range(kv_heads)]
    out = []
    for stream in (STREAM_K, STREAM_V):
        g = torch.Generator(device=device)
        g.manual_seed(seed * 1000 + stream + 10000 * layer)
        x = torch.randn((batch, kv_heads, T, HEAD_DIM), generator=g, device=device,
                        dtype=torch.float32)
        for h in range(kv_heads):
            x[:, h, :, torch.as_tensor(chans[h], device=device)] *= factor
        out.append(x.to(torch.float16))
    return out[0], out[1]
