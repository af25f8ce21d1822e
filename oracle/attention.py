"""Attention over the paged 4-bit KV pool, in fp64 (test infrastructure).

Every function reads the pool through ``gather_head``, so it serves both KV
formats: affine 4-bit group-64 and TQ4 (Sec. 3.1 Eq. 4).

Only tests, smoke() and the bench CPU baseline use this module.

* ``paged_decode`` is the plain definition of single-query attention read from
  the paged cache (Sec. 3.1: decode reads the compressed pages where they are
  used instead of expanding the whole cache).  For request b and query head h
  with KV head kv = floor(h / G), G = Hq / Hkv (contiguous head groups, the
  grouping of Eq. 5), logical positions t < ctx_b:
      s_t = softmax_scale * <q_{b,h}, K_hat_t>,  o = sum_t softmax(s)_t V_hat_t.
  ``context_lens`` count positions already appended, including the current
  token (append, then attend).  An empty context gives a zero output.
* ``split_partials`` / ``merge_partials`` are the bounded-workspace form of the
  same result (Sec. 2 Eq. 3 motivates never sizing temporaries by the history
  length; Sec. 3.1): positions are cut into contiguous splits, each split keeps
  (m_s, l_s, O_s) with m_s its max logit, l_s = sum exp(s_t - m_s) and
  O_s = sum exp(s_t - m_s) V_hat_t, and the merge is
      o = sum_s e^{m_s - m*} O_s / sum_s e^{m_s - m*} l_s,  m* = max_s m_s.
* ``prefill_chunk`` is causal attention of a chunk of C queries at absolute
  positions q_start .. q_start+C-1 against positions 0 .. q_start+i of the
  reconstructed cache (Sec. 3.1 and Eq. 5: prefill attention consumes K/V
  reconstructed from the pool; the chunk's own rows are appended first).
"""
from __future__ import annotations

import numpy as np

from . import affine4, tq4
from .affine4 import KIND_K, KIND_V, bf16_to_f64


def gather_head(pool, layout, page_table_row, ctx, head, kind):
    """Reconstructed K or V of one KV head, fp64 [ctx, D], for either format:
    an affine ``PoolLayout`` or a TQ4 ``Tq4Layout`` (which carries its codec)."""
    if isinstance(layout, tq4.Tq4Layout):
        return tq4.gather_head(pool, layout, page_table_row, ctx, head, kind)
    return affine4.gather_head(pool, layout, page_table_row, ctx, head, kind)


def _softmax_weighted(s: np.ndarray, v: np.ndarray) -> np.ndarray:
    """softmax(s) @ v for s [..., T] and v [T, D], fp64, max-subtracted."""
    m = s.max(axis=-1, keepdims=True)
    p = np.exp(s - m)
    return (p @ v) / p.sum(axis=-1, keepdims=True)


def paged_decode(pool: np.ndarray, layout, page_table: np.ndarray,
                 context_lens, q_bits: np.ndarray, softmax_scale: float,
                 heads=None) -> np.ndarray:
    """Single-query paged decode attention.

    q_bits: bf16 bit patterns [B, Hq, D].  Returns fp64 [B, Hq, D].
    ``heads`` optionally restricts the computed query heads (others stay 0).
    """
    q = bf16_to_f64(q_bits)
    B, Hq, D = q.shape
    G = Hq // layout.num_kv_heads
    out = np.zeros((B, Hq, D), dtype=np.float64)
    want = set(range(Hq)) if heads is None else set(heads)
    for b in range(B):
        ctx = int(context_lens[b])
        if ctx == 0:
            continue
        for kv in range(layout.num_kv_heads):
            hs = [h for h in range(kv * G, (kv + 1) * G) if h in want]
            if not hs:
                continue
            k = gather_head(pool, layout, page_table[b], ctx, kv, KIND_K)
            v = gather_head(pool, layout, page_table[b], ctx, kv, KIND_V)
            s = softmax_scale * (q[b, hs] @ k.T)                 # [len(hs), ctx]
            out[b, hs] = _softmax_weighted(s, v)
    return out


def split_bounds(ctx: int, num_splits: int):
    """Contiguous, near-equal position ranges [lo, hi) covering [0, ctx)."""
    edges = [(ctx * s) // num_splits for s in range(num_splits + 1)]
    return [(edges[s], edges[s + 1]) for s in range(num_splits) if edges[s + 1] > edges[s]]


def split_partials(s: np.ndarray, v: np.ndarray, num_splits: int):
    """Per-split (m_s, l_s, O_s) of logits s [T] and values v [T, D]."""
    parts = []
    for lo, hi in split_bounds(len(s), num_splits):
        m = s[lo:hi].max()
        p = np.exp(s[lo:hi] - m)
        parts.append((m, p.sum(), p @ v[lo:hi]))
    return parts


def merge_partials(parts) -> np.ndarray:
    m_star = max(m for m, _, _ in parts)
    num = sum(np.exp(m - m_star) * o for m, _, o in parts)
    den = sum(np.exp(m - m_star) * l for m, l, _ in parts)
    return num / den


def paged_decode_split(pool: np.ndarray, layout, page_table: np.ndarray,
                       context_lens, q_bits: np.ndarray, softmax_scale: float,
                       num_splits: int) -> np.ndarray:
    """The same result as ``paged_decode`` through split partials + merge."""
    q = bf16_to_f64(q_bits)
    B, Hq, D = q.shape
    G = Hq // layout.num_kv_heads
    out = np.zeros((B, Hq, D), dtype=np.float64)
    for b in range(B):
        ctx = int(context_lens[b])
        if ctx == 0:
            continue
        for kv in range(layout.num_kv_heads):
            k = gather_head(pool, layout, page_table[b], ctx, kv, KIND_K)
            v = gather_head(pool, layout, page_table[b], ctx, kv, KIND_V)
            for h in range(kv * G, (kv + 1) * G):
                s = softmax_scale * (k @ q[b, h])
                out[b, h] = merge_partials(split_partials(s, v, num_splits))
    return out


def prefill_chunk(pool: np.ndarray, layout, page_table_row: np.ndarray,
                  q_bits: np.ndarray, q_start: int, softmax_scale: float,
                  causal: bool = True) -> np.ndarray:
    """Chunk attention.  q_bits [C, Hq, D] at absolute positions q_start + i.

    Causal: query i attends positions [0, q_start + i].  Non-causal: every
    query attends [0, q_start + C).  Returns fp64 [C, Hq, D].
    """
    q = bf16_to_f64(q_bits)
    C, Hq, D = q.shape
    G = Hq // layout.num_kv_heads
    total = q_start + C
    out = np.zeros((C, Hq, D), dtype=np.float64)
    if C == 0:
        return out
    t = np.arange(total)
    limit = (q_start + np.arange(C) + 1) if causal else np.full(C, total)
    mask = t[None, :] < limit[:, None]                                  # [C, total]
    for kv in range(layout.num_kv_heads):
        k = gather_head(pool, layout, page_table_row, total, kv, KIND_K)
        v = gather_head(pool, layout, page_table_row, total, kv, KIND_V)
        for h in range(kv * G, (kv + 1) * G):
            s = softmax_scale * (q[:, h] @ k.T)                          # [C, total]
            s = np.where(mask, s, -np.inf)
            out[:, h] = _softmax_weighted(s, v)
    return out
