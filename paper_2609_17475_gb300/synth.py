"""Seeded synthetic inputs for the paged 4-bit KV path.

This module only draws random inputs and lays out page tables.  It holds no
quantization, attention or checkpoint arithmetic, so that the CPU oracle and
the CUDA path can both consume exactly the same bytes without sharing any of
the method's code.

Input recipe (the paper's workloads are repeated-word prompts on a 27B GQA
model; no dataset or weights are needed for the KV path):

* K and V rows are drawn fp32 N(0, 1) from a ``torch.Generator`` seeded per
  workload, then cast to bf16 with round-to-nearest-even.
* "Outlier" workloads multiply 4 seeded head_dim channels per KV head of K by
  20 before the bf16 cast (per-channel key outliers).
* Queries are drawn the same way, N(0, 1) bf16.
* Physical page ids are a seeded random permutation of the pool, so logical
  token order never matches physical order.
* The TQ4 random-sign vectors are NumPy draws (``tq4_signs``); both the
  oracle and the CUDA path take them as inputs.

The head geometry follows the paper's evaluated model (Sec. 2; App. A.1):
24 query heads, 4 KV heads, head_dim 256, 256-position pages.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Sequence

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Geometry:
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    page_size: int

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads


def generator(seed: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    return g


def normal_bf16(gen: torch.Generator, shape: Sequence[int]) -> torch.Tensor:
    """fp32 N(0,1) draws cast to bf16 (RNE), on the CPU."""
    return torch.randn(*shape, generator=gen, dtype=torch.float32).to(torch.bfloat16)


def outlier_channels(gen: torch.Generator, num_kv_heads: int, head_dim: int,
                     count: int = 4) -> torch.Tensor:
    """``count`` distinct head_dim channel indices per KV head, int64 [Hkv, count]."""
    rows = [torch.randperm(head_dim, generator=gen)[:count].sort().values
            for _ in range(num_kv_heads)]
    return torch.stack(rows)


def kv_rows(gen: torch.Generator, n: int, num_kv_heads: int, head_dim: int,
            channels: Optional[torch.Tensor] = None,
            outlier_scale: float = 20.0):
    """K and V rows, bf16 [n, Hkv, D].  ``channels`` (from ``outlier_channels``)
    selects K channels multiplied by ``outlier_scale`` before the bf16 cast."""
    k = torch.randn(n, num_kv_heads, head_dim, generator=gen, dtype=torch.float32)
    v = torch.randn(n, num_kv_heads, head_dim, generator=gen, dtype=torch.float32)
    if channels is not None:
        for h in range(num_kv_heads):
            k[:, h, channels[h]] *= outlier_scale
    return k.to(torch.bfloat16), v.to(torch.bfloat16)


def page_permutation(gen: torch.Generator, num_pages: int) -> torch.Tensor:
    return torch.randperm(num_pages, generator=gen).to(torch.int32)


def pages_for(ctx: int, page_size: int) -> int:
    return (ctx + page_size - 1) // page_size


def page_tables(gen: torch.Generator, context_lens: Sequence[int], page_size: int,
                num_pages: Optional[int] = None, pad_value: int = -1):
    """Assign each request's logical pages to distinct physical pages drawn from
    a seeded permutation of a pool of ``num_pages`` pages (default: exactly the
    pages needed).  Returns (page_table int32 [B, maxP] padded with
    ``pad_value``, num_pages)."""
    need = [pages_for(c, page_size) for c in context_lens]
    total = sum(need)
    if num_pages is None:
        num_pages = total
    assert num_pages >= total
    perm = page_permutation(gen, num_pages)
    max_p = max(max(need), 1)
    table = torch.full((len(need), max_p), pad_value, dtype=torch.int32)
    off = 0
    for b, n in enumerate(need):
        table[b, :n] = perm[off:off + n]
        off += n
    return table, num_pages


def interleaved_page_tables(gen: torch.Generator, context_lens: Sequence[int],
                            page_size: int, num_pages: int):
    """Physical pages of several requests interleaved at random: each physical
    page is owned by a request chosen in proportion to what it still needs."""
    need = [pages_for(c, page_size) for c in context_lens]
    assert sum(need) <= num_pages
    owners: List[int] = []
    for b, n in enumerate(need):
        owners += [b] * n
    owners_t = torch.tensor(owners, dtype=torch.int64)
    order = torch.randperm(len(owners), generator=gen)
    owners_t = owners_t[order]
    phys = torch.randperm(num_pages, generator=gen)[: len(owners)]
    max_p = max(need)
    table = torch.full((len(need), max_p), -1, dtype=torch.int32)
    fill = [0] * len(need)
    for i in range(len(owners)):
        b = int(owners_t[i])
        table[b, fill[b]] = int(phys[i])
        fill[b] += 1
    return table


def append_rows_for(context_lens: Sequence[int]):
    """(row_req, row_pos) int32 listing every position of every request in
    logical order, used to fill a pool from scratch."""
    req, pos = [], []
    for b, c in enumerate(context_lens):
        req.append(torch.full((c,), b, dtype=torch.int32))
        pos.append(torch.arange(c, dtype=torch.int32))
    if not req:
        return torch.zeros(0, dtype=torch.int32), torch.zeros(0, dtype=torch.int32)
    return torch.cat(req), torch.cat(pos)


def tq4_signs(seed: int, head_dim: int) -> np.ndarray:
    """The random-sign diagonal S of the TQ4 rotation (App. A.1 Table 3):
    NumPy ``default_rng(seed + d * 7919)`` drawing one of (-1, +1) per
    coordinate, int8 [d].  K uses seed 0 and V seed 1 by default."""
    rng = np.random.default_rng(int(seed) + int(head_dim) * 7919)
    return rng.choice(np.array([-1, 1], dtype=np.int8), size=int(head_dim))


TQ4_SEED_K, TQ4_SEED_V = 0, 1


def context_lengths(gen: torch.Generator, batch: int, lo: int, hi: int) -> List[int]:
    """Context lengths uniform on the integers [lo, hi]."""
    return [int(x) for x in torch.randint(lo, hi + 1, (batch,), generator=gen)]


# Named workloads: shapes, seeds and sizes.  Sizes in positions.
WORKLOADS = {
    "tiny": dict(seed=1, geometry=Geometry(8, 2, 128, 256), context_lens=[4096],
                 outliers=False, append_rows=256),
    "full_window_256k": dict(seed=2, geometry=Geometry(24, 4, 256, 256),
                             context_lens=[262144], outliers=True, layers=64),
    "two_request_320k": dict(seed=3, geometry=Geometry(24, 4, 256, 256),
                             context_lens=[196608, 131072], num_pages=1280,
                             outliers=False, num_splits=32),
    "prefill_decode_32k_6k": dict(seed=4, geometry=Geometry(24, 4, 256, 256),
                                  prompt=32768, chunk=2048, decode_steps=6144,
                                  outliers=False),
    "mixed_batch_32": dict(seed=5, geometry=Geometry(24, 4, 256, 256), batch=32,
                           ctx_lo=1024, ctx_hi=65536, outliers=True,
                           page_sizes=[64, 128, 256]),
}
