"""Shared construction of seeded test cases for GPU-vs-oracle parity tests.

Inputs come from the seeded generators in ``paper_2609_17475_gb300.synth``;
the oracle builds its own pool from the same bf16 rows, the GPU builds its pool
with the quantize-append kernel (or receives a copy of the oracle's pool when a
test isolates the attention kernel).
"""
import dataclasses
from typing import List, Optional

import numpy as np
import torch

from oracle import affine4 as OA
from paper_2609_17475_gb300 import synth

MAX_ABS = 2e-2      # bf16 attention output vs fp64 oracle, unit-variance inputs
MEAN_ABS = 2e-3


def bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


@dataclasses.dataclass
class Case:
    Hq: int
    Hkv: int
    D: int
    P: int
    ctx: List[int]
    k: torch.Tensor           # bf16 [N, Hkv, D] (all requests' rows, logical order)
    v: torch.Tensor
    req: torch.Tensor         # int32 [N]
    pos: torch.Tensor         # int32 [N]
    page_table: torch.Tensor  # int32 [B, maxP]
    num_pages: int
    q: torch.Tensor           # bf16 [B, Hq, D]

    @property
    def layout(self):
        return OA.PoolLayout(self.Hkv, self.P, self.D)

    def oracle_pool(self, fill: int = 0) -> np.ndarray:
        pool = OA.new_pool(self.layout, self.num_pages, fill=fill)
        OA.append(pool, self.layout, self.page_table.numpy(), self.req.numpy(), self.pos.numpy(),
                  bits(self.k), bits(self.v))
        return pool


def make_case(seed: int, Hq: int, Hkv: int, D: int, P: int, ctx: List[int],
              num_pages: Optional[int] = None, outliers: bool = False) -> Case:
    gen = synth.generator(seed)
    channels = synth.outlier_channels(gen, Hkv, D) if outliers else None
    total = sum(ctx)
    k, v = synth.kv_rows(gen, total, Hkv, D, channels)
    pt, npages = synth.page_tables(gen, ctx, P, num_pages=num_pages)
    q = synth.normal_bf16(gen, (len(ctx), Hq, D))
    req, pos = synth.append_rows_for(ctx)
    return Case(Hq, Hkv, D, P, list(ctx), k, v, req, pos, pt, npages, q)


def assert_attention_close(got: torch.Tensor, ref: np.ndarray, max_abs=MAX_ABS, mean_abs=MEAN_ABS):
    g = got.float().cpu().numpy()
    assert np.isfinite(g).all(), "non-finite output"
    err = np.abs(g - ref)
    assert err.max() <= max_abs and err.mean() <= mean_abs, (float(err.max()), float(err.mean()))
    return float(err.max()), float(err.mean())
