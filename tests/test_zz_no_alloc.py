"""The decode entry point that allocates nothing (for callers that cannot
allocate device memory) must match the workspace entry point.

Collected last so a failure here never hides the other tests' results."""
import math

import numpy as np
import pytest
import torch

import paper_2609_17475_gb300 as jf
from tests.cases import MAX_ABS, MEAN_ABS, make_case

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _pool(case):
    pool = jf.KVPool.allocate(case.num_pages, case.P, case.Hkv, case.D, device=DEV)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_quantize_append(pool, case.page_table.to(DEV), case.req.to(DEV), case.pos.to(DEV),
                             case.k.to(DEV), case.v.to(DEV), err)
    return pool


def test_noalloc_matches_workspace_entry_point_twice():
    case = make_case(901, 24, 4, 256, 256, [9000, 130])
    pool = _pool(case)
    pt = case.page_table.to(DEV)
    ctx = torch.tensor(case.ctx, dtype=torch.int32, device=DEV)
    q = case.q.to(DEV)
    scale = 1 / math.sqrt(case.D)
    splits = 16
    ref = torch.empty(2, 24, 256, dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(2, 24, 4, 256, splits, device=DEV)
    jf.jf_paged_decode_attn(pool, pt, ctx, q, scale, ref, ws, splits)
    err = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    for call in range(2):
        out = torch.full_like(ref, float("nan"))
        jf.jf_paged_decode_attn_noalloc(pool, pt, ctx, q, scale, out, splits, err)
        torch.cuda.synchronize()
        assert int(err.item()) == 0
        d = (out.float() - ref.float()).abs()
        assert torch.isfinite(out.float()).all()
        assert d.max().item() <= MAX_ABS and d.mean().item() <= MEAN_ABS, call


def test_noalloc_rejects_requests_beyond_its_array():
    case = make_case(902, 8, 2, 128, 64, [100])
    pool = _pool(case)
    too_many = 1 + jf.binding.JF_STATIC_WORKSPACE_BYTES // (8 * (4 * 128 + 8))
    out = torch.empty(1, 8, 128, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(jf.JfError) as e:
        jf.jf_paged_decode_attn_noalloc(pool, case.page_table.to(DEV),
                                         torch.tensor([100], dtype=torch.int32, device=DEV),
                                         case.q.to(DEV), 0.1, out, int(too_many))
    assert e.value.status == jf.binding.JF_ERR_WORKSPACE_TOO_SMALL
