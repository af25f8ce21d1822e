"""The decode entry point that allocates nothing (for callers that cannot
allocate device memory) must match the workspace entry point.

Collected last so a failure here never hides the other tests' results."""
import math

import numpy as np
import pytest
import torch

import paper_2609_17475_gb300 as jf
from oracle import attention as OT
from tests.cases import MAX_ABS, MEAN_ABS, assert_attention_close, bits, make_case

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
    oref = OT.paged_decode(case.oracle_pool(), case.layout, case.page_table.numpy(), case.ctx,
                           bits(case.q), scale)
    for call in range(2):
        out = torch.full_like(ref, float("nan"))
        jf.jf_paged_decode_attn_noalloc(pool, pt, ctx, q, scale, out, splits, err)
        torch.cuda.synchronize()
        assert int(err.item()) == 0
        d = (out.float() - ref.float()).abs()
        assert torch.isfinite(out.float()).all()
        assert d.max().item() <= MAX_ABS and d.mean().item() <= MEAN_ABS, call
        assert_attention_close(out, oref)      # and against the oracle itself


def test_noalloc_single_request_after_a_larger_batch():
    """A one-request call (per-request split plan) right after a larger batch
    call (batch plan) that filled more of the shared array: nothing the earlier
    call left behind may reach the later call's output."""
    big = make_case(903, 24, 4, 256, 128, [20000, 7000, 333])
    small = make_case(904, 24, 4, 256, 128, [5000])
    scale = 1 / math.sqrt(256)
    err = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    pool_b = _pool(big)
    out_b = torch.empty(3, 24, 256, dtype=torch.bfloat16, device=DEV)
    jf.jf_paged_decode_attn_noalloc(pool_b, big.page_table.to(DEV),
                                     torch.tensor(big.ctx, dtype=torch.int32, device=DEV),
                                     big.q.to(DEV), scale, out_b, 40, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    pool_s = _pool(small)
    pt, ctx, q = (small.page_table.to(DEV), torch.tensor(small.ctx, dtype=torch.int32, device=DEV),
                  small.q.to(DEV))
    splits = 8
    ref = torch.empty(1, 24, 256, dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(1, 24, 4, 256, splits, device=DEV)
    jf.jf_paged_decode_attn(pool_s, pt, ctx, q, scale, ref, ws, splits)
    out = torch.full_like(ref, float("nan"))
    jf.jf_paged_decode_attn_noalloc(pool_s, pt, ctx, q, scale, out, splits, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0 and jf.workspace_status(ws) == 0
    assert torch.equal(out, ref)          # same kernels, same split plan: same bits
    oref = OT.paged_decode(small.oracle_pool(), small.layout, small.page_table.numpy(), small.ctx,
                           bits(small.q), scale)
    assert_attention_close(out, oref)
    oref_b = OT.paged_decode(big.oracle_pool(), big.layout, big.page_table.numpy(), big.ctx,
                             bits(big.q), scale)
    assert_attention_close(out_b, oref_b)


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
