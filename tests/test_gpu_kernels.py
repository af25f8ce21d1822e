"""GPU parity tests: quantize-append and checkpoint bit-exact, paged decode
attention within tolerance of the fp64 oracle, plus invariants and edge cases.
All calls go through the C ABI (libjfkv.so) via the thin binding."""
import math

import numpy as np
import pytest
import torch

import paper_2609_17475_gb300 as jf
from oracle import affine4 as OA
from oracle import attention as OT
from oracle import checkpoint as OC
from tests.cases import assert_attention_close, bits, make_case

pytestmark = pytest.mark.gpu
DEV = "cuda"


def gpu_append(case, fill=0):
    pool = jf.KVPool.allocate(case.num_pages, case.P, case.Hkv, case.D, device=DEV, fill=fill)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_quantize_append(pool, case.page_table.to(DEV), case.req.to(DEV), case.pos.to(DEV),
                             case.k.to(DEV), case.v.to(DEV), err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    return pool


def pool_from_numpy(case, arr):
    pool = jf.KVPool.allocate(case.num_pages, case.P, case.Hkv, case.D, device=DEV, fill=None)
    pool.data.copy_(torch.from_numpy(arr))
    return pool


def gpu_decode(case, pool, splits, ctx=None, q=None, scale=None, page_table=None):
    ctx = case.ctx if ctx is None else ctx
    q = case.q if q is None else q
    pt = case.page_table if page_table is None else page_table
    B = len(ctx)
    out = torch.full((B, case.Hq, case.D), float("nan"), dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(B, case.Hq, case.Hkv, case.D, splits, device=DEV)
    ws[256:] = 0xFF    # NaN partials: rows past the split plan must never be used
    scale = 1 / math.sqrt(case.D) if scale is None else scale
    jf.jf_paged_decode_attn(pool, pt.to(DEV), torch.tensor(ctx, dtype=torch.int32, device=DEV),
                            q.to(DEV), scale, out, ws, splits)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    return out


# --------------------------------------------------------------------------
# quantize-append: bit-exact against the oracle
# --------------------------------------------------------------------------
@pytest.mark.parametrize("Hkv,D,P,ctx,outliers", [
    (2, 128, 256, [256], False),                   # the tiny workload's 256-row append
    (2, 128, 64, [1, 63, 130], False),
    (4, 256, 256, [1000, 517], True),
    (3, 256, 128, [300], True),
    (1, 128, 128, [4096], False),
])
def test_append_bit_exact(Hkv, D, P, ctx, outliers):
    case = make_case(100 + sum(ctx), 2 * Hkv, Hkv, D, P, ctx, outliers=outliers,
                     num_pages=sum(-(-c // P) for c in ctx) + 2)
    ref = case.oracle_pool(fill=0x5A)
    pool = gpu_append(case, fill=0x5A)
    got = pool.data.cpu().numpy()
    assert np.array_equal(got, ref)


def test_append_special_groups_bit_exact():
    """Constant groups, signed zeros, exact midpoints, subnormals, huge ranges."""
    D, Hkv, P = 256, 2, 64
    rng = np.random.default_rng(4)
    n = 64
    x = rng.standard_normal((2, n, Hkv, D)).astype(np.float32)
    x[:, 0] = 3.0                                        # constant
    x[:, 1] = 0.0
    x[:, 1, :, ::3] = -0.0                               # signed zeros
    x[:, 2] = np.tile(np.arange(64) % 16 + 0.5, D // 64)  # midpoints
    x[:, 2, :, ::64] = 0.0
    x[:, 2, :, 1::64] = 15.0
    x[:, 3] *= 1e-39                                     # subnormal range
    x[:, 4] *= 1e30                                      # huge range
    x[:, 5, :, :32] = 1e20
    kv = torch.from_numpy(x).to(torch.bfloat16)
    case = make_case(7, 2 * Hkv, Hkv, D, P, [n])
    case.k, case.v = kv[0].contiguous(), kv[1].contiguous()
    ref = case.oracle_pool(fill=0)
    pool = gpu_append(case, fill=0)
    assert np.array_equal(pool.data.cpu().numpy(), ref)


def test_append_flags_bad_rows_and_skips_them():
    case = make_case(9, 4, 2, 128, 64, [100], num_pages=3)
    pool = jf.KVPool.allocate(case.num_pages, 64, 2, 128, device=DEV, fill=0x11)
    pt = case.page_table.clone()
    pt[0, 1] = 999                                       # page id outside the pool
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_quantize_append(pool, pt.to(DEV), case.req.to(DEV), case.pos.to(DEV),
                             case.k.to(DEV), case.v.to(DEV), err)
    torch.cuda.synchronize()
    assert int(err.item()) & jf.binding.JF_DEV_ERR_PAGE_ID
    got = pool.data.cpu().numpy()
    L = case.layout
    ref = OA.new_pool(L, case.num_pages, fill=0x11)
    OA.append(ref, L, case.page_table.numpy(), case.req.numpy()[:64], case.pos.numpy()[:64],
              bits(case.k[:64]), bits(case.v[:64]))
    assert np.array_equal(got, ref)                      # rows 64..99 skipped
    pos = case.pos.clone()
    pos[5] = 10_000                                      # beyond the page-table row
    err.zero_()
    jf.jf_kv_quantize_append(pool, case.page_table.to(DEV), case.req.to(DEV), pos.to(DEV),
                             case.k.to(DEV), case.v.to(DEV), err)
    torch.cuda.synchronize()
    assert int(err.item()) & jf.binding.JF_DEV_ERR_POSITION


# --------------------------------------------------------------------------
# checkpoint / restore: bit-exact
# --------------------------------------------------------------------------
@pytest.mark.parametrize("Hkv,D,P,ctx", [(2, 128, 256, [3000]), (4, 256, 64, [700]),
                                         (4, 256, 256, [38912])])
def test_checkpoint_and_restore_bit_exact(Hkv, D, P, ctx):
    case = make_case(11, 2 * Hkv, Hkv, D, P, ctx, num_pages=-(-ctx[0] // P) + 3)
    ref = case.oracle_pool(fill=0x33)
    pool = pool_from_numpy(case, ref)
    n = -(-ctx[0] // P)
    blob = torch.empty(n * pool.page_bytes, dtype=torch.uint8, device=DEV)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_checkpoint(pool, case.page_table[0].to(DEV), n, blob, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    assert np.array_equal(blob.cpu().numpy(), OC.checkpoint(ref, case.page_table[0].numpy(), n))
    fresh = jf.KVPool.allocate(case.num_pages, P, Hkv, D, device=DEV, fill=0)
    jf.jf_kv_restore(fresh, case.page_table[0].to(DEV), n, blob, err)
    torch.cuda.synchronize()
    exp = OA.new_pool(case.layout, case.num_pages, fill=0)
    OC.restore(exp, case.page_table[0].numpy(), n, OC.checkpoint(ref, case.page_table[0].numpy(), n))
    assert np.array_equal(fresh.data.cpu().numpy(), exp)


# --------------------------------------------------------------------------
# paged decode attention
# --------------------------------------------------------------------------
@pytest.mark.parametrize("Hq,Hkv,D,P,ctx,splits,outliers", [
    (8, 2, 128, 256, [4096], 1, False),            # tiny workload, one split
    (8, 2, 128, 256, [4096], 8, False),            # tiny workload, split-K + merge
    (8, 2, 128, 64, [1, 33, 517, 2000], 4, False),  # ragged batch, partial pages
    (24, 4, 256, 256, [5000], 3, True),            # paper geometry, outliers
    (24, 4, 256, 128, [777, 1], 16, True),
    (4, 4, 256, 64, [1500], 2, False),             # G = 1
    (16, 2, 256, 256, [2500], 5, False),           # G = 8
    (12, 2, 128, 128, [999], 64, False),           # more splits than needed
    (8, 2, 128, 256, [70000, 3000], 150, False),   # > 128 live splits: merge loops
    (8, 2, 128, 64, [20000, 70, 1, 3000], 8, False),   # batch plan: the long request
                                                       # takes more than num_splits
    (24, 4, 256, 128, [9000, 0, 40], 3, True),     # batch plan with an empty request
])
def test_decode_matches_oracle(Hq, Hkv, D, P, ctx, splits, outliers):
    case = make_case(200 + Hq + sum(ctx), Hq, Hkv, D, P, ctx, outliers=outliers)
    ref_pool = case.oracle_pool()
    pool = pool_from_numpy(case, ref_pool)
    out = gpu_decode(case, pool, splits)
    ref = OT.paged_decode(ref_pool, case.layout, case.page_table.numpy(), ctx, bits(case.q),
                          1 / math.sqrt(D))
    assert_attention_close(out, ref)


@pytest.mark.parametrize("Hq,Hkv,D,P,splits", [(8, 2, 128, 64, 2), (24, 4, 256, 128, 3)])
def test_decode_batch_pieces_spanning_many_requests(Hq, Hkv, D, P, splits):
    """Batches cut the requests' chunks, laid end to end, into equal pieces:
    with few splits and many short requests a piece crosses many request
    boundaries (empty requests, single positions, exact chunk and page
    multiples), and every request still matches the oracle."""
    ctx = [0, 1, 31, 32, 33, 64, 65, 500, 0, 2048, 7, 1000, 3, 4096, 129, 1, 0, 777, 256, 5000,
           31, 33, 96, 97, 1500, 2, 640, 2049, 15, 300]
    case = make_case(700 + D, Hq, Hkv, D, P, ctx, outliers=True)
    ref_pool = case.oracle_pool()
    pool = pool_from_numpy(case, ref_pool)
    out = gpu_decode(case, pool, splits)
    ref = OT.paged_decode(ref_pool, case.layout, case.page_table.numpy(), ctx, bits(case.q),
                          1 / math.sqrt(D))
    assert_attention_close(out, ref)
    for b, c in enumerate(ctx):
        if c == 0:
            assert (out[b].float() == 0).all()


@pytest.mark.parametrize("Hq,Hkv,D,P,ctx,splits", [
    (24, 4, 256, 256, [5000, 257, 1], 76),   # new rows mid-page, at slot 0 of a page, alone
    (8, 2, 128, 64, [64, 65, 999], 4),
    (16, 2, 256, 128, [3000], 1),            # one split writes and reads directly
    (8, 2, 128, 64, [1, 40, 2, 33, 700, 65, 3], 2),   # pieces spanning requests
])
def test_fused_append_decode_equals_append_then_decode(Hq, Hkv, D, P, ctx, splits):
    """jf_paged_decode_append_attn leaves the same pool bytes and output as
    jf_kv_quantize_append of each request's newest row followed by
    jf_paged_decode_attn, and both match the oracle."""
    case = make_case(900 + sum(ctx), Hq, Hkv, D, P, ctx)
    req, pos = case.req.numpy(), case.pos.numpy()
    last = np.array([np.nonzero(req == b)[0].max() for b in range(len(ctx))])
    keep = np.setdiff1d(np.arange(len(req)), last)
    prefix = OA.new_pool(case.layout, case.num_pages, fill=0xFF)
    OA.append(prefix, case.layout, case.page_table.numpy(), req[keep], pos[keep],
              bits(case.k[keep]), bits(case.v[keep]))
    full = case.oracle_pool(fill=0xFF)
    k_new = case.k[last].contiguous()
    v_new = case.v[last].contiguous()
    B = len(ctx)
    pt = case.page_table.to(DEV)
    ctx_t = torch.tensor(ctx, dtype=torch.int32, device=DEV)
    scale = 1 / math.sqrt(D)

    pool_a = pool_from_numpy(case, prefix)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_quantize_append(pool_a, pt, torch.arange(B, dtype=torch.int32, device=DEV),
                             (ctx_t - 1).contiguous(), k_new.to(DEV), v_new.to(DEV), err)
    out_a = torch.full((B, Hq, D), float("nan"), dtype=torch.bfloat16, device=DEV)
    ws_a = jf.decode_workspace(B, Hq, Hkv, D, splits, device=DEV)
    jf.jf_paged_decode_attn(pool_a, pt, ctx_t, case.q.to(DEV), scale, out_a, ws_a, splits)

    pool_b = pool_from_numpy(case, prefix)
    out_b = torch.full((B, Hq, D), float("nan"), dtype=torch.bfloat16, device=DEV)
    ws_b = jf.decode_workspace(B, Hq, Hkv, D, splits, device=DEV)
    ws_b[256:] = 0xFF
    jf.jf_paged_decode_append_attn(pool_b, pt, ctx_t, k_new.to(DEV), v_new.to(DEV),
                                   case.q.to(DEV), scale, out_b, ws_b, splits)
    torch.cuda.synchronize()
    assert int(err.item()) == 0 and jf.workspace_status(ws_a) == 0 and jf.workspace_status(ws_b) == 0
    assert torch.equal(pool_a.data, pool_b.data)
    assert np.array_equal(pool_b.data.cpu().numpy(), full)       # bit-exact quantize-append
    assert torch.equal(out_a, out_b)
    ref = OT.paged_decode(full, case.layout, case.page_table.numpy(), ctx, bits(case.q), scale)
    assert_attention_close(out_b, ref)


def test_fused_append_decode_reports_bad_page_id():
    case = make_case(911, 8, 2, 128, 64, [100])
    pool = pool_from_numpy(case, case.oracle_pool())
    pt = case.page_table.clone()
    pt[0, 1] = 10 ** 6                      # the page of position 99 (and 64..98)
    out = torch.zeros((1, 8, 128), dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(1, 8, 2, 128, 2, device=DEV)
    before = pool.data.clone()
    ctx_t = torch.tensor([100], dtype=torch.int32, device=DEV)
    jf.jf_paged_decode_append_attn(pool, pt.to(DEV), ctx_t, case.k[99:100].contiguous().to(DEV),
                                   case.v[99:100].contiguous().to(DEV), case.q.to(DEV), 0.1, out,
                                   ws, 2)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) & jf.binding.JF_DEV_ERR_PAGE_ID
    assert torch.equal(pool.data, before)    # nothing written anywhere


@pytest.mark.parametrize("Hq,Hkv,D,P,ctx,L,splits", [
    (24, 4, 256, 256, [5000], 2, None),          # 12 (token, head) rows: 2 row groups, one CTA
    (24, 4, 256, 128, [3000, 777], 4, None),     # 24 rows, batch plan
    (24, 4, 256, 256, [4096], 3, 1),             # one split: rows written directly
    (8, 2, 128, 64, [3, 65, 300, 2001], 3, 5),   # a context equal to q_len, partial pages
    (16, 2, 256, 64, [1000], 4, 7),              # G = 8: 32 rows, two CTAs (3 + 1 groups)
    (14, 2, 256, 64, [2500], 4, 6),              # G = 7: 28 rows, two CTAs (3 + 1 groups)
    (12, 2, 128, 128, [9000], 4, 1),             # D = 128, 3 groups, 70 chunks per warp pair
    (8, 4, 128, 64, [700, 31], 4, 3),            # 8 rows: one group (the 6-warp kernel)
])
def test_verifier_matches_oracle(Hq, Hkv, D, P, ctx, L, splits):
    """Token i of each request attends positions up to ctx - L + i; the oracle
    is the causal prefill of those L queries (Sec. 3.1 packed verifier)."""
    from paper_2609_17475_gb300 import synth
    case = make_case(500 + sum(ctx) + L, Hq, Hkv, D, P, ctx)
    ref_pool = case.oracle_pool()
    pool = pool_from_numpy(case, ref_pool)
    B = len(ctx)
    q = synth.normal_bf16(synth.generator(600 + L), (B, L, Hq, D))
    if splits is None:
        splits = jf.default_verify_splits(B, L, Hq, Hkv)
    ws = jf.verify_workspace(B, L, Hq, Hkv, D, splits, device=DEV)
    ws[256:] = 0xFF
    out = torch.full((B, L, Hq, D), float("nan"), dtype=torch.bfloat16, device=DEV)
    scale = 1 / math.sqrt(D)
    jf.jf_paged_verify_attn(pool, case.page_table.to(DEV), torch.tensor(ctx, dtype=torch.int32,
                            device=DEV), q.to(DEV), scale, out, ws, splits)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    ref = np.stack([OT.prefill_chunk(ref_pool, case.layout, case.page_table[b].numpy(), bits(q[b]),
                                     ctx[b] - L, scale) for b in range(B)])
    assert_attention_close(out, ref)


@pytest.mark.parametrize("splits", [1, 3])
def test_verifier_context_shorter_than_q_len(splits):
    """A request whose context is shorter than q_len: token i sees positions
    < ctx - q_len + 1 + i, so the first tokens see nothing and their rows are
    zero (the oracle's softmax over an empty set is undefined, NaN); the
    others match the oracle.  Warp-pair kernel (24 rows per KV head)."""
    from paper_2609_17475_gb300 import synth
    Hq, Hkv, D, P, L = 24, 4, 256, 64, 4
    case = make_case(5151 + splits, Hq, Hkv, D, P, [2, 900])
    ref_pool = case.oracle_pool()
    pool = pool_from_numpy(case, ref_pool)
    q = synth.normal_bf16(synth.generator(5252), (2, L, Hq, D))
    ws = jf.verify_workspace(2, L, Hq, Hkv, D, splits, device=DEV)
    out = torch.full((2, L, Hq, D), float("nan"), dtype=torch.bfloat16, device=DEV)
    scale = 1 / math.sqrt(D)
    jf.jf_paged_verify_attn(pool, case.page_table.to(DEV),
                            torch.tensor(case.ctx, dtype=torch.int32, device=DEV), q.to(DEV),
                            scale, out, ws, splits)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    got = out.float().cpu()
    assert (got[0, :2] == 0).all()                       # tokens 0, 1 of the 2-position request
    with np.errstate(invalid="ignore"):   # the rows of tokens 0, 1 are NaN in the oracle
        ref0 = OT.prefill_chunk(ref_pool, case.layout, case.page_table[0].numpy(), bits(q[0]),
                                2 - L, scale)
    assert_attention_close(out[0, 2:], ref0[2:])
    ref1 = OT.prefill_chunk(ref_pool, case.layout, case.page_table[1].numpy(), bits(q[1]),
                            900 - L, scale)
    assert_attention_close(out[1], ref1)


@pytest.mark.parametrize("Hq,Hkv,D,L,splits", [(24, 4, 256, 4, 5), (24, 4, 256, 2, 3),
                                                (12, 2, 128, 3, 1)])
def test_verifier_warp_pairs_are_deterministic(Hq, Hkv, D, L, splits):
    """The two warps of a pair swap partial logits through double-buffered
    shared memory once per chunk: repeated calls on the same inputs give the
    same bits (a buffer reused too early would show up as run-to-run noise)."""
    from paper_2609_17475_gb300 import synth
    case = make_case(4242 + L, Hq, Hkv, D, 64, [7000, 3001])
    pool = pool_from_numpy(case, case.oracle_pool())
    q = synth.normal_bf16(synth.generator(4343 + L), (2, L, Hq, D)).to(DEV)
    ws = jf.verify_workspace(2, L, Hq, Hkv, D, splits, device=DEV)
    ctx = torch.tensor(case.ctx, dtype=torch.int32, device=DEV)
    outs = []
    for _ in range(3):
        out = torch.empty(2, L, Hq, D, dtype=torch.bfloat16, device=DEV)
        jf.jf_paged_verify_attn(pool, case.page_table.to(DEV), ctx, q, 1 / math.sqrt(D), out, ws,
                                splits)
        outs.append(out)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


def test_verifier_with_one_token_is_decode():
    case = make_case(77, 24, 4, 256, 256, [3333, 1234])
    pool = pool_from_numpy(case, case.oracle_pool())
    splits = 9
    out_d = gpu_decode(case, pool, splits)
    ws = jf.verify_workspace(2, 1, 24, 4, 256, splits, device=DEV)
    out_v = torch.empty((2, 1, 24, 256), dtype=torch.bfloat16, device=DEV)
    jf.jf_paged_verify_attn(pool, case.page_table.to(DEV),
                            torch.tensor(case.ctx, dtype=torch.int32, device=DEV),
                            case.q.view(2, 1, 24, 256).to(DEV), 1 / 16, out_v, ws, splits)
    torch.cuda.synchronize()
    assert torch.equal(out_v.view(2, 24, 256), out_d)


def test_decode_edge_contexts():
    case = make_case(5, 8, 2, 128, 64, [0, 1, 64, 65])
    ref_pool = case.oracle_pool()
    pool = pool_from_numpy(case, ref_pool)
    for splits in (1, 4):
        out = gpu_decode(case, pool, splits)
        assert (out[0].float() == 0).all()                        # empty context -> zeros
        ref = OT.paged_decode(ref_pool, case.layout, case.page_table.numpy(), case.ctx,
                              bits(case.q), 1 / math.sqrt(128))
        assert_attention_close(out, ref)
        # ctx = 1: the output is the single reconstructed V row (up to bf16 rounding)
        v0 = OA.gather_head(ref_pool, case.layout, case.page_table.numpy()[1], 1, 0, OA.KIND_V)[0]
        assert np.abs(out[1, 0].float().cpu().numpy() - v0).max() <= 2 ** -8 * np.abs(v0).max()


def test_decode_page_permutation_is_bitwise_invariant():
    case = make_case(31, 24, 4, 256, 256, [3000], num_pages=20)
    ref_pool = case.oracle_pool()
    out_a = gpu_decode(case, pool_from_numpy(case, ref_pool), 4)
    perm = np.random.default_rng(2).permutation(20)
    moved = np.empty_like(ref_pool)
    moved[perm] = ref_pool
    pt = case.page_table.clone()
    n = -(-3000 // 256)
    pt[0, :n] = torch.from_numpy(perm[case.page_table[0, :n].numpy()].astype(np.int32))
    out_b = gpu_decode(case, pool_from_numpy(case, moved), 4, page_table=pt)
    assert torch.equal(out_a, out_b)


def test_decode_split_count_changes_only_rounding():
    case = make_case(41, 24, 4, 256, 256, [20000], outliers=True)
    ref_pool = case.oracle_pool()
    pool = pool_from_numpy(case, ref_pool)
    ref = OT.paged_decode(ref_pool, case.layout, case.page_table.numpy(), case.ctx, bits(case.q),
                          1 / 16)
    outs = [gpu_decode(case, pool, s) for s in (1, 2, 7, 39)]
    for o in outs:
        assert_attention_close(o, ref)
    for o in outs[1:]:
        assert (o.float() - outs[0].float()).abs().max().item() <= 1e-2


def test_decode_head_subset_is_bitwise_identical():
    """A pool holding only KV heads {1, 2} gives bitwise the same outputs for
    their query heads as the full 4-head pool (Eq. 5: heads are independent)."""
    full = make_case(51, 24, 4, 256, 256, [3333])
    sub = make_case(51, 12, 2, 256, 256, [3333])
    sub.k, sub.v = full.k[:, 1:3].contiguous(), full.v[:, 1:3].contiguous()
    sub.page_table, sub.num_pages = full.page_table, full.num_pages
    sub.q = full.q[:, 6:18].contiguous()
    out_full = gpu_decode(full, gpu_append(full), 5)
    out_sub = gpu_decode(sub, gpu_append(sub), 5)
    assert torch.equal(out_full[:, 6:18], out_sub)


def test_decode_poison_pages_and_tail_never_leak():
    """NaN scales in pages outside the page table and in tail slots beyond the
    context must not reach the output (App. E.4 poison-page protocol)."""
    case = make_case(61, 8, 2, 128, 64, [200], num_pages=10)
    ref_pool = case.oracle_pool(fill=0xFF)        # 0xFFFF scale/bias = NaN everywhere unwritten
    used = set(case.page_table[0, :4].tolist())
    assert any(p not in used for p in range(10))
    pool = pool_from_numpy(case, ref_pool)
    out = gpu_decode(case, pool, 2)
    ref = OT.paged_decode(ref_pool, case.layout, case.page_table.numpy(), case.ctx, bits(case.q),
                          1 / math.sqrt(128))
    assert_attention_close(out, ref)


def test_decode_reports_bad_page_id():
    case = make_case(71, 8, 2, 128, 64, [300])
    pool = pool_from_numpy(case, case.oracle_pool())
    pt = case.page_table.clone()
    pt[0, 2] = 12345
    out = torch.empty(1, 8, 128, dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(1, 8, 2, 128, 2, device=DEV)
    jf.jf_paged_decode_attn(pool, pt.to(DEV), torch.tensor([300], dtype=torch.int32, device=DEV),
                            case.q.to(DEV), 0.1, out, ws, 2)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) & jf.binding.JF_DEV_ERR_PAGE_ID


@pytest.mark.parametrize("splits", [1, 4])
@pytest.mark.parametrize("bad", ["past_row", "negative"])
def test_decode_flags_a_bad_context_of_a_later_request(splits, bad):
    """A context length outside [0, pt_stride * P] of the last request of a
    batch sets JF_DEV_ERR_POSITION (per-request and batch split plans)."""
    case = make_case(81, 8, 2, 128, 64, [300, 500, 200])
    pool = pool_from_numpy(case, case.oracle_pool())
    pt = case.page_table
    ctx = [300, 500, pt.shape[1] * 64 + 1 if bad == "past_row" else -5]
    out = torch.empty(3, 8, 128, dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(3, 8, 2, 128, splits, device=DEV)
    jf.jf_paged_decode_attn(pool, pt.to(DEV), torch.tensor(ctx, dtype=torch.int32, device=DEV),
                            case.q.to(DEV), 0.1, out, ws, splits)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) & jf.binding.JF_DEV_ERR_POSITION
    # the valid requests are still right
    ref = OT.paged_decode(case.oracle_pool(), case.layout, case.page_table.numpy(),
                          [300, 500, 0], bits(case.q), 0.1)
    assert_attention_close(out[:2], ref[:2])


def test_bounded_wait_gives_up_and_reports_timeout():
    """The give-up path of the kernels' bounded waits: a barrier nobody
    arrives at makes the wait run out, JF_DEV_ERR_TIMEOUT is reported, and the
    context stays usable (a decode afterwards is still right)."""
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.binding.jf_selftest_bounded_wait(st, True)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    jf.binding.jf_selftest_bounded_wait(st, False)
    torch.cuda.synchronize()
    assert int(st.item()) == jf.binding.JF_DEV_ERR_TIMEOUT
    case = make_case(93, 8, 2, 128, 64, [500])
    ref_pool = case.oracle_pool()
    out = gpu_decode(case, pool_from_numpy(case, ref_pool), 3)
    ref = OT.paged_decode(ref_pool, case.layout, case.page_table.numpy(), case.ctx, bits(case.q),
                          1 / math.sqrt(128))
    assert_attention_close(out, ref)


def test_decode_full_window_256k_sampled_heads():
    """The 256K full-window workload (24/4/256, 1,024 pages in a random physical
    order, 4 K channels per KV head x20) at full size, in the launch shape the
    benchmark uses; KV heads 0 and 3 checked against the oracle."""
    from paper_2609_17475_gb300 import synth
    w = synth.WORKLOADS["full_window_256k"]
    geo = w["geometry"]
    ctx = w["context_lens"][0]
    gen = synth.generator(w["seed"])
    channels = synth.outlier_channels(gen, geo.num_kv_heads, geo.head_dim)
    k, v = synth.kv_rows(gen, ctx, geo.num_kv_heads, geo.head_dim, channels)
    pt, npages = synth.page_tables(gen, [ctx], geo.page_size)
    q = synth.normal_bf16(gen, (1, geo.num_q_heads, geo.head_dim))
    req, pos = synth.append_rows_for([ctx])
    pool = jf.KVPool.allocate(npages, geo.page_size, geo.num_kv_heads, geo.head_dim, device=DEV)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_quantize_append(pool, pt.to(DEV), req.to(DEV), pos.to(DEV), k.to(DEV), v.to(DEV), err)
    splits = jf.default_num_splits(1, geo.num_kv_heads)
    out = torch.empty(1, geo.num_q_heads, geo.head_dim, dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(1, geo.num_q_heads, geo.num_kv_heads, geo.head_dim, splits, device=DEV)
    scale = 1 / math.sqrt(geo.head_dim)
    jf.jf_paged_decode_attn(pool, pt.to(DEV), torch.tensor([ctx], dtype=torch.int32, device=DEV),
                            q.to(DEV), scale, out, ws, splits)
    torch.cuda.synchronize()
    assert int(err.item()) == 0 and jf.workspace_status(ws) == 0
    G = geo.group
    for kvh in (0, 3):
        # oracle pool holding only this KV head, built from the same bf16 rows
        L1 = OA.PoolLayout(1, geo.page_size, geo.head_dim)
        opool = OA.new_pool(L1, npages)
        OA.append(opool, L1, pt.numpy(), req.numpy(), pos.numpy(),
                  bits(k[:, kvh:kvh + 1]), bits(v[:, kvh:kvh + 1]))
        ref = OT.paged_decode(opool, L1, pt.numpy(), [ctx], bits(q[:, kvh * G:(kvh + 1) * G]),
                              scale)
        assert_attention_close(out[:, kvh * G:(kvh + 1) * G], ref)
        # sampled pages: the GPU's bytes for this head decode to the oracle's vectors
        gp = pool.data.cpu().numpy()
        for page in pt[0, [0, 511, 1023]].tolist():
            for kind in (OA.KIND_K, OA.KIND_V):
                L4 = OA.PoolLayout(geo.num_kv_heads, geo.page_size, geo.head_dim)
                o4 = L4.codes_offset(kind, kvh, 0)
                o1 = L1.codes_offset(kind, 0, 0)
                n = geo.page_size * L4.code_bytes
                assert np.array_equal(gp[page, o4:o4 + n], opool[page, o1:o1 + n])


@pytest.mark.parametrize("L", [2, 4])
def test_verifier_full_window_256k_sampled_heads(L):
    """The packed verifier on the 256K full-window workload (24/4/256, 1,024
    pages in a random physical order) in the launch shape the benchmark uses
    (default split cap, warp pairs sharing the unpacking); KV heads 0 and 3
    against the oracle's causal chunk attention of the L tokens."""
    from paper_2609_17475_gb300 import synth
    w = synth.WORKLOADS["full_window_256k"]
    geo = w["geometry"]
    ctx = w["context_lens"][0]
    gen = synth.generator(w["seed"] + 17)
    channels = synth.outlier_channels(gen, geo.num_kv_heads, geo.head_dim)
    k, v = synth.kv_rows(gen, ctx, geo.num_kv_heads, geo.head_dim, channels)
    pt, npages = synth.page_tables(gen, [ctx], geo.page_size)
    q = synth.normal_bf16(gen, (1, L, geo.num_q_heads, geo.head_dim))
    req, pos = synth.append_rows_for([ctx])
    pool = jf.KVPool.allocate(npages, geo.page_size, geo.num_kv_heads, geo.head_dim, device=DEV)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_quantize_append(pool, pt.to(DEV), req.to(DEV), pos.to(DEV), k.to(DEV), v.to(DEV), err)
    Hq, Hkv, D = geo.num_q_heads, geo.num_kv_heads, geo.head_dim
    splits = jf.default_verify_splits(1, L, Hq, Hkv)
    ws = jf.verify_workspace(1, L, Hq, Hkv, D, splits, device=DEV)
    out = torch.empty(1, L, Hq, D, dtype=torch.bfloat16, device=DEV)
    scale = 1 / math.sqrt(D)
    jf.jf_paged_verify_attn(pool, pt.to(DEV), torch.tensor([ctx], dtype=torch.int32, device=DEV),
                            q.to(DEV), scale, out, ws, splits)
    torch.cuda.synchronize()
    assert int(err.item()) == 0 and jf.workspace_status(ws) == 0
    G = geo.group
    for kvh in (0, 3):
        L1 = OA.PoolLayout(1, geo.page_size, D)
        opool = OA.new_pool(L1, npages)
        OA.append(opool, L1, pt.numpy(), req.numpy(), pos.numpy(),
                  bits(k[:, kvh:kvh + 1]), bits(v[:, kvh:kvh + 1]))
        ref = OT.prefill_chunk(opool, L1, pt[0].numpy(), bits(q[0, :, kvh * G:(kvh + 1) * G]),
                               ctx - L, scale)
        assert_attention_close(out[0, :, kvh * G:(kvh + 1) * G], ref)


# --------------------------------------------------------------------------
# prefill chunk attention (tcgen05)
# --------------------------------------------------------------------------
def gpu_prefill(case, pool, q, q_start, causal, scale):
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device=DEV)
    ws = torch.zeros(jf.jf_prefill_workspace_bytes(), dtype=torch.uint8, device=DEV)
    jf.jf_prefill_chunk_attn(pool, case.page_table[0].to(DEV), q.to(DEV), q_start, scale, causal,
                             out, ws)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    return out


@pytest.mark.parametrize("Hq,Hkv,D,P,q_start,C,causal", [
    (8, 2, 128, 256, 0, 256, True),          # tiny geometry, first chunk
    (8, 2, 128, 64, 300, 77, True),           # ragged chunk, partial pages
    (24, 4, 256, 256, 0, 130, True),          # G = 6: 21 queries per CTA
    (24, 4, 256, 256, 1000, 64, True),
    (24, 4, 256, 128, 517, 200, False),       # non-causal
    (4, 4, 256, 64, 100, 129, True),          # G = 1: 128 queries per CTA
    (16, 2, 128, 128, 64, 40, True),          # G = 8
])
def test_prefill_matches_oracle(Hq, Hkv, D, P, q_start, C, causal):
    total = q_start + C
    case = make_case(300 + Hq + total, Hq, Hkv, D, P, [total], outliers=True)
    ref_pool = case.oracle_pool()
    pool = pool_from_numpy(case, ref_pool)
    from paper_2609_17475_gb300 import synth
    q = synth.normal_bf16(synth.generator(7 + C), (C, Hq, D))
    scale = 1 / math.sqrt(D)
    out = gpu_prefill(case, pool, q, q_start, causal, scale)
    ref = OT.prefill_chunk(ref_pool, case.layout, case.page_table[0].numpy(), bits(q), q_start,
                           scale, causal=causal)
    assert_attention_close(out, ref)


@pytest.mark.parametrize("D", [128, 256])
@pytest.mark.parametrize("total", [1, 64, 65, 128, 192, 257, 320, 450, 576])
def test_prefill_history_tile_counts(D, total):
    """1 to 9 history tiles of 64 positions: S runs over tile pairs (a lone
    last tile, pair buffers reused once and twice), P over single tiles."""
    Hq, Hkv, P = (24, 4, 256) if D == 256 else (8, 2, 128)
    C = min(total, 24)
    case = make_case(700 + total + D, Hq, Hkv, D, P, [total], outliers=True)
    ref_pool = case.oracle_pool()
    pool = pool_from_numpy(case, ref_pool)
    from paper_2609_17475_gb300 import synth
    q = synth.normal_bf16(synth.generator(701 + total), (C, Hq, D))
    scale = 1 / math.sqrt(D)
    out = gpu_prefill(case, pool, q, total - C, True, scale)
    ref = OT.prefill_chunk(ref_pool, case.layout, case.page_table[0].numpy(), bits(q), total - C,
                           scale, causal=True)
    assert_attention_close(out, ref)


def test_prefill_32k_prefix_sampled_rows():
    """The last 2,048-query chunk of the 32K prompt (24/4/256, P 256): sampled
    query rows checked against the oracle's decode at ctx = position + 1."""
    Hq, Hkv, D, P, C = 24, 4, 256, 256, 2048
    q_start = 32768 - C
    case = make_case(404, Hq, Hkv, D, P, [32768])
    pool = gpu_append(case)
    from paper_2609_17475_gb300 import synth
    q = synth.normal_bf16(synth.generator(405), (C, Hq, D))
    out = gpu_prefill(case, pool, q, q_start, True, 1 / 16)
    G = Hq // Hkv
    for kvh in (0, 3):
        L1 = OA.PoolLayout(1, P, D)
        opool = OA.new_pool(L1, case.num_pages)
        OA.append(opool, L1, case.page_table.numpy(), case.req.numpy(), case.pos.numpy(),
                  bits(case.k[:, kvh:kvh + 1]), bits(case.v[:, kvh:kvh + 1]))
        for i in (0, 1, 20, 21, 1000, C - 1):
            ref = OT.paged_decode(opool, L1, case.page_table.numpy(), [q_start + i + 1],
                                  bits(q[i:i + 1, kvh * G:(kvh + 1) * G]), 1 / 16)
            assert_attention_close(out[i:i + 1, kvh * G:(kvh + 1) * G], ref)


def _whole_waves(pairs):
    slots = torch.cuda.get_device_properties(0).multi_processor_count // 2
    return pairs <= slots or pairs % slots == 0


# rows on both sides of the head/tail boundaries the wave balance can choose
# for this chunk (1,596 on 152 SMs) and the chunk's ends
BALANCE_ROWS = (0, 1, 1511, 1512, 1553, 1554, 1595, 1596, 1597, 1800, 2047)


def test_prefill_wave_balanced_chunk():
    """2,048 queries after 30,720 positions (24/4/256, P 256): 196 CTA pairs,
    not whole waves of the pairs the GPU runs at once.  With the workspace
    jf_prefill_chunk_workspace_bytes asks for, the chunk runs as whole waves
    plus a tail whose histories are split; sampled rows against the oracle,
    every row against the one-launch form (minimal workspace)."""
    Hq, Hkv, D, P, C = 24, 4, 256, 256, 2048
    q_start = 32768 - C
    if _whole_waves(Hkv * -(-C // 42)):
        pytest.skip("the chunk fills whole waves on this GPU")
    case = make_case(406, Hq, Hkv, D, P, [32768])
    pool = gpu_append(case)
    from paper_2609_17475_gb300 import synth
    q = synth.normal_bf16(synth.generator(407), (C, Hq, D))
    ws = jf.prefill_chunk_workspace(pool, q_start, C, Hq, device=DEV)
    assert ws.numel() > jf.jf_prefill_workspace_bytes()
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device=DEV)
    jf.jf_prefill_chunk_attn(pool, case.page_table[0].to(DEV), q.to(DEV), q_start, 1 / 16, True,
                             out, ws)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    one = gpu_prefill(case, pool, q, q_start, True, 1 / 16)
    assert torch.isfinite(out.float()).all()
    diff = (out.float() - one.float()).abs()
    assert diff.max().item() <= 1e-2 and diff.mean().item() <= 1e-4, (diff.max(), diff.mean())
    G = Hq // Hkv
    for kvh in (0, 3):
        L1 = OA.PoolLayout(1, P, D)
        opool = OA.new_pool(L1, case.num_pages)
        OA.append(opool, L1, case.page_table.numpy(), case.req.numpy(), case.pos.numpy(),
                  bits(case.k[:, kvh:kvh + 1]), bits(case.v[:, kvh:kvh + 1]))
        for i in BALANCE_ROWS:
            ref = OT.paged_decode(opool, L1, case.page_table.numpy(), [q_start + i + 1],
                                  bits(q[i:i + 1, kvh * G:(kvh + 1) * G]), 1 / 16)
            assert_attention_close(out[i:i + 1, kvh * G:(kvh + 1) * G], ref)


def test_prefill_poison_pages_never_leak():
    case = make_case(77, 8, 2, 128, 64, [300], num_pages=12)
    ref_pool = case.oracle_pool(fill=0xFF)
    pool = pool_from_numpy(case, ref_pool)
    from paper_2609_17475_gb300 import synth
    q = synth.normal_bf16(synth.generator(78), (100, 8, 128))
    out = gpu_prefill(case, pool, q, 200, True, 0.1)
    ref = OT.prefill_chunk(ref_pool, case.layout, case.page_table[0].numpy(), bits(q), 200, 0.1)
    assert_attention_close(out, ref)


def test_prefill_flags_groups_beyond_fp16_range():
    """A K group scaled far past the fp16 range sets JF_DEV_ERR_RANGE (the
    call still completes); the same cache without it leaves the status clear."""
    from paper_2609_17475_gb300 import synth
    case = make_case(91, 8, 2, 128, 64, [300])
    q = synth.normal_bf16(synth.generator(92), (40, 8, 128))
    out = gpu_prefill(case, pool_from_numpy(case, case.oracle_pool()), q, 260, True, 0.1)
    assert torch.isfinite(out.float()).all()
    big = case.k.clone()
    big[123, 1, 64:128] = (big[123, 1, 64:128].float() * 40000.0).to(torch.bfloat16)
    case.k = big
    pool = pool_from_numpy(case, case.oracle_pool())
    ws = torch.zeros(jf.jf_prefill_workspace_bytes(), dtype=torch.uint8, device=DEV)
    jf.jf_prefill_chunk_attn(pool, case.page_table[0].to(DEV), q.to(DEV), 260, 0.1, True,
                             torch.empty_like(q, device=DEV), ws)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == jf.binding.JF_DEV_ERR_RANGE


# --------------------------------------------------------------------------
# prefill chunks of several requests in one launch
# --------------------------------------------------------------------------
@pytest.mark.parametrize("Hq,Hkv,D,P,spans,causal,splits", [
    # (q_start, chunk_len) per request
    (24, 4, 256, 256, [(1000, 64), (0, 256), (4000, 130), (300, 0), (17, 1)], True, 1),
    (8, 2, 128, 64, [(70, 200), (0, 21), (500, 77)], True, 1),
    (24, 4, 256, 128, [(200, 64), (900, 33)], False, 1),
    # history splits: more splits than some query tiles have history tiles
    (24, 4, 256, 256, [(5000, 64), (0, 40), (2000, 300)], True, 7),
    (8, 2, 128, 64, [(3000, 21), (100, 130)], False, 3),
])
def test_prefill_batch_matches_oracle_and_single_calls(Hq, Hkv, D, P, spans, causal, splits):
    from paper_2609_17475_gb300 import synth
    totals = [qs + c for qs, c in spans]
    case = make_case(600 + sum(totals), Hq, Hkv, D, P, totals, outliers=True)
    ref_pool = case.oracle_pool()
    pool = pool_from_numpy(case, ref_pool)
    C = [c for _, c in spans]
    qs = [q for q, _ in spans]
    q = synth.normal_bf16(synth.generator(601), (sum(C), Hq, D))
    scale = 1 / math.sqrt(D)
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device=DEV)
    ws = jf.prefill_batch_workspace(sum(C), Hq, D, splits, device=DEV)
    ws[256:] = 0xFF    # NaN partials: every one the merge reads must be written
    jf.jf_prefill_batch_attn(pool, case.page_table.to(DEV), qs, C, q.to(DEV), scale, causal,
                             out, ws, num_splits=splits)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    row = 0
    for b, (q0, c) in enumerate(spans):
        if c:
            ref = OT.prefill_chunk(ref_pool, case.layout, case.page_table[b].numpy(),
                                   bits(q[row:row + c]), q0, scale, causal=causal)
            assert_attention_close(out[row:row + c], ref)
            one = torch.empty(c, Hq, D, dtype=torch.bfloat16, device=DEV)
            pws = torch.zeros(jf.jf_prefill_workspace_bytes(), dtype=torch.uint8, device=DEV)
            jf.jf_prefill_chunk_attn(pool, case.page_table[b].to(DEV), q[row:row + c].to(DEV),
                                     q0, scale, causal, one, pws)
            torch.cuda.synchronize()
            if splits == 1:
                assert torch.equal(one, out[row:row + c])   # same tiles, same arithmetic
            else:   # another summation order: at most one bf16 rounding step apart
                a, b2 = one.float(), out[row:row + c].float()
                assert ((a - b2).abs() <= 2 ** -7 * torch.maximum(a.abs(), b2.abs()) + 1e-3).all()
        row += c
