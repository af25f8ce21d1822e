"""GPU parity for the TQ4 format (Sec. 3.1 Eq. 4; App. A.1 Table 3): encode on
append bit-exact against the oracle (indices and fp16 norms), page-native
decode attention within tolerance of the fp64 oracle, checkpoint/restore byte
identity.  Every call goes through the C ABI (libjfkv.so)."""
import math

import numpy as np
import pytest
import torch

import paper_2609_17475_gb300 as jf
from oracle import attention as OT
from oracle import checkpoint as OC
from oracle import tq4 as OQ
from paper_2609_17475_gb300 import synth
from tests.cases import assert_attention_close, bits, make_case

pytestmark = pytest.mark.gpu
DEV = "cuda"


def signs(D):
    """Sign vectors for the CUDA path (seeded inputs; equal to the oracle's
    ``sign_vector`` by a CPU test)."""
    return synth.tq4_signs(synth.TQ4_SEED_K, D), synth.tq4_signs(synth.TQ4_SEED_V, D)


def oracle_codec(D):
    return OQ.make_codec(D, OQ.sign_vector(OQ.SEED_K, D), OQ.sign_vector(OQ.SEED_V, D))


def oracle_layout(case):
    return OQ.Tq4Layout(case.Hkv, case.P, case.D, oracle_codec(case.D))


def oracle_pool(case, fill=0):
    lay = oracle_layout(case)
    pool = OQ.new_pool(lay, case.num_pages, fill=fill)
    OQ.append(pool, lay, case.page_table.numpy(), case.req.numpy(), case.pos.numpy(),
              bits(case.k), bits(case.v))
    return lay, pool


def gpu_pool(case, fill=0):
    sk, sv = signs(case.D)
    return jf.KVPool.allocate(case.num_pages, case.P, case.Hkv, case.D, device=DEV, fill=fill,
                              format=jf.JF_FMT_TQ4, codec=jf.Tq4Codec(case.D, sk, sv))


def gpu_append(case, fill=0, k=None, v=None):
    pool = gpu_pool(case, fill)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_quantize_append(pool, case.page_table.to(DEV), case.req.to(DEV), case.pos.to(DEV),
                             (case.k if k is None else k).to(DEV),
                             (case.v if v is None else v).to(DEV), err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    return pool


def pool_from_numpy(case, arr):
    pool = gpu_pool(case, fill=None)
    pool.data.copy_(torch.from_numpy(arr))
    return pool


def gpu_decode(case, pool, splits, ctx=None):
    ctx = case.ctx if ctx is None else ctx
    B = len(ctx)
    out = torch.full((B, case.Hq, case.D), float("nan"), dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(B, case.Hq, case.Hkv, case.D, splits, device=DEV)
    ws[256:] = 0xFF    # NaN partials: rows past the split plan must never be used
    jf.jf_paged_decode_attn(pool, case.page_table.to(DEV),
                            torch.tensor(ctx, dtype=torch.int32, device=DEV), case.q.to(DEV),
                            1 / math.sqrt(case.D), out, ws, splits)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    return out


# --------------------------------------------------------------------------
# codebook: the library's construction equals the oracle's, bit for bit
# --------------------------------------------------------------------------
@pytest.mark.parametrize("D", [128, 256])
def test_tq4_codebook_bit_exact(D):
    assert np.array_equal(jf.jf_tq4_codebook(D), OQ.codebook(D))


# --------------------------------------------------------------------------
# encode on append: bit-exact against the oracle
# --------------------------------------------------------------------------
@pytest.mark.parametrize("Hkv,D,P,ctx,outliers", [
    (2, 128, 256, [256], False),
    (2, 128, 64, [1, 63, 130], False),
    (4, 256, 256, [1000, 517], True),
    (3, 256, 128, [300], True),
    (1, 256, 64, [2048], False),
])
def test_tq4_append_bit_exact(Hkv, D, P, ctx, outliers):
    case = make_case(300 + sum(ctx), 2 * Hkv, Hkv, D, P, ctx, outliers=outliers,
                     num_pages=sum(-(-c // P) for c in ctx) + 2)
    _, ref = oracle_pool(case, fill=0x5A)
    pool = gpu_append(case, fill=0x5A)
    assert np.array_equal(pool.data.cpu().numpy(), ref)


def test_tq4_append_special_vectors_bit_exact():
    """Zero vectors, one-hot vectors, norms past the fp16 range (saturated),
    tiny magnitudes, a 2^30 magnitude spread, signed zeros."""
    D, Hkv, P = 256, 2, 64
    n = 64
    rng = np.random.default_rng(5)
    x = rng.standard_normal((2, n, Hkv, D)).astype(np.float32)
    x[:, 0] = 0.0
    x[:, 1] = 0.0
    x[:, 1, :, 7] = -2.5                                   # one-hot
    x[:, 2] *= 5000.0                                      # norm ~80000 > 65504
    x[:, 3] *= 1e-20                                       # tiny
    x[:, 4, :, ::2] *= 2.0 ** -30                          # wide spread
    x[:, 5, :, ::3] = -0.0
    x[:, 6] = 1.0                                          # all equal
    kb = torch.from_numpy(x[0]).to(torch.bfloat16)
    vb = torch.from_numpy(x[1]).to(torch.bfloat16)
    case = make_case(9, 2 * Hkv, Hkv, D, P, [n], num_pages=2)
    case.k, case.v = kb, vb
    _, ref = oracle_pool(case, fill=0x11)
    pool = gpu_append(case, fill=0x11)
    assert np.array_equal(pool.data.cpu().numpy(), ref)


def test_tq4_append_many_rows_exercises_both_decision_paths():
    """8,192 vectors: some lie within 2^-15 rho of a threshold and take the
    exact fp64 path; all must match the oracle."""
    case = make_case(77, 8, 4, 256, 256, [1024], outliers=True)
    _, ref = oracle_pool(case)
    pool = gpu_append(case)
    assert np.array_equal(pool.data.cpu().numpy(), ref)


def test_tq4_append_close_thresholds_take_the_exact_path_everywhere():
    """A codebook with two thresholds closer than the fast path's margins:
    every index is decided in fp64, still bit-exact against the oracle."""
    D, Hkv = 256, 2
    c = OQ.codebook(D).copy()
    c[8] = np.float32(c[7] + np.float32(2e-7))            # c_7, c_8, c_9 within 4e-7:
    c[9] = np.float32(c[8] + np.float32(2e-7))            # t_7 and t_8 nearly equal
    assert np.all(np.diff(c) > 0)
    assert np.diff(np.float32(16) * OQ.thresholds(c)).min() < 2 ** -12
    sk, sv = signs(D)
    case = make_case(21, 2 * Hkv, Hkv, D, 64, [300], num_pages=6)
    lay = OQ.Tq4Layout(Hkv, 64, D, OQ.Codec(D, c, OQ.sign_vector(OQ.SEED_K, D),
                                            OQ.sign_vector(OQ.SEED_V, D)))
    ref = OQ.new_pool(lay, case.num_pages)
    OQ.append(ref, lay, case.page_table.numpy(), case.req.numpy(), case.pos.numpy(),
              bits(case.k), bits(case.v))
    pool = jf.KVPool.allocate(case.num_pages, 64, Hkv, D, device=DEV, format=jf.JF_FMT_TQ4,
                              codec=jf.Tq4Codec(D, sk, sv, centroids=c))
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_quantize_append(pool, case.page_table.to(DEV), case.req.to(DEV), case.pos.to(DEV),
                             case.k.to(DEV), case.v.to(DEV), err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    assert np.array_equal(pool.data.cpu().numpy(), ref)


def test_tq4_append_flags_bad_rows_and_skips_them():
    case = make_case(13, 8, 2, 128, 64, [100], num_pages=3)
    pool = gpu_pool(case, fill=0x77)
    before = pool.data.clone()
    pos = case.pos.clone()
    pos[5] = 10 ** 6                     # beyond the page-table row
    pt = case.page_table.clone()
    pt[0, 1] = 999                       # page id outside the pool
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_quantize_append(pool, pt.to(DEV), case.req.to(DEV), pos.to(DEV), case.k.to(DEV),
                             case.v.to(DEV), err)
    torch.cuda.synchronize()
    e = int(err.item())
    assert e & jf.binding.JF_DEV_ERR_POSITION and e & jf.binding.JF_DEV_ERR_PAGE_ID
    # rows 64..99 went to the bad page id and were skipped: the page they
    # would have used under the original table is untouched
    orig = int(case.page_table[0, 1])
    assert torch.equal(before[orig], pool.data[orig])


# --------------------------------------------------------------------------
# checkpoint / restore
# --------------------------------------------------------------------------
def test_tq4_checkpoint_and_restore_bit_exact():
    case = make_case(17, 8, 4, 256, 128, [1500], num_pages=15)
    _, ref = oracle_pool(case, fill=0x33)
    pool = pool_from_numpy(case, ref)
    n = -(-1500 // 128)
    blob = torch.empty(n * pool.page_bytes, dtype=torch.uint8, device=DEV)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_checkpoint(pool, case.page_table[0].to(DEV), n, blob, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    want = OC.checkpoint(ref, case.page_table[0].numpy(), n)
    assert np.array_equal(blob.cpu().numpy(), want)
    fresh = gpu_pool(case, fill=0)
    jf.jf_kv_restore(fresh, case.page_table[0].to(DEV), n, blob, err)
    torch.cuda.synchronize()
    exp = np.zeros_like(ref)
    OC.restore(exp, case.page_table[0].numpy(), n, want)
    assert np.array_equal(fresh.data.cpu().numpy(), exp)


# --------------------------------------------------------------------------
# decode attention
# --------------------------------------------------------------------------
@pytest.mark.parametrize("Hq,Hkv,D,P,ctx,splits,outliers", [
    (8, 2, 128, 256, [4096], 1, False),            # tiny geometry, one split
    (8, 2, 128, 256, [4096], 8, False),            # split-K + merge
    (8, 2, 128, 64, [1, 33, 517, 2000], 4, False),  # ragged batch, partial pages
    (24, 4, 256, 256, [5000], 3, True),            # paper geometry, outliers
    (24, 4, 256, 128, [777, 1], 16, True),
    (4, 4, 256, 64, [1500], 2, False),             # G = 1
    (16, 2, 256, 256, [2500], 5, False),           # G = 8
    (8, 2, 128, 256, [70000, 3000], 150, False),   # > 128 live splits
    (24, 4, 256, 128, [9000, 0, 40], 3, True),     # batch plan with an empty request
])
def test_tq4_decode_matches_oracle(Hq, Hkv, D, P, ctx, splits, outliers):
    case = make_case(400 + Hq + sum(ctx), Hq, Hkv, D, P, ctx, outliers=outliers)
    lay, ref_pool = oracle_pool(case)
    pool = pool_from_numpy(case, ref_pool)
    out = gpu_decode(case, pool, splits)
    ref = OT.paged_decode(ref_pool, lay, case.page_table.numpy(), ctx, bits(case.q),
                          1 / math.sqrt(D))
    assert_attention_close(out, ref)


def test_tq4_decode_edge_contexts():
    case = make_case(6, 8, 2, 128, 64, [0, 1, 64, 65])
    lay, ref_pool = oracle_pool(case)
    pool = pool_from_numpy(case, ref_pool)
    for splits in (1, 4):
        out = gpu_decode(case, pool, splits)
        assert (out[0].float() == 0).all()
        ref = OT.paged_decode(ref_pool, lay, case.page_table.numpy(), case.ctx, bits(case.q),
                              1 / math.sqrt(128))
        assert_attention_close(out, ref)
        v0 = OT.gather_head(ref_pool, lay, case.page_table.numpy()[1], 1, 0, OQ.KIND_V)[0]
        assert np.abs(out[1, 0].float().cpu().numpy() - v0).max() <= 2 ** -7 * np.abs(v0).max()


def test_tq4_decode_poison_pages_and_tail_never_leak():
    """0xFF bytes (fp16 norm NaN) in unwritten pages and tail slots stay out."""
    case = make_case(62, 8, 2, 128, 64, [200], num_pages=10)
    lay, ref_pool = oracle_pool(case, fill=0xFF)
    pool = pool_from_numpy(case, ref_pool)
    out = gpu_decode(case, pool, 2)
    ref = OT.paged_decode(ref_pool, lay, case.page_table.numpy(), case.ctx, bits(case.q),
                          1 / math.sqrt(128))
    assert_attention_close(out, ref)


def test_tq4_decode_after_gpu_append_and_split_invariance():
    case = make_case(81, 24, 4, 256, 256, [12000], outliers=True)
    lay, ref_pool = oracle_pool(case)
    pool = gpu_append(case)
    assert np.array_equal(pool.data.cpu().numpy(), ref_pool)
    ref = OT.paged_decode(ref_pool, lay, case.page_table.numpy(), case.ctx, bits(case.q), 1 / 16)
    outs = [gpu_decode(case, pool, s) for s in (1, 2, 7, 38)]
    for o in outs:
        assert_attention_close(o, ref)


def test_tq4_no_workspace_decode_is_rejected():
    case = make_case(3, 8, 2, 128, 64, [100])
    pool = gpu_pool(case)
    q = torch.zeros(1, 8, 128, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(jf.JfError) as e:
        jf.jf_paged_decode_attn_noalloc(pool, case.page_table.to(DEV),
                                        torch.tensor([100], dtype=torch.int32, device=DEV), q,
                                        0.1, torch.empty_like(q), 2)
    assert e.value.status == jf.binding.JF_ERR_UNSUPPORTED


@pytest.mark.parametrize("Hq,Hkv,D,P,ctx,L,splits", [
    (24, 4, 256, 256, [5000], 2, None),
    (24, 4, 256, 128, [3000, 40], 4, None),       # G * L = 24: 3 n-tiles, batch plan
    (8, 2, 128, 64, [700], 3, 5),
    (16, 2, 256, 256, [2100, 4], 4, 3),           # G * L = 32; a context of exactly q_len
    (24, 4, 256, 64, [9000], 3, 1),               # one split written directly, 70 chunks per pair
    (14, 2, 128, 128, [6000], 4, 1),              # G = 7, D = 128: 28 rows, two CTAs (3 + 1 groups)
    (8, 4, 128, 64, [500, 33], 4, 2),             # 8 rows: one group (one CTA per n-tile kernel)
])
def test_tq4_verifier_matches_oracle(Hq, Hkv, D, P, ctx, L, splits):
    case = make_case(900 + sum(ctx) + L, Hq, Hkv, D, P, ctx)
    lay, ref_pool = oracle_pool(case)
    pool = pool_from_numpy(case, ref_pool)
    B = len(ctx)
    q = synth.normal_bf16(synth.generator(910 + L), (B, L, Hq, D))
    if splits is None:
        splits = jf.default_verify_splits(B, L, Hq, Hkv, format=jf.JF_FMT_TQ4)
    ws = jf.verify_workspace(B, L, Hq, Hkv, D, splits, device=DEV)
    ws[256:] = 0xFF
    out = torch.full((B, L, Hq, D), float("nan"), dtype=torch.bfloat16, device=DEV)
    scale = 1 / math.sqrt(D)
    jf.jf_paged_verify_attn(pool, case.page_table.to(DEV),
                            torch.tensor(ctx, dtype=torch.int32, device=DEV), q.to(DEV), scale,
                            out, ws, splits)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    ref = np.stack([OT.prefill_chunk(ref_pool, lay, case.page_table[b].numpy(), bits(q[b]),
                                     ctx[b] - L, scale) for b in range(B)])
    assert_attention_close(out, ref)


def test_tq4_verifier_warp_pairs_are_deterministic():
    """Repeated TQ4 verifier calls on the same inputs give the same bits (the
    warp pairs' per-chunk exchange of partial dot products)."""
    case = make_case(4444, 24, 4, 256, 64, [6000, 2500])
    _, ref_pool = oracle_pool(case)
    pool = pool_from_numpy(case, ref_pool)
    q = synth.normal_bf16(synth.generator(4545), (2, 3, 24, 256)).to(DEV)
    ws = jf.verify_workspace(2, 3, 24, 4, 256, 4, device=DEV)
    ctx = torch.tensor(case.ctx, dtype=torch.int32, device=DEV)
    outs = []
    for _ in range(3):
        out = torch.empty(2, 3, 24, 256, dtype=torch.bfloat16, device=DEV)
        jf.jf_paged_verify_attn(pool, case.page_table.to(DEV), ctx, q, 1 / 16, out, ws, 4)
        outs.append(out)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


def test_tq4_verifier_with_one_token_is_decode():
    case = make_case(78, 24, 4, 256, 256, [3333, 1234])
    _, ref_pool = oracle_pool(case)
    pool = pool_from_numpy(case, ref_pool)
    out_d = gpu_decode(case, pool, 9)
    ws = jf.verify_workspace(2, 1, 24, 4, 256, 9, device=DEV)
    out_v = torch.empty((2, 1, 24, 256), dtype=torch.bfloat16, device=DEV)
    jf.jf_paged_verify_attn(pool, case.page_table.to(DEV),
                            torch.tensor(case.ctx, dtype=torch.int32, device=DEV),
                            case.q.view(2, 1, 24, 256).to(DEV), 1 / 16, out_v, ws, 9)
    torch.cuda.synchronize()
    assert torch.equal(out_v.view(2, 24, 256), out_d)


@pytest.mark.parametrize("Hq,Hkv,D,P,ctx,splits", [
    (24, 4, 256, 256, [5000, 257, 1], 38),   # new rows mid-page, at slot 0 of a page, alone
    (8, 2, 128, 64, [64, 65, 999], 4),
    (16, 2, 256, 128, [3000], 1),            # one split writes and reads directly
])
def test_tq4_fused_append_decode_equals_append_then_decode(Hq, Hkv, D, P, ctx, splits):
    case = make_case(950 + sum(ctx), Hq, Hkv, D, P, ctx)
    lay = oracle_layout(case)
    req, pos = case.req.numpy(), case.pos.numpy()
    last = np.array([np.nonzero(req == b)[0].max() for b in range(len(ctx))])
    keep = np.setdiff1d(np.arange(len(req)), last)
    prefix = OQ.new_pool(lay, case.num_pages, fill=0xFF)
    OQ.append(prefix, lay, case.page_table.numpy(), req[keep], pos[keep], bits(case.k[keep]),
              bits(case.v[keep]))
    full = OQ.new_pool(lay, case.num_pages, fill=0xFF)
    OQ.append(full, lay, case.page_table.numpy(), req, pos, bits(case.k), bits(case.v))
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
    assert np.array_equal(pool_b.data.cpu().numpy(), full)       # bit-exact encode on append
    assert torch.equal(out_a, out_b)
    ref = OT.paged_decode(full, lay, case.page_table.numpy(), ctx, bits(case.q), scale)
    assert_attention_close(out_b, ref)


def test_tq4_decode_full_window_256k_one_head():
    """The 256K full-window workload (24/4/256, 1,024 pages in a random physical
    order, K outlier channels) in TQ4 at full size and in the benchmark's launch
    shape; KV head 2 checked against the oracle, bytes of sampled pages too,
    then the packed verifier (4 tokens, warp pairs) on the same pages."""
    w = synth.WORKLOADS["full_window_256k"]
    geo = w["geometry"]
    ctx = w["context_lens"][0]
    gen = synth.generator(w["seed"])
    channels = synth.outlier_channels(gen, geo.num_kv_heads, geo.head_dim)
    k, v = synth.kv_rows(gen, ctx, geo.num_kv_heads, geo.head_dim, channels)
    pt, npages = synth.page_tables(gen, [ctx], geo.page_size)
    q = synth.normal_bf16(gen, (1, geo.num_q_heads, geo.head_dim))
    req, pos = synth.append_rows_for([ctx])
    sk, sv = signs(geo.head_dim)
    pool = jf.KVPool.allocate(npages, geo.page_size, geo.num_kv_heads, geo.head_dim, device=DEV,
                              format=jf.JF_FMT_TQ4, codec=jf.Tq4Codec(geo.head_dim, sk, sv))
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    jf.jf_kv_quantize_append(pool, pt.to(DEV), req.to(DEV), pos.to(DEV), k.to(DEV), v.to(DEV), err)
    splits = jf.default_num_splits(1, geo.num_kv_heads, format=jf.JF_FMT_TQ4)
    out = torch.empty(1, geo.num_q_heads, geo.head_dim, dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(1, geo.num_q_heads, geo.num_kv_heads, geo.head_dim, splits, device=DEV)
    scale = 1 / math.sqrt(geo.head_dim)
    jf.jf_paged_decode_attn(pool, pt.to(DEV), torch.tensor([ctx], dtype=torch.int32, device=DEV),
                            q.to(DEV), scale, out, ws, splits)
    torch.cuda.synchronize()
    assert int(err.item()) == 0 and jf.workspace_status(ws) == 0
    G, kvh = geo.group, 2
    L1 = OQ.Tq4Layout(1, geo.page_size, geo.head_dim, oracle_codec(geo.head_dim))
    opool = OQ.new_pool(L1, npages)
    OQ.append(opool, L1, pt.numpy(), req.numpy(), pos.numpy(),
              bits(k[:, kvh:kvh + 1]), bits(v[:, kvh:kvh + 1]))
    ref = OT.paged_decode(opool, L1, pt.numpy(), [ctx], bits(q[:, kvh * G:(kvh + 1) * G]), scale)
    assert_attention_close(out[:, kvh * G:(kvh + 1) * G], ref)
    gp = pool.data.cpu().numpy()
    L4 = OQ.Tq4Layout(geo.num_kv_heads, geo.page_size, geo.head_dim, L1.codec)
    for page in pt[0, [0, 511, 1023]].tolist():
        for kind in (OQ.KIND_K, OQ.KIND_V):
            o4, o1 = L4.codes_offset(kind, kvh, 0), L1.codes_offset(kind, 0, 0)
            n = geo.page_size * L4.code_bytes
            assert np.array_equal(gp[page, o4:o4 + n], opool[page, o1:o1 + n])
            o4, o1 = L4.norm_offset(kind, kvh, 0), L1.norm_offset(kind, 0, 0)
            assert np.array_equal(gp[page, o4:o4 + 2 * geo.page_size],
                                  opool[page, o1:o1 + 2 * geo.page_size])
    # packed verifier: tokens ctx - 4 .. ctx - 1 against the oracle's causal chunk
    Lq = 4
    qv = synth.normal_bf16(gen, (1, Lq, geo.num_q_heads, geo.head_dim))
    sv = jf.default_verify_splits(1, Lq, geo.num_q_heads, geo.num_kv_heads,
                                  format=jf.JF_FMT_TQ4)
    wv = jf.verify_workspace(1, Lq, geo.num_q_heads, geo.num_kv_heads, geo.head_dim, sv,
                             device=DEV)
    ov = torch.empty(1, Lq, geo.num_q_heads, geo.head_dim, dtype=torch.bfloat16, device=DEV)
    jf.jf_paged_verify_attn(pool, pt.to(DEV), torch.tensor([ctx], dtype=torch.int32, device=DEV),
                            qv.to(DEV), scale, ov, wv, sv)
    torch.cuda.synchronize()
    assert jf.workspace_status(wv) == 0
    ref_v = OT.prefill_chunk(opool, L1, pt[0].numpy(), bits(qv[0, :, kvh * G:(kvh + 1) * G]),
                             ctx - Lq, scale)
    assert_attention_close(ov[0, :, kvh * G:(kvh + 1) * G], ref_v)


def test_tq4_prefill_wave_balanced_chunk():
    """2,048 queries after 30,720 TQ4 positions (24/4/256, P 256): 196 CTA
    pairs, not whole waves, and the TQ4 minimum workspace already holds the
    balanced form (whole waves, then a tail with split histories), so the
    plain call runs it; sampled rows against the oracle's decode."""
    Hq, Hkv, D, P, C = 24, 4, 256, 256, 2048
    q_start = 32768 - C
    slots = torch.cuda.get_device_properties(0).multi_processor_count // 2
    pairs = Hkv * -(-C // 42)
    if pairs <= slots or pairs % slots == 0:
        pytest.skip("the chunk fills whole waves on this GPU")
    case = make_case(408, Hq, Hkv, D, P, [32768])
    pool = gpu_append(case)
    q = synth.normal_bf16(synth.generator(409), (C, Hq, D))
    ws = jf.prefill_batch_workspace(C, Hq, D, 1, device=DEV, format=jf.JF_FMT_TQ4)
    assert jf.jf_prefill_chunk_workspace_bytes(pool, q_start, C, Hq) == ws.numel()
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device=DEV)
    jf.jf_prefill_chunk_attn(pool, case.page_table[0].to(DEV), q.to(DEV), q_start, 1 / 16, True,
                             out, ws)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    assert torch.isfinite(out.float()).all()
    sk, sv = signs(D)
    G = Hq // Hkv
    L1 = OQ.Tq4Layout(1, P, D, oracle_codec(D))
    for kvh in (1, 2):
        opool = OQ.new_pool(L1, case.num_pages)
        OQ.append(opool, L1, case.page_table.numpy(), case.req.numpy(), case.pos.numpy(),
                  bits(case.k[:, kvh:kvh + 1]), bits(case.v[:, kvh:kvh + 1]))
        for i in (0, 1511, 1512, 1553, 1554, 1595, 1596, 1597, 2047):
            ref = OT.paged_decode(opool, L1, case.page_table.numpy(), [q_start + i + 1],
                                  bits(q[i:i + 1, kvh * G:(kvh + 1) * G]), 1 / 16)
            assert_attention_close(out[i:i + 1, kvh * G:(kvh + 1) * G], ref)


# --------------------------------------------------------------------------
# prefill chunk attention over TQ4 pages
# --------------------------------------------------------------------------
@pytest.mark.parametrize("Hq,Hkv,D,P,q_start,C,causal", [
    (8, 2, 128, 256, 0, 256, True),
    (8, 2, 128, 64, 300, 77, True),
    (24, 4, 256, 256, 1000, 130, True),
    (24, 4, 256, 128, 517, 200, False),
    (4, 4, 256, 64, 100, 129, True),      # G = 1
])
def test_tq4_prefill_matches_oracle(Hq, Hkv, D, P, q_start, C, causal):
    total = q_start + C
    case = make_case(700 + Hq + total, Hq, Hkv, D, P, [total], outliers=True)
    lay, ref_pool = oracle_pool(case)
    pool = pool_from_numpy(case, ref_pool)
    q = synth.normal_bf16(synth.generator(8 + C), (C, Hq, D))
    scale = 1 / math.sqrt(D)
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device=DEV)
    ws = jf.prefill_batch_workspace(C, Hq, D, 1, device=DEV, format=jf.JF_FMT_TQ4)
    jf.jf_prefill_chunk_attn(pool, case.page_table[0].to(DEV), q.to(DEV), q_start, scale, causal,
                             out, ws)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    ref = OT.prefill_chunk(ref_pool, lay, case.page_table[0].numpy(), bits(q), q_start, scale,
                           causal=causal)
    assert_attention_close(out, ref)


@pytest.mark.parametrize("total", [1, 65, 257, 450, 833])
def test_tq4_prefill_history_tile_counts(total):
    """1 to 14 history tiles on the TQ4 instance (three V buffers): a lone
    last tile of a pair, buffers reused several times."""
    Hq, Hkv, D, P = 24, 4, 256, 256
    C = min(total, 24)
    case = make_case(750 + total, Hq, Hkv, D, P, [total], outliers=True)
    lay, ref_pool = oracle_pool(case)
    pool = pool_from_numpy(case, ref_pool)
    q = synth.normal_bf16(synth.generator(9 + total), (C, Hq, D))
    scale = 1 / math.sqrt(D)
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device=DEV)
    ws = jf.prefill_batch_workspace(C, Hq, D, 1, device=DEV, format=jf.JF_FMT_TQ4)
    jf.jf_prefill_chunk_attn(pool, case.page_table[0].to(DEV), q.to(DEV), total - C, scale, True,
                             out, ws)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    ref = OT.prefill_chunk(ref_pool, lay, case.page_table[0].numpy(), bits(q), total - C, scale,
                           causal=True)
    assert_attention_close(out, ref)


@pytest.mark.parametrize("spans,splits", [
    ([(3000, 64), (0, 40), (700, 150)], 1),
    ([(3000, 64), (0, 40), (700, 150)], 5),
])
def test_tq4_prefill_batch_with_splits_matches_oracle(spans, splits):
    Hq, Hkv, D, P = 24, 4, 256, 256
    totals = [a + c for a, c in spans]
    case = make_case(800 + splits, Hq, Hkv, D, P, totals)
    lay, ref_pool = oracle_pool(case)
    pool = pool_from_numpy(case, ref_pool)
    C = [c for _, c in spans]
    qs = [a for a, _ in spans]
    q = synth.normal_bf16(synth.generator(801), (sum(C), Hq, D))
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device=DEV)
    ws = jf.prefill_batch_workspace(sum(C), Hq, D, splits, device=DEV, format=jf.JF_FMT_TQ4)
    ws[256:] = 0xFF
    jf.jf_prefill_batch_attn(pool, case.page_table.to(DEV), qs, C, q.to(DEV), 1 / 16, True, out,
                             ws, num_splits=splits)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    row = 0
    for b, (a0, c) in enumerate(spans):
        ref = OT.prefill_chunk(ref_pool, lay, case.page_table[b].numpy(), bits(q[row:row + c]), a0,
                               1 / 16)
        assert_attention_close(out[row:row + c], ref)
        row += c
