"""Pins for the oracle's paged decode, split merge, prefill chunk and checkpoint.

Independent anchors:
* exactly quantizable K/V (every group is bias + c * 2^e), so the pool holds the
  original values and the paged oracle must agree with torch's
  scaled_dot_product_attention on the dense fp64 values (GQA, softmax scale,
  page-table indirection and layout all checked at once);
* closed forms: constant K -> mean of V; ctx = 1 -> V_0; a dominant logit;
* a pure-Python brute-force loop on tiny inputs;
* invariants: page permutation (bitwise), split count, head subset (bitwise),
  GQA head grouping, causal prefill row i == decode at ctx q_start + i + 1;
* checkpoint byte identity and restore round trip.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import affine4 as A
from oracle import attention as T
from oracle import checkpoint as C
from tests.helpers import bf16_bits, exact_groups, f64_to_bf16_tensor


def _pool_from_dense(L, k, v, ctx_list, rng, num_pages=None, fill=0):
    """Append dense bf16 K/V rows ([B][ctx, Hkv, D] bits) into a pool with a
    shuffled page assignment.  Returns pool, page_table."""
    P = L.page_size
    need = [-(-c // P) for c in ctx_list]
    total = sum(need)
    num_pages = num_pages or total + 3
    perm = rng.permutation(num_pages)
    pt = np.full((len(ctx_list), max(max(need), 1)), -1, dtype=np.int32)
    off = 0
    for b, n in enumerate(need):
        pt[b, :n] = perm[off:off + n]
        off += n
    pool = A.new_pool(L, num_pages, fill=fill)
    for b, c in enumerate(ctx_list):
        if c == 0:
            continue
        A.append(pool, L, pt, np.full(c, b, np.int32), np.arange(c, dtype=np.int32), k[b], v[b])
    return pool, pt


def _exact_case(seed, B, Hq, Hkv, D, P, ctx_list):
    rng = np.random.default_rng(seed)
    L = A.PoolLayout(Hkv, P, D)
    kd = [exact_groups(rng, (c, Hkv, D)) for c in ctx_list]
    vd = [exact_groups(rng, (c, Hkv, D)) for c in ctx_list]
    kb = [bf16_bits(f64_to_bf16_tensor(x)) for x in kd]
    vb = [bf16_bits(f64_to_bf16_tensor(x)) for x in vd]
    pool, pt = _pool_from_dense(L, kb, vb, ctx_list, rng)
    q = torch.randn(B, Hq, D, generator=torch.Generator().manual_seed(seed)).to(torch.bfloat16)
    return L, pool, pt, kd, vd, q


def _sdpa_ref(q_bf16, kd, vd, ctx_list, Hq, Hkv, scale):
    """torch SDPA over dense fp64 values, one request at a time."""
    G = Hq // Hkv
    out = []
    for b, c in enumerate(ctx_list):
        qb = q_bf16[b].to(torch.float64)[:, None, :]                       # [Hq, 1, D]
        k = torch.from_numpy(kd[b]).permute(1, 0, 2).repeat_interleave(G, 0)  # [Hq, c, D]
        v = torch.from_numpy(vd[b]).permute(1, 0, 2).repeat_interleave(G, 0)
        out.append(F.scaled_dot_product_attention(qb, k, v, scale=scale)[:, 0].numpy())
    return np.stack(out)


@pytest.mark.parametrize("Hq,Hkv,D,P,ctx", [
    (8, 2, 128, 64, [300, 64, 1]),
    (24, 4, 256, 256, [700]),
    (6, 6, 128, 128, [129, 5]),
])
def test_decode_matches_sdpa_on_exact_values(Hq, Hkv, D, P, ctx):
    L, pool, pt, kd, vd, q = _exact_case(11, len(ctx), Hq, Hkv, D, P, ctx)
    scale = 1 / math.sqrt(D)
    ours = T.paged_decode(pool, L, pt, ctx, bf16_bits(q), scale)
    ref = _sdpa_ref(q, kd, vd, ctx, Hq, Hkv, scale)
    np.testing.assert_allclose(ours, ref, rtol=1e-11, atol=1e-12)


def test_constant_k_gives_mean_of_v():
    rng = np.random.default_rng(2)
    L = A.PoolLayout(2, 64, 128)
    ctx = 200
    krow = exact_groups(rng, (1, 2, 128))
    kd = np.repeat(krow, ctx, axis=0)
    vd = exact_groups(rng, (ctx, 2, 128))
    pool, pt = _pool_from_dense(L, [bf16_bits(f64_to_bf16_tensor(kd))],
                                [bf16_bits(f64_to_bf16_tensor(vd))], [ctx], rng)
    q = torch.randn(1, 4, 128).to(torch.bfloat16)
    out = T.paged_decode(pool, L, pt, [ctx], bf16_bits(q), 0.3)
    for h in range(4):
        np.testing.assert_allclose(out[0, h], vd[:, h // 2].mean(axis=0), rtol=0, atol=1e-12)


def test_single_position_returns_v0_and_empty_context_is_zero():
    L, pool, pt, kd, vd, q = _exact_case(4, 2, 4, 2, 128, 64, [1, 0])
    out = T.paged_decode(pool, L, pt, [1, 0], bf16_bits(q), 0.1)
    for h in range(4):
        assert np.array_equal(out[0, h], vd[0][0, h // 2])
    assert (out[1] == 0).all()


def test_dominant_logit_selects_its_row():
    rng = np.random.default_rng(8)
    L = A.PoolLayout(1, 64, 128)
    ctx = 90
    kd = rng.standard_normal((ctx, 1, 128)) * 0.01
    qv = np.sign(rng.standard_normal(128))
    kd[37, 0] = qv * 4.0                                   # aligned with q, large
    vd = exact_groups(rng, (ctx, 1, 128))
    kb = bf16_bits(torch.from_numpy(kd).to(torch.bfloat16))
    pool, pt = _pool_from_dense(L, [kb], [bf16_bits(f64_to_bf16_tensor(vd))], [ctx], rng)
    q = f64_to_bf16_tensor(qv[None, None, :])
    out = T.paged_decode(pool, L, pt, [ctx], bf16_bits(q), 1.0)
    np.testing.assert_allclose(out[0, 0], vd[37, 0], rtol=0, atol=1e-12)


def test_brute_force_tiny():
    """Pure-Python loops over positions and dims (no NumPy linear algebra)."""
    L, pool, pt, kd, vd, q = _exact_case(21, 1, 4, 2, 128, 64, [7])
    scale = 0.125
    qf = q.to(torch.float64).numpy()
    ours = T.paged_decode(pool, L, pt, [7], bf16_bits(q), scale)
    for h in range(4):
        kv = h // 2
        logits = []
        for t in range(7):
            acc = 0.0
            for d in range(128):
                acc += float(qf[0, h, d]) * float(kd[0][t, kv, d])
            logits.append(scale * acc)
        m = max(logits)
        w = [math.exp(s - m) for s in logits]
        z = sum(w)
        for d in range(128):
            o = sum(w[t] * float(vd[0][t, kv, d]) for t in range(7)) / z
            assert abs(o - ours[0, h, d]) <= 1e-12 * (1 + abs(o))


def _random_pool(seed, Hq, Hkv, D, P, ctx_list, outliers=False, num_pages=None):
    g = torch.Generator().manual_seed(seed)
    rng = np.random.default_rng(seed)
    L = A.PoolLayout(Hkv, P, D)
    kb, vb = [], []
    for c in ctx_list:
        k = torch.randn(c, Hkv, D, generator=g)
        if outliers:
            k[:, :, :4] *= 20
        kb.append(bf16_bits(k.to(torch.bfloat16)))
        vb.append(bf16_bits(torch.randn(c, Hkv, D, generator=g).to(torch.bfloat16)))
    pool, pt = _pool_from_dense(L, kb, vb, ctx_list, rng, num_pages=num_pages)
    q = torch.randn(len(ctx_list), Hq, D, generator=g).to(torch.bfloat16)
    return L, pool, pt, bf16_bits(q), kb, vb


def test_random_decode_matches_sdpa_on_dequantized_values():
    Hq, Hkv, D, P, ctx = 8, 2, 256, 128, [333, 1000]
    L, pool, pt, qb, kb, vb = _random_pool(5, Hq, Hkv, D, P, ctx, outliers=True)
    scale = 1 / 16
    ours = T.paged_decode(pool, L, pt, ctx, qb, scale)
    q = torch.from_numpy(qb.view(np.int16)).view(torch.bfloat16)
    kd = [A.decode_vectors(*A.encode_vectors(x)) for x in kb]       # dense dequantized rows
    vd = [A.decode_vectors(*A.encode_vectors(x)) for x in vb]
    ref = _sdpa_ref(q, kd, vd, ctx, Hq, Hkv, scale)
    np.testing.assert_allclose(ours, ref, rtol=1e-11, atol=1e-12)


def test_page_permutation_invariance_is_exact():
    Hq, Hkv, D, P, ctx = 8, 2, 128, 64, [500]
    L, pool, pt, qb, _, _ = _random_pool(7, Hq, Hkv, D, P, ctx, num_pages=12)
    rng = np.random.default_rng(1)
    perm = rng.permutation(12)                    # move every page somewhere else
    pool2 = np.empty_like(pool)
    pool2[perm] = pool
    pt2 = pt.copy()
    pt2[0, :8] = perm[pt[0, :8]]
    a = T.paged_decode(pool, L, pt, ctx, qb, 0.1)
    b = T.paged_decode(pool2, L, pt2, ctx, qb, 0.1)
    assert np.array_equal(a, b)


def test_page_size_invariance_is_exact():
    """The same logical rows in pools of 64-, 128- and 256-position pages
    (each with its own shuffled page order) give bitwise the same output."""
    Hq, Hkv, D, ctx = 8, 2, 256, [700, 130]
    rng = np.random.default_rng(21)
    kb = [bf16_bits(torch.randn(c, Hkv, D, generator=torch.Generator().manual_seed(c))
                    .to(torch.bfloat16)) for c in ctx]
    vb = [bf16_bits(torch.randn(c, Hkv, D, generator=torch.Generator().manual_seed(c + 1))
                    .to(torch.bfloat16)) for c in ctx]
    qb = bf16_bits(torch.randn(len(ctx), Hq, D, generator=torch.Generator().manual_seed(3))
                   .to(torch.bfloat16))
    outs = []
    for P in (64, 128, 256):
        L = A.PoolLayout(Hkv, P, D)
        pool, pt = _pool_from_dense(L, kb, vb, ctx, rng)
        outs.append(T.paged_decode(pool, L, pt, ctx, qb, 1 / 16))
    assert np.array_equal(outs[0], outs[1]) and np.array_equal(outs[0], outs[2])


@pytest.mark.parametrize("splits", [1, 2, 3, 7, 64])
def test_split_merge_equals_plain_softmax(splits):
    Hq, Hkv, D, P, ctx = 4, 2, 128, 64, [257, 40]
    L, pool, pt, qb, _, _ = _random_pool(9, Hq, Hkv, D, P, ctx)
    a = T.paged_decode(pool, L, pt, ctx, qb, 0.2)
    b = T.paged_decode_split(pool, L, pt, ctx, qb, 0.2, splits)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-13)


def test_split_bounds_cover_exactly():
    for ctx in [1, 5, 64, 1000]:
        for s in [1, 3, 32, 2000]:
            bounds = T.split_bounds(ctx, s)
            assert bounds[0][0] == 0 and bounds[-1][1] == ctx
            assert all(b[1] == c[0] for b, c in zip(bounds, bounds[1:]))


def test_head_subset_is_bitwise_identical_and_gqa_grouping():
    Hq, Hkv, D, P, ctx = 6, 3, 128, 64, [150]
    L, pool, pt, qb, kb, vb = _random_pool(13, Hq, Hkv, D, P, ctx)
    full = T.paged_decode(pool, L, pt, ctx, qb, 0.1)
    part = T.paged_decode(pool, L, pt, ctx, qb, 0.1, heads=[2, 3])
    assert np.array_equal(full[:, 2:4], part[:, 2:4]) and (part[:, :2] == 0).all()
    # query head h uses KV head h // 2: rebuild each KV head as its own 1-head pool
    for kv in range(Hkv):
        L1 = A.PoolLayout(1, P, D)
        rng = np.random.default_rng(0)
        pool1, pt1 = _pool_from_dense(L1, [kb[0][:, kv:kv + 1]], [vb[0][:, kv:kv + 1]], ctx, rng)
        one = T.paged_decode(pool1, L1, pt1, ctx, qb[:, 2 * kv:2 * kv + 2], 0.1)
        np.testing.assert_allclose(one, full[:, 2 * kv:2 * kv + 2], rtol=1e-13, atol=1e-14)


@pytest.mark.parametrize("q_start,Cq", [(0, 40), (100, 70), (64, 64)])
def test_prefill_rows_equal_decode_and_sdpa(q_start, Cq):
    Hq, Hkv, D, P = 4, 2, 128, 64
    total = q_start + Cq
    L, pool, pt, _, kb, vb = _random_pool(17, Hq, Hkv, D, P, [total])
    g = torch.Generator().manual_seed(3)
    q = torch.randn(Cq, Hq, D, generator=g).to(torch.bfloat16)
    qb = bf16_bits(q)
    scale = 0.09
    out = T.prefill_chunk(pool, L, pt[0], qb, q_start, scale, causal=True)
    for i in [0, Cq // 2, Cq - 1]:
        dec = T.paged_decode(pool, L, pt, [q_start + i + 1], qb[i][None], scale)
        np.testing.assert_allclose(out[i], dec[0], rtol=1e-12, atol=1e-13)
    # library reference with an explicit offset-causal mask
    kd = torch.from_numpy(A.decode_vectors(*A.encode_vectors(kb[0]))).permute(1, 0, 2)
    vd = torch.from_numpy(A.decode_vectors(*A.encode_vectors(vb[0]))).permute(1, 0, 2)
    kd = kd.repeat_interleave(2, 0)
    vd = vd.repeat_interleave(2, 0)
    mask = torch.arange(total)[None, :] <= (q_start + torch.arange(Cq))[:, None]
    ref = F.scaled_dot_product_attention(q.to(torch.float64).permute(1, 0, 2), kd, vd,
                                         attn_mask=mask, scale=scale).permute(1, 0, 2)
    np.testing.assert_allclose(out, ref.numpy(), rtol=1e-11, atol=1e-12)
    nc = T.prefill_chunk(pool, L, pt[0], qb, q_start, scale, causal=False)
    ref2 = F.scaled_dot_product_attention(q.to(torch.float64).permute(1, 0, 2), kd, vd,
                                          scale=scale).permute(1, 0, 2)
    np.testing.assert_allclose(nc, ref2.numpy(), rtol=1e-11, atol=1e-12)


def test_checkpoint_bytes_and_restore_round_trip():
    L, pool, pt, _, _, _ = _random_pool(19, 4, 2, 128, 64, [300, 100], num_pages=9)
    n = 5
    blob = C.checkpoint(pool, pt[0], n)
    assert blob.shape == (n * L.page_bytes,)
    for k in range(n):
        assert np.array_equal(blob[k * L.page_bytes:(k + 1) * L.page_bytes], pool[pt[0, k]])
    fresh = A.new_pool(L, 9, fill=0x5A)
    C.restore(fresh, pt[0], n, blob)
    for k in range(n):
        assert np.array_equal(fresh[pt[0, k]], pool[pt[0, k]])
    assert C.checkpoint(pool, pt[0], 0).shape == (0,)
