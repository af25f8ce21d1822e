"""Pins for the oracle's TQ4 format (Sec. 3.1 Eq. 4; App. A.1 Table 3; Eq. 2).

Each pin ties the oracle to something other than itself:
* the Hadamard matrix to scipy's Sylvester construction;
* the codebook's quantile start to scipy's Beta quantiles (a coordinate of a
  uniform point on the sphere is (2 B - 1), B ~ Beta((d-1)/2, (d-1)/2));
* each Lloyd update, and the whole run of updates, to the same iteration on
  the continuous density integrated by scipy.integrate.quad;
* d = 3 (a flat density) to the uniform quantizer's closed form;
* the distortion to the published 16-level Gaussian Lloyd-Max value;
* the one-hot vectors of tests/golden/tq4_cases.json to the published
  Gaussian Lloyd-Max thresholds;
* exactness of H S x to integer arithmetic, the norm to exact rationals;
* the byte counts to Eq. 2 and the MiB figures printed in Sec. 2.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch
from scipy import integrate, linalg, stats

from oracle import attention as T
from oracle import tq4
from oracle.affine4 import KIND_K, KIND_V, f32_to_bf16, pack_nibbles, unpack_nibbles
from paper_2609_17475_gb300 import synth
from tests.helpers import bf16_bits

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "tq4_cases.json")))


def _codec(d=256):
    return tq4.make_codec(d, tq4.sign_vector(tq4.SEED_K, d), tq4.sign_vector(tq4.SEED_V, d))


def _density(d):
    return lambda u: (1.0 - u * u) ** ((d - 3) / 2.0)


def _continuous_update(c, d):
    f = _density(d)
    t = np.concatenate([[-1.0], (c[:-1] + c[1:]) / 2.0, [1.0]])
    out = np.empty(len(c))
    for k in range(len(c)):
        num = integrate.quad(lambda u: u * f(u), t[k], t[k + 1], epsabs=1e-15, epsrel=1e-13)[0]
        den = integrate.quad(f, t[k], t[k + 1], epsabs=1e-15, epsrel=1e-13)[0]
        out[k] = num / den
    return out


# -- random signs (Table 3) ------------------------------------------------------
@pytest.mark.parametrize("d", [3, 64, 128, 256])
@pytest.mark.parametrize("seed", [0, 1, 7])
def test_seeded_input_signs_equal_the_oracle_rule(seed, d):
    """The sign vectors handed to the CUDA path (the seeded-input module) are
    the oracle's reading of Table 3's rule, entry for entry."""
    s = synth.tq4_signs(seed, d)
    assert s.dtype == np.int8
    assert np.array_equal(s.astype(np.float64), tq4.sign_vector(seed, d))
    assert (synth.TQ4_SEED_K, synth.TQ4_SEED_V) == (tq4.SEED_K, tq4.SEED_V) == (0, 1)


def test_sign_rule_seed_offset_is_d_times_7919():
    """Table 3 seeds the generator with seed + d * 7919: the draw for (seed, d)
    and for (seed + 7919, d - 1) start from the same generator state, so the
    shorter vector is a prefix of the longer one; any other offset breaks it."""
    for d in (64, 128, 256):
        a = tq4.sign_vector(3, d)
        b = tq4.sign_vector(3 + 7919, d - 1)
        assert np.array_equal(a[:d - 1], b)
        assert not np.array_equal(a[:d - 1], tq4.sign_vector(3 + 7918, d - 1))
        assert set(np.unique(a)) == {-1.0, 1.0}
        # K and V (seeds 0 and 1) get different diagonals; about half the signs are negative
        k, v = tq4.sign_vector(0, d), tq4.sign_vector(1, d)
        assert not np.array_equal(k, v)
        assert abs(int((k < 0).sum()) - d // 2) < 4 * math.sqrt(d)


# -- rotation ------------------------------------------------------------------
@pytest.mark.parametrize("d", [2, 8, 64, 128, 256])
def test_hadamard_is_sylvester(d):
    assert np.array_equal(tq4.hadamard(d), linalg.hadamard(d).astype(np.float64))


def test_rotation_is_orthogonal_and_preserves_norms():
    d = 256
    c = _codec(d)
    R = tq4.hadamard(d) @ np.diag(c.signs_k) / np.sqrt(d)       # y = R x / rho
    assert np.abs(R @ R.T - np.eye(d)).max() < 1e-13
    x = np.random.default_rng(1).standard_normal((50, d))
    assert np.allclose(np.linalg.norm(x @ R.T, axis=1), np.linalg.norm(x, axis=1), rtol=1e-13)


# -- codebook ------------------------------------------------------------------
@pytest.mark.parametrize("d", [64, 256])
def test_quantile_start_is_the_beta_quantile(d):
    x, w = tq4.grid_and_weights(d)
    a = (d - 1) / 2.0
    ref = 2.0 * stats.beta.ppf((np.arange(16) + 0.5) / 16, a, a) - 1.0
    spacing = x[1] - x[0]
    assert np.abs(tq4.quantile_init(x, w) - ref).max() < spacing


def test_codebook_for_a_flat_density_is_the_uniform_quantizer():
    # d = 3: (1 - x^2)^0 is flat on [-1, 1]; Lloyd-Max levels are the cell centres
    c = tq4.codebook(3).astype(np.float64)
    assert np.abs(c - (-1.0 + (2 * np.arange(16) + 1) / 16.0)).max() < 1e-4


@pytest.mark.parametrize("d", [64, 256])
def test_lloyd_update_matches_the_continuous_conditional_means(d):
    x, w = tq4.grid_and_weights(d)
    c, _ = tq4.codebook_f64(d)
    # from the final state and from the start: within the grid's resolution
    for state in (c, tq4.quantile_init(x, w)):
        assert np.abs(tq4.lloyd_update(x, w, state) - _continuous_update(state, d)).max() < 4e-5


@pytest.mark.parametrize("d", [64, 256])
def test_codebook_follows_the_continuous_lloyd_run(d):
    c, n = tq4.codebook_f64(d)
    a = (d - 1) / 2.0
    ref = 2.0 * stats.beta.ppf((np.arange(16) + 0.5) / 16, a, a) - 1.0
    for _ in range(n):
        ref = _continuous_update(ref, d)
    assert 1 <= n <= tq4.MAX_UPDATES
    assert np.abs(c - ref).max() < 1.5e-4


@pytest.mark.parametrize("d", [64, 128, 256])
def test_codebook_is_ascending_and_symmetric(d):
    c = tq4.codebook(d)
    assert c.dtype == np.float32 and c.shape == (16,)
    assert np.all(np.diff(c) > 0)
    assert np.abs(c + c[::-1]).max() <= 2 * np.spacing(np.abs(c)).max()
    t = tq4.thresholds(c)
    assert np.all((t > c[:-1]) & (t < c[1:]))


def test_codebook_distortion_matches_gaussian_lloyd_max():
    # per unit vector, d x (per-coordinate MSE) tends to the 16-level Gaussian
    # Lloyd-Max distortion as d grows; at d = 256 it is within 2 %
    d = 256
    c = tq4.codebook(d).astype(np.float64)
    f = _density(d)
    t = np.concatenate([[-1.0], (c[:-1] + c[1:]) / 2.0, [1.0]])
    Z = integrate.quad(f, -1, 1, epsabs=1e-15)[0]
    D = sum(integrate.quad(lambda u: (u - c[k]) ** 2 * f(u), t[k], t[k + 1], epsabs=1e-16)[0]
            for k in range(16)) / Z
    ref = GOLD["gaussian_max_distortion_N16"]
    assert abs(d * D - ref) / ref < 0.02


# -- encode / decode ----------------------------------------------------------
def test_one_hot_vectors_get_the_gaussian_lloyd_max_indices():
    g = GOLD["one_hot"]
    d = g["head_dim"]
    codec = _codec(d)
    H = linalg.hadamard(d)
    for case in g["cases"]:
        i, a = case["i"], case["a"]
        x = np.zeros(d, dtype=np.float32)
        x[i] = a
        for kind in (KIND_K, KIND_V):
            z, nb = tq4.encode(f32_to_bf16(x), codec, kind)
            sgn = np.sign(a) * codec.signs(kind)[i] * H[:, i]
            want = np.where(sgn > 0, g["index_for_plus_one_sigma"], g["index_for_minus_one_sigma"])
            assert np.array_equal(z.astype(np.int64), want)
            assert np.float16(abs(a)).view(np.uint16) == nb


def test_indices_are_nearest_centroids():
    d = 256
    codec = _codec(d)
    x = synth.normal_bf16(synth.generator(7), (300, d))
    xb = bf16_bits(x)
    z, _ = tq4.encode(xb, codec, KIND_V)
    xf = x.double().numpy()
    rho = tq4.norms_f32(xf).astype(np.float64)
    y = (xf * codec.signs_v) @ linalg.hadamard(d).T / (16.0 * rho[:, None])
    c = codec.centroids.astype(np.float64)
    err = np.abs(y - c[z])
    for dz in (-1, 1):
        zz = np.clip(z.astype(np.int64) + dz, 0, 15)
        assert np.all(err <= np.abs(y - c[zz]) + 1e-12)


def test_rotated_coordinates_are_exact_in_fp64():
    # H S x from integers: x = m 2^e with integer m, summed exactly in Python ints
    d = 256
    codec = _codec(d)
    x = synth.normal_bf16(synth.generator(8), (20, d)).double().numpy()
    x[:, :4] *= 20.0
    e = -40
    m = (x * 2.0 ** -e)
    assert np.all(m == np.round(m))
    H = linalg.hadamard(d).astype(object)
    s = codec.signs_k.astype(np.int64).astype(object)
    for row, mi in zip(x, m.astype(np.int64).astype(object)):
        exact = (H @ (s * mi)).astype(object)
        got = (row * codec.signs_k) @ tq4.hadamard(d).T
        assert all(Fraction(float(g)) == Fraction(int(v)) * Fraction(2) ** e for g, v in zip(got, exact))


def test_norm_is_the_nearest_fp32_to_the_exact_norm():
    d = 256
    x = synth.normal_bf16(synth.generator(9), (40, d)).double().numpy()
    rho = tq4.norms_f32(x)
    for row, r in zip(x, rho):
        s = sum(Fraction(float(v)) ** 2 for v in row)
        r = np.float32(r)
        lo = Fraction(float(r)) - Fraction(float(np.spacing(r))) / 2
        hi = Fraction(float(r)) + Fraction(float(np.spacing(r))) / 2
        assert lo * lo <= s <= hi * hi


def test_zero_and_huge_vectors():
    d = 256
    codec = _codec(d)
    z, nb = tq4.encode(np.zeros((2, d), dtype=np.uint16), codec, KIND_K)
    assert np.all(z == 0) and np.all(nb == 0)
    assert np.all(tq4.decode(z, nb, codec, KIND_K) == 0.0)
    big = np.full(d, 30000.0, dtype=np.float32)                 # norm 480000 > fp16 max
    _, nb = tq4.encode(f32_to_bf16(big), codec, KIND_K)
    assert nb == np.float16(65504.0).view(np.uint16)


def test_round_trip_error_matches_the_codebook_distortion():
    d = 256
    codec = _codec(d)
    x = synth.normal_bf16(synth.generator(10), (2000, d))
    xf = x.double().numpy()
    for kind in (KIND_K, KIND_V):
        z, nb = tq4.encode(bf16_bits(x), codec, kind)
        xh = tq4.decode(z, nb, codec, kind)
        rel = ((xf - xh) ** 2).sum(1) / (xf ** 2).sum(1)
        # the codebook's own distortion at d = 256 (quad), about 0.00941
        assert 0.0090 < rel.mean() < 0.0098
        # norms: ||x_hat|| = rho_hat ||c[z]||
        cz = codec.centroids.astype(np.float64)[z]
        assert np.allclose(np.linalg.norm(xh, axis=1),
                           tq4.fp16_to_f64(nb) * np.linalg.norm(cz, axis=1), rtol=1e-12)


def test_decode_by_explicit_matrices():
    d = 64
    codec = _codec(d)
    rng = np.random.default_rng(3)
    z = rng.integers(0, 16, size=(5, d)).astype(np.uint8)
    nb = np.float16(rng.uniform(0.5, 4.0, 5)).view(np.uint16)
    got = tq4.decode(z, nb, codec, KIND_V)
    H = linalg.hadamard(d).astype(np.float64)
    S = np.diag(codec.signs_v)
    for r in range(5):
        want = float(np.float16(nb[r].view(np.float16))) * (S @ H @ codec.centroids[z[r]].astype(np.float64)) / 8.0
        assert np.allclose(got[r], want, rtol=0, atol=1e-14)


# -- layout and byte accounting (Eq. 2, Sec. 2) -------------------------------
def test_bytes_per_position_match_eq2():
    b = GOLD["byte_accounting"]
    lay = tq4.Tq4Layout(b["num_kv_heads"], 256, b["head_dim"], _codec(b["head_dim"]))
    per = lay.bytes_per_position * b["layers"]
    assert per == b["bytes_per_position_all_layers"]
    assert per * 262144 == b["mib_at_262144"] * 2 ** 20
    assert per * 327680 == b["mib_at_327680"] * 2 ** 20
    fp16 = b["layers"] * 2 * b["num_kv_heads"] * b["head_dim"] * 2
    assert round(100.0 * per / fp16, 1) == b["fraction_of_fp16_percent"]
    assert lay.page_bytes == 256 * lay.bytes_per_position


def test_append_then_gather_round_trips_through_permuted_pages():
    d, Hkv, P = 64, 2, 16
    codec = _codec(d)
    lay = tq4.Tq4Layout(Hkv, P, d, codec)
    gen = synth.generator(11)
    ctx = [40, 17]
    table, num_pages = synth.page_tables(gen, ctx, P, num_pages=9)
    req, pos = synth.append_rows_for(ctx)
    k, v = synth.kv_rows(gen, len(req), Hkv, d)
    pool = tq4.new_pool(lay, num_pages, fill=0xAB)
    tq4.append(pool, lay, table.numpy(), req.numpy(), pos.numpy(), bf16_bits(k), bf16_bits(v))
    kb, vb = bf16_bits(k), bf16_bits(v)
    off = 0
    for b, c in enumerate(ctx):
        for h in range(Hkv):
            for kind, xb in ((KIND_K, kb), (KIND_V, vb)):
                z, nb = tq4.encode(xb[off:off + c, h], codec, kind)
                want = tq4.decode(z, nb, codec, kind)
                got = T.gather_head(pool, lay, table[b].numpy(), c, h, kind)
                assert np.array_equal(got, want)
                # bytes where the layout says: indices then norms
                for t in (0, c - 1):
                    page, slot = int(table[b, t // P]), t % P
                    rec = pool[page]
                    co = lay.codes_offset(kind, h, slot)
                    assert np.array_equal(unpack_nibbles(rec[co:co + d // 2]), z[t])
                    no = lay.norm_offset(kind, h, slot)
                    assert int(rec[no]) | (int(rec[no + 1]) << 8) == int(nb[t])
        off += c


# -- attention over TQ4 pages -------------------------------------------------
def _tq4_pool(seed, ctx, Hkv=2, d=64, P=16):
    codec = _codec(d)
    lay = tq4.Tq4Layout(Hkv, P, d, codec)
    gen = synth.generator(seed)
    table, num_pages = synth.page_tables(gen, ctx, P)
    req, pos = synth.append_rows_for(ctx)
    k, v = synth.kv_rows(gen, len(req), Hkv, d)
    pool = tq4.new_pool(lay, num_pages)
    tq4.append(pool, lay, table.numpy(), req.numpy(), pos.numpy(), bf16_bits(k), bf16_bits(v))
    return lay, pool, table.numpy(), gen


def test_tq4_decode_equals_sdpa_on_reconstructed_rows():
    lay, pool, table, gen = _tq4_pool(12, [37, 5])
    q = synth.normal_bf16(gen, (2, 4, 64))
    out = T.paged_decode(pool, lay, table, [37, 5], bf16_bits(q), 0.125)
    for b, c in enumerate([37, 5]):
        for h in range(4):
            kv = h // 2
            K = torch.from_numpy(T.gather_head(pool, lay, table[b], c, kv, KIND_K))
            V = torch.from_numpy(T.gather_head(pool, lay, table[b], c, kv, KIND_V))
            qq = q[b, h].double()[None, None, None]
            ref = torch.nn.functional.scaled_dot_product_attention(qq, K[None, None], V[None, None],
                                                                   scale=0.125)
            assert np.allclose(out[b, h], ref[0, 0, 0].numpy(), rtol=1e-12, atol=1e-13)
    split = T.paged_decode_split(pool, lay, table, [37, 5], bf16_bits(q), 0.125, num_splits=3)
    assert np.allclose(split, out, rtol=1e-12, atol=1e-13)
