"""Pins for the oracle's affine 4-bit group-64 quantizer, packing and layout.

The oracle defines the bit-exact contract the CUDA append kernel must meet, so
it is pinned here against things other than itself: torch's own bf16 rounding,
hand-derived golden groups (tests/golden/affine4_cases.json), the error bound
|x - x_hat| <= scale/2 and nearest-level optimality checked in fp64, and
exactly quantizable groups that must round-trip unchanged.
"""
import json
import os

import numpy as np
import pytest
import torch

from oracle import affine4 as A
from tests.helpers import bf16_bits, exact_groups, f64_to_bf16_tensor

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "affine4_cases.json")))


def _expand(pattern, n=64):
    return [pattern[i % len(pattern)] for i in range(n)]


# -- bf16 rounding against torch's RNE cast ---------------------------------
def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([
        rng.standard_normal(20000).astype(np.float32),
        (rng.standard_normal(2000) * 1e-39).astype(np.float32),       # subnormals
        (rng.standard_normal(2000) * 1e30).astype(np.float32),
        np.array([0.0, -0.0, 1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1 / 15, 3.3895314e38],
                 dtype=np.float32),
    ])
    # exact ties: bf16 value plus half an ulp, both parities of the kept lsb
    base = (rng.integers(0x3000, 0x5000, 4000).astype(np.uint32) << 16) | 0x8000
    x = np.concatenate([x, base.view(np.float32)])
    ours = A.f32_to_bf16(x)
    ref = bf16_bits(torch.from_numpy(x).to(torch.bfloat16))
    assert np.array_equal(ours, ref)


def test_bf16_widening_is_exact():
    bits = np.arange(0, 0x7F80, 7, dtype=np.uint16)
    ref = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(A.bf16_to_f32(bits), ref)


# -- golden groups -------------------------------------------------------------
@pytest.mark.parametrize("case", GOLD["groups"], ids=[c["name"] for c in GOLD["groups"]])
def test_golden_group(case):
    x = np.array(_expand(case["x"]), dtype=np.float64)
    xb = bf16_bits(f64_to_bf16_tensor(x))
    if case["name"] == "signed_zeros":          # keep the sign bits of -0.0
        xb = np.where(np.signbit(x), np.uint16(0x8000), np.uint16(0)).astype(np.uint16)
    codes, sbits, bbits = A.quantize_groups(xb)
    assert int(sbits) == int(case["scale_bits"], 16)
    assert int(bbits) == int(case["bias_bits"], 16)
    assert codes.tolist() == _expand(case["codes"])


def test_golden_packing():
    codes = np.array(GOLD["packing"]["codes"], dtype=np.uint8)
    packed = A.pack_nibbles(codes)
    assert packed.tolist() == [int(b, 16) for b in GOLD["packing"]["bytes"]]
    assert A.unpack_nibbles(packed).tolist() == codes.tolist()


@pytest.mark.parametrize("lay", GOLD["layouts"], ids=lambda l: f"h{l['num_kv_heads']}p{l['page_size']}d{l['head_dim']}")
def test_golden_layout(lay):
    L = A.PoolLayout(lay["num_kv_heads"], lay["page_size"], lay["head_dim"])
    assert L.page_bytes == lay["page_bytes"]
    if "bytes_per_position" in lay:
        assert L.bytes_per_position == lay["bytes_per_position"]
        assert 16 * L.bytes_per_position == lay["bytes_per_position_16_layers"]
    for o in lay["offsets"]:
        f = L.codes_offset if o["what"] == "codes" else L.sb_offset
        assert f(o["kind"], o["head"], o["slot"]) == o["offset"]


def test_sb_bytes_are_scale_then_bias_little_endian():
    x = np.array(_expand([-8.0 + 0.25 * k for k in range(16)]), dtype=np.float64)
    xb = bf16_bits(f64_to_bf16_tensor(x))
    cb, sb = A.encode_vectors(xb)
    assert sb.tolist() == [0x80, 0x3E, 0x00, 0xC1]      # 0x3E80, 0xC100 little-endian
    assert cb[:2].tolist() == [0x10, 0x32]


# -- properties on random data ----------------------------------------------------
def _random_groups(seed, n):
    g = torch.Generator().manual_seed(seed)
    base = torch.randn(n, 64, generator=g)
    scales = torch.exp2(torch.randint(-12, 12, (n, 1), generator=g).float())
    x = (base * scales)
    x[: n // 8, :4] *= 20.0                                      # outlier channels
    x[n // 8: n // 4] = x[n // 8: n // 4].abs() + 3.0 * scales[n // 8: n // 4]  # offset groups
    return bf16_bits(x.to(torch.bfloat16))


def test_error_bound_and_nearest_level():
    xb = _random_groups(1, 4096)
    codes, sbits, bbits = A.quantize_groups(xb)
    x = A.bf16_to_f64(xb)
    s = A.bf16_to_f64(sbits)[:, None]
    b = A.bf16_to_f64(bbits)[:, None]
    xhat = codes * s + b
    err = np.abs(x - xhat)
    assert (s > 0).all()
    assert (err <= 0.5 * s * (1 + 2 ** -16)).all(), float((err / s).max())
    # nearest level among the 16: no other code is strictly closer
    levels = np.arange(16)[None, None, :] * s[..., None] + b[..., None]
    best = np.abs(x[..., None] - levels).min(axis=-1)
    assert (err <= best * (1 + 2 ** -20) + 1e-300).all()
    # codes span the range: min element -> 0, max element -> 15
    assert (codes.min(axis=1) == 0).all() and (codes.max(axis=1) == 15).all()


def test_exact_groups_round_trip():
    rng = np.random.default_rng(3)
    x = exact_groups(rng, (512, 256))
    xb = bf16_bits(f64_to_bf16_tensor(x))
    cb, sb = A.encode_vectors(xb)
    assert cb.shape == (512, 128) and sb.shape == (512, 16)
    assert np.array_equal(A.decode_vectors(cb, sb), x)


def test_constant_and_zero_groups():
    x = np.zeros((3, 64), dtype=np.float64)
    x[1] = -2.5
    x[2] = 1e-3
    xb = bf16_bits(torch.from_numpy(x).to(torch.bfloat16))
    codes, sbits, bbits = A.quantize_groups(xb)
    assert (codes == 0).all() and (sbits == 0).all()
    assert np.array_equal(A.dequantize(codes[:, None], sbits[:, None], bbits[:, None])[:, 0],
                          A.bf16_to_f64(xb))


def test_append_places_rows_through_page_table():
    L = A.PoolLayout(2, 64, 128)
    rng = np.random.default_rng(5)
    ctx = [150, 64]
    pt = np.array([[3, 0, 5], [1, -1, -1]], dtype=np.int32)
    pool = A.new_pool(L, 6, fill=0xAB)
    n = sum(ctx)
    req = np.array([0] * ctx[0] + [1] * ctx[1], dtype=np.int32)
    pos = np.concatenate([np.arange(c) for c in ctx]).astype(np.int32)
    x = exact_groups(rng, (2, n, 2, 128))
    kb = bf16_bits(f64_to_bf16_tensor(x[0]))
    vb = bf16_bits(f64_to_bf16_tensor(x[1]))
    A.append(pool, L, pt, req, pos, kb, vb, chunk=37)
    # every row reads back exactly at (page_table[req, pos//P], pos % P)
    for i in range(n):
        page = pt[req[i], pos[i] // 64]
        for kind, src in ((A.KIND_K, x[0]), (A.KIND_V, x[1])):
            for h in range(2):
                o = L.codes_offset(kind, h, pos[i] % 64)
                so = L.sb_offset(kind, h, pos[i] % 64)
                v = A.decode_vectors(pool[page, o:o + 64], pool[page, so:so + 8])
                assert np.array_equal(v, src[i, h])
    # untouched bytes keep their fill: page 2 and 4 unused, tail slots of page 5
    assert (pool[2] == 0xAB).all() and (pool[4] == 0xAB).all()
    tail = L.codes_offset(A.KIND_K, 0, 150 - 128)
    assert (pool[5, tail:L.codes_offset(A.KIND_K, 1, 0)] == 0xAB).all()
