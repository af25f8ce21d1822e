"""The oracle's pins must catch plausible mistakes.

Each case plants one mistake in the oracle (on the CPU, via monkeypatch) and
checks that at least one pin test now fails: a dropped term, a wrong divisor,
the wrong tie direction, swapped nibbles, a transposed GQA map, a missing
softmax scale, an off-by-one causal bound, a wrong page lookup.
"""
import numpy as np
import pytest

import oracle.affine4 as A
import oracle.attention as T
from tests import test_oracle_attention as TA
from tests import test_oracle_quantizer as TQ


def _fails(fn, *args, **kw):
    try:
        fn(*args, **kw)
    except AssertionError:
        return True
    return False


def _golden(name):
    return next(c for c in TQ.GOLD["groups"] if c["name"] == name)


def test_scale_divisor_16_is_caught(monkeypatch):
    orig = A.quantize_groups

    def bad(x_bits):
        x = A.bf16_to_f32(np.asarray(x_bits, dtype=np.uint16))
        codes, sbits, bbits = orig(x_bits)
        rng = (x.max(axis=-1) - x.min(axis=-1)).astype(np.float32)
        return codes, A.f32_to_bf16(rng / np.float32(16)), bbits
    monkeypatch.setattr(A, "quantize_groups", bad)
    assert _fails(TQ.test_golden_group, _golden("ramp_unit"))


def test_ties_rounding_up_is_caught(monkeypatch):
    orig = A.quantize_groups

    def bad(x_bits):
        codes, sbits, bbits = orig(x_bits)
        x = A.bf16_to_f32(np.asarray(x_bits, dtype=np.uint16))
        s = A.bf16_to_f32(sbits)[..., None]
        b = A.bf16_to_f32(bbits)[..., None]
        with np.errstate(divide="ignore", invalid="ignore"):
            r = (x - b) / s
        up = np.clip(np.floor(r + np.float32(0.5)), 0, 15).astype(np.uint8)   # ties up
        up[(s == 0).squeeze(-1)] = 0
        return up, sbits, bbits
    monkeypatch.setattr(A, "quantize_groups", bad)
    assert _fails(TQ.test_golden_group, _golden("midpoints_go_down"))


def test_swapped_nibbles_are_caught(monkeypatch):
    def bad(codes):
        codes = np.asarray(codes, dtype=np.uint8)
        return (codes[..., 1::2] | (codes[..., 0::2] << 4)).astype(np.uint8)
    monkeypatch.setattr(A, "pack_nibbles", bad)
    assert _fails(TQ.test_golden_packing)


def test_dropped_bias_is_caught(monkeypatch):
    monkeypatch.setattr(A, "dequantize",
                        lambda c, s, b: c.astype(np.float64) * A.bf16_to_f64(s)[..., None])
    assert _fails(TA.test_decode_matches_sdpa_on_exact_values, 8, 2, 128, 64, [300, 64, 1])


def test_wrong_gqa_map_is_caught(monkeypatch):
    def bad(pool, layout, page_table, context_lens, q_bits, softmax_scale, heads=None):
        q = A.bf16_to_f64(q_bits)
        B, Hq, D = q.shape
        out = np.zeros((B, Hq, D))
        for b in range(B):
            ctx = int(context_lens[b])
            if ctx == 0:
                continue
            for h in range(Hq):
                kv = h % layout.num_kv_heads                         # interleaved, not grouped
                k = A.gather_head(pool, layout, page_table[b], ctx, kv, A.KIND_K)
                v = A.gather_head(pool, layout, page_table[b], ctx, kv, A.KIND_V)
                out[b, h] = T._softmax_weighted(softmax_scale * (k @ q[b, h]), v)
        return out
    monkeypatch.setattr(T, "paged_decode", bad)
    assert _fails(TA.test_decode_matches_sdpa_on_exact_values, 8, 2, 128, 64, [300, 64, 1])


def test_missing_softmax_scale_is_caught(monkeypatch):
    orig = T.paged_decode
    monkeypatch.setattr(T, "paged_decode",
                        lambda pool, L, pt, ctx, q, scale, heads=None: orig(pool, L, pt, ctx, q, 1.0, heads))
    assert _fails(TA.test_decode_matches_sdpa_on_exact_values, 24, 4, 256, 256, [700])


def test_off_by_one_causal_bound_is_caught(monkeypatch):
    orig = T.prefill_chunk

    def bad(pool, layout, pt_row, q_bits, q_start, scale, causal=True):
        if not causal:
            return orig(pool, layout, pt_row, q_bits, q_start, scale, causal=False)
        C = q_bits.shape[0]
        out = np.zeros(q_bits.shape)
        for i in range(C):                                        # excludes the own position
            if q_start + i == 0:
                continue
            out[i] = T.paged_decode(pool, layout, np.asarray(pt_row)[None], [q_start + i],
                                    q_bits[i][None], scale)[0]
        return out
    monkeypatch.setattr(T, "prefill_chunk", bad)
    assert _fails(TA.test_prefill_rows_equal_decode_and_sdpa, 100, 70)


def test_ignored_page_table_is_caught(monkeypatch):
    orig = A.gather_head

    def bad(pool, layout, page_table_row, ctx, head, kind):
        identity = np.arange(len(page_table_row), dtype=np.int64)
        return orig(pool, layout, identity, ctx, head, kind)
    monkeypatch.setattr(A, "gather_head", bad)
    monkeypatch.setattr(T, "gather_head", bad)
    assert _fails(TA.test_decode_matches_sdpa_on_exact_values, 8, 2, 128, 64, [300, 64, 1])


def test_unmutated_pins_pass():
    TQ.test_golden_group(_golden("ramp_unit"))
    TQ.test_golden_packing()
    TA.test_decode_matches_sdpa_on_exact_values(8, 2, 128, 64, [300, 64, 1])
    TA.test_prefill_rows_equal_decode_and_sdpa(100, 70)
