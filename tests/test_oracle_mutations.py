"""The oracle's pins must catch plausible mistakes.

Each case plants one mistake in the oracle (on the CPU, via monkeypatch) and
checks that at least one pin test now fails: a dropped term, a wrong divisor,
the wrong tie direction, swapped nibbles, a transposed GQA map, a missing
softmax scale, an off-by-one causal bound, a wrong page lookup, a merge
without the max rescale, split ranges that drop a position, checkpoint
records in physical instead of logical order, restore into the wrong pages,
and a reservation without the output cap or rounded down.
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


# -- TQ4 (Sec. 3.1 Eq. 4; App. A.1 Table 3) -----------------------------------
import oracle.tq4 as Q
from tests import test_oracle_tq4 as TT


def test_tq4_dropped_signs_are_caught(monkeypatch):
    orig = Q.encode

    def bad(x_bits, codec, kind):
        ones = np.ones(codec.head_dim)
        return orig(x_bits, Q.Codec(codec.head_dim, codec.centroids, ones, ones), kind)
    monkeypatch.setattr(Q, "encode", bad)
    assert _fails(TT.test_one_hot_vectors_get_the_gaussian_lloyd_max_indices)


def test_tq4_wrong_density_exponent_is_caught(monkeypatch):
    def bad(d):
        x = np.linspace(-1.0 + Q.GRID_EPS, 1.0 - Q.GRID_EPS, Q.GRID_POINTS)
        w = (1.0 - x * x) ** ((d - 1) / 2.0)
        return x, w / w.sum()
    monkeypatch.setattr(Q, "grid_and_weights", bad)
    assert _fails(TT.test_lloyd_update_matches_the_continuous_conditional_means, 256)


def test_tq4_unweighted_cell_means_are_caught(monkeypatch):
    orig = Q.lloyd_update

    def bad(x, w, c):
        return orig(x, np.full_like(w, 1.0 / len(w)), c)
    monkeypatch.setattr(Q, "lloyd_update", bad)
    assert _fails(TT.test_lloyd_update_matches_the_continuous_conditional_means, 256)


def test_tq4_thresholds_at_centroids_are_caught(monkeypatch):
    monkeypatch.setattr(Q, "thresholds", lambda c32: np.asarray(c32, dtype=np.float32)[1:])
    assert _fails(TT.test_indices_are_nearest_centroids)


def test_tq4_missing_sqrt_d_in_decode_is_caught(monkeypatch):
    orig = Q.decode

    def bad(z, nb, codec, kind):
        return orig(z, nb, codec, kind) * np.sqrt(codec.head_dim)
    monkeypatch.setattr(Q, "decode", bad)
    assert _fails(TT.test_round_trip_error_matches_the_codebook_distortion)


def test_tq4_rotation_order_swapped_in_decode_is_caught(monkeypatch):
    def bad(z, nb, codec, kind):
        d = codec.head_dim
        cz = codec.centroids.astype(np.float64)[np.asarray(z, dtype=np.int64)]
        rot = (cz * codec.signs(kind)) @ Q.hadamard(d).T          # H S c instead of S H c
        return Q.fp16_to_f64(nb)[..., None] * rot / np.sqrt(np.float64(d))
    monkeypatch.setattr(Q, "decode", bad)
    assert _fails(TT.test_round_trip_error_matches_the_codebook_distortion)


def test_tq4_bf16_norm_is_caught(monkeypatch):
    monkeypatch.setattr(Q, "norm_to_fp16",
                        lambda rho: A.f32_to_bf16(np.asarray(rho, dtype=np.float32)))
    assert _fails(TT.test_one_hot_vectors_get_the_gaussian_lloyd_max_indices)


def test_tq4_quantile_offset_is_caught(monkeypatch):
    def bad(x, w):
        cdf = np.cumsum(w)
        return np.array([x[np.searchsorted(cdf, k / 16.0)] for k in range(16)])
    monkeypatch.setattr(Q, "quantile_init", bad)
    assert _fails(TT.test_quantile_start_is_the_beta_quantile, 256)


# -- split merge (Eq. 3 workspace), checkpoint / restore (Sec. 3.4), Eq. 7 -----
import oracle.checkpoint as C
import oracle.reservation as R
from tests import test_oracle_reservation as TR


def test_merge_without_max_rescale_is_caught(monkeypatch):
    def bad(parts):
        return sum(o for _, _, o in parts) / sum(l for _, l, _ in parts)
    monkeypatch.setattr(T, "merge_partials", bad)
    assert _fails(TA.test_split_merge_equals_plain_softmax, 3)


def test_merge_rescaling_only_the_sums_is_caught(monkeypatch):
    def bad(parts):
        m_star = max(m for m, _, _ in parts)
        return (sum(o for _, _, o in parts) /
                sum(np.exp(m - m_star) * l for m, l, _ in parts))
    monkeypatch.setattr(T, "merge_partials", bad)
    assert _fails(TA.test_split_merge_equals_plain_softmax, 2)


def test_split_bounds_dropping_the_last_position_are_caught(monkeypatch):
    orig = T.split_bounds

    def bad(ctx, num_splits):
        b = orig(ctx, num_splits)
        return b[:-1] + [(b[-1][0], b[-1][1] - 1)] if b[-1][1] - 1 > b[-1][0] else b
    monkeypatch.setattr(T, "split_bounds", bad)
    assert _fails(TA.test_split_bounds_cover_exactly)


def test_checkpoint_in_physical_page_order_is_caught(monkeypatch):
    orig = C.checkpoint

    def bad(pool, page_table_row, num_pages):
        return orig(pool, np.sort(np.asarray(page_table_row)[:num_pages]), num_pages)
    monkeypatch.setattr(C, "checkpoint", bad)
    assert _fails(TA.test_checkpoint_bytes_and_restore_round_trip)


def test_restore_to_logical_slots_is_caught(monkeypatch):
    def bad(pool, page_table_row, num_pages, blob):
        pb = pool.shape[1]
        for k in range(num_pages):
            pool[k] = blob[k * pb:(k + 1) * pb]
    monkeypatch.setattr(C, "restore", bad)
    assert _fails(TA.test_checkpoint_bytes_and_restore_round_trip)


def test_reservation_without_the_output_cap_is_caught(monkeypatch):
    monkeypatch.setattr(R, "reservation_pages",
                        lambda p, o, g_out=8192, page_size=256: -(-(p + o) // page_size))
    assert _fails(TR.test_paper_policy_numbers)


def test_reservation_rounding_down_is_caught(monkeypatch):
    monkeypatch.setattr(R, "reservation_pages",
                        lambda p, o, g_out=8192, page_size=256: (p + min(o, g_out)) // page_size)
    assert _fails(TR.test_reservation_matches_brute_force_and_library, 257, 0, 8192, 256)
