"""Host-only checks of the C ABI: the library loads, exports every symbol the
header declares, and rejects bad arguments before launching anything (these
calls never touch the GPU, so they run on CPU-only machines)."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2609_17475_gb300 import binding as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "jfkv.h")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(jf_[a-z0-9_]+)\s*\(", text)))


def test_library_exports_every_declared_symbol():
    L = B.lib()
    names = _declared()
    assert "jf_paged_decode_attn" in names and len(names) >= 10
    for n in names:
        assert hasattr(L, n), n
    assert sorted(B.EXPORTS) == names


def test_sizes():
    assert B.jf_kv_page_bytes(4, 256, 256) == 294912
    assert B.jf_kv_page_bytes(2, 256, 128) == 73728
    assert B.jf_kv_page_bytes(2, 64, 128) == 18432
    assert B.jf_kv_page_bytes(4, 256, 64) == 0
    # fixed workspace: independent of context length, linear in splits
    w1 = B.jf_attn_workspace_bytes(1, 24, 4, 256, 32)
    w2 = B.jf_attn_workspace_bytes(1, 24, 4, 256, 64)
    assert w1 >= 24 * 32 * (4 * 256 + 8)
    assert w2 - w1 == 24 * 32 * 4 * 256 + (24 * 64 * 8 - 24 * 32 * 8)
    assert B.jf_attn_workspace_bytes(2, 24, 5, 256, 4) == 0     # Hq % Hkv != 0
    assert B.jf_attn_workspace_bytes(1, 8, 2, 96, 4) == 0        # unsupported head_dim
    assert B.jf_prefill_workspace_bytes() >= 4
    assert B.status_string(-3) == "JF_ERR_WORKSPACE_TOO_SMALL"
    assert "sm_103a" in B.version()


def _pool(**kw):
    d = dict(base=0x10000, num_pages=8, page_size=256, num_kv_heads=2, head_dim=128,
             group_size=64, format=0)
    d.update(kw)
    return B._Pool(**d)


FAKE = ctypes.c_void_p(0x20000)   # aligned, never dereferenced: validation fails first


@pytest.mark.parametrize("kw,expect", [
    (dict(base=None), B.JF_ERR_INVALID_ARG),
    (dict(base=0x10004), B.JF_ERR_INVALID_ARG),
    (dict(head_dim=96), B.JF_ERR_UNSUPPORTED),
    (dict(page_size=100), B.JF_ERR_UNSUPPORTED),
    (dict(group_size=32), B.JF_ERR_UNSUPPORTED),
    (dict(format=1), B.JF_ERR_INVALID_ARG),        # TQ4 without its codec
    (dict(format=2), B.JF_ERR_UNSUPPORTED),
    (dict(num_pages=0), B.JF_ERR_INVALID_ARG),
])
def test_decode_rejects_bad_pool(kw, expect):
    p = _pool(**kw)
    st = B.lib().jf_paged_decode_attn(ctypes.byref(p), FAKE, 4, FAKE, 1, FAKE, 8, 0.1, FAKE,
                                       FAKE, 1 << 20, 4, None)
    assert st == expect


def test_decode_rejects_bad_arguments():
    p = _pool()
    L = B.lib()
    call = lambda **kw: L.jf_paged_decode_attn(
        ctypes.byref(p), kw.get("pt", FAKE), 4, FAKE, kw.get("batch", 1), FAKE,
        kw.get("hq", 8), kw.get("scale", 0.1), FAKE, kw.get("ws", FAKE),
        kw.get("wsb", 1 << 20), kw.get("splits", 4), None)
    assert call(pt=None) == B.JF_ERR_INVALID_ARG
    assert call(hq=7) == B.JF_ERR_INVALID_ARG            # Hq % Hkv
    assert call(hq=18) == B.JF_ERR_UNSUPPORTED           # G = 9 > 8
    assert call(splits=0) == B.JF_ERR_INVALID_ARG
    assert call(batch=0) == B.JF_ERR_INVALID_ARG
    assert call(scale=float("nan")) == B.JF_ERR_INVALID_ARG
    assert call(wsb=100) == B.JF_ERR_WORKSPACE_TOO_SMALL
    assert call(ws=ctypes.c_void_p(0x20010)) == B.JF_ERR_INVALID_ARG   # not 256-aligned


def test_append_checkpoint_prefill_reject_bad_arguments():
    p = _pool()
    L = B.lib()
    assert L.jf_kv_quantize_append(ctypes.byref(p), FAKE, 4, 1, FAKE, FAKE, FAKE, FAKE, -1,
                                   None, None) == B.JF_ERR_INVALID_ARG
    assert L.jf_kv_quantize_append(ctypes.byref(p), FAKE, 4, 1, FAKE, FAKE, FAKE, FAKE, 0,
                                   None, None) == B.JF_OK          # empty append: no-op
    assert L.jf_kv_quantize_append(ctypes.byref(p), FAKE, 4, 1, FAKE, FAKE,
                                   ctypes.c_void_p(0x20002), FAKE, 5, None,
                                   None) == B.JF_ERR_INVALID_ARG  # misaligned k
    pb = B.jf_kv_page_bytes(2, 256, 128)
    assert L.jf_kv_checkpoint(ctypes.byref(p), FAKE, 3, FAKE, 3 * pb - 1, None,
                              None) == B.JF_ERR_INVALID_ARG       # dst too small
    assert L.jf_kv_checkpoint(ctypes.byref(p), FAKE, 0, FAKE, 0, None, None) == B.JF_OK
    assert L.jf_kv_restore(ctypes.byref(p), FAKE, -1, FAKE, 0, None,
                           None) == B.JF_ERR_INVALID_ARG
    assert L.jf_prefill_chunk_attn(ctypes.byref(p), FAKE, FAKE, 0, 16, 8, 0.1, 1, FAKE, FAKE, 0,
                                   None) == B.JF_ERR_WORKSPACE_TOO_SMALL
    assert L.jf_prefill_chunk_attn(ctypes.byref(p), FAKE, FAKE, -1, 16, 8, 0.1, 1, FAKE, FAKE,
                                   256, None) == B.JF_ERR_INVALID_ARG
    assert L.jf_prefill_chunk_attn(ctypes.byref(p), FAKE, FAKE, 0, 0, 8, 0.1, 1, FAKE, FAKE,
                                   256, None) == B.JF_OK           # empty chunk: no-op


# -- TQ4 (Sec. 3.1 Eq. 4; App. A.1 Table 3): host-side logic --------------------
def _tq4_pool(codec, **kw):
    p = _pool(format=B.JF_FMT_TQ4, **kw)
    p.tq4 = ctypes.pointer(codec._c)
    return p


def _codec(d=128):
    from paper_2609_17475_gb300 import synth
    return B.Tq4Codec(d, synth.tq4_signs(0, d), synth.tq4_signs(1, d))


@pytest.mark.parametrize("d", [3, 64, 128, 256])
def test_tq4_codebook_equals_the_oracle_bit_for_bit(d):
    from oracle import tq4
    assert np.array_equal(B.jf_tq4_codebook(d), tq4.codebook(d))


def test_tq4_page_bytes_follow_eq2():
    assert B.jf_kv_page_bytes_fmt(B.JF_FMT_TQ4, 4, 256, 256) == 256 * 1040
    assert B.jf_kv_page_bytes_fmt(B.JF_FMT_AFFINE4_G64, 4, 256, 256) == B.jf_kv_page_bytes(4, 256, 256)
    assert B.jf_kv_page_bytes_fmt(7, 4, 256, 256) == 0
    assert B.lib().jf_tq4_codebook(2, (ctypes.c_float * 16)()) == B.JF_ERR_INVALID_ARG


def test_tq4_bad_codecs_and_unsupported_entry_points():
    L = B.lib()
    c = _codec()
    p = _tq4_pool(c)
    dec = lambda pool: L.jf_paged_decode_attn(ctypes.byref(pool), FAKE, 4, FAKE, 1, FAKE, 8, 0.1,
                                               FAKE, FAKE, 1 << 20, 4, None)
    bad = _codec()
    bad._c.centroids[3] = bad._c.centroids[2]          # not strictly ascending
    assert dec(_tq4_pool(bad)) == B.JF_ERR_INVALID_ARG
    bad = _codec()
    bad._c.signs_v[5] = 0                              # not +-1
    assert dec(_tq4_pool(bad)) == B.JF_ERR_INVALID_ARG
    assert L.jf_kv_quantize_append(ctypes.byref(_tq4_pool(bad)), FAKE, 4, 1, FAKE, FAKE, FAKE,
                                   FAKE, 5, None, None) == B.JF_ERR_INVALID_ARG
    # the verifier and the fused step validate the codec too; the no-workspace
    # decode does not take TQ4 pools
    assert L.jf_paged_verify_attn(ctypes.byref(_tq4_pool(bad)), FAKE, 4, FAKE, 1, FAKE, 2, 8, 0.1,
                                  FAKE, FAKE, 1 << 20, 4, None) == B.JF_ERR_INVALID_ARG
    assert L.jf_paged_decode_append_attn(ctypes.byref(_tq4_pool(bad)), FAKE, 4, FAKE, 1, FAKE,
                                         FAKE, FAKE, 8, 0.1, FAKE, FAKE, 1 << 20, 4,
                                         None) == B.JF_ERR_INVALID_ARG
    assert L.jf_prefill_chunk_attn(ctypes.byref(p), FAKE, FAKE, 0, 16, 8, 0.1, 1, FAKE, FAKE, 256,
                                   None) == B.JF_ERR_WORKSPACE_TOO_SMALL   # TQ4 needs more
    assert L.jf_paged_decode_attn_noalloc(ctypes.byref(p), FAKE, 4, FAKE, 1, FAKE, 8, 0.1, FAKE, 4,
                                          None, None) == B.JF_ERR_UNSUPPORTED
    # checkpoint sizes use the TQ4 page record
    pb = B.jf_kv_page_bytes_fmt(B.JF_FMT_TQ4, 2, 256, 128)
    assert L.jf_kv_checkpoint(ctypes.byref(p), FAKE, 3, FAKE, 3 * pb - 1, None,
                              None) == B.JF_ERR_INVALID_ARG


def test_prefill_batch_rejects_bad_arguments():
    L = B.lib()
    p = _pool()
    I = ctypes.c_int32
    qs = (I * 2)(0, 100)
    cl = (I * 2)(16, 16)
    call = lambda batch=2, stride=4, q_start=qs, clen=cl, wsb=256, splits=1: L.jf_prefill_batch_attn(
        ctypes.byref(p), FAKE, stride, batch, q_start, clen, FAKE, 8, 0.1, 1, splits, FAKE, FAKE,
        wsb, None)
    assert call(batch=0) == B.JF_ERR_INVALID_ARG
    assert call(batch=65, q_start=(I * 65)(), clen=(I * 65)()) == B.JF_ERR_UNSUPPORTED
    assert call(wsb=0) == B.JF_ERR_WORKSPACE_TOO_SMALL
    assert call(stride=1, q_start=(I * 2)(0, 250), clen=(I * 2)(4, 16)) == B.JF_ERR_INVALID_ARG
    assert call(q_start=(I * 2)(-1, 0)) == B.JF_ERR_INVALID_ARG
    assert call(clen=(I * 2)(0, 0)) == B.JF_OK                     # nothing to do
    assert call(splits=0) == B.JF_ERR_INVALID_ARG
    need = L.jf_prefill_batch_workspace_bytes
    n = need(0, 32, 8, 128, 4)
    assert n == 256 + (32 * 8 * 4 * 8 + 255) // 256 * 256 + 32 * 8 * 4 * 128 * 4
    assert need(0, 32, 8, 128, 1) == 256 and need(0, 32, 8, 96, 4) == 0
    # TQ4: partials even unsplit, plus the rotated queries
    assert need(1, 32, 8, 128, 1) == 256 + (32 * 8 * 8 + 255) // 256 * 256 + 2 * 32 * 8 * 128 * 4
    assert need(5, 32, 8, 128, 1) == 0
    assert call(splits=4, wsb=n - 1) == B.JF_ERR_WORKSPACE_TOO_SMALL


def test_prefill_chunk_workspace_plans_the_wave_balance():
    """Host-only (num_sms given): a 2,048-query chunk after 30,720 positions at
    24/4/256 has 49 CTA pairs per KV head, 196 in all; 152 SMs run 76 at a time,
    so the last wave would hold 44.  The tail of 11 pairs per KV head (the last
    452 queries) is split 3 ways: its workspace holds 3 partials per row."""
    p = _pool(num_kv_heads=4, head_dim=256, num_pages=128)
    f = lambda qs, c, hq=24, sms=152: B.lib().jf_prefill_chunk_workspace_bytes(
        ctypes.byref(p), qs, c, hq, sms)
    rows = 452 * 24 * 3
    assert f(30720, 2048) == 256 + -(-rows * 8 // 256) * 256 + rows * 256 * 4
    assert f(30720, 2048) == B.lib().jf_prefill_batch_workspace_bytes(0, 452, 24, 256, 3)
    minimal = B.jf_prefill_workspace_bytes()
    assert f(0, 2048) == minimal            # short prefix: unequal pairs, one launch
    assert f(30720, 798) == minimal         # 76 pairs: one wave
    assert f(30720, 1596) == minimal        # 152 pairs: two whole waves
    assert f(30720, 2394) == minimal        # 228 pairs: three whole waves
    assert f(30720, 2048, sms=196 * 2) == minimal   # all pairs at once
    assert f(30720, 2048, hq=23) == 0       # Hq % Hkv
    assert f(-1, 2048) == 0
    # a TQ4 pool's minimum (its rotated queries and partials) already covers
    # the balanced form's two launches
    codec = _codec(256)
    t = _tq4_pool(codec, num_kv_heads=4, head_dim=256, num_pages=128)
    g = B.lib().jf_prefill_chunk_workspace_bytes(ctypes.byref(t), 30720, 2048, 24, 152)
    assert g == B.lib().jf_prefill_batch_workspace_bytes(1, 2048, 24, 256, 1)


def test_split_planners_on_a_152_sm_gpu():
    """The host split planners with the SM count given (no device touched),
    against the split counts the benchmark runs on a 152-SM GB300."""
    # decode: one wave of 2 split CTAs per SM (affine), 1 per SM (TQ4)
    assert B.default_num_splits(1, 4, num_sms=152) == 76
    assert B.default_num_splits(1, 4, num_sms=152, format=B.JF_FMT_TQ4) == 38
    assert B.default_num_splits(2, 4, num_sms=152) == 38 + 2      # batch: even share + 2
    # verifier (affine): 24 / 4 heads give 2, 3, 3 row groups, all in one
    # 8-warp CTA per split and KV head, one CTA per SM; 8 / 4 heads at q_len 2
    # fit one group (6-warp CTAs, two per SM); 32 / 2 heads at q_len 4 give
    # 8 groups, 3 CTAs per split
    assert [B.default_verify_splits(1, L, 24, 4, num_sms=152) for L in (2, 3, 4)] == [38, 38, 38]
    assert B.default_verify_splits(1, 2, 8, 4, num_sms=152) == 76
    assert B.default_verify_splits(1, 4, 32, 2, num_sms=152) == 25
    # TQ4 verifier: the same warp-pair CTAs (one per SM) for two or more groups
    assert [B.default_verify_splits(1, L, 24, 4, num_sms=152, format=B.JF_FMT_TQ4)
            for L in (2, 3, 4)] == [38, 38, 38]
    assert B.default_verify_splits(1, 2, 8, 4, num_sms=152, format=B.JF_FMT_TQ4) == 38
    # prefill history splits (24 / 4 heads, 42 queries per CTA pair)
    ps = lambda qs, cl: B.default_prefill_splits(qs, cl, 24, 4, num_sms=152)
    assert ps([32704], [64]) == 9          # 4 pairs walking 512 tiles each
    assert ps([30720], [2048]) == 3
    assert ps([4096 * (b + 1) - 64 for b in range(8)], [64] * 8) == 2
    assert ps([4096 * (b + 1) - 512 for b in range(8)], [512] * 8) == 1
    assert ps([0], [0]) == 1               # nothing to schedule


def test_nvtx_ranges_wrap_every_enqueueing_call_when_enabled():
    """JFKV_NVTX=1 wraps each call that enqueues work in an NVTX range named
    after its C entry point; unset, the functions stay unwrapped."""
    import subprocess
    import sys
    names = ["jf_kv_quantize_append", "jf_paged_decode_attn", "jf_paged_decode_append_attn",
             "jf_paged_verify_attn", "jf_paged_decode_attn_noalloc", "jf_prefill_chunk_attn",
             "jf_prefill_batch_attn", "jf_kv_checkpoint", "jf_kv_restore"]
    code = ("import paper_2609_17475_gb300.binding as B; "
            f"print(all(hasattr(getattr(B, n), '__wrapped__') for n in {names!r}), "
            f"any(hasattr(getattr(B, n), '__wrapped__') for n in {names!r}))")
    import os
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    on = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, cwd=root,
                        env=dict(os.environ, JFKV_NVTX="1"))
    off = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, cwd=root,
                         env=dict(os.environ, JFKV_NVTX="0"))
    assert on.stdout.split() == ["True", "True"], on.stderr
    assert off.stdout.split() == ["False", "False"], off.stderr


SPAN_HDR = 32   # decode.cuh: places standing for a segment's start


def _span_segments(ctx, budget, dtok=32, min_cps=16, hdr=SPAN_HDR):
    """The span plan's segments as the decode kernels work them out
    (decode.cuh: span_nch, span_width, span_find, span_rows): each request a
    run of hdr places then its chunks, the runs laid end to end, pieces of W
    places, segment (piece x, request b) -> row x + b and real chunks
    [max(v0 - hdr, 0), max(v1 - hdr, 0))."""
    nch = [(max(0, c) + dtok - 1) // dtok for c in ctx]
    run = [n + hdr if n else 0 for n in nch]
    T = sum(run)
    W = max(min_cps, -(-T // max(budget, 1)))
    starts = [sum(run[:b]) for b in range(len(run))]
    segs = []
    for x in range(budget):
        pos, end = x * W, min((x + 1) * W, T)
        while pos < end:
            b = next(b for b in range(len(run)) if run[b] and starts[b] <= pos < starts[b] + run[b])
            v1 = min(end, starts[b] + run[b]) - starts[b]
            v0 = pos - starts[b]
            segs.append((x, b, max(v0 - hdr, 0), max(v1 - hdr, 0), v1 - v0))
            pos = starts[b] + v1
    merge = {}
    for b in range(len(run)):
        if run[b]:
            x0, x1 = starts[b] // W, (starts[b] + run[b] - 1) // W
            merge[b] = (x0 + b, x1 - x0 + 1)
    return nch, W, segs, merge


@pytest.mark.parametrize("seed", range(6))
def test_span_plan_rows_are_unique_contiguous_and_inside_the_workspace(seed):
    """Every request's chunks are covered exactly once by segments; each
    segment's partial row x + b is distinct, a request's rows are the
    contiguous run the merge reads, and every row fits the workspace's
    B * num_splits rows when budget <= B (num_splits - 1) + 1."""
    rng = np.random.default_rng(seed)
    B = int(rng.integers(2, 40))
    num_splits = int(rng.integers(2, 8))
    ctx = [int(c) for c in rng.choice([0, 1, 31, 32, 33, 500, 4096, 70000], size=B)]
    ctx = [c if rng.random() < 0.5 else int(rng.integers(0, 90000)) for c in ctx]
    slots = 38
    budget = min(slots, B * (num_splits - 1) + 1)
    nch, W, segs, merge = _span_segments(ctx, budget)
    rows = [x + b for (x, b, c0, c1, _) in segs]
    assert len(rows) == len(set(rows))
    assert max(rows, default=0) < B * num_splits
    for b in range(B):
        mine = sorted((c0, c1, x + b) for (x, bb, c0, c1, _) in segs if bb == b)
        covered = [c for c0, c1, _ in mine for c in range(c0, c1)]
        assert covered == list(range(nch[b]))
        if nch[b]:
            first, n = merge[b]
            assert sorted(r for _, _, r in mine) == list(range(first, first + n))
        else:
            assert b not in merge
    # the pieces carry equal work: every piece but the last holds exactly W
    # places (a request's start counts SPAN_HDR places before its chunks)
    per_piece = {}
    for (x, b, c0, c1, places) in segs:
        per_piece[x] = per_piece.get(x, 0) + places
    full = [per_piece[x] for x in sorted(per_piece)][:-1]
    assert all(w == W for w in full)
