"""Oracle parity at the benchmark workloads' own shapes and launch shapes.

* two requests of 196,608 and 131,072 positions whose pages are interleaved at
  random in one 1,280-page pool, decoded in one call with the fixed 32-split
  workspace (the batch split plan);
* 32 requests with contexts uniform in [1,024, 65,536] and K channel
  outliers, at page sizes 64, 128 and 256 (the split count the benchmark uses);
* the 32K + 6K workload: a 32,768-position prompt appended in 2,048-row
  chunks, then 6,144 fused append + decode steps captured in one CUDA graph,
  then a checkpoint of all 152 pages.

The oracle is too slow for every KV head of these sizes, so attention is
checked on sampled KV heads (0 and 3) or sampled decode steps; each sample is
compared element by element at the attention tolerance, and checkpoint bytes
are compared in full.  The oracle's reference for a KV head is built from the
same bf16 rows in a pool that holds only that head (head independence, Eq. 5,
is pinned on the CPU and checked bitwise on the GPU).
"""
import math

import numpy as np
import pytest
import torch

import paper_2609_17475_gb300 as jf
from oracle import affine4 as OA
from oracle import attention as OT
from oracle import checkpoint as OC
from paper_2609_17475_gb300 import synth
from tests.cases import assert_attention_close, bits

pytestmark = pytest.mark.gpu
DEV = "cuda"
SAMPLED_KV_HEADS = (0, 3)


def head_reference(k, v, kvh, page_table, context_lens, q_bits, P, num_pages, scale):
    """fp64 oracle decode of the G query heads of KV head kvh (q_bits holds
    just those heads), from a pool that holds only that KV head."""
    D = k.shape[-1]
    L1 = OA.PoolLayout(1, P, D)
    pool = OA.new_pool(L1, num_pages)
    req, pos = synth.append_rows_for(context_lens)
    OA.append(pool, L1, page_table, req.numpy(), pos.numpy(),
              bits(k[:, kvh:kvh + 1]), bits(v[:, kvh:kvh + 1]))
    return OT.paged_decode(pool, L1, page_table, context_lens, q_bits, scale)


def gpu_fill(pool, page_table, context_lens, k, v, rows_per_call=65536):
    """Quantize-append every row of every request (logical order)."""
    req, pos = synth.append_rows_for(context_lens)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    for s0 in range(0, len(req), rows_per_call):
        s1 = min(len(req), s0 + rows_per_call)
        jf.jf_kv_quantize_append(pool, page_table, req[s0:s1].to(DEV), pos[s0:s1].to(DEV),
                                 k[s0:s1].to(DEV), v[s0:s1].to(DEV), err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0


@pytest.mark.parametrize("heads", ["24/4/256", "8/2/128"])
def test_two_requests_interleaved_pool_32_splits(heads):
    """196,608 + 131,072 positions, pages interleaved in a 1,280-page pool,
    one batched decode call with a workspace of 32 splits per (request, head);
    at the paper's model shape and at the tiny workload's head shape (the
    workload statement's "same head shape as config 1" read both ways)."""
    w = synth.WORKLOADS["two_request_320k"]
    ctxs, S = w["context_lens"], w["num_splits"]
    geo = w["geometry"] if heads == "24/4/256" else synth.WORKLOADS["tiny"]["geometry"]
    Hq, Hkv, D, P, G = geo.num_q_heads, geo.num_kv_heads, geo.head_dim, geo.page_size, geo.group
    gen = synth.generator(w["seed"])
    pt = synth.interleaved_page_tables(gen, ctxs, P, w["num_pages"])
    k, v = synth.kv_rows(gen, sum(ctxs), Hkv, D)
    q = synth.normal_bf16(gen, (len(ctxs), Hq, D))
    # the two requests' pages really alternate in the pool
    owner = np.full(w["num_pages"], -1)
    for b, c in enumerate(ctxs):
        owner[pt[b, :synth.pages_for(c, P)].numpy()] = b
    used = owner[owner >= 0]
    assert (np.diff(used) != 0).sum() > 100

    pool = jf.KVPool.allocate(w["num_pages"], P, Hkv, D, device=DEV, fill=0xFF)
    ptd = pt.to(DEV)
    gpu_fill(pool, ptd, ctxs, k, v)
    out = torch.full((len(ctxs), Hq, D), float("nan"), dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(len(ctxs), Hq, Hkv, D, S, device=DEV)
    ws[256:] = 0xFF     # NaN partials: rows past the split plan must never be read
    scale = 1 / math.sqrt(D)
    jf.jf_paged_decode_attn(pool, ptd, torch.tensor(ctxs, dtype=torch.int32, device=DEV),
                            q.to(DEV), scale, out, ws, S)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    assert torch.isfinite(out.float()).all()
    for kvh in (0, Hkv - 1):          # the first and last KV heads
        hs = slice(kvh * G, (kvh + 1) * G)
        ref = head_reference(k, v, kvh, pt.numpy(), ctxs, bits(q[:, hs]), P, w["num_pages"],
                             scale)
        assert_attention_close(out[:, hs], ref)


@pytest.fixture(scope="module")
def mixed_batch():
    """The 32-request batch (contexts, rows with K outliers, queries) and the
    oracle's outputs for the sampled KV heads.  The oracle's result depends
    only on the logical rows, not on the page size or the physical page order
    (both pinned on the CPU), so one reference serves every page size."""
    w = synth.WORKLOADS["mixed_batch_32"]
    geo = w["geometry"]
    Hkv, D, G = geo.num_kv_heads, geo.head_dim, geo.group
    gen = synth.generator(w["seed"])
    ctxs = synth.context_lengths(gen, w["batch"], w["ctx_lo"], w["ctx_hi"])
    chans = synth.outlier_channels(gen, Hkv, D)
    k, v = synth.kv_rows(gen, sum(ctxs), Hkv, D, chans)
    q = synth.normal_bf16(gen, (w["batch"], geo.num_q_heads, D))
    scale = 1 / math.sqrt(D)
    pt, npages = synth.page_tables(synth.generator(w["seed"] + 1000), ctxs, 256)
    refs = {kvh: head_reference(k, v, kvh, pt.numpy(), ctxs,
                                bits(q[:, kvh * G:(kvh + 1) * G]), 256, npages, scale)
            for kvh in SAMPLED_KV_HEADS}
    return dict(w=w, ctxs=ctxs, k=k, v=v, q=q, scale=scale, refs=refs)


@pytest.mark.parametrize("P", [64, 128, 256])
def test_mixed_batch_32_requests(mixed_batch, P):
    m = mixed_batch
    geo = m["w"]["geometry"]
    Hq, Hkv, D, G = geo.num_q_heads, geo.num_kv_heads, geo.head_dim, geo.group
    ctxs = m["ctxs"]
    assert len(ctxs) == 32 and min(ctxs) >= 1024 and max(ctxs) <= 65536
    assert any(c % P for c in ctxs)                 # partial tail pages at every page size
    pt, npages = synth.page_tables(synth.generator(m["w"]["seed"] + P), ctxs, P)
    pool = jf.KVPool.allocate(npages, P, Hkv, D, device=DEV, fill=0xFF)
    ptd = pt.to(DEV)
    gpu_fill(pool, ptd, ctxs, m["k"], m["v"])
    S = jf.default_num_splits(len(ctxs), Hkv)
    out = torch.full((len(ctxs), Hq, D), float("nan"), dtype=torch.bfloat16, device=DEV)
    ws = jf.decode_workspace(len(ctxs), Hq, Hkv, D, S, device=DEV)
    ws[256:] = 0xFF
    jf.jf_paged_decode_attn(pool, ptd, torch.tensor(ctxs, dtype=torch.int32, device=DEV),
                            m["q"].to(DEV), m["scale"], out, ws, S)
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    assert torch.isfinite(out.float()).all()
    for kvh in SAMPLED_KV_HEADS:
        assert_attention_close(out[:, kvh * G:(kvh + 1) * G], m["refs"][kvh])


def test_prompt_32k_then_6k_fused_decode_steps_then_checkpoint():
    """The 32K + 6K workload's decode phase as the benchmark runs it: 6,144
    fused append + decode steps in one CUDA graph, each step appending its
    own K/V row at position ctx - 1 and attending ctx = 32,769 .. 38,912
    positions.  Sampled steps are compared with the oracle at their contexts,
    every step's output with the eager run bitwise, and the final 152-page
    checkpoint with the oracle's bytes."""
    w = synth.WORKLOADS["prefill_decode_32k_6k"]
    geo = w["geometry"]
    Hq, Hkv, D, P = geo.num_q_heads, geo.num_kv_heads, geo.head_dim, geo.page_size
    prompt, chunk, steps = w["prompt"], w["chunk"], w["decode_steps"]
    total = prompt + steps
    gen = synth.generator(w["seed"])
    k, v = synth.kv_rows(gen, total, Hkv, D)
    pt, npages = synth.page_tables(gen, [total], P)
    assert npages == 152
    qd = synth.normal_bf16(gen, (steps, 1, Hq, D))
    scale = 1 / math.sqrt(D)

    pool = jf.KVPool.allocate(npages, P, Hkv, D, device=DEV, fill=0)
    ptd = pt.to(DEV)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    zero_req = torch.zeros(chunk, dtype=torch.int32, device=DEV)
    for c in range(prompt // chunk):
        pos = torch.arange(c * chunk, (c + 1) * chunk, dtype=torch.int32, device=DEV)
        jf.jf_kv_quantize_append(pool, ptd, zero_req, pos, k[c * chunk:(c + 1) * chunk].to(DEV),
                                 v[c * chunk:(c + 1) * chunk].to(DEV), err)
    kd = k[prompt:].to(DEV).view(steps, 1, Hkv, D)
    vd = v[prompt:].to(DEV).view(steps, 1, Hkv, D)
    qdd = qd.to(DEV)
    out = torch.full((steps, 1, Hq, D), float("nan"), dtype=torch.bfloat16, device=DEV)
    ctx_all = torch.arange(prompt + 1, total + 1, dtype=torch.int32, device=DEV)
    S = jf.default_num_splits(1, Hkv)
    ws = jf.decode_workspace(1, Hq, Hkv, D, S, device=DEV)
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())

    def loop():
        for t in range(steps):
            jf.jf_paged_decode_append_attn(pool, ptd, ctx_all[t:t + 1], kd[t], vd[t], qdd[t],
                                           scale, out[t], ws, S, stream=stream)

    with torch.cuda.stream(stream):
        loop()                                   # eager: fills the pool step by step
    stream.synchronize()
    assert int(err.item()) == 0 and jf.workspace_status(ws) == 0
    eager = out.clone()
    out.fill_(float("nan"))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(graph, stream=stream):
            loop()
    graph.replay()
    torch.cuda.synchronize()
    assert jf.workspace_status(ws) == 0
    assert torch.equal(out, eager)               # the graph replays the same bits

    L = OA.PoolLayout(Hkv, P, D)
    opool = OA.new_pool(L, npages)
    req, pos = synth.append_rows_for([total])
    OA.append(opool, L, pt.numpy(), req.numpy(), pos.numpy(), bits(k), bits(v))
    for t in (0, 1, steps // 2 - 1, steps - 1):
        ref = OT.paged_decode(opool, L, pt.numpy(), [prompt + t + 1], bits(qd[t]), scale)
        assert_attention_close(out[t], ref)
    assert torch.isfinite(out.float()).all()

    blob = torch.empty(npages * pool.page_bytes, dtype=torch.uint8, device=DEV)
    jf.jf_kv_checkpoint(pool, ptd[0], npages, blob, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    assert np.array_equal(blob.cpu().numpy(), OC.checkpoint(opool, pt[0].numpy(), npages))
