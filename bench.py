"""Benchmark: 4-bit paged decode attention at 256K context on GB300.

Workload (default): the full-window single request -- 24 query / 4 KV heads,
head_dim 256, 262,144 positions in 1,024 pages of 256 positions with a random
physical page order, K/V drawn N(0,1) bf16 with 4 K channels per KV head
scaled x20, quantized to affine 4-bit group 64 -- over a 64-layer stack of
independent caches (19.3 GB of packed KV, far larger than L2, so no flush is
needed between steps).

One step = one decode token through the stack: per layer, quantize-append the
token's K/V row at the last position (append, then attend), then paged decode
attention with the split-K workspace (split kernel + merge kernel).

Prints one JSON line (rank 0).  ``--impl reference`` times the CPU oracle on a
bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

METRIC = "4-bit paged decode attention KV positions/s and HBM GB/s vs GB300 peak at 256K"
UNIT = "positions/s"


def measured_traffic(kernel):
    """DRAM bytes per launch of `kernel` from the committed ncu record, or None
    when any of the kernel's source files changed since the capture."""
    import hashlib
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    rec = json.load(open(p)).get(kernel)
    if not rec:
        return None
    for name, sha in rec["sources"].items():
        src = os.path.join(ROOT, name)
        if not os.path.exists(src) or hashlib.sha256(open(src, "rb").read()).hexdigest() != sha:
            return None
    return rec["dram_read"] + rec["dram_write"]


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during a region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except FileNotFoundError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), float(parts[3]), parts[4:]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        loaded = [r for r in rows if r[2] > 200.0] or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in loaded:
            for n, flag in zip(names, r[3][1:]):
                if flag.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(r[0] for r in loaded),
                "sm_max_mhz": max(r[1] for r in loaded),
                "power_w_max": max(r[2] for r in loaded),
                "samples": len(loaded), "reasons": sorted(reasons)}


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(value, world, device):
    """The largest `value` over all ranks (the slowest replica's time); the
    value itself when one process runs."""
    if world <= 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
def build_stack(jf, synth, layers, seed, dev):
    w = synth.WORKLOADS["full_window_256k"]
    geo = w["geometry"]
    ctx = w["context_lens"][0]
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    gcpu = synth.generator(seed)
    pools, tables = [], []
    req = torch.zeros(ctx, dtype=torch.int32, device=dev)
    pos = torch.arange(ctx, dtype=torch.int32, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    chunk = 65536
    for layer in range(layers):
        pt, npages = synth.page_tables(gcpu, [ctx], geo.page_size)
        pt = pt.to(dev)
        chans = synth.outlier_channels(gcpu, geo.num_kv_heads, geo.head_dim).to(dev)
        pool = jf.KVPool.allocate(npages, geo.page_size, geo.num_kv_heads, geo.head_dim,
                                  device=dev, fill=None)
        for s in range(0, ctx, chunk):
            n = min(chunk, ctx - s)
            k = torch.randn(n, geo.num_kv_heads, geo.head_dim, generator=g, device=dev)
            v = torch.randn(n, geo.num_kv_heads, geo.head_dim, generator=g, device=dev)
            for h in range(geo.num_kv_heads):
                k[:, h, chans[h]] *= 20.0
            jf.jf_kv_quantize_append(pool, pt, req[s:s + n], pos[s:s + n],
                                     k.to(torch.bfloat16), v.to(torch.bfloat16), err)
        pools.append(pool)
        tables.append(pt)
    torch.cuda.synchronize()
    assert int(err.item()) == 0, "append reported a device error"
    return geo, ctx, pools, tables


def run_ours(args, world, rank, local):
    import paper_2609_17475_gb300 as jf
    from paper_2609_17475_gb300 import synth

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    layers = args.layers
    geo, ctx, pools, tables = build_stack(jf, synth, layers, 1000 + rank, dev)
    Hq, Hkv, D = geo.num_q_heads, geo.num_kv_heads, geo.head_dim
    splits = args.splits or jf.default_num_splits(1, Hkv)
    scale = 1.0 / math.sqrt(D)
    g = torch.Generator(device=dev)
    g.manual_seed(77 + rank)
    # per-step inputs: one query and one new K/V row per layer
    q = torch.randn(layers, 1, Hq, D, generator=g, device=dev).to(torch.bfloat16)
    knew = torch.randn(layers, 1, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
    vnew = torch.randn(layers, 1, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
    out = torch.empty(layers, 1, Hq, D, dtype=torch.bfloat16, device=dev)
    ctx_t = torch.tensor([ctx], dtype=torch.int32, device=dev)
    ws = jf.decode_workspace(1, Hq, Hkv, D, splits, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def step(qs=q, ks=knew, vs=vnew, outs=out):
        # per layer: append the step's K/V row at position ctx - 1, then attend
        # over [0, ctx) -- one fused call (split kernel with the append + merge)
        for l in range(layers):
            jf.jf_paged_decode_append_attn(pools[l], tables[l], ctx_t, ks[l], vs[l], qs[l], scale,
                                           outs[l], ws, splits, stream=stream)

    with torch.cuda.stream(stream):
        for _ in range(2):
            step()
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(graph, stream=stream):
            step()
    stream.synchronize()

    # ---- device-timed steps (inputs resident in HBM) ----
    for _ in range(args.warmup):
        graph.replay()
    stream.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(args.steps):
                graph.replay()
            e1.record(stream)
        stream.synchronize()
    torch.cuda.synchronize()
    ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    if world > 1:
        torch.distributed.barrier()
    clocks = clk.summary()

    # ---- the same step over a region of at least one second (more graph
    # replays), so that run-to-run spread can be assessed on a longer window
    n_long = max(args.steps, int(math.ceil(1000.0 / max(ms / args.steps, 1e-3))))
    with ClockSampler(local) as clk_long:
        with torch.cuda.stream(stream):
            s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            s0.record(stream)
            for _ in range(n_long):
                graph.replay()
            s1.record(stream)
        stream.synchronize()
    long_ms = max_over_ranks(s0.elapsed_time(s1), world, dev)

    # ---- dominant call alone: decode (split + merge) for every layer, captured
    # as one CUDA graph and timed with events on its stream; the average call
    # is the graph time / layers (64 caches of 302 MB: inputs larger than L2)
    dgraph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(dgraph, stream=stream):
            for l in range(layers):
                jf.jf_paged_decode_attn(pools[l], tables[l], ctx_t, q[l], scale, out[l], ws,
                                        splits, stream=stream)
    stream.synchronize()
    reps = max(3, min(20, args.steps))
    with torch.cuda.stream(stream):
        dgraph.replay()
        d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        d0.record(stream)
        for _ in range(reps):
            dgraph.replay()
        d1.record(stream)
    stream.synchronize()
    decode_ms = d0.elapsed_time(d1) / (reps * layers)
    del dgraph
    app_ms = None

    # ---- end-to-end through the public API with host buffers ----
    # Every step copies its inputs (q, new K/V rows of all layers) from pinned
    # host memory and reads its outputs back, as a serving loop would: two
    # sets of device buffers, the copies of step i + 1 and the read-back of
    # step i - 1 on a copy stream overlapping step i's eager API calls on the
    # compute stream.  The timed region runs from before the first step's
    # copies to the end of the last step's read-back.
    nb = 2
    qh = [q.cpu().pin_memory() for _ in range(nb)]
    kh = [knew.cpu().pin_memory() for _ in range(nb)]
    vh = [vnew.cpu().pin_memory() for _ in range(nb)]
    oh = [torch.empty(out.shape, dtype=out.dtype).pin_memory() for _ in range(nb)]
    qd = [torch.empty_like(q) for _ in range(nb)]
    kd = [torch.empty_like(knew) for _ in range(nb)]
    vd = [torch.empty_like(vnew) for _ in range(nb)]
    od = [torch.empty_like(out) for _ in range(nb)]
    cstream = torch.cuda.Stream(device=dev)
    e2e_steps = max(3, min(args.steps, 50))

    def e2e_run(n):
        loaded = [torch.cuda.Event() for _ in range(n)]
        computed = [torch.cuda.Event() for _ in range(n)]
        read = [torch.cuda.Event() for _ in range(n)]

        def load(i):
            j = i % nb
            with torch.cuda.stream(cstream):
                if i >= nb:   # step i - nb has consumed these inputs
                    cstream.wait_event(computed[i - nb])
                qd[j].copy_(qh[j], non_blocking=True)
                kd[j].copy_(kh[j], non_blocking=True)
                vd[j].copy_(vh[j], non_blocking=True)
                loaded[i].record(cstream)

        def readback(i):
            j = i % nb
            with torch.cuda.stream(cstream):
                cstream.wait_event(computed[i])
                oh[j].copy_(od[j], non_blocking=True)
                read[i].record(cstream)

        load(0)
        for i in range(n):
            if i + 1 < n:
                load(i + 1)
            j = i % nb
            with torch.cuda.stream(stream):
                stream.wait_event(loaded[i])
                if i >= nb:   # the read-back of step i - nb has left od[j]
                    stream.wait_event(read[i - nb])
                step(qd[j], kd[j], vd[j], od[j])
                computed[i].record(stream)
            if i >= 1:
                readback(i - 1)
        readback(n - 1)

    e2e_run(2)
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record(cstream)
    stream.wait_event(f0)
    e2e_run(e2e_steps)
    f1.record(cstream)   # after the last read-back, which follows every step
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(f0.elapsed_time(f1) / e2e_steps, world, dev)
    h2d = qh[0].numel() * 2 + kh[0].numel() * 2 + vh[0].numel() * 2
    d2h = oh[0].numel() * 2
    torch.cuda.synchronize()
    assert int(err.item()) == 0 and jf.workspace_status(ws) == 0, "device error flag set"

    positions_per_step = ctx * layers
    ms_per_step = ms / args.steps
    value = positions_per_step * world / (ms_per_step / 1e3)
    bytes_per_pos = 2 * Hkv * (D // 2 + 4 * (D // 64))
    alg_bytes = ctx * bytes_per_pos + 2 * Hq * D * 2 + tables[0].numel() * 4 + 4
    hbm, src = peaks()
    achieved = alg_bytes / (decode_ms / 1e3) / 1e9
    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u4/bf16 (fp16 MMA, fp32 softmax)",
        "data": "synthetic: seeded N(0,1) bf16 K/V with x20 K outlier channels, affine 4-bit g64",
        "config": {"workload": "full_window_256k", "num_q_heads": Hq, "num_kv_heads": Hkv,
                   "head_dim": D, "page_size": geo.page_size, "context": ctx,
                   "layers": layers, "num_splits": splits, "batch": 1,
                   "l2": "inputs larger than L2 (64 independent 302 MB caches per step)",
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                   "step": "per layer: quantize-append 1 row + split-K decode + merge, "
                           "jf_paged_decode_append_attn (2 launches), CUDA graph"},
        "hbm_gbs_step": positions_per_step * bytes_per_pos / (ms_per_step / 1e3) / 1e9,
        "roofline": {"bound": "hbm", "kernel": "jf_paged_decode_attn (split + merge launches)",
                     "achieved": achieved, "peak": hbm, "peak_source": src, "unit": "GB/s",
                     "frac": achieved / hbm,
                     "traffic": measured_traffic("decode_split_kernel<256>"),
                     "alg_bytes_per_launch": alg_bytes, "avg_call_us": decode_ms * 1e3,
                     "frac_of_8tbs": achieved / 8000.0},
        "e2e": {"value": positions_per_step * world / (e2e_ms / 1e3), "unit": UNIT,
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_ms},
        "gpu_launches": args.steps * layers * 2,
        "clocks": clocks,
        "steady": {"steps": n_long, "seconds": long_ms / 1e3, "ms_per_step": long_ms / n_long,
                   "value": positions_per_step * world / (long_ms / n_long / 1e3),
                   "clocks": clk_long.summary()},
    }
    if args.rows:
        import json as _json
        pk = os.path.join(ROOT, "MEASURED_PEAKS.json")
        peak_tf = float(_json.load(open(pk))["bf16_tflops"]) if os.path.exists(pk) else 1900.0
        result["rows"] = bench_rows(jf, synth, dev, stream, hbm, peak_tf)
        result["rows"]["peak_tensor_tflops_f16"] = peak_tf
    if rank == 0 and args.cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(args)
    return result


# ---------------------------------------------------------------------------
# the other rows of the path, each on its own workload shape
# ---------------------------------------------------------------------------
def _event_time(fn, reps, stream):
    """Mean milliseconds per call of fn() on `stream`, CUDA events, after 2 warm calls."""
    with torch.cuda.stream(stream):
        for _ in range(2):
            fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
    stream.synchronize()
    return e0.elapsed_time(e1) / reps


ROW_GROUPS = ("tiny", "prompt", "two_request", "mixed", "verify", "tq4", "prefill_batch",
              "checkpoint")


def bench_rows(jf, synth, dev, stream, peaks_gbs, peak_tf, only=None, tq4_copies=8):
    """Tiny decode, append, prefill chunk, decode loop, checkpoint, two-request and
    mixed-batch decode (`only` selects one group of ROW_GROUPS).  Every tensor is
    allocated on `stream`, the stream the kernels run on, so the caching allocator
    never hands a buffer back out while a kernel still reads it."""
    with torch.cuda.stream(stream):
        out = _bench_rows(jf, synth, dev, stream, peaks_gbs, peak_tf, only)
        if only is None or only == "verify":
            out["verify_256k"] = _bench_verify(jf, dev, stream)
        if only is None or only == "tq4":
            out["tq4_256k"] = _bench_tq4(jf, synth, dev, stream, peaks_gbs, copies=tq4_copies)
        if only is None or only == "prefill_batch":
            out["prefill_batch"] = _bench_prefill_batch(jf, dev, stream, peak_tf)
        if only is None or only == "checkpoint":
            out["a5_checkpoint_256k_1024_pages"] = _bench_checkpoint(jf, dev, stream, peaks_gbs)
        return out


def _bench_checkpoint(jf, dev, stream, peaks_gbs):
    """Checkpoint of a whole 256K request (24/4/256, page 256): its 1,024 page
    records (301,989,888 B, random physical order) gathered in logical order
    into one contiguous buffer, and the restore scatter back into the pool.
    Each call moves 302 MB each way, more than twice the L2, so it runs from
    HBM (the 152-page row of the 32K + 6K workload largely fits in L2)."""
    Hkv, D, P, ctx = 4, 256, 256, 262144
    g = torch.Generator(device=dev)
    g.manual_seed(99)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    npg = ctx // P
    pool = jf.KVPool.allocate(npg, P, Hkv, D, device=dev, fill=None)
    pt = torch.randperm(npg, device=dev, generator=g).to(torch.int32).view(1, -1)
    for s0 in range(0, ctx, 65536):
        kk = torch.randn(65536, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vv = torch.randn(65536, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        jf.jf_kv_quantize_append(pool, pt, torch.zeros(65536, dtype=torch.int32, device=dev),
                                 torch.arange(s0, s0 + 65536, dtype=torch.int32, device=dev),
                                 kk, vv, err, stream=stream)
    blob = torch.empty(npg * pool.page_bytes, dtype=torch.uint8, device=dev)
    t_ck = _event_time(lambda: jf.jf_kv_checkpoint(pool, pt[0], npg, blob, err, stream=stream),
                       20, stream)
    t_rs = _event_time(lambda: jf.jf_kv_restore(pool, pt[0], npg, blob, err, stream=stream),
                       20, stream)
    stream.synchronize()
    assert int(err.item()) == 0, "checkpoint reported a device error"
    nbytes = 2 * npg * pool.page_bytes
    res = {"pages": npg, "page_bytes": pool.page_bytes, "alg_bytes": nbytes,
           "checkpoint_us": t_ck * 1e3, "checkpoint_GBps": nbytes / (t_ck / 1e3) / 1e9,
           "restore_us": t_rs * 1e3, "restore_GBps": nbytes / (t_rs / 1e3) / 1e9}
    res["frac_hbm"] = res["checkpoint_GBps"] / peaks_gbs
    res["roofline"] = {"bound": "hbm", "achieved": res["checkpoint_GBps"], "peak": peaks_gbs,
                       "unit": "GB/s", "frac": res["frac_hbm"],
                       "traffic": measured_traffic("page_copy_kernel")}
    del pool, blob
    return res


def _bench_prefill_batch(jf, dev, stream, peak_tf):
    """Prefill chunks of 8 requests (24/4/256, P 256, prefixes 4K..32K of
    32,768-position caches) in one jf_prefill_batch_attn launch against one
    jf_prefill_chunk_attn launch per request: 64-query chunks (the cadence the
    scheduler uses beside active decoders, Sec. 3.3) and 512-query chunks."""
    Hq, Hkv, D, P, B, ctx = 24, 4, 256, 256, 8, 32768
    g = torch.Generator(device=dev)
    g.manual_seed(31)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    npg = B * ctx // P
    pool = jf.KVPool.allocate(npg, P, Hkv, D, device=dev, fill=None)
    pt = torch.randperm(npg, device=dev, generator=g).to(torch.int32).view(B, ctx // P)
    for b in range(B):
        kk = torch.randn(ctx, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vv = torch.randn(ctx, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        jf.jf_kv_quantize_append(pool, pt, torch.full((ctx,), b, dtype=torch.int32, device=dev),
                                 torch.arange(ctx, dtype=torch.int32, device=dev), kk, vv, err,
                                 stream=stream)
    ws = torch.zeros(jf.jf_prefill_workspace_bytes(), dtype=torch.uint8, device=dev)
    scale = 1 / math.sqrt(D)
    res = {}
    # one request: a 64-query chunk after a 32,704-position prefix, whole history
    # per CTA pair vs the history split across CTA pairs and merged
    q1 = torch.randn(64, Hq, D, generator=g, device=dev).to(torch.bfloat16)
    o1 = torch.empty_like(q1)
    s1 = jf.default_prefill_splits([ctx - 64], [64], Hq, Hkv)
    w1 = jf.prefill_batch_workspace(64, Hq, D, s1, device=dev)
    t_one = _event_time(lambda: jf.jf_prefill_chunk_attn(pool, pt[0], q1, ctx - 64, scale, True,
                                                         o1, ws, stream=stream), 20, stream)
    t_one_s = _event_time(lambda: jf.jf_prefill_batch_attn(pool, pt[:1], [ctx - 64], [64], q1,
                                                           scale, True, o1, w1, num_splits=s1,
                                                           stream=stream), 20, stream)
    fl1 = 4 * Hq * D * (64 * (ctx - 64) + 64 * 65 // 2)
    res["one_chunk_64_at_32704"] = {"whole_history_us": t_one * 1e3, "splits": s1,
                                    "split_us": t_one_s * 1e3, "speedup": t_one / t_one_s,
                                    "TFLOPs_split": fl1 / (t_one_s / 1e3) / 1e12}
    # a large chunk: 2,048 queries after 30,720 positions, unsplit vs the default split
    q2 = torch.randn(2048, Hq, D, generator=g, device=dev).to(torch.bfloat16)
    o2 = torch.empty_like(q2)
    s2 = jf.default_prefill_splits([ctx - 2048], [2048], Hq, Hkv)
    w2 = jf.prefill_batch_workspace(2048, Hq, D, s2, device=dev)
    t2 = _event_time(lambda: jf.jf_prefill_chunk_attn(pool, pt[0], q2, ctx - 2048, scale, True,
                                                      o2, ws, stream=stream), 5, stream)
    t2s = _event_time(lambda: jf.jf_prefill_batch_attn(pool, pt[:1], [ctx - 2048], [2048], q2,
                                                       scale, True, o2, w2, num_splits=s2,
                                                       stream=stream), 5, stream)
    fl2 = 4 * Hq * D * (2048 * (ctx - 2048) + 2048 * 2049 // 2)
    res["one_chunk_2048_at_30720"] = {"unsplit_ms": t2, "splits": s2, "split_ms": t2s,
                                      "TFLOPs_unsplit": fl2 / (t2 / 1e3) / 1e12,
                                      "TFLOPs_split": fl2 / (t2s / 1e3) / 1e12}
    del w2
    for C in (64, 512):
        starts = [4096 * (b + 1) - C for b in range(B)]
        q = torch.randn(B * C, Hq, D, generator=g, device=dev).to(torch.bfloat16)
        o = torch.empty_like(q)
        tb = _event_time(lambda: jf.jf_prefill_batch_attn(pool, pt, starts, [C] * B, q, scale,
                                                          True, o, ws, stream=stream), 20, stream)
        sp = jf.default_prefill_splits(starts, [C] * B, Hq, Hkv)
        wsp = jf.prefill_batch_workspace(B * C, Hq, D, sp, device=dev)
        tbs = _event_time(lambda: jf.jf_prefill_batch_attn(pool, pt, starts, [C] * B, q, scale,
                                                           True, o, wsp, num_splits=sp,
                                                           stream=stream), 20, stream)

        def singles():
            for b in range(B):
                jf.jf_prefill_chunk_attn(pool, pt[b], q[b * C:(b + 1) * C], starts[b], scale,
                                         True, o[b * C:(b + 1) * C], ws, stream=stream)
        ts = _event_time(singles, 20, stream)
        stream.synchronize()
        assert jf.workspace_status(ws) == 0 and jf.workspace_status(wsp) == 0
        assert int(err.item()) == 0
        flops = sum(4 * Hq * D * (C * s0 + C * (C + 1) // 2) for s0 in starts)
        res[f"chunk_{C}"] = {"batched_us": tb * 1e3, "separate_us": ts * 1e3,
                             "speedup": ts / tb, "TFLOPs_batched": flops / (tb / 1e3) / 1e12,
                             "frac_tensor": flops / (tb / 1e3) / 1e12 / peak_tf,
                             "splits": sp, "batched_split_us": tbs * 1e3,
                             "TFLOPs_batched_split": flops / (tbs / 1e3) / 1e12}
    del pool
    return res


def _bench_tq4(jf, synth, dev, stream, peaks_gbs, copies=8):
    """TQ4 format (Sec. 3.1 Eq. 4) on the 256K full-window shape (24/4/256,
    page 256, random physical pages, 4 K channels per KV head x20): encode on
    append of a 2,048-row chunk, and single-query decode over `copies`
    independent caches taken in turn (2.2 GB in all, so no call finds the
    previous one's pages in L2)."""
    Hq, Hkv, D, P, ctx = 24, 4, 256, 256, 262144
    g = torch.Generator(device=dev)
    g.manual_seed(777)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    codec = jf.Tq4Codec(D, synth.tq4_signs(synth.TQ4_SEED_K, D), synth.tq4_signs(synth.TQ4_SEED_V, D))
    ch = torch.randperm(D, device=dev, generator=g)[:4]
    pools, tables = [], []
    for _ in range(copies):
        pt = torch.randperm(ctx // P, device=dev, generator=g).to(torch.int32).view(1, -1)
        pool = jf.KVPool.allocate(ctx // P, P, Hkv, D, device=dev, fill=None,
                                  format=jf.JF_FMT_TQ4, codec=codec)
        for s0 in range(0, ctx, 65536):
            kk = torch.randn(65536, Hkv, D, generator=g, device=dev)
            kk[:, :, ch] *= 20.0
            vv = torch.randn(65536, Hkv, D, generator=g, device=dev)
            jf.jf_kv_quantize_append(pool, pt, torch.zeros(65536, dtype=torch.int32, device=dev),
                                     torch.arange(s0, s0 + 65536, dtype=torch.int32, device=dev),
                                     kk.to(torch.bfloat16), vv.to(torch.bfloat16), err,
                                     stream=stream)
        pools.append(pool)
        tables.append(pt)
    c = torch.tensor([ctx], dtype=torch.int32, device=dev)
    q = torch.randn(1, Hq, D, generator=g, device=dev).to(torch.bfloat16)
    o = torch.empty_like(q)
    splits = jf.default_num_splits(1, Hkv, format=jf.JF_FMT_TQ4)
    ws = jf.decode_workspace(1, Hq, Hkv, D, splits, device=dev)
    it = [0]

    def call():
        i = it[0] % copies
        it[0] += 1
        jf.jf_paged_decode_attn(pools[i], tables[i], c, q, 1 / 16, o, ws, splits, stream=stream)
    t = _event_time(call, 8 * copies, stream)
    # encode on append: one 2,048-row chunk (8,192 vectors) into the first cache
    kk = torch.randn(2048, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
    vv = torch.randn(2048, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
    rr = torch.zeros(2048, dtype=torch.int32, device=dev)
    pp = torch.arange(0, 2048, dtype=torch.int32, device=dev)
    ta = _event_time(lambda: jf.jf_kv_quantize_append(pools[0], tables[0], rr, pp, kk, vv, err,
                                                      stream=stream), 20, stream)
    # prefill over TQ4 pages: 2,048 causal queries after a 30,720-position
    # prefix of the first cache (rotated queries, centroid tiles, merge with
    # the inverse rotation)
    Cq, q0 = 2048, 30720
    qp = torch.randn(Cq, Hq, D, generator=g, device=dev).to(torch.bfloat16)
    op = torch.empty_like(qp)
    wp = jf.prefill_batch_workspace(Cq, Hq, D, 1, device=dev, format=jf.JF_FMT_TQ4)
    tp = _event_time(lambda: jf.jf_prefill_chunk_attn(pools[0], tables[0][0], qp, q0, 1 / 16, True,
                                                      op, wp, stream=stream), 5, stream)
    fl = 4 * Hq * D * (Cq * q0 + Cq * (Cq + 1) // 2)
    # packed verifier over the first cache: q_len 2-4 tokens in one call
    ver = {}
    for Lq in (2, 3, 4):
        qv = torch.randn(1, Lq, Hq, D, generator=g, device=dev).to(torch.bfloat16)
        ov = torch.empty_like(qv)
        sv = jf.default_verify_splits(1, Lq, Hq, Hkv, format=jf.JF_FMT_TQ4)
        wv = jf.verify_workspace(1, Lq, Hq, Hkv, D, sv, device=dev)
        tv = _event_time(lambda: jf.jf_paged_verify_attn(pools[0], tables[0], c, qv, 1 / 16, ov,
                                                         wv, sv, stream=stream), 10, stream)
        stream.synchronize()
        assert jf.workspace_status(wv) == 0
        ver[f"q_len_{Lq}"] = {"us": tv * 1e3, "splits": sv}
    stream.synchronize()
    assert jf.workspace_status(ws) == 0 and int(err.item()) == 0 and jf.workspace_status(wp) == 0
    bpp = 2 * Hkv * (D // 2 + 2)
    alg = ctx * bpp + 2 * Hq * D * 2 + (ctx // P) * 4
    gbs = alg / (t / 1e3) / 1e9
    res = {"decode_us": t * 1e3, "positions_per_s": ctx / (t / 1e3), "GBps": gbs,
           "frac_of_measured": gbs / peaks_gbs, "splits": splits, "bytes_per_position": bpp,
           "alg_bytes_per_call": alg, "traffic": measured_traffic("tq4_split_kernel<256>"),
           "append_2048_rows_us": ta * 1e3,
           "append_GBps": (2048 * Hkv * D * 2 * 2 + 2048 * bpp) / (ta / 1e3) / 1e9,
           "prefill_2048_at_30720_ms": tp, "prefill_TFLOPs": fl / (tp / 1e3) / 1e12,
           "verify": ver}
    del pools
    return res


def _bench_verify(jf, dev, stream):
    """Packed verifier on one 262,144-position request (24/4/256, page 256):
    q_len 2-4 tokens in one call against q_len separate decode calls."""
    Hq, Hkv, D, P, ctx = 24, 4, 256, 256, 262144
    g = torch.Generator(device=dev)
    g.manual_seed(99)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    pt = torch.randperm(ctx // P, device=dev, generator=g).to(torch.int32).view(1, -1)
    pool = jf.KVPool.allocate(ctx // P, P, Hkv, D, device=dev, fill=None)
    for s0 in range(0, ctx, 65536):
        kk = torch.randn(65536, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        vv = torch.randn(65536, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
        jf.jf_kv_quantize_append(pool, pt, torch.zeros(65536, dtype=torch.int32, device=dev),
                                 torch.arange(s0, s0 + 65536, dtype=torch.int32, device=dev),
                                 kk, vv, err, stream=stream)
    c = torch.tensor([ctx], dtype=torch.int32, device=dev)
    bpp = 2 * Hkv * (D // 2 + 4 * D // 64)
    q1 = torch.randn(1, Hq, D, generator=g, device=dev).to(torch.bfloat16)
    o1 = torch.empty_like(q1)
    s1 = jf.default_num_splits(1, Hkv)
    w1 = jf.decode_workspace(1, Hq, Hkv, D, s1, device=dev)
    t1 = _event_time(lambda: jf.jf_paged_decode_attn(pool, pt, c, q1, 1 / 16, o1, w1, s1,
                                                     stream=stream), 20, stream)
    res = {"decode_us": t1 * 1e3}
    for L in (2, 3, 4):
        qv = torch.randn(1, L, Hq, D, generator=g, device=dev).to(torch.bfloat16)
        ov = torch.empty_like(qv)
        sv = jf.default_verify_splits(1, L, Hq, Hkv)
        wv = jf.verify_workspace(1, L, Hq, Hkv, D, sv, device=dev)
        tv = _event_time(lambda: jf.jf_paged_verify_attn(pool, pt, c, qv, 1 / 16, ov, wv, sv,
                                                         stream=stream), 20, stream)
        stream.synchronize()
        assert jf.workspace_status(wv) == 0 and int(err.item()) == 0
        res[f"q_len_{L}"] = {"us": tv * 1e3, "splits": sv,
                             "GBps_kv_once": ctx * bpp / (tv / 1e3) / 1e9,
                             "speedup_vs_separate_decodes": L * t1 / tv}
    del pool
    return res


def _bench_rows(jf, synth, dev, stream, peaks_gbs, peak_tf, only=None):
    out = {}
    want = lambda name: only is None or only == name

    def check(section, *words):
        stream.synchronize()
        bad = {"err": int(err.item())}
        for i, w in enumerate(words):
            bad[f"ws{i}"] = jf.workspace_status(w)
        assert not any(bad.values()), f"device status set in {section}: {bad}"

    g = torch.Generator(device=dev)
    g.manual_seed(4242)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    if want("tiny"):
        # ---- tiny workload: 8/2/128, P 256, one request of 4,096 positions in
        # 16 shuffled pages (L2-resident: a latency figure, not a bandwidth one)
        gt = synth.generator(1)
        geo = synth.WORKLOADS["tiny"]["geometry"]
        kt, vt = synth.kv_rows(gt, 4096, geo.num_kv_heads, geo.head_dim)
        ptt, npt = synth.page_tables(gt, [4096], geo.page_size)
        poolt = jf.KVPool.allocate(npt, geo.page_size, geo.num_kv_heads, geo.head_dim, device=dev)
        jf.jf_kv_quantize_append(poolt, ptt.to(dev), torch.zeros(4096, dtype=torch.int32, device=dev),
                                 torch.arange(4096, dtype=torch.int32, device=dev), kt.to(dev),
                                 vt.to(dev), err, stream=stream)
        qt = synth.normal_bf16(gt, (1, geo.num_q_heads, geo.head_dim)).to(dev)
        ot = torch.empty_like(qt)
        st = jf.default_num_splits(1, geo.num_kv_heads)
        wst = jf.decode_workspace(1, geo.num_q_heads, geo.num_kv_heads, geo.head_dim, st, device=dev)
        ct = torch.tensor([4096], dtype=torch.int32, device=dev)
        ptt = ptt.to(dev)
        tt = _event_time(lambda: jf.jf_paged_decode_attn(poolt, ptt, ct, qt, 1 / math.sqrt(128), ot,
                                                         wst, st, stream=stream), 50, stream)
        check("tiny", wst)
        out["tiny_4096_8q_2kv_128d"] = {"us": tt * 1e3, "positions_per_s": 4096 / (tt / 1e3)}
        del poolt
    if not want("prompt"):
        return _bench_rows_rest(jf, synth, dev, stream, peaks_gbs, peak_tf, only, out, g, err,
                                check, want)
    # ---- prefill-then-decode shapes: 24/4/256, P 256, 32K prompt + 6K decode
    Hq, Hkv, D, P = 24, 4, 256, 256
    prompt, chunk, steps = 32768, 2048, 6144
    total = prompt + steps
    npages = total // P
    pt = torch.randperm(npages, device=dev, generator=g).to(torch.int32).view(1, -1)
    pool = jf.KVPool.allocate(npages, P, Hkv, D, device=dev, fill=0)
    zero_req = torch.zeros(chunk, dtype=torch.int32, device=dev)
    kc = torch.randn(chunk, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
    vc = torch.randn(chunk, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
    qc = torch.randn(chunk, Hq, D, generator=g, device=dev).to(torch.bfloat16)
    oc = torch.empty_like(qc)
    pws = torch.zeros(jf.jf_prefill_workspace_bytes(), dtype=torch.uint8, device=dev)
    scale = 1 / math.sqrt(D)
    # a1: append of one 2,048-row chunk (positions 0..2047)
    pos0 = torch.arange(chunk, dtype=torch.int32, device=dev)
    t_app = _event_time(lambda: jf.jf_kv_quantize_append(pool, pt, zero_req, pos0, kc, vc, err,
                                                         stream=stream), 50, stream)
    app_bytes = 2 * chunk * Hkv * D * 2 + chunk * 2 * Hkv * (D // 2 + 4 * D // 64) + chunk * 8
    check("a1 append")
    out["a1_append_2048_rows"] = {"us": t_app * 1e3, "GBps": app_bytes / (t_app / 1e3) / 1e9,
                                  "frac_hbm": app_bytes / (t_app / 1e3) / 1e9 / peaks_gbs,
                                  "alg_bytes": app_bytes}
    # fill the whole prompt: 16 appends, each followed by its prefill chunk (timed end to end)
    def prefill_all():
        for c in range(prompt // chunk):
            pos = torch.arange(c * chunk, (c + 1) * chunk, dtype=torch.int32, device=dev)
            jf.jf_kv_quantize_append(pool, pt, zero_req, pos, kc, vc, err, stream=stream)
            jf.jf_prefill_chunk_attn(pool, pt[0], qc, c * chunk, scale, True, oc, pws,
                                     stream=stream)
    t_pf_all = _event_time(prefill_all, 3, stream)
    check("a1+a4 prompt", pws)
    flops_all = sum(4 * Hq * D * (chunk * c * chunk + chunk * (chunk + 1) // 2)
                    for c in range(prompt // chunk))
    # a4: the last chunk alone (2,048 causal queries over a 30,720-position prefix)
    q_last = prompt - chunk
    t_pf = _event_time(lambda: jf.jf_prefill_chunk_attn(pool, pt[0], qc, q_last, scale, True, oc,
                                                        pws, stream=stream), 10, stream)
    flops = 4 * Hq * D * (chunk * q_last + chunk * (chunk + 1) // 2)
    out["a4_prefill_chunk_2048_at_30720"] = {
        "ms": t_pf, "TFLOPs": flops / (t_pf / 1e3) / 1e12,
        "frac_tensor": flops / (t_pf / 1e3) / 1e12 / peak_tf, "flops": flops,
        "roofline": {"bound": "tensor", "achieved": flops / (t_pf / 1e3) / 1e12, "peak": peak_tf,
                     "unit": "TFLOP/s", "frac": flops / (t_pf / 1e3) / 1e12 / peak_tf,
                     "traffic": measured_traffic("prefill_kernel<256>")}}
    out["a1a4_prompt_32k_16_chunks"] = {
        "ms": t_pf_all, "TFLOPs_attention": flops_all / (t_pf_all / 1e3) / 1e12,
        "prompt_positions_per_s": prompt / (t_pf_all / 1e3)}
    # the same calls with the workspace that lets a chunk balance its waves
    # (whole waves of CTA pairs, then the last query tiles with split histories)
    pwb = torch.zeros(max(jf.jf_prefill_chunk_workspace_bytes(pool, c * chunk, chunk, Hq)
                          for c in range(prompt // chunk)), dtype=torch.uint8, device=dev)
    t_bal = _event_time(lambda: jf.jf_prefill_chunk_attn(pool, pt[0], qc, q_last, scale, True, oc,
                                                         pwb, stream=stream), 10, stream)

    def prefill_all_balanced():
        for c in range(prompt // chunk):
            pos = torch.arange(c * chunk, (c + 1) * chunk, dtype=torch.int32, device=dev)
            jf.jf_kv_quantize_append(pool, pt, zero_req, pos, kc, vc, err, stream=stream)
            jf.jf_prefill_chunk_attn(pool, pt[0], qc, c * chunk, scale, True, oc, pwb,
                                     stream=stream)
    t_all_bal = _event_time(prefill_all_balanced, 3, stream)
    check("a1+a4 prompt, balanced", pwb)
    out["a4_prefill_chunk_2048_at_30720"]["balanced"] = {
        "ms": t_bal, "TFLOPs": flops / (t_bal / 1e3) / 1e12,
        "frac_tensor": flops / (t_bal / 1e3) / 1e12 / peak_tf,
        "workspace_bytes": pwb.numel(), "launches": "prefill (whole waves) + prefill (split "
                                                    "tail) + merge"}
    out["a1a4_prompt_32k_16_chunks"]["balanced"] = {
        "ms": t_all_bal, "TFLOPs_attention": flops_all / (t_all_bal / 1e3) / 1e12,
        "prompt_positions_per_s": prompt / (t_all_bal / 1e3)}
    del pwb
    # decode loop of the 32K+6K workload: 6,144 x (append 1 row, decode) in one CUDA graph
    q1 = torch.randn(1, Hq, D, generator=g, device=dev).to(torch.bfloat16)
    o1 = torch.empty_like(q1)
    k1 = torch.randn(1, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
    v1 = torch.randn(1, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
    splits = jf.default_num_splits(1, Hkv)
    dws = jf.decode_workspace(1, Hq, Hkv, D, splits, device=dev)
    ctx_all = torch.arange(prompt + 1, total + 1, dtype=torch.int32, device=dev)

    def decode_loop():
        for t in range(steps):
            jf.jf_paged_decode_append_attn(pool, pt, ctx_all[t:t + 1], k1, v1, q1, scale, o1,
                                           dws, splits, stream=stream)
    with torch.cuda.stream(stream):
        decode_loop()
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(graph, stream=stream):
            decode_loop()
    t_dec = _event_time(graph.replay, 2, stream)
    check("decode loop", dws)
    pos_sum = int((prompt + 1 + total) * steps // 2)
    bpp = 2 * Hkv * (D // 2 + 4 * D // 64)
    out["a2a3_decode_6144_steps_32k_to_38k"] = {
        "ms": t_dec, "us_per_step": t_dec * 1e3 / steps,
        "positions_per_s": pos_sum / (t_dec / 1e3),
        "GBps": pos_sum * bpp / (t_dec / 1e3) / 1e9}
    del graph
    # a5: checkpoint of all 152 pages
    blob = torch.empty(npages * pool.page_bytes, dtype=torch.uint8, device=dev)
    t_ck = _event_time(lambda: jf.jf_kv_checkpoint(pool, pt[0], npages, blob, err,
                                                   stream=stream), 20, stream)
    check("checkpoint")
    ck_bytes = 2 * npages * pool.page_bytes
    out["a5_checkpoint_152_pages"] = {"us": t_ck * 1e3, "GBps": ck_bytes / (t_ck / 1e3) / 1e9,
                                      "frac_hbm": ck_bytes / (t_ck / 1e3) / 1e9 / peaks_gbs,
                                      "alg_bytes": ck_bytes}
    del pool, blob
    return _bench_rows_rest(jf, synth, dev, stream, peaks_gbs, peak_tf, only, out, g, err, check,
                            want)


def _bench_rows_rest(jf, synth, dev, stream, peaks_gbs, peak_tf, only, out, g, err, check, want):
    Hq, Hkv, D, P = 24, 4, 256, 256
    scale = 1 / math.sqrt(D)
    bpp = 2 * Hkv * (D // 2 + 4 * D // 64)
    if not want("two_request"):
        return _bench_rows_mixed(jf, synth, dev, stream, out, g, err, check, want)
    # ---- two requests, 196,608 + 131,072 positions, 1,280-page pool, 32 splits
    ctxs = [196608, 131072]
    gc = synth.generator(3)
    pt2 = synth.interleaved_page_tables(gc, ctxs, P, 1280).to(dev)
    pool2 = jf.KVPool.allocate(1280, P, Hkv, D, device=dev, fill=None)
    for b, c in enumerate(ctxs):
        for s0 in range(0, c, 65536):
            n = min(65536, c - s0)
            kk = torch.randn(n, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
            vv = torch.randn(n, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
            jf.jf_kv_quantize_append(pool2, pt2, torch.full((n,), b, dtype=torch.int32, device=dev),
                                     torch.arange(s0, s0 + n, dtype=torch.int32, device=dev),
                                     kk, vv, err, stream=stream)
    q2 = torch.randn(2, Hq, D, generator=g, device=dev).to(torch.bfloat16)
    o2 = torch.empty_like(q2)
    ws2 = jf.decode_workspace(2, Hq, Hkv, D, 32, device=dev)
    c2 = torch.tensor(ctxs, dtype=torch.int32, device=dev)
    t2 = _event_time(lambda: jf.jf_paged_decode_attn(pool2, pt2, c2, q2, scale, o2, ws2, 32,
                                                     stream=stream), 20, stream)
    check("two-request", ws2)
    out["two_request_320k_32_splits"] = {"us": t2 * 1e3, "positions_per_s": sum(ctxs) / (t2 / 1e3),
                                         "GBps": sum(ctxs) * bpp / (t2 / 1e3) / 1e9}
    del pool2
    return _bench_rows_mixed(jf, synth, dev, stream, out, g, err, check, want)


def _bench_rows_mixed(jf, synth, dev, stream, out, g, err, check, want):
    if not want("mixed"):
        return out
    Hq, Hkv, D = 24, 4, 256
    scale = 1 / math.sqrt(D)
    bpp = 2 * Hkv * (D // 2 + 4 * D // 64)
    # ---- 32 requests, contexts uniform in [1,024, 65,536], page size sweep
    gm = synth.generator(5)
    ctxm = synth.context_lengths(gm, 32, 1024, 65536)
    qm = torch.randn(32, Hq, D, generator=g, device=dev).to(torch.bfloat16)
    om = torch.empty_like(qm)
    cm = torch.tensor(ctxm, dtype=torch.int32, device=dev)
    sweep = {}
    for PS in (64, 128, 256):
        ptm, npm = synth.page_tables(gm, ctxm, PS)
        ptm = ptm.to(dev)
        poolm = jf.KVPool.allocate(npm, PS, Hkv, D, device=dev, fill=None)
        for b, c in enumerate(ctxm):
            kk = torch.randn(c, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
            vv = torch.randn(c, Hkv, D, generator=g, device=dev).to(torch.bfloat16)
            jf.jf_kv_quantize_append(poolm, ptm, torch.full((c,), b, dtype=torch.int32, device=dev),
                                     torch.arange(c, dtype=torch.int32, device=dev), kk, vv, err,
                                     stream=stream)
        sm_ = jf.default_num_splits(32, Hkv)
        wsm = jf.decode_workspace(32, Hq, Hkv, D, sm_, device=dev)
        tm = _event_time(lambda: jf.jf_paged_decode_attn(poolm, ptm, cm, qm, scale, om, wsm, sm_,
                                                         stream=stream), 20, stream)
        check(f"mixed batch P={PS}", wsm)
        sweep[f"page_{PS}"] = {"us": tm * 1e3, "positions_per_s": sum(ctxm) / (tm / 1e3),
                               "GBps": sum(ctxm) * bpp / (tm / 1e3) / 1e9}
        del poolm
    out["mixed_batch_32"] = {"sum_context": sum(ctxm), **sweep}
    return out


# ---------------------------------------------------------------------------
# CPU oracle (reference arm and cpu_baseline)
# ---------------------------------------------------------------------------
def _blas_threads():
    """(threads, library) of the BLAS NumPy is running, asked from the loaded
    library itself; (None, None) when it cannot be found."""
    try:
        from threadpoolctl import threadpool_info
        for info in threadpool_info():
            if info.get("user_api") == "blas":
                return int(info["num_threads"]), info.get("internal_api")
    except ImportError:
        pass
    import ctypes
    try:
        maps = open("/proc/self/maps").read().splitlines()
    except OSError:
        return None, None
    seen = set()
    for line in maps:
        path = line.split()[-1] if "/" in line else ""
        if "openblas" not in os.path.basename(path).lower() or path in seen:
            continue
        seen.add(path)
        try:
            lib = ctypes.CDLL(path)
        except OSError:
            continue
        for sym in ("scipy_openblas_get_num_threads64_", "scipy_openblas_get_num_threads",
                    "openblas_get_num_threads64_", "openblas_get_num_threads"):
            f = getattr(lib, sym, None)
            if f is not None:
                f.restype = ctypes.c_int
                return int(f()), "openblas"
    return None, None


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else platform)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.processor() or platform.machine()


def _oracle_sample(sample_heads=1):
    """Oracle decode of one layer's full 262,144-position window for
    ``sample_heads`` KV head(s) in this process; seconds and BLAS threads."""
    import numpy as np

    from oracle import affine4 as OA
    from oracle import attention as OT
    from paper_2609_17475_gb300 import synth

    w = synth.WORKLOADS["full_window_256k"]
    geo = w["geometry"]
    ctx = w["context_lens"][0]
    gen = synth.generator(w["seed"])
    chans = synth.outlier_channels(gen, geo.num_kv_heads, geo.head_dim)
    k, v = synth.kv_rows(gen, ctx, sample_heads, geo.head_dim, chans[:sample_heads])
    pt, npages = synth.page_tables(gen, [ctx], geo.page_size)
    q = synth.normal_bf16(gen, (1, geo.group * sample_heads, geo.head_dim))
    req, pos = synth.append_rows_for([ctx])
    bits = lambda t: t.contiguous().view(torch.int16).numpy().view(np.uint16)
    L = OA.PoolLayout(sample_heads, geo.page_size, geo.head_dim)
    pool = OA.new_pool(L, npages)
    OA.append(pool, L, pt.numpy(), req.numpy(), pos.numpy(), bits(k), bits(v))
    t0 = time.perf_counter()
    OT.paged_decode(pool, L, pt.numpy(), [ctx], bits(q), 1 / math.sqrt(geo.head_dim))
    dt = time.perf_counter() - t0
    threads, blas = _blas_threads()
    return {"seconds": dt, "blas_threads": threads, "blas": blas, "ctx": ctx,
            "frac": sample_heads / geo.num_kv_heads, "num_kv_heads": geo.num_kv_heads,
            "group": geo.group}


def _oracle_in_child(threads, sample_heads=1):
    """Run _oracle_sample in a fresh process whose BLAS / OpenMP pools are
    capped at `threads` (the cap must be set before NumPy loads its BLAS)."""
    env = dict(os.environ)
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[var] = str(threads)
    env.pop("RANK", None)
    env.pop("WORLD_SIZE", None)
    code = ("import json, sys; sys.path.insert(0, %r); import bench; "
            "print('ORACLE ' + json.dumps(bench._oracle_sample(%d)))" % (ROOT, sample_heads))
    p = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                       cwd=ROOT, timeout=600)
    for line in p.stdout.splitlines():
        if line.startswith("ORACLE "):
            return json.loads(line[7:])
    raise RuntimeError(f"oracle child failed ({p.returncode}): {p.stderr[-2000:]}")


def cpu_baseline(args, sample_heads=1):
    """The oracle on a bounded sample of the benchmark workload (one layer's
    262,144-position window, ``sample_heads`` of 4 KV heads, positions/s scaled
    to the full layer), timed twice on the host: BLAS capped at one thread and
    at every core.  The headline value is the all-cores run."""
    ncpu = os.cpu_count() or 1
    runs = {}
    for label, threads in (("one_thread", 1), ("all_cores", ncpu)):
        r = _oracle_in_child(threads, sample_heads)
        runs[label] = {"value": r["ctx"] * r["frac"] / r["seconds"], "seconds": r["seconds"],
                       "threads_requested": threads, "blas_threads": r["blas_threads"],
                       "blas": r["blas"]}
    best = runs["all_cores"]
    used = best["blas_threads"] if best["blas_threads"] is not None else ncpu
    return {"value": best["value"], "unit": UNIT, "cores": used, "kind": "oracle",
            "seconds": best["seconds"], "cpu_model": cpu_model(), "host_cpus": ncpu,
            "runs": runs,
            "sample": f"one layer, 262144 positions, {sample_heads} of 4 KV heads "
                      f"({6 * sample_heads} query heads), NumPy fp64 paged_decode; "
                      f"positions/s scaled to the full 4-head layer; BLAS capped at 1 thread "
                      f"and at all {ncpu} host CPUs in separate processes"}


def run_reference(args, world, rank):
    """The CPU oracle on a bounded sample of the benchmark workload (rank 0):
    each step is one oracle decode of the sample with BLAS on every host CPU
    (the first step also runs the one-thread comparison)."""
    if rank != 0:
        return None
    t0 = time.perf_counter()
    base = cpu_baseline(args)
    samples = [base["seconds"]]
    for _ in range(max(1, min(args.steps, 3)) - 1):
        samples.append(_oracle_in_child(os.cpu_count() or 1)["seconds"])
    sec = statistics.median(samples)
    value = 262144 * 0.25 / sec
    base = dict(base, value=value, seconds=sec, steps=len(samples))
    return {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": len(samples), "warmup": 0, "ms_per_step": sec * 1e3 * 4,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic: seeded N(0,1) bf16 K/V, affine 4-bit g64 (oracle's own quantizer)",
            "config": {"workload": "full_window_256k", "num_q_heads": 24, "num_kv_heads": 4,
                       "head_dim": 256, "page_size": 256, "context": 262144},
            "impl": "reference", "cpu_baseline": base,
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
            "wall_s": time.perf_counter() - t0}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--layers", type=int, default=64)
    ap.add_argument("--splits", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", dest="cpu_baseline", action="store_false")
    ap.add_argument("--no-rows", dest="rows", action="store_false",
                    help="skip the append / prefill / checkpoint / multi-request measurements")
    ap.add_argument("--row", choices=ROW_GROUPS, default=None,
                    help="run only this group of the row measurements (for profiling) and "
                         "print it; no bench line")
    ap.add_argument("--copies", type=int, default=8,
                    help="independent 256K caches the tq4 row cycles through (1 for profiling)")
    args = ap.parse_args()
    if args.row:
        import paper_2609_17475_gb300 as jf
        from paper_2609_17475_gb300 import synth
        dev = torch.device("cuda", 0)
        torch.cuda.set_device(dev)
        hbm, _ = peaks()
        pk = os.path.join(ROOT, "MEASURED_PEAKS.json")
        peak_tf = float(json.load(open(pk))["bf16_tflops"]) if os.path.exists(pk) else 1900.0
        stream = torch.cuda.Stream(device=dev)
        print(json.dumps(bench_rows(jf, synth, dev, stream, hbm, peak_tf, only=args.row,
                                    tq4_copies=args.copies)))
        return
    args.warmup = max(3, args.warmup)
    world, rank, local = dist_env()
    if world > 1 and args.impl == "ours":
        torch.distributed.init_process_group("nccl")
    if args.impl == "reference":
        res = run_reference(args, world, rank)
    else:
        res = run_ours(args, world, rank, local)
    if rank == 0 and res is not None:
        print(json.dumps(res))
    if world > 1 and args.impl == "ours":
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
