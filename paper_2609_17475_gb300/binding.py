"""Thin Python binding over libjfkv.so (include/jfkv.h).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  PyTorch supplies device memory and the current stream.  There is no
CPU fallback: if the library is missing or a call fails, this module raises.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libjfkv.so")

JF_OK = 0
JF_ERR_INVALID_ARG = -1
JF_ERR_UNSUPPORTED = -2
JF_ERR_WORKSPACE_TOO_SMALL = -3
JF_ERR_CUDA = -4
JF_DEV_ERR_PAGE_ID = 1
JF_DEV_ERR_POSITION = 2
JF_DEV_ERR_TIMEOUT = 4
JF_DEV_ERR_LAYOUT = 8
JF_DEV_ERR_RANGE = 16
JF_FMT_AFFINE4_G64 = 0
JF_FMT_TQ4 = 1

EXPORTS = [
    "jf_kv_page_bytes", "jf_attn_workspace_bytes", "jf_prefill_workspace_bytes",
    "jf_kv_quantize_append", "jf_paged_decode_attn", "jf_prefill_chunk_attn",
    "jf_kv_checkpoint", "jf_kv_restore", "jf_status_string", "jf_version",
    "jf_paged_decode_attn_noalloc", "jf_paged_decode_append_attn", "jf_paged_verify_attn",
    "jf_kv_page_bytes_fmt", "jf_tq4_codebook", "jf_prefill_batch_attn", "jf_reservation_pages",
    "jf_prefill_batch_workspace_bytes", "jf_prefill_chunk_workspace_bytes",
    "jf_selftest_bounded_wait",
]
JF_STATIC_WORKSPACE_BYTES = 8 << 20


class JfError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} failed: {status} ({status_string(status)})")


class _Tq4Codec(ctypes.Structure):
    _fields_ = [("centroids", ctypes.c_float * 16), ("signs_k", ctypes.c_int8 * 256),
                ("signs_v", ctypes.c_int8 * 256)]


class _Pool(ctypes.Structure):
    _fields_ = [("base", ctypes.c_void_p), ("num_pages", ctypes.c_int64),
                ("page_size", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("group_size", ctypes.c_int32),
                ("format", ctypes.c_int32), ("tq4", ctypes.POINTER(_Tq4Codec))]


_lib = None


def lib() -> ctypes.CDLL:
    """Load libjfkv.so (built in-tree by __graft_entry__.build())."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        P, I32, I64, SZ, F32 = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                                ctypes.c_size_t, ctypes.c_float)
        PP = ctypes.POINTER(_Pool)
        sig = {
            "jf_kv_page_bytes": (SZ, [I32, I32, I32]),
            "jf_attn_workspace_bytes": (SZ, [I32, I32, I32, I32, I32]),
            "jf_prefill_workspace_bytes": (SZ, []),
            "jf_kv_quantize_append": (ctypes.c_int, [PP, P, I32, I32, P, P, P, P, I32, P, P]),
            "jf_paged_decode_attn": (ctypes.c_int, [PP, P, I32, P, I32, P, I32, F32, P, P, SZ,
                                                    I32, P]),
            "jf_prefill_chunk_attn": (ctypes.c_int, [PP, P, P, I32, I32, I32, F32, I32, P, P,
                                                     SZ, P]),
            "jf_kv_checkpoint": (ctypes.c_int, [PP, P, I32, P, SZ, P, P]),
            "jf_kv_restore": (ctypes.c_int, [PP, P, I32, P, SZ, P, P]),
            "jf_paged_decode_attn_noalloc": (ctypes.c_int, [PP, P, I32, P, I32, P, I32, F32, P,
                                                            I32, P, P]),
            "jf_paged_decode_append_attn": (ctypes.c_int, [PP, P, I32, P, I32, P, P, P, I32, F32,
                                                           P, P, SZ, I32, P]),
            "jf_paged_verify_attn": (ctypes.c_int, [PP, P, I32, P, I32, P, I32, I32, F32, P, P,
                                                    SZ, I32, P]),
            "jf_kv_page_bytes_fmt": (SZ, [I32, I32, I32, I32]),
            "jf_tq4_codebook": (ctypes.c_int, [I32, ctypes.POINTER(ctypes.c_float)]),
            "jf_prefill_batch_attn": (ctypes.c_int, [PP, P, I32, I32, P, P, P, I32, F32, I32, I32,
                                                     P, P, SZ, P]),
            "jf_prefill_batch_workspace_bytes": (SZ, [I32, I64, I32, I32, I32]),
            "jf_prefill_chunk_workspace_bytes": (SZ, [PP, I32, I32, I32, I32]),
            "jf_reservation_pages": (I64, [I64, I64, I64, I32]),
            "jf_selftest_bounded_wait": (ctypes.c_int, [P, I32, P]),
            "jf_status_string": (ctypes.c_char_p, [ctypes.c_int]),
            "jf_version": (ctypes.c_char_p, []),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().jf_status_string(int(status)).decode()


def version() -> str:
    return lib().jf_version().decode()


# NVTX ranges around every call that enqueues work (named after the C entry
# point), for timelines in Nsight tools: enabled by JFKV_NVTX=1 in the
# environment when this module is imported; otherwise the functions are left
# unwrapped and cost nothing.
NVTX = os.environ.get("JFKV_NVTX", "0") not in ("", "0")


def _traced(fn):
    if not NVTX:
        return fn
    import functools

    @functools.wraps(fn)
    def wrapper(*args, **kwargs):
        torch.cuda.nvtx.range_push(fn.__name__)
        try:
            return fn(*args, **kwargs)
        finally:
            torch.cuda.nvtx.range_pop()
    return wrapper


def _check(fn: str, status: int) -> None:
    if status != JF_OK:
        raise JfError(fn, status)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _need(t: torch.Tensor, dtype, name: str) -> None:
    if not isinstance(t, torch.Tensor) or t.dtype != dtype or not t.is_cuda or not t.is_contiguous():
        raise TypeError(f"{name} must be a contiguous CUDA tensor of dtype {dtype}")


def jf_tq4_codebook(head_dim: int):
    """The 16 ascending fp32 TQ4 centroids for head_dim (computed by the library)."""
    import numpy as np
    buf = (ctypes.c_float * 16)()
    _check("jf_tq4_codebook", lib().jf_tq4_codebook(int(head_dim), buf))
    return np.frombuffer(bytes(buf), dtype=np.float32).copy()


class Tq4Codec:
    """TQ4 codec (Sec. 3.1 Eq. 4): the library's centroids for head_dim and the
    K and V random-sign vectors (+1 / -1, length head_dim), which the caller
    draws (synth.tq4_signs gives the paper's NumPy draw)."""

    def __init__(self, head_dim: int, signs_k, signs_v, centroids=None):
        """``centroids`` (16 ascending fp32 values, |c| < 1) replaces the
        library's Lloyd-Max codebook when given."""
        import numpy as np
        sk = np.asarray(signs_k).astype(np.int64)
        sv = np.asarray(signs_v).astype(np.int64)
        if sk.shape != (head_dim,) or sv.shape != (head_dim,):
            raise ValueError("sign vectors must have head_dim entries")
        if not (np.isin(sk, (-1, 1)).all() and np.isin(sv, (-1, 1)).all()):
            raise ValueError("signs must be +1 or -1")
        self.head_dim = int(head_dim)
        if centroids is None:
            self.centroids = jf_tq4_codebook(head_dim)
        else:
            self.centroids = np.asarray(centroids, dtype=np.float32).copy()
            if self.centroids.shape != (16,):
                raise ValueError("a TQ4 codebook has 16 centroids")
        self.signs_k, self.signs_v = sk, sv
        c = _Tq4Codec()
        for i in range(16):
            c.centroids[i] = float(self.centroids[i])
        for j in range(head_dim):
            c.signs_k[j] = int(sk[j])
            c.signs_v[j] = int(sv[j])
        self._c = c


@dataclasses.dataclass
class KVPool:
    """A paged 4-bit KV pool: ``data`` is a CUDA uint8 tensor [num_pages, page_bytes].
    ``codec`` is required for the TQ4 format."""
    data: torch.Tensor
    page_size: int
    num_kv_heads: int
    head_dim: int
    group_size: int = 64
    format: int = JF_FMT_AFFINE4_G64
    codec: Optional[Tq4Codec] = None

    @staticmethod
    def allocate(num_pages: int, page_size: int, num_kv_heads: int, head_dim: int,
                 device="cuda", fill: Optional[int] = 0, format: int = JF_FMT_AFFINE4_G64,
                 codec: Optional[Tq4Codec] = None) -> "KVPool":
        pb = jf_kv_page_bytes_fmt(format, num_kv_heads, page_size, head_dim)
        if pb == 0:
            raise ValueError("unsupported pool geometry")
        if format == JF_FMT_TQ4 and (codec is None or codec.head_dim != head_dim):
            raise ValueError("a TQ4 pool needs a codec for its head_dim")
        if fill is None:
            data = torch.empty(num_pages, pb, dtype=torch.uint8, device=device)
        else:
            data = torch.full((num_pages, pb), fill, dtype=torch.uint8, device=device)
        return KVPool(data, page_size, num_kv_heads, head_dim, format=format, codec=codec)

    @property
    def num_pages(self) -> int:
        return self.data.shape[0]

    @property
    def page_bytes(self) -> int:
        return self.data.shape[1]

    def c_struct(self) -> _Pool:
        p = _Pool(self.data.data_ptr(), self.num_pages, self.page_size, self.num_kv_heads,
                  self.head_dim, self.group_size, self.format)
        if self.codec is not None:
            p.tq4 = ctypes.pointer(self.codec._c)
        return p


def jf_kv_page_bytes(num_kv_heads: int, page_size: int, head_dim: int) -> int:
    return int(lib().jf_kv_page_bytes(num_kv_heads, page_size, head_dim))


def jf_kv_page_bytes_fmt(format: int, num_kv_heads: int, page_size: int, head_dim: int) -> int:
    return int(lib().jf_kv_page_bytes_fmt(format, num_kv_heads, page_size, head_dim))


def jf_attn_workspace_bytes(batch: int, num_q_heads: int, num_kv_heads: int, head_dim: int,
                            num_splits: int) -> int:
    return int(lib().jf_attn_workspace_bytes(batch, num_q_heads, num_kv_heads, head_dim,
                                             num_splits))


def jf_prefill_workspace_bytes() -> int:
    return int(lib().jf_prefill_workspace_bytes())


def decode_workspace(batch, num_q_heads, num_kv_heads, head_dim, num_splits, device="cuda"):
    n = jf_attn_workspace_bytes(batch, num_q_heads, num_kv_heads, head_dim, num_splits)
    if n == 0:
        raise ValueError("invalid workspace geometry")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def workspace_status(workspace: torch.Tensor) -> int:
    """Device status word (JF_DEV_* bits) stored in the first 4 bytes."""
    return int(workspace[:4].view(torch.int32).item())


@_traced
def jf_kv_quantize_append(pool: KVPool, page_table: torch.Tensor, row_req: torch.Tensor,
                          row_pos: torch.Tensor, k: torch.Tensor, v: torch.Tensor,
                          err_flag: Optional[torch.Tensor] = None, stream=None) -> None:
    _need(page_table, torch.int32, "page_table")
    _need(row_req, torch.int32, "row_req")
    _need(row_pos, torch.int32, "row_pos")
    _need(k, torch.bfloat16, "k")
    _need(v, torch.bfloat16, "v")
    n = row_req.numel()
    if row_pos.numel() != n or k.shape != (n, pool.num_kv_heads, pool.head_dim) or v.shape != k.shape:
        raise ValueError("shape mismatch")
    if err_flag is not None:
        _need(err_flag, torch.int32, "err_flag")
    pt = page_table if page_table.dim() == 2 else page_table.view(1, -1)
    st = lib().jf_kv_quantize_append(ctypes.byref(pool.c_struct()), _ptr(pt), pt.shape[1],
                                      pt.shape[0], _ptr(row_req), _ptr(row_pos), _ptr(k), _ptr(v),
                                      n, _ptr(err_flag), _stream(stream))
    _check("jf_kv_quantize_append", st)


@_traced
def jf_paged_decode_attn(pool: KVPool, page_table: torch.Tensor, context_lens: torch.Tensor,
                         q: torch.Tensor, softmax_scale: float, out: torch.Tensor,
                         workspace: torch.Tensor, num_splits: int, stream=None) -> None:
    _need(page_table, torch.int32, "page_table")
    _need(context_lens, torch.int32, "context_lens")
    _need(q, torch.bfloat16, "q")
    _need(out, torch.bfloat16, "out")
    _need(workspace, torch.uint8, "workspace")
    B, Hq, D = q.shape
    if out.shape != q.shape or D != pool.head_dim or page_table.shape[0] != B or context_lens.numel() != B:
        raise ValueError("shape mismatch")
    st = lib().jf_paged_decode_attn(ctypes.byref(pool.c_struct()), _ptr(page_table),
                                     page_table.shape[1], _ptr(context_lens), B, _ptr(q), Hq,
                                     float(softmax_scale), _ptr(out), _ptr(workspace),
                                     workspace.numel(), int(num_splits), _stream(stream))
    _check("jf_paged_decode_attn", st)


@_traced
def jf_paged_decode_append_attn(pool: KVPool, page_table: torch.Tensor,
                                context_lens: torch.Tensor, k_new: torch.Tensor,
                                v_new: torch.Tensor, q: torch.Tensor, softmax_scale: float,
                                out: torch.Tensor, workspace: torch.Tensor, num_splits: int,
                                stream=None) -> None:
    """Append the step's K/V row of every request at position context_lens[b] - 1,
    then decode: the same pool bytes and output as jf_kv_quantize_append followed
    by jf_paged_decode_attn, in one launch pair."""
    _need(page_table, torch.int32, "page_table")
    _need(context_lens, torch.int32, "context_lens")
    _need(k_new, torch.bfloat16, "k_new")
    _need(v_new, torch.bfloat16, "v_new")
    _need(q, torch.bfloat16, "q")
    _need(out, torch.bfloat16, "out")
    _need(workspace, torch.uint8, "workspace")
    B, Hq, D = q.shape
    if out.shape != q.shape or D != pool.head_dim or page_table.shape[0] != B or context_lens.numel() != B:
        raise ValueError("shape mismatch")
    if tuple(k_new.shape) != (B, pool.num_kv_heads, D) or v_new.shape != k_new.shape:
        raise ValueError("k_new / v_new must be [batch, Hkv, D]")
    st = lib().jf_paged_decode_append_attn(ctypes.byref(pool.c_struct()), _ptr(page_table),
                                            page_table.shape[1], _ptr(context_lens), B,
                                            _ptr(k_new), _ptr(v_new), _ptr(q), Hq,
                                            float(softmax_scale), _ptr(out), _ptr(workspace),
                                            workspace.numel(), int(num_splits), _stream(stream))
    _check("jf_paged_decode_append_attn", st)


@_traced
def jf_paged_verify_attn(pool: KVPool, page_table: torch.Tensor, context_lens: torch.Tensor,
                         q: torch.Tensor, softmax_scale: float, out: torch.Tensor,
                         workspace: torch.Tensor, num_splits: int, stream=None) -> None:
    """Packed verifier: q, out are [batch, q_len, Hq, D]; token i of request b
    sees positions up to context_lens[b] - q_len + i."""
    _need(page_table, torch.int32, "page_table")
    _need(context_lens, torch.int32, "context_lens")
    _need(q, torch.bfloat16, "q")
    _need(out, torch.bfloat16, "out")
    _need(workspace, torch.uint8, "workspace")
    B, L, Hq, D = q.shape
    if out.shape != q.shape or D != pool.head_dim or page_table.shape[0] != B or context_lens.numel() != B:
        raise ValueError("shape mismatch")
    st = lib().jf_paged_verify_attn(ctypes.byref(pool.c_struct()), _ptr(page_table),
                                     page_table.shape[1], _ptr(context_lens), B, _ptr(q), L, Hq,
                                     float(softmax_scale), _ptr(out), _ptr(workspace),
                                     workspace.numel(), int(num_splits), _stream(stream))
    _check("jf_paged_verify_attn", st)


def verify_workspace(batch, q_len, num_q_heads, num_kv_heads, head_dim, num_splits, device="cuda"):
    return decode_workspace(batch, q_len * num_q_heads, num_kv_heads, head_dim, num_splits,
                            device=device)


def _num_sms(device, num_sms) -> int:
    """num_sms when given (planning for a GPU of that size), else the SM count
    of `device` (the current one when None)."""
    if num_sms is not None:
        return int(num_sms)
    dev = device if device is not None else torch.cuda.current_device()
    return torch.cuda.get_device_properties(dev).multi_processor_count


def default_verify_splits(batch: int, q_len: int, num_q_heads: int, num_kv_heads: int,
                          device=None, format: int = JF_FMT_AFFINE4_G64,
                          num_sms: Optional[int] = None) -> int:
    """Split cap for the verifier, one full wave of split CTAs.  The G * q_len
    (token, head) rows of a KV head form nt = ceil(G * q_len / 8) groups of 8.
    With nt >= 2 each split of a KV head runs ceil(nt / 3) CTAs, one per SM
    (warp pairs sharing the unpacking or the centroid lookups, either
    format); with nt = 1 one CTA, two per SM (affine) or one (TQ4)."""
    nt = -(-(num_q_heads // num_kv_heads) * q_len // 8)
    sms = _num_sms(device, num_sms)
    if nt >= 2:
        slots, per_head = sms, -(-nt // min(nt, 3))
    elif format == JF_FMT_TQ4:
        slots, per_head = sms, 1
    else:
        slots, per_head = 2 * sms, 1
    per = slots // (batch * num_kv_heads * per_head)   # one full wave
    return max(1, per if batch == 1 else per + 2)


@_traced
def jf_paged_decode_attn_noalloc(pool: KVPool, page_table: torch.Tensor,
                                 context_lens: torch.Tensor, q: torch.Tensor, softmax_scale: float,
                                 out: torch.Tensor, num_splits: int,
                                 err_flag: Optional[torch.Tensor] = None, stream=None) -> None:
    """Decode attention for callers that cannot allocate device memory: the
    split partials live in a fixed device array inside libjfkv.so
    (JF_STATIC_WORKSPACE_BYTES), shared by every call on the device, so calls
    that overlap on the GPU race.  The first call on a device sets the array up
    and should come before any stream capture."""
    _need(page_table, torch.int32, "page_table")
    _need(context_lens, torch.int32, "context_lens")
    _need(q, torch.bfloat16, "q")
    _need(out, torch.bfloat16, "out")
    if err_flag is not None:
        _need(err_flag, torch.int32, "err_flag")
    B, Hq, D = q.shape
    if out.shape != q.shape or D != pool.head_dim or page_table.shape[0] != B or context_lens.numel() != B:
        raise ValueError("shape mismatch")
    st = lib().jf_paged_decode_attn_noalloc(ctypes.byref(pool.c_struct()), _ptr(page_table),
                                             page_table.shape[1], _ptr(context_lens), B, _ptr(q),
                                             Hq, float(softmax_scale), _ptr(out), int(num_splits),
                                             _ptr(err_flag), _stream(stream))
    _check("jf_paged_decode_attn_noalloc", st)


@_traced
def jf_prefill_chunk_attn(pool: KVPool, page_table_row: torch.Tensor, q: torch.Tensor,
                          q_start: int, softmax_scale: float, causal: bool, out: torch.Tensor,
                          workspace: torch.Tensor, stream=None) -> None:
    _need(page_table_row, torch.int32, "page_table_row")
    _need(q, torch.bfloat16, "q")
    _need(out, torch.bfloat16, "out")
    _need(workspace, torch.uint8, "workspace")
    C, Hq, D = q.shape
    if out.shape != q.shape or D != pool.head_dim:
        raise ValueError("shape mismatch")
    st = lib().jf_prefill_chunk_attn(ctypes.byref(pool.c_struct()), _ptr(page_table_row), _ptr(q),
                                      int(q_start), C, Hq, float(softmax_scale), int(bool(causal)),
                                      _ptr(out), _ptr(workspace), workspace.numel(),
                                      _stream(stream))
    _check("jf_prefill_chunk_attn", st)


JF_PREFILL_MAX_BATCH = 64


def prefill_batch_workspace(total_rows: int, num_q_heads: int, head_dim: int, num_splits: int,
                            device="cuda", format: int = JF_FMT_AFFINE4_G64) -> torch.Tensor:
    n = int(lib().jf_prefill_batch_workspace_bytes(int(format), int(total_rows), num_q_heads,
                                                   head_dim, num_splits))
    if n == 0:
        raise ValueError("invalid workspace geometry")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def jf_prefill_chunk_workspace_bytes(pool: "KVPool", q_start: int, chunk_len: int,
                                     num_q_heads: int, num_sms: int = 0) -> int:
    """Workspace bytes for jf_prefill_chunk_attn's wave-balanced form (the
    plain minimum when the chunk runs as one launch); num_sms 0: the current
    device's."""
    return int(lib().jf_prefill_chunk_workspace_bytes(ctypes.byref(pool.c_struct()), int(q_start),
                                                      int(chunk_len), int(num_q_heads),
                                                      int(num_sms)))


def prefill_chunk_workspace(pool: "KVPool", q_start: int, chunk_len: int, num_q_heads: int,
                            device="cuda") -> torch.Tensor:
    """A zeroed workspace with which jf_prefill_chunk_attn balances its waves."""
    n = jf_prefill_chunk_workspace_bytes(pool, q_start, chunk_len, num_q_heads)
    if n == 0:
        raise ValueError("invalid workspace geometry")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def default_prefill_splits(q_start, chunk_len, num_q_heads: int, num_kv_heads: int,
                           device=None, num_sms: Optional[int] = None) -> int:
    """History splits for a launch.  The kernel runs one CTA per SM, two per
    pair, so SMs / 2 pairs run at once; each candidate split count is scored
    by its makespan when the pairs' history tiles (64 positions each, plus a
    fixed cost per pair) are list-scheduled longest first onto those slots,
    and the best is returned (no split below 8 tiles; a 2 % margin keeps the
    smaller count on a near tie, splits costing partial writes and a merge)."""
    import heapq
    G = num_q_heads // num_kv_heads
    qpc = max(1, 128 // G)
    work = []   # history tiles of every CTA pair (per KV head)
    for s0, c in zip(q_start, chunk_len):
        c = int(c)
        for k in range((-(-c // qpc) + 1) // 2 if c else 0):
            last = min(c, (2 * k + 2) * qpc)
            work += [-(-(int(s0) + last) // 64)] * num_kv_heads
    if not work:
        return 1
    slots = max(1, _num_sms(device, num_sms) // 2)
    longest = max(work)
    scores = []
    for S in [1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 12, 14, 16, 20, 24, 32, 48, 64]:
        if S > 1 and longest // S < 8:
            break
        items = sorted((-(-w // S) + 2 for w in work for _ in range(S)), reverse=True)
        if len(items) <= slots:
            t = items[0]
        else:
            heap = [0] * slots
            for it in items:
                heapq.heapreplace(heap, heap[0] + it)
            t = max(heap)
        t += 2 if S > 1 else 0   # the merge pass
        scores.append((S, t))
    best_t = min(t for _, t in scores)
    return next(S for S, t in scores if t <= 1.02 * best_t)


@_traced
def jf_prefill_batch_attn(pool: KVPool, page_table: torch.Tensor, q_start, chunk_len,
                          q: torch.Tensor, softmax_scale: float, causal: bool, out: torch.Tensor,
                          workspace: torch.Tensor, num_splits: int = 1, stream=None) -> None:
    """Prefill chunks of several requests in one launch.  ``q`` / ``out`` are
    the requests' chunks concatenated, [sum(chunk_len), Hq, D]; ``q_start`` and
    ``chunk_len`` are host sequences (one entry per page-table row).  With
    ``num_splits`` > 1 each query tile's history is split across CTA pairs and
    merged (workspace from prefill_batch_workspace)."""
    _need(page_table, torch.int32, "page_table")
    _need(q, torch.bfloat16, "q")
    _need(out, torch.bfloat16, "out")
    _need(workspace, torch.uint8, "workspace")
    B = page_table.shape[0]
    if len(q_start) != B or len(chunk_len) != B:
        raise ValueError("one q_start and chunk_len per page-table row")
    N, Hq, D = q.shape
    if out.shape != q.shape or D != pool.head_dim or N != sum(int(c) for c in chunk_len):
        raise ValueError("shape mismatch")
    qs = (ctypes.c_int32 * B)(*[int(x) for x in q_start])
    cl = (ctypes.c_int32 * B)(*[int(x) for x in chunk_len])
    st = lib().jf_prefill_batch_attn(ctypes.byref(pool.c_struct()), _ptr(page_table),
                                      page_table.shape[1], B, qs, cl, _ptr(q), Hq,
                                      float(softmax_scale), int(bool(causal)), int(num_splits),
                                      _ptr(out), _ptr(workspace), workspace.numel(),
                                      _stream(stream))
    _check("jf_prefill_batch_attn", st)


def jf_reservation_pages(prompt_len: int, output_len: int, g_out: int = 8192,
                         page_size: int = 256) -> int:
    """Eq. 7: ceil((prompt_len + min(output_len, g_out)) / page_size)."""
    r = int(lib().jf_reservation_pages(int(prompt_len), int(output_len), int(g_out),
                                       int(page_size)))
    if r < 0:
        raise ValueError("invalid reservation arguments")
    return r


def jf_selftest_bounded_wait(status: torch.Tensor, arrive: bool, stream=None) -> None:
    """Run the bounded-wait give-up path alone (include/jfkv.h): with
    arrive=False the wait runs out and JF_DEV_ERR_TIMEOUT is ORed into status."""
    _need(status, torch.int32, "status")
    _check("jf_selftest_bounded_wait",
           lib().jf_selftest_bounded_wait(_ptr(status), 1 if arrive else 0, _stream(stream)))


@_traced
def jf_kv_checkpoint(pool: KVPool, page_table_row: torch.Tensor, num_pages: int,
                     dst: torch.Tensor, err_flag: Optional[torch.Tensor] = None,
                     stream=None) -> None:
    _need(page_table_row, torch.int32, "page_table_row")
    _need(dst, torch.uint8, "dst")
    if err_flag is not None:
        _need(err_flag, torch.int32, "err_flag")
    st = lib().jf_kv_checkpoint(ctypes.byref(pool.c_struct()), _ptr(page_table_row),
                                 int(num_pages), _ptr(dst), dst.numel(), _ptr(err_flag),
                                 _stream(stream))
    _check("jf_kv_checkpoint", st)


@_traced
def jf_kv_restore(pool: KVPool, page_table_row: torch.Tensor, num_pages: int,
                  src: torch.Tensor, err_flag: Optional[torch.Tensor] = None,
                  stream=None) -> None:
    _need(page_table_row, torch.int32, "page_table_row")
    _need(src, torch.uint8, "src")
    if err_flag is not None:
        _need(err_flag, torch.int32, "err_flag")
    st = lib().jf_kv_restore(ctypes.byref(pool.c_struct()), _ptr(page_table_row), int(num_pages),
                              _ptr(src), src.numel(), _ptr(err_flag), _stream(stream))
    _check("jf_kv_restore", st)


def default_num_splits(batch: int, num_kv_heads: int, device=None,
                       format: int = JF_FMT_AFFINE4_G64, num_sms: Optional[int] = None) -> int:
    """Split cap per (request, KV head) so the split grid fills every SM slot
    once (two split CTAs per SM for the affine format, one for TQ4, whose
    centroid table takes a CTA's spare shared memory).  A batch plans its
    splits over all requests together, and its workspace then needs room for
    about two more splits per request than an even share (rounding up per
    request)."""
    target = (1 if format == JF_FMT_TQ4 else 2) * _num_sms(device, num_sms)
    per = -(-target // (batch * num_kv_heads))
    return max(1, per if batch == 1 else per + 2)
