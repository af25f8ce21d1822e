"""Affine 4-bit group-64 KV format: layout, quantizer, packing, dequant, append.

Test infrastructure (see ``oracle/__init__.py``): only tests, smoke() and the
bench CPU baseline use this module.

What the paper fixes and what is read into it
---------------------------------------------
* Sec. 2 (paged KV pool, Eq. 2): K/V live in a fixed pool of pages of
  ``page_size`` positions; a per-request page table maps logical token order to
  physical pages.  Eq. 2 counts packed bytes per position per layer.
* App. A.1, Table 3 (quantization rule): 4-bit indices select one of 16
  ordered levels; an element takes the level chosen by midpoint thresholds
  between consecutive levels, compared with strict ``>``.  Here the 16 levels
  of a 64-element group are ``bias + k * scale`` (k = 0..15), so the thresholds
  are ``k + 0.5`` in units of ``scale`` and an exact midpoint goes to the lower
  code.  Table 3 also packs eight 4-bit indices per 32-bit word; read
  little-endian, element 2i is the low nibble of byte i.
* The affine group format itself (group 64 along head_dim, bf16 scale and
  bias) is the workload's stated format; the paper defines only TQ4 for KV.
  Readings taken where nothing is printed:
    - bias = group minimum (as bf16, exact), with -0 canonicalised to +0;
    - scale = bf16_rne(fp32(max - min) / 15), all fp32 operations IEEE
      round-to-nearest-even with no fused multiply-add;
    - r = fp32(x - bias) / scale (IEEE division), code = #{k in 0..14 :
      r > k + 0.5}; a zero scale gives all codes 0;
    - reconstruction x_hat = code * scale + bias (exact in fp64).

Page record layout (one physical page, ``page_bytes`` bytes):
    [K codes: Hkv x P x D/2 u8][V codes: same]
    [K scale/bias: Hkv x P x (D/64) x (scale bf16, bias bf16)][V scale/bias: same]
all little-endian; within a code row, element 2i is the low nibble of byte i.
"""
from __future__ import annotations

import dataclasses

import numpy as np

GROUP = 64          # elements per affine group along head_dim
LEVELS = 16         # 4-bit codes
KIND_K, KIND_V = 0, 1


# --------------------------------------------------------------------------
# Layout (Sec. 2: fixed page pool addressed through a page table)
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class PoolLayout:
    num_kv_heads: int
    page_size: int
    head_dim: int

    @property
    def n_groups(self) -> int:
        return self.head_dim // GROUP

    @property
    def code_bytes(self) -> int:      # packed codes of one vector
        return self.head_dim // 2

    @property
    def sb_bytes(self) -> int:        # scale+bias pairs of one vector
        return self.n_groups * 4

    @property
    def codes_region(self) -> int:    # bytes of K (or V) codes in a page
        return self.num_kv_heads * self.page_size * self.code_bytes

    @property
    def sb_region(self) -> int:       # bytes of K (or V) scale/bias in a page
        return self.num_kv_heads * self.page_size * self.sb_bytes

    @property
    def page_bytes(self) -> int:
        return 2 * self.codes_region + 2 * self.sb_region

    @property
    def bytes_per_position(self) -> int:
        """Packed K+V bytes per position per layer (analogue of Eq. 2)."""
        return 2 * self.num_kv_heads * (self.code_bytes + self.sb_bytes)

    def codes_offset(self, kind: int, head: int, slot: int) -> int:
        return kind * self.codes_region + (head * self.page_size + slot) * self.code_bytes

    def sb_offset(self, kind: int, head: int, slot: int) -> int:
        return (2 * self.codes_region + kind * self.sb_region
                + (head * self.page_size + slot) * self.sb_bytes)


def new_pool(layout: PoolLayout, num_pages: int, fill: int = 0) -> np.ndarray:
    return np.full((num_pages, layout.page_bytes), fill, dtype=np.uint8)


# --------------------------------------------------------------------------
# bf16 <-> fp32 (bit-level, round-to-nearest-even)
# --------------------------------------------------------------------------
def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float32."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns, round to nearest, ties to even.
    (Finite inputs; NaN is outside the format's contract.)"""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    return ((u + 0x7FFF + lsb) >> 16).astype(np.uint16)


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return bf16_to_f32(bits).astype(np.float64)


# --------------------------------------------------------------------------
# Quantizer (App. A.1 Table 3: midpoint thresholds, strict >)
# --------------------------------------------------------------------------
def quantize_groups(x_bits: np.ndarray):
    """Quantize bf16 groups.

    x_bits: uint16 [..., 64] (bf16 bit patterns).
    Returns (codes uint8 [..., 64], scale_bits uint16 [...], bias_bits uint16 [...]).
    """
    x_bits = np.asarray(x_bits, dtype=np.uint16)
    assert x_bits.shape[-1] == GROUP
    x = bf16_to_f32(x_bits)                                   # exact
    mn = x.min(axis=-1)
    mx = x.max(axis=-1)
    bias = (mn + np.float32(0.0)).astype(np.float32)          # -0 -> +0
    rng = (mx - mn).astype(np.float32)                        # fp32 RNE
    scale_bits = f32_to_bf16(rng / np.float32(LEVELS - 1))    # IEEE div, then bf16 RNE
    scale = bf16_to_f32(scale_bits)
    bias_bits = f32_to_bf16(bias)                             # exact (bias is a bf16 value)

    diff = (x - bias[..., None]).astype(np.float32)           # fp32 RNE
    with np.errstate(divide="ignore", invalid="ignore"):
        r = (diff / scale[..., None]).astype(np.float32)      # IEEE division
    codes = np.zeros(x.shape, dtype=np.uint8)
    for k in range(LEVELS - 1):                               # thresholds k + 1/2
        codes += (r > np.float32(k + 0.5)).astype(np.uint8)
    codes[scale == 0] = 0
    return codes, scale_bits, bias_bits


def dequantize(codes: np.ndarray, scale_bits: np.ndarray, bias_bits: np.ndarray) -> np.ndarray:
    """x_hat = code * scale + bias in fp64.  codes [..., n_g, 64]; scale/bias [..., n_g]."""
    s = bf16_to_f64(scale_bits)[..., None]
    b = bf16_to_f64(bias_bits)[..., None]
    return codes.astype(np.float64) * s + b


# --------------------------------------------------------------------------
# Packing (App. A.1 Table 3: eight 4-bit indices per U32 word, little-endian)
# --------------------------------------------------------------------------
def pack_nibbles(codes: np.ndarray) -> np.ndarray:
    codes = np.asarray(codes, dtype=np.uint8)
    lo = codes[..., 0::2] & 0xF
    hi = codes[..., 1::2] & 0xF
    return (lo | (hi << 4)).astype(np.uint8)


def unpack_nibbles(packed: np.ndarray) -> np.ndarray:
    packed = np.asarray(packed, dtype=np.uint8)
    out = np.empty(packed.shape[:-1] + (packed.shape[-1] * 2,), dtype=np.uint8)
    out[..., 0::2] = packed & 0xF
    out[..., 1::2] = packed >> 4
    return out


def encode_vectors(x_bits: np.ndarray):
    """Encode bf16 vectors [..., D] -> (code bytes [..., D/2], sb bytes [..., D/64*4])."""
    x_bits = np.asarray(x_bits, dtype=np.uint16)
    d = x_bits.shape[-1]
    g = x_bits.reshape(x_bits.shape[:-1] + (d // GROUP, GROUP))
    codes, sbits, bbits = quantize_groups(g)
    code_bytes = pack_nibbles(codes.reshape(x_bits.shape))
    sb = np.stack([sbits, bbits], axis=-1)                    # [..., n_g, 2] uint16
    sb_bytes = np.ascontiguousarray(sb.astype("<u2")).view(np.uint8)
    sb_bytes = sb_bytes.reshape(x_bits.shape[:-1] + (d // GROUP * 4,))
    return code_bytes, sb_bytes


def decode_vectors(code_bytes: np.ndarray, sb_bytes: np.ndarray) -> np.ndarray:
    """Inverse of encode_vectors up to quantization: fp64 [..., D]."""
    codes = unpack_nibbles(code_bytes)
    d = codes.shape[-1]
    n_g = d // GROUP
    sb = np.ascontiguousarray(sb_bytes).view("<u2").reshape(sb_bytes.shape[:-1] + (n_g, 2))
    xg = dequantize(codes.reshape(codes.shape[:-1] + (n_g, GROUP)), sb[..., 0], sb[..., 1])
    return xg.reshape(codes.shape)


# --------------------------------------------------------------------------
# Quantize-on-append (Sec. 3.3: pending cache writes land in the request's
# page slots; Sec. 2: page table maps logical position -> physical page)
# --------------------------------------------------------------------------
def append(pool: np.ndarray, layout: PoolLayout, page_table: np.ndarray,
           row_req: np.ndarray, row_pos: np.ndarray,
           k_bits: np.ndarray, v_bits: np.ndarray, chunk: int = 8192) -> None:
    """Quantize rows k/v (bf16 bits [n, Hkv, D]) into ``pool`` in place.

    Row i is logical position row_pos[i] of request row_req[i]; it lands in
    physical page page_table[row_req[i], row_pos[i] // P], slot row_pos[i] % P.
    """
    P = layout.page_size
    n = len(row_req)
    heads = np.arange(layout.num_kv_heads)
    flat = pool.reshape(-1)
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        req = np.asarray(row_req[s:e], dtype=np.int64)
        pos = np.asarray(row_pos[s:e], dtype=np.int64)
        page = np.asarray(page_table, dtype=np.int64)[req, pos // P]
        slot = pos % P
        assert (page >= 0).all() and (page < pool.shape[0]).all()
        for kind, x in ((KIND_K, k_bits), (KIND_V, v_bits)):
            cb, sb = encode_vectors(np.asarray(x[s:e], dtype=np.uint16))
            base = page[:, None] * layout.page_bytes                     # [m, 1]
            row = (heads[None, :] * P + slot[:, None])                   # [m, Hkv]
            c_off = base + kind * layout.codes_region + row * layout.code_bytes
            s_off = (base + 2 * layout.codes_region + kind * layout.sb_region
                     + row * layout.sb_bytes)
            flat[c_off[..., None] + np.arange(layout.code_bytes)] = cb
            flat[s_off[..., None] + np.arange(layout.sb_bytes)] = sb


def gather_head(pool: np.ndarray, layout: PoolLayout, page_table_row: np.ndarray,
                ctx: int, head: int, kind: int) -> np.ndarray:
    """Dequantized K (kind 0) or V (kind 1) of one KV head, logical positions
    [0, ctx), fp64 [ctx, D]."""
    P = layout.page_size
    t = np.arange(ctx, dtype=np.int64)
    page = np.asarray(page_table_row, dtype=np.int64)[t // P]
    slot = t % P
    flat = pool.reshape(-1)
    base = page * layout.page_bytes
    row = head * P + slot
    c_off = base + kind * layout.codes_region + row * layout.code_bytes
    s_off = base + 2 * layout.codes_region + kind * layout.sb_region + row * layout.sb_bytes
    cb = flat[c_off[:, None] + np.arange(layout.code_bytes)]
    sb = flat[s_off[:, None] + np.arange(layout.sb_bytes)]
    return decode_vectors(cb, sb)
