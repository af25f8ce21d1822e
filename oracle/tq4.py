"""TQ4 KV format: codebook, rotation, encode, decode, page layout, append.

Test infrastructure (see ``oracle/__init__.py``): only tests, smoke() and the
bench CPU baseline use this module.

What the paper fixes (Sec. 3.1 Eq. 4; App. A.1 Table 3; Sec. 2 Eq. 2)
----------------------------------------------------------------------
* Encoding of a vector x of length d with norm rho = ||x||_2, unnormalized
  Hadamard matrix H_d and random-sign diagonal S:
      y = H_d S x / (sqrt(d) rho),   x_hat = rho_hat S H_d c[z] / sqrt(d),
  z the 4-bit indices into 16 shared centroids c, rho_hat the stored FP16
  norm (computed from an FP32 norm).
* Codebook: 16 FP32 centroids for the density proportional to
  (1 - x^2)^((d-3)/2) on [-1, 1] (the law of one coordinate of a uniform
  point on the unit sphere), built by Lloyd iteration on a 32,768-point grid
  over [-1 + 1e-6, 1 - 1e-6], quantile initialization, at most 100 centroid
  updates, stopping once the largest change is below 1e-6.
* Quantization: midpoint thresholds between the ordered centroids, strict >.
* Storage per vector: 32 U32 words of eight 4-bit indices (d = 256) and one
  FP16 norm; Eq. 2 counts 16 * 2 * 4 * (128 + 2) bytes per position for the
  paper's 16 layers x 4 KV heads.
* Signs: NumPy ``default_rng(seed + d * 7919)`` sampling +-1; K seed 0, V
  seed 1.  ``sign_vector`` is this module's reading of that rule; the codec
  functions take sign vectors as arguments, and the tests require the seeded
  inputs the CUDA path is given to equal ``sign_vector``'s.

Readings taken where the paper is silent
----------------------------------------
* Quantile initialization: centroid k starts at the first grid point whose
  cumulative normalized weight reaches (k + 1/2) / 16.
* Lloyd update: thresholds are the fp64 midpoints of the current centroids; a
  grid point x belongs to cell #{k : x > t_k} (the strict > of Table 3); each
  centroid moves to the weighted mean of its cell (an empty cell keeps its
  centroid); the loop ends after the update whose largest change is below
  1e-6, or after 100 updates.  The fp64 result is rounded to fp32.
* Encoding thresholds are fp32: t_k = fp32(fp32(c_k + c_{k+1}) * 0.5).
* Sign draw: one ``rng.integers(0, 2)`` per coordinate, 0 -> -1 and 1 -> +1
  (``2 * rng.integers(0, 2, size=d) - 1``, which is also the draw
  ``rng.choice([-1, 1], size=d)`` makes).
* H_d is Sylvester's ordering, H[i, j] = (-1)^popcount(i & j).
* The index decision is exact: with u = H_d S x (exact in fp64 for bf16
  inputs whose nonzero magnitudes span less than 2^37) and
  T_k = fp64(fp64(sqrt(d) * rho) * t_k), z_j = #{k : u_j > T_k}.  For
  d = 64 and 256, sqrt(d) * rho * t_k is exact, so this is y_j > t_k in real
  arithmetic.  A zero vector gets rho = 0, T_k = +-0 and z = 0 everywhere.
* rho = fp32 round-to-nearest of sqrt(s), s the correctly rounded fp64 sum
  of the squares (each square of a bf16 value is exact in fp64, and so is
  their sum whenever the vector's nonzero magnitudes span less than 2^14);
  rho_hat = fp16 round-to-nearest of rho, saturated at 65504.
* Index j of a vector sits in word j // 8 at nibble j % 8 (low nibble
  first), so element 2i is the low nibble of byte i, as in the affine format.

Page record layout (one physical page, ``page_bytes`` bytes):
    [K indices: Hkv x P x d/2 u8][V indices: same]
    [K norms: Hkv x P x fp16][V norms: same]
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

from .affine4 import KIND_K, KIND_V, bf16_to_f64, pack_nibbles, unpack_nibbles

LEVELS = 16
GRID_POINTS = 32768
GRID_EPS = 1e-6
MAX_UPDATES = 100
TOL = 1e-6
FP16_MAX = 65504.0


# --------------------------------------------------------------------------
# Codebook (App. A.1 Table 3: Lloyd-Max for the sphere-coordinate density)
# --------------------------------------------------------------------------
def grid_and_weights(d: int):
    """The 32,768-point grid and its normalized density weights."""
    x = np.linspace(-1.0 + GRID_EPS, 1.0 - GRID_EPS, GRID_POINTS)
    w = (1.0 - x * x) ** ((d - 3) / 2.0)
    return x, w / w.sum()


def quantile_init(x: np.ndarray, w: np.ndarray) -> np.ndarray:
    cdf = np.cumsum(w)
    return np.array([x[np.searchsorted(cdf, (k + 0.5) / LEVELS)] for k in range(LEVELS)])


def lloyd_update(x: np.ndarray, w: np.ndarray, c: np.ndarray) -> np.ndarray:
    """One centroid update: cells from the midpoint thresholds (strict >),
    then each centroid to its cell's weighted mean."""
    t = (c[:-1] + c[1:]) / 2.0
    cell = (x[:, None] > t[None, :]).sum(axis=1)
    new = c.copy()
    for k in range(LEVELS):
        m = cell == k
        mass = w[m].sum()
        if mass > 0:
            new[k] = (w[m] * x[m]).sum() / mass
    return new


def codebook_f64(d: int):
    """(fp64 centroids, number of updates made)."""
    x, w = grid_and_weights(d)
    c = quantile_init(x, w)
    n = 0
    for n in range(1, MAX_UPDATES + 1):
        new = lloyd_update(x, w, c)
        change = np.abs(new - c).max()
        c = new
        if change < TOL:
            break
    return c, n


def codebook(d: int) -> np.ndarray:
    """The 16 ascending fp32 centroids for head dimension d."""
    return codebook_f64(d)[0].astype(np.float32)


def thresholds(c32: np.ndarray) -> np.ndarray:
    """fp32 midpoints t_k = fp32(fp32(c_k + c_{k+1}) * 0.5), k = 0..14."""
    c32 = np.asarray(c32, dtype=np.float32)
    return ((c32[:-1] + c32[1:]).astype(np.float32) * np.float32(0.5)).astype(np.float32)


# --------------------------------------------------------------------------
# Rotation (Eq. 4)
# --------------------------------------------------------------------------
def hadamard(d: int) -> np.ndarray:
    """Unnormalized Sylvester Hadamard matrix, fp64 [d, d]."""
    i = np.arange(d)
    bits = np.bitwise_and(i[:, None], i[None, :])
    pop = np.zeros_like(bits)
    while bits.any():
        pop += bits & 1
        bits >>= 1
    return np.where(pop % 2 == 0, 1.0, -1.0)


SEED_K, SEED_V = 0, 1   # Table 3's default K and V seeds


def sign_vector(seed: int, d: int) -> np.ndarray:
    """The random-sign diagonal S of Table 3 for head_dim d, fp64 [d] of +-1:
    NumPy ``default_rng(seed + d * 7919)``, one uniform bit per coordinate,
    0 -> -1 and 1 -> +1 (module header: sign draw)."""
    rng = np.random.default_rng(int(seed) + int(d) * 7919)
    return (2 * rng.integers(0, 2, size=int(d)) - 1).astype(np.float64)


@dataclasses.dataclass(frozen=True)
class Codec:
    """Everything the encoding needs: d, fp32 centroids, K and V sign vectors."""
    head_dim: int
    centroids: np.ndarray     # fp32 [16], ascending
    signs_k: np.ndarray       # fp64 [d], entries +-1
    signs_v: np.ndarray

    def signs(self, kind: int) -> np.ndarray:
        return self.signs_k if kind == KIND_K else self.signs_v


def make_codec(head_dim: int, signs_k, signs_v) -> Codec:
    sk = np.asarray(signs_k, dtype=np.float64)
    sv = np.asarray(signs_v, dtype=np.float64)
    assert sk.shape == (head_dim,) and sv.shape == (head_dim,)
    assert np.all(np.abs(sk) == 1) and np.all(np.abs(sv) == 1)
    return Codec(head_dim, codebook(head_dim), sk, sv)


# --------------------------------------------------------------------------
# Encode / decode of vectors (Eq. 4, Table 3)
# --------------------------------------------------------------------------
def norms_f32(x: np.ndarray) -> np.ndarray:
    """rho = fp32(sqrt(s)) per row of fp64 x [..., d], s the correctly rounded
    fp64 sum of the squares."""
    s = np.array([math.fsum(v) for v in (x * x).reshape(-1, x.shape[-1])])
    return np.sqrt(s).astype(np.float32).reshape(x.shape[:-1])


def norm_to_fp16(rho: np.ndarray) -> np.ndarray:
    """fp16 bit patterns of rho (round to nearest even, saturated at 65504)."""
    r = np.minimum(np.asarray(rho, dtype=np.float64), FP16_MAX)
    h = np.asarray(r, dtype=np.float32).astype(np.float16)
    return np.where(np.isinf(h), np.float16(FP16_MAX), h).view(np.uint16)


def encode(x_bits: np.ndarray, codec: Codec, kind: int):
    """Encode bf16 vectors [..., d] -> (indices uint8 [..., d], norm fp16 bits [...])."""
    x = bf16_to_f64(np.asarray(x_bits, dtype=np.uint16))
    d = codec.head_dim
    assert x.shape[-1] == d
    rho = norms_f32(x)
    u = (x * codec.signs(kind)) @ hadamard(d).T                  # H S x, fp64
    r = np.float64(np.sqrt(np.float64(d))) * rho.astype(np.float64)
    t = thresholds(codec.centroids).astype(np.float64)
    T = r[..., None] * t                                           # [..., 15]
    z = (u[..., :, None] > T[..., None, :]).sum(axis=-1)
    return z.astype(np.uint8), norm_to_fp16(rho)


def fp16_to_f64(bits: np.ndarray) -> np.ndarray:
    return np.asarray(bits, dtype=np.uint16).view(np.float16).astype(np.float64)


def decode(z: np.ndarray, norm_bits: np.ndarray, codec: Codec, kind: int) -> np.ndarray:
    """x_hat = rho_hat S H c[z] / sqrt(d), fp64 [..., d]."""
    d = codec.head_dim
    cz = codec.centroids.astype(np.float64)[np.asarray(z, dtype=np.int64)]
    rot = cz @ hadamard(d).T                                       # H c[z]
    return fp16_to_f64(norm_bits)[..., None] * codec.signs(kind) * rot / np.sqrt(np.float64(d))


# --------------------------------------------------------------------------
# Page layout (Sec. 2 paged pool; Eq. 2 byte count)
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class Tq4Layout:
    num_kv_heads: int
    page_size: int
    head_dim: int
    codec: Codec

    @property
    def code_bytes(self) -> int:      # packed indices of one vector
        return self.head_dim // 2

    @property
    def codes_region(self) -> int:
        return self.num_kv_heads * self.page_size * self.code_bytes

    @property
    def norm_region(self) -> int:
        return self.num_kv_heads * self.page_size * 2

    @property
    def page_bytes(self) -> int:
        return 2 * self.codes_region + 2 * self.norm_region

    @property
    def bytes_per_position(self) -> int:
        """Packed K+V bytes per position per layer (Eq. 2 without the layer factor)."""
        return 2 * self.num_kv_heads * (self.code_bytes + 2)

    def codes_offset(self, kind: int, head: int, slot: int) -> int:
        return kind * self.codes_region + (head * self.page_size + slot) * self.code_bytes

    def norm_offset(self, kind: int, head: int, slot: int) -> int:
        return 2 * self.codes_region + kind * self.norm_region + (head * self.page_size + slot) * 2


def new_pool(layout: Tq4Layout, num_pages: int, fill: int = 0) -> np.ndarray:
    return np.full((num_pages, layout.page_bytes), fill, dtype=np.uint8)


def append(pool: np.ndarray, layout: Tq4Layout, page_table: np.ndarray,
           row_req: np.ndarray, row_pos: np.ndarray,
           k_bits: np.ndarray, v_bits: np.ndarray, chunk: int = 4096) -> None:
    """Encode rows k/v (bf16 bits [n, Hkv, d]) into ``pool`` in place; row i is
    logical position row_pos[i] of request row_req[i] (page table lookup)."""
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
            z, nb = encode(np.asarray(x[s:e], dtype=np.uint16), layout.codec, kind)
            cb = pack_nibbles(z)
            nbytes = np.ascontiguousarray(nb.astype("<u2")).view(np.uint8).reshape(nb.shape + (2,))
            base = page[:, None] * layout.page_bytes
            row = heads[None, :] * P + slot[:, None]
            c_off = base + kind * layout.codes_region + row * layout.code_bytes
            n_off = base + 2 * layout.codes_region + kind * layout.norm_region + row * 2
            flat[c_off[..., None] + np.arange(layout.code_bytes)] = cb
            flat[n_off[..., None] + np.arange(2)] = nbytes


def gather_head(pool: np.ndarray, layout: Tq4Layout, page_table_row: np.ndarray,
                ctx: int, head: int, kind: int) -> np.ndarray:
    """Reconstructed K (kind 0) or V (kind 1) of one KV head, logical positions
    [0, ctx), fp64 [ctx, d]."""
    P = layout.page_size
    t = np.arange(ctx, dtype=np.int64)
    page = np.asarray(page_table_row, dtype=np.int64)[t // P]
    slot = t % P
    flat = pool.reshape(-1)
    base = page * layout.page_bytes
    row = head * P + slot
    c_off = base + kind * layout.codes_region + row * layout.code_bytes
    n_off = base + 2 * layout.codes_region + kind * layout.norm_region + row * 2
    cb = flat[c_off[:, None] + np.arange(layout.code_bytes)]
    nb = flat[n_off[:, None] + np.arange(2)].copy().view("<u2")[:, 0]
    return decode(unpack_nibbles(cb), nb, layout.codec, kind)
