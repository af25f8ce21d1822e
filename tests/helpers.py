"""Small test helpers: dtype plumbing and exactly-quantizable inputs.

Nothing here implements the quantizer or attention; the exact-vector builder
only composes values ``bias + c * 2**e`` that any correct affine 4-bit group
quantizer must reproduce exactly, so attention over them can be checked
against library routines on the original fp64 values.
"""
import numpy as np
import torch


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """bf16 torch tensor -> numpy uint16 bit patterns (CPU copy)."""
    assert t.dtype == torch.bfloat16
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def bits_to_bf16(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits, dtype=np.uint16).view(np.int16)).view(torch.bfloat16)


def exact_groups(rng: np.random.Generator, shape, group=64):
    """fp64 values [..., D] whose every 64-group is {bias + c*step : c in 0..15}
    with c = 0 and c = 15 both present, step a power of two and bias a small
    multiple of step, so bf16 holds them exactly and an affine 4-bit quantizer
    (min/max, 15 steps) reproduces them exactly."""
    shape = tuple(shape)
    d = shape[-1]
    lead = shape[:-1]
    n_g = d // group
    c = rng.integers(0, 16, size=lead + (n_g, group))
    c[..., 0] = 0
    c[..., 1] = 15
    # shuffle positions of the forced extremes inside the group
    perm = np.argsort(rng.random(lead + (n_g, group)), axis=-1)
    c = np.take_along_axis(c, perm, axis=-1)
    e = rng.integers(-4, 0, size=lead + (n_g, 1)).astype(np.float64)
    step = np.exp2(e)
    bias = rng.integers(-16, 1, size=lead + (n_g, 1)) * step
    x = bias + c * step
    return x.reshape(shape)


def f64_to_bf16_tensor(x: np.ndarray) -> torch.Tensor:
    t = torch.from_numpy(np.asarray(x, dtype=np.float64)).to(torch.float32)
    b = t.to(torch.bfloat16)
    assert torch.equal(b.to(torch.float64), torch.from_numpy(np.asarray(x, dtype=np.float64))), \
        "value not exactly representable in bf16"
    return b
