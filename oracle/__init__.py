"""CPU oracle for the paged 4-bit KV path (test infrastructure).

Plain, slow, obviously correct NumPy code: fp32 IEEE emulation for the
quantizer (the bit-exact contract) and fp64 for attention.  It shares no code
with the CUDA library and imports nothing from the product package.

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import or run anything in this package.  The product path
never calls it; there is no CPU fallback.

Modules
-------
affine4     page-record layout, bf16 rounding, affine 4-bit group-64 quantizer,
            nibble packing, dequantization, quantize-on-append.
attention   paged decode attention (plain softmax definition), split partials
            and their merge, causal prefill-chunk attention.
tq4         TQ4 format (Sec. 3.1 Eq. 4; App. A.1 Table 3): Lloyd-Max
            codebook, Hadamard rotation with random signs, exact index
            decision, FP16 norms, page layout, append and reconstruction.
checkpoint  page-gather checkpoint and its inverse (restore scatter).
reservation the page reservation rule of Eq. 7.

Parity status: every function here is pinned by the ``-m "not gpu"`` tests in
``tests/test_oracle_*.py`` (closed forms, invariants, brute force on tiny
inputs, library routines on special cases, hand-derived fixtures in
``tests/golden/``).  The TQ4 codebook is pinned to the continuous-density
Lloyd iteration to within the grid's resolution (about 1e-4), not bit for bit.
"""
from . import affine4, attention, checkpoint, reservation, tq4  # noqa: F401
