"""Page reservation of a request (Sec. 3.3, Eq. 7) -- test infrastructure.

Only tests may import this module.

An unshared request with prompt length p, requested output o and output
guarantee g_out reserves R = ceil((p + min(o, g_out)) / P) page equivalents
(P = 256 and g_out = 8,192 in the paper's four-lane policy).  Written here as
the plain definition with integer arithmetic.
"""
from __future__ import annotations

PAGE = 256
G_OUT = 8192


def reservation_pages(prompt_len: int, output_len: int, g_out: int = G_OUT,
                      page_size: int = PAGE) -> int:
    assert prompt_len >= 0 and output_len >= 0 and g_out >= 0 and page_size >= 1
    need = prompt_len + min(output_len, g_out)
    return -(-need // page_size)
