"""Pins for the Eq. 7 reservation rule and the library's host implementation.

The oracle's ceiling formula is checked against a brute-force search for the
smallest page count that holds the prompt plus the guaranteed output, against
the paper's numbers (page 256, g_out 8,192, a four-lane policy that permits
16,384 output tokens while reserving the first 8,192), and the library's
jf_reservation_pages is checked against the oracle (host call, no GPU).
"""
import pytest

from oracle import reservation as R
from paper_2609_17475_gb300 import binding as B


def _brute(p, o, g, page):
    n = 0
    while n * page < p + min(o, g):
        n += 1
    return n


@pytest.mark.parametrize("p,o,g,page", [
    (0, 0, 8192, 256), (1, 0, 8192, 256), (256, 0, 8192, 256), (257, 0, 8192, 256),
    (32768, 6144, 8192, 256), (262144, 16384, 8192, 256), (131072, 16384, 8192, 256),
    (1000, 100000, 8192, 64), (5, 7, 3, 2),
])
def test_reservation_matches_brute_force_and_library(p, o, g, page):
    want = _brute(p, o, g, page)
    assert R.reservation_pages(p, o, g, page) == want
    assert B.jf_reservation_pages(p, o, g, page) == want


def test_paper_policy_numbers():
    # 32K prompt + 6K output (the evolution workload) -> 152 pages of 256
    assert R.reservation_pages(32768, 6144) == 152
    # a 16,384-token request reserves only its first 8,192 output positions
    assert R.reservation_pages(0, 16384) == 8192 // 256 == 32
    assert R.reservation_pages(262144, 16384) == (262144 + 8192) // 256


def test_library_rejects_invalid_arguments():
    L = B.lib()
    assert L.jf_reservation_pages(-1, 0, 8192, 256) == -1
    assert L.jf_reservation_pages(0, 0, 8192, 0) == -1
    assert L.jf_reservation_pages(2 ** 62, 0, 2 ** 62, 256) >= 0
    assert L.jf_reservation_pages(2 ** 63 - 10, 100, 8192, 256) == -1
