"""Page-gather checkpoint and its inverse (test infrastructure).

Only tests, smoke() and the bench CPU baseline use this module.

Sec. 3.4 (and App. A.1's persistence path): a checkpoint reads the request's
page runs in place, while the request keeps ownership, and writes them out as
one contiguous packed stream; restoration writes the packed runs back into the
existing pool.  Here the unit is the whole page record, so the checkpoint of
``num_pages`` logical pages is the concatenation of the page records the page
table names, in logical order, tail bytes of the last page included.
"""
from __future__ import annotations

import numpy as np


def checkpoint(pool: np.ndarray, page_table_row: np.ndarray, num_pages: int) -> np.ndarray:
    """bytes [num_pages * page_bytes]: record page_table_row[k] at offset k * page_bytes."""
    out = [pool[int(page_table_row[k])] for k in range(num_pages)]
    if not out:
        return np.zeros(0, dtype=np.uint8)
    return np.concatenate(out).astype(np.uint8)


def restore(pool: np.ndarray, page_table_row: np.ndarray, num_pages: int,
            blob: np.ndarray) -> None:
    """Inverse of ``checkpoint``: write record k of ``blob`` into page page_table_row[k]."""
    page_bytes = pool.shape[1]
    for k in range(num_pages):
        pool[int(page_table_row[k])] = blob[k * page_bytes:(k + 1) * page_bytes]
