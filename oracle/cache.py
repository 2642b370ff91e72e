"""Paged KV cache model (oracle; test infrastructure).

Sec. 3 defines one cache KV^i_{<t} per layer and leaves its updates implicit;
Alg. 2 grows it by the k+1 verify rows and truncates it after acceptance.  The
paper does not fix a memory layout.  The reading used throughout: per layer,
K and V are each stored as pages of `page_size` tokens, array
[num_pages, Hkv, page_size, D]; sequence b's logical position `pos` lives in
page page_table[b, pos // page_size] at offset pos % page_size, i.e. in slot

    slot = page_table[b, pos // page_size] * page_size + pos % page_size.
"""

from __future__ import annotations

import numpy as np


def slot(page_table_row: np.ndarray, pos: int, page_size: int) -> int:
    return int(page_table_row[pos // page_size]) * page_size + pos % page_size


def gather_rows(cache: np.ndarray, page_table_row: np.ndarray, n: int) -> np.ndarray:
    """Rows 0..n-1 of one sequence: cache [num_pages, Hkv, P, D] -> [n, Hkv, D]."""
    P = cache.shape[2]
    out = np.empty((n, cache.shape[1], cache.shape[3]), dtype=cache.dtype)
    for pos in range(n):
        out[pos] = cache[int(page_table_row[pos // P]), :, pos % P, :]
    return out


def write_rows(cache: np.ndarray, page_table_row: np.ndarray, start: int,
               rows: np.ndarray) -> None:
    """Write rows [m, Hkv, D] at logical positions start..start+m-1."""
    P = cache.shape[2]
    for i in range(rows.shape[0]):
        pos = start + i
        cache[int(page_table_row[pos // P]), :, pos % P, :] = rows[i]


def poison_from(cache: np.ndarray, page_table_row: np.ndarray, start: int,
                capacity: int) -> None:
    """Set positions start..capacity-1 of a sequence to NaN (rolled-back or
    never-written rows; a read of any of them turns a result into NaN)."""
    P = cache.shape[2]
    for pos in range(start, capacity):
        cache[int(page_table_row[pos // P]), :, pos % P, :] = np.nan
