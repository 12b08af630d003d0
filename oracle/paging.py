"""Plain references for the paged-KV bookkeeping around fork decode (test infrastructure only):
appending one decode step's K/V to paged suffixes, and packing / unpacking a
sequence's pages for the remote prefix cache.

What is computed and where it comes from
----------------------------------------
After a fork event every fork decodes its own continuation while the reasoning
prefix stays shared (Algorithm 1, "Fork K spec. generations"; Section 4.2):
each decode step adds one key/value row per fork to that fork's private
suffix.  In the paged layout (token j of a sequence at page ``table[j // B]``,
slot ``j % B``), the new token of fork f with S_f tokens already in its suffix
goes to slot ``S_f % B`` of page ``table[S_f // B]``; when ``S_f % B == 0`` that
page does not exist yet and the fork takes the next id of a free list, in fork
order, and records it in its block table.

Readings where the paper is silent (listed in the design notes): the free list
is consumed in increasing fork order; a fork's block table has a fixed capacity
(its CSR range) and an append past it is an error; the latent pool (no value
pool) stores only the key row.

Deliberately plain: one fork at a time, numpy copies of whole rows.
"""

from __future__ import annotations

import numpy as np


def append_kv(k_pages, v_pages, suffix_table, suffix_bt_offsets, suffix_lens, k_new, v_new,
              free_pages, page_size):
    """Return (k_pages, v_pages, suffix_table, pages_taken) after one append.

    k_pages / v_pages: [num_pages, Hkv, B, width] bf16 bits (v_pages may be None);
    suffix_table / suffix_bt_offsets: CSR block tables (capacity per fork);
    suffix_lens[f]: tokens already in fork f's suffix; k_new / v_new:
    [F, Hkv, width] rows to append; free_pages: ids to take, in order.
    The inputs are not modified.
    """
    k = np.array(k_pages, copy=True)
    v = None if v_pages is None else np.array(v_pages, copy=True)
    table = np.array(suffix_table, copy=True)
    offs = np.asarray(suffix_bt_offsets)
    taken = 0
    for f in range(len(suffix_lens)):
        n = int(suffix_lens[f])
        page_index, slot = divmod(n, page_size)
        start, cap = int(offs[f]), int(offs[f + 1] - offs[f])
        if page_index >= cap:
            raise ValueError(f"fork {f}: block table full ({cap} pages)")
        if slot == 0:
            if taken >= len(free_pages):
                raise ValueError("free list exhausted")
            page = int(free_pages[taken])
            taken += 1
            table[start + page_index] = page
        else:
            page = int(table[start + page_index])
        k[page, :, slot, :] = k_new[f]
        if v is not None:
            v[page, :, slot, :] = v_new[f]
    return k, v, table, taken


def pack_pages(k_pages, v_pages, table):
    """Contiguous copy of the pages ``table[0..n)`` of a paged sequence.

    The remote prefix cache (Section 6.2.3) moves a suspended trace's prefix KV
    off the GPU and back; its device side gathers the sequence's pages into one
    buffer and scatters them back under a new block table.  Layout of the
    buffer: the K blocks of the n pages in table order ([n, Hkv, B, Dk] bf16
    bits), then the V blocks ([n, Hkv, B, Dv]) when there is a value pool.
    Returns a flat uint16 array.
    """
    t = np.asarray(table, dtype=np.int64)
    parts = [np.asarray(k_pages)[t].reshape(-1)]
    if v_pages is not None:
        parts.append(np.asarray(v_pages)[t].reshape(-1))
    return np.concatenate(parts) if parts else np.zeros(0, np.uint16)


def unpack_pages(k_pages, v_pages, table, packed):
    """Pools with page ``table[i]`` overwritten by page i of ``packed`` (the
    layout of pack_pages); the inputs are not modified.  Returns (k, v)."""
    k = np.array(k_pages, copy=True)
    v = None if v_pages is None else np.array(v_pages, copy=True)
    t = np.asarray(table, dtype=np.int64)
    n = len(t)
    nk = n * int(np.prod(k.shape[1:]))
    k[t] = np.asarray(packed[:nk]).reshape((n,) + k.shape[1:])
    if v is not None:
        v[t] = np.asarray(packed[nk: nk + n * int(np.prod(v.shape[1:]))]).reshape((n,) + v.shape[1:])
    return k, v
