"""Plain fp64 definition of fork-decode attention (test infrastructure only).

What is computed and where it comes from
----------------------------------------
SpecGen forks K non-reasoning generations from the reasoning prefix pi of a
running reasoning generation: each fork's prompt is the concatenation of the
iteration prompt and pi (Algorithm 1, "Fork K spec. generations"; Section 6.1.1),
and the forks reuse the reasoning generation's KV cache for that shared prefix
(Section 4.2; Section 8.6, "prefix caching").  When the K forks then decode, each
fork's single new query attends to the shared prefix tokens followed by its own
private continuation tokens.  The paper prints no attention formula; the
quantity itself is ordinary softmax attention, written out here:

    s_i   = sigma * <q, k_i>                        (scores, i over all keys)
    m     = max_i s_i
    l     = sum_i exp(s_i - m)
    O     = sum_i exp(s_i - m) v_i / l
    LSE   = m + ln l                                (natural log of the scaled scores)

with keys/values taken in logical order: prefix tokens 0..P-1 of the fork's
trace, then the fork's own suffix tokens 0..S-1.  Token j of a paged sequence
lives in physical page ``table[j // B]`` at slot ``j % B`` (paged KV cache, the
serving layout the paper relies on through vLLM, Section 8.1).

Readings where the paper is silent (each is listed in the design notes):
  * GQA head map: query head h reads kv head h // (Hq // Hkv).
  * Latent (MLA-style) keys: when no separate value pool is given, the value row
    is the first ``dv`` columns of the key row.
  * An empty key set gives O = 0 and LSE = -inf.

Inputs are bf16 bit patterns (uint16); they are widened exactly to float64 and
all arithmetic is float64.  The functions are deliberately slow and direct: one
(fork, kv-head) group at a time, a library matrix product for the dot products,
no blocking or reordering beyond the definition.
"""

from __future__ import annotations

import numpy as np

NEG_INF = float("-inf")


def bf16_bits_to_f64(bits) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64.

    A bf16 value is the upper 16 bits of an IEEE binary32 value, so shifting
    the pattern left by 16 gives the binary32 value exactly; binary32 widens
    to binary64 exactly.
    """
    b = np.asarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def gather_logical(pool: np.ndarray, table, length: int, page_size: int,
                   head: int) -> np.ndarray:
    """Rows 0..length-1 of one paged sequence for one kv head, in logical order.

    ``pool`` has shape [num_pages, Hkv, page_size, width] (bf16 bits);
    token j is stored in page ``table[j // page_size]`` at slot
    ``j % page_size``.  Returns float64 [length, width].
    """
    j = np.arange(int(length))
    pages = np.asarray(table, dtype=np.int64)[j // page_size]
    return bf16_bits_to_f64(pool[pages, head, j % page_size])


def attention_rows(q: np.ndarray, k: np.ndarray, v: np.ndarray,
                   scale: float) -> tuple[np.ndarray, np.ndarray]:
    """Softmax attention of several query rows over one key/value set, fp64.

    q: [R, Dqk], k: [N, Dqk], v: [N, Dv]  (float64)
    Returns O [R, Dv] and LSE [R]; N = 0 gives O = 0 and LSE = -inf.
    """
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    rows, dv = q.shape[0], v.shape[1]
    if k.shape[0] == 0:
        return np.zeros((rows, dv)), np.full(rows, NEG_INF)
    s = scale * (q @ k.T)                      # s_i = sigma <q, k_i>
    m = s.max(axis=1, keepdims=True)           # m = max_i s_i
    w = np.exp(s - m)                          # exp(s_i - m)
    l = w.sum(axis=1, keepdims=True)           # l = sum_i exp(s_i - m)
    o = (w @ v) / l                            # O = sum_i w_i v_i / l
    lse = m[:, 0] + np.log(l[:, 0])            # LSE = m + ln l
    return o, lse


def lse_merge(o_a, lse_a, o_b, lse_b) -> tuple[np.ndarray, np.ndarray]:
    """Combine two partial attentions over disjoint key sets into one.

    If (O_a, LSE_a) and (O_b, LSE_b) are the attentions of the same queries
    over key sets A and B, the attention over A u B is
        m   = max(LSE_a, LSE_b)
        w_x = exp(LSE_x - m)
        O   = (w_a O_a + w_b O_b) / (w_a + w_b)
        LSE = m + ln(w_a + w_b)
    (the normaliser of A u B is the sum of the two normalisers).  A part with
    LSE = -inf is empty and contributes nothing; both empty gives O = 0,
    LSE = -inf.
    """
    o_a = np.asarray(o_a, dtype=np.float64)
    o_b = np.asarray(o_b, dtype=np.float64)
    lse_a = np.asarray(lse_a, dtype=np.float64)
    lse_b = np.asarray(lse_b, dtype=np.float64)
    o = np.zeros(np.broadcast_shapes(o_a.shape, o_b.shape))
    lse = np.full(np.broadcast_shapes(lse_a.shape, lse_b.shape), NEG_INF)
    for r in np.ndindex(lse.shape):
        a, b = lse_a[r], lse_b[r]
        if a == NEG_INF and b == NEG_INF:
            continue
        m = max(a, b)
        wa = 0.0 if a == NEG_INF else np.exp(a - m)
        wb = 0.0 if b == NEG_INF else np.exp(b - m)
        o[r] = (wa * o_a[r] + wb * o_b[r]) / (wa + wb)
        lse[r] = m + np.log(wa + wb)
    return o, lse


def _fork_kv(k_pages, v_pages, dv, page_size, prefix_table, prefix_len,
             suffix_table, suffix_len, g, parts=("prefix", "suffix")):
    """Keys and values one fork attends to for kv head g (logical order)."""
    ks, vs = [], []
    if "prefix" in parts:
        ks.append(gather_logical(k_pages, prefix_table, prefix_len, page_size, g))
        if v_pages is not None:
            vs.append(gather_logical(v_pages, prefix_table, prefix_len, page_size, g))
    if "suffix" in parts:
        ks.append(gather_logical(k_pages, suffix_table, suffix_len, page_size, g))
        if v_pages is not None:
            vs.append(gather_logical(v_pages, suffix_table, suffix_len, page_size, g))
    k = np.concatenate(ks, axis=0)
    v = np.concatenate(vs, axis=0) if v_pages is not None else k[:, :dv]
    return k, v


def _check(w):
    if w["hq"] % w["hkv"] != 0:
        raise ValueError("hq must be a multiple of hkv")


def fork_attn_decode_rows(w: dict, rows) -> tuple[np.ndarray, np.ndarray]:
    """(O, LSE) for selected (fork, q-head) rows of a fork-decode workload.

    ``w`` holds the workload as host numpy arrays (see ``fork_attn_decode``).
    ``rows`` is an iterable of (fork, head) pairs.  Returns O [len, dv] and
    LSE [len] in float64.
    """
    _check(w)
    rows = list(rows)
    g_size = w["hq"] // w["hkv"]
    dv = w["dv"]
    out_o = np.zeros((len(rows), dv))
    out_lse = np.zeros(len(rows))
    # group requested rows by (fork, kv head) so each key set is gathered once
    groups: dict[tuple[int, int], list[int]] = {}
    for idx, (f, h) in enumerate(rows):
        groups.setdefault((int(f), int(h) // g_size), []).append(idx)
    fork_offsets = w["fork_offsets"]
    trace_of = np.searchsorted(fork_offsets, np.arange(w["total_forks"]), side="right") - 1
    for (f, g), idxs in groups.items():
        t = int(trace_of[f])
        pt = w["prefix_table"][w["prefix_bt_offsets"][t]:w["prefix_bt_offsets"][t + 1]]
        st = w["suffix_table"][w["suffix_bt_offsets"][f]:w["suffix_bt_offsets"][f + 1]]
        k, v = _fork_kv(w["k_pages"], w.get("v_pages"), dv, w["page_size"], pt,
                        int(w["prefix_lens"][t]), st, int(w["suffix_lens"][f]), g)
        heads = [int(rows[i][1]) for i in idxs]
        q = bf16_bits_to_f64(w["q"][f, heads, :])
        o, lse = attention_rows(q, k, v, w["scale"])
        out_o[idxs] = o
        out_lse[idxs] = lse
    return out_o, out_lse


def fork_attn_decode(w: dict) -> tuple[np.ndarray, np.ndarray]:
    """Full fork-decode attention, every fork and every query head.

    Workload dict keys (host numpy arrays, bf16 as uint16 bits):
      q            [total_forks, hq, dqk]
      k_pages      [num_pages, hkv, page_size, dqk]
      v_pages      [num_pages, hkv, page_size, dv] or None (V = K[..., :dv])
      prefix_table, prefix_bt_offsets [T+1], prefix_lens [T]
      fork_offsets [T+1]   forks of trace t are fork_offsets[t]..fork_offsets[t+1]-1
      suffix_table, suffix_bt_offsets [F+1], suffix_lens [F]
      hq, hkv, dv, page_size, scale, total_forks
    Returns O [total_forks, hq, dv] and LSE [total_forks, hq] (float64).
    """
    nf, hq = w["total_forks"], w["hq"]
    rows = [(f, h) for f in range(nf) for h in range(hq)]
    o, lse = fork_attn_decode_rows(w, rows)
    return o.reshape(nf, hq, w["dv"]), lse.reshape(nf, hq)


def fork_attn_split_merge(w: dict) -> tuple[np.ndarray, np.ndarray]:
    """Prefix-only and suffix-only attention, combined with ``lse_merge``.

    This is the two-stage form of the same quantity (prefix stage, suffix
    stage, log-sum-exp merge); it must agree with ``fork_attn_decode``.
    """
    _check(w)
    nf, hq, hkv, dv = w["total_forks"], w["hq"], w["hkv"], w["dv"]
    g_size = hq // hkv
    trace_of = np.searchsorted(w["fork_offsets"], np.arange(nf), side="right") - 1
    o = np.zeros((nf, hq, dv))
    lse = np.zeros((nf, hq))
    for f in range(nf):
        t = int(trace_of[f])
        pt = w["prefix_table"][w["prefix_bt_offsets"][t]:w["prefix_bt_offsets"][t + 1]]
        st = w["suffix_table"][w["suffix_bt_offsets"][f]:w["suffix_bt_offsets"][f + 1]]
        for g in range(hkv):
            heads = list(range(g * g_size, (g + 1) * g_size))
            q = bf16_bits_to_f64(w["q"][f, heads, :])
            args = (w["k_pages"], w.get("v_pages"), dv, w["page_size"], pt,
                    int(w["prefix_lens"][t]), st, int(w["suffix_lens"][f]), g)
            kp, vp = _fork_kv(*args, parts=("prefix",))
            ks, vs = _fork_kv(*args, parts=("suffix",))
            o_p, l_p = attention_rows(q, kp, vp, w["scale"])
            o_s, l_s = attention_rows(q, ks, vs, w["scale"])
            o[f, heads], lse[f, heads] = lse_merge(o_p, l_p, o_s, l_s)
    return o, lse


def fork_prefill(w: dict, chunk_lens, q_rows) -> tuple[np.ndarray, np.ndarray]:
    """Causal prefill of every fork's newest suffix tokens (Algorithm 1: the
    fork's prompt follows the shared prefix and is processed before it decodes).

    ``w`` is a fork-decode workload whose suffix lengths already count the
    chunk; fork f's chunk is its last ``chunk_lens[f]`` suffix tokens.  Query
    row r = (f, j), fork by fork and j < chunk_lens[f] (``q_rows`` [R, hq, dqk]
    bf16 bits), attends to the trace's prefix and the fork's suffix tokens
    0 .. S_f - chunk_lens[f] + j: its own token and everything before it.
    Returns O [R, hq, dv] and LSE [R, hq] (float64).
    """
    _check(w)
    hq, g_size, dv = w["hq"], w["hq"] // w["hkv"], w["dv"]
    chunk_lens = np.asarray(chunk_lens)
    n_rows = int(chunk_lens.sum())
    out_o = np.zeros((n_rows, hq, dv))
    out_lse = np.zeros((n_rows, hq))
    fo = w["fork_offsets"]
    trace_of = np.searchsorted(fo, np.arange(w["total_forks"]), side="right") - 1
    r = 0
    for f in range(w["total_forks"]):
        t = int(trace_of[f])
        pt = w["prefix_table"][w["prefix_bt_offsets"][t]:w["prefix_bt_offsets"][t + 1]]
        st = w["suffix_table"][w["suffix_bt_offsets"][f]:w["suffix_bt_offsets"][f + 1]]
        before = int(w["suffix_lens"][f]) - int(chunk_lens[f])
        for j in range(int(chunk_lens[f])):
            for g in range(w["hkv"]):
                k, v = _fork_kv(w["k_pages"], w.get("v_pages"), dv, w["page_size"], pt,
                                int(w["prefix_lens"][t]), st, before + j + 1, g)
                heads = list(range(g * g_size, (g + 1) * g_size))
                q = bf16_bits_to_f64(np.asarray(q_rows)[r, heads, :])
                o, lse = attention_rows(q, k, v, w["scale"])
                out_o[r, heads] = o
                out_lse[r, heads] = lse
            r += 1
    return out_o, out_lse


def fork_cascade_decode(w: dict) -> tuple[np.ndarray, np.ndarray]:
    """Decode over a tree of shared prefix segments (repeated fork events at
    growing prefixes, Algorithm 1: pi_1 is a prefix of pi_2 ...).

    ``w`` is a fork-decode workload whose prefix tables are *segments*:
    segment s has ``prefix_lens[s]`` tokens at pages ``prefix_table[
    prefix_bt_offsets[s]:prefix_bt_offsets[s+1]]`` (its token 0 at slot 0 of its
    first page) and serves the forks ``segment_rows[s][0] <= f < segment_rows[s][1]``.
    Fork f attends to every segment that serves it and then to its own suffix;
    the key set is a union, so the order of segments does not matter.
    Returns O [F, hq, dv] and LSE [F, hq].
    """
    _check(w)
    F, hq, dv, B = w["total_forks"], w["hq"], w["dv"], w["page_size"]
    g_size = hq // w["hkv"]
    seg_rows = np.asarray(w["segment_rows"]).reshape(-1, 2)
    out_o = np.zeros((F, hq, dv))
    out_lse = np.zeros((F, hq))
    for f in range(F):
        st = w["suffix_table"][w["suffix_bt_offsets"][f]:w["suffix_bt_offsets"][f + 1]]
        for g in range(w["hkv"]):
            ks, vs = [], []
            for s in range(len(seg_rows)):
                if seg_rows[s][0] <= f < seg_rows[s][1]:
                    pt = w["prefix_table"][w["prefix_bt_offsets"][s]:w["prefix_bt_offsets"][s + 1]]
                    k, v = _fork_kv(w["k_pages"], w.get("v_pages"), dv, B, pt,
                                    int(w["prefix_lens"][s]), pt, 0, g)
                    ks.append(k)
                    vs.append(v)
            k, v = _fork_kv(w["k_pages"], w.get("v_pages"), dv, B, st, 0, st,
                            int(w["suffix_lens"][f]), g)
            ks.append(k)
            vs.append(v)
            heads = list(range(g * g_size, (g + 1) * g_size))
            q = bf16_bits_to_f64(w["q"][f, heads, :])
            o, lse = attention_rows(q, np.concatenate(ks), np.concatenate(vs), w["scale"])
            out_o[f, heads] = o
            out_lse[f, heads] = lse
    return out_o, out_lse
