"""Seeded synthetic fork-decode workloads (inputs only, no attention arithmetic).

The workloads stand in for the paper's serving load, which is not available
here: reasoning traces of GLM-5.1 / DeepSeek-V4-Pro on KernelBench tasks
(Section 8.1).  Their shape follows the paper's description of speculative
generation: one long reasoning prefix per trace, K forks per fork event that
share it (Algorithm 1), fork points between 14% and 70% of the trace
(Section 4.2), and short private continuations per fork.

This module is shared by the CUDA path's tests/benchmark and by the oracle's
tests.  It only draws random numbers, rounds them to bf16, lays them out in
the paged pool and builds block tables; it computes nothing of the method.

Recipe (fixed per workload, seed = the workload's index unless overridden):
  1. rng = numpy.random.default_rng(seed) (PCG64).
  2. Integer lengths are drawn uniformly with inclusive bounds, in this order:
     prefix lengths (per trace), fork counts (per trace), suffix lengths (per fork).
  3. Logical pages: each trace's prefix needs ceil(P/B) pages, each fork's
     suffix ceil(S/B) pages, plus ``sentinel_pages`` pages nobody references.
     Physical ids are a seeded permutation of the pool when ``shuffle``.
  4. K, V (and Q) values are float32 N(0,1) draws rounded to bf16
     (round-to-nearest-even).  Slots past a sequence's length inside its last
     page, and every sentinel page, hold a quiet NaN so that reading them is
     detectable.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, asdict

import numpy as np

BF16_QNAN = 0x7FC0


@dataclass(frozen=True)
class WorkloadSpec:
    name: str
    num_traces: int
    prefix_len: tuple[int, int]       # inclusive uniform bounds per trace
    forks: tuple[int, int]            # inclusive uniform bounds per trace
    suffix_len: tuple[int, int]       # inclusive uniform bounds per fork
    hq: int
    hkv: int
    dqk: int
    dv: int
    page_size: int
    separate_v: bool = True           # False: V = first dv columns of K (latent KV)
    shuffle: bool = True
    seed: int = 0
    sentinel_pages: int = 2

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.dqk)


# The five workloads.  Sizes are the ones the fork-decode benchmark is quoted on.
WORKLOADS = {
    "tiny_p512_f4": WorkloadSpec(
        "tiny_p512_f4", 1, (512, 512), (4, 4), (32, 32), hq=8, hkv=2, dqk=64, dv=64,
        page_size=16, shuffle=False, seed=0),
    "fork_p8k_f8": WorkloadSpec(
        "fork_p8k_f8", 1, (8192, 8192), (8, 8), (64, 512), hq=64, hkv=8, dqk=128, dv=128,
        page_size=16, seed=1),
    "long_p32k_f16": WorkloadSpec(
        "long_p32k_f16", 1, (32768, 32768), (16, 16), (256, 2048), hq=64, hkv=8, dqk=128,
        dv=128, page_size=16, seed=2),
    "ragged_t8": WorkloadSpec(
        "ragged_t8", 8, (4096, 32768), (4, 16), (32, 1024), hq=64, hkv=8, dqk=128, dv=128,
        page_size=16, seed=3),
    "mla_p16k_f8": WorkloadSpec(
        "mla_p16k_f8", 1, (16384, 16384), (8, 8), (128, 1024), hq=128, hkv=1, dqk=576,
        dv=512, page_size=64, separate_v=False, seed=4),
}
WORKLOAD_ORDER = list(WORKLOADS)

# Diagnostic workloads (not benchmark configurations): the suffix-stage kernel
# alone on a call large enough that its fixed per-call latency is amortised,
# 64 forks of one trace with 2048-token suffixes and no prefix (538 MB of KV).
DIAGNOSTIC = {
    "suffix_only_f64_s2048": WorkloadSpec(
        "suffix_only_f64_s2048", 1, (0, 0), (64, 64), (2048, 2048), hq=64, hkv=8, dqk=128,
        dv=128, page_size=16, seed=5),
    # the latent kernel's prefix chunks are shared by the forks' items through L2:
    # four times the forks, and a prefix larger than L2 (151 MB of latent KV)
    "mla_p16k_f32": WorkloadSpec(
        "mla_p16k_f32", 1, (16384, 16384), (32, 32), (128, 1024), hq=128, hkv=1, dqk=576,
        dv=512, page_size=64, separate_v=False, seed=6),
    "mla_p128k_f8": WorkloadSpec(
        "mla_p128k_f8", 1, (131072, 131072), (8, 8), (128, 1024), hq=128, hkv=1, dqk=576,
        dv=512, page_size=64, separate_v=False, seed=7),
}


def spec_of(name: str) -> WorkloadSpec:
    """A benchmark workload or a diagnostic one, by name."""
    return WORKLOADS[name] if name in WORKLOADS else DIAGNOSTIC[name]


def round_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns, round-to-nearest-even (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    return ((u + np.uint32(0x7FFF) + lsb) >> np.uint32(16)).astype(np.uint16)


def bf16_normal(rng: np.random.Generator, shape) -> np.ndarray:
    return round_to_bf16_bits(rng.standard_normal(shape, dtype=np.float32))


def _uniform(rng, lo_hi, n):
    lo, hi = lo_hi
    return rng.integers(lo, hi + 1, size=n, dtype=np.int64)


def _draw_lengths(rng, spec: WorkloadSpec):
    """The first draws of a workload: prefix lengths, forks per trace, suffix lengths."""
    prefix_lens = _uniform(rng, spec.prefix_len, spec.num_traces)
    forks = _uniform(rng, spec.forks, spec.num_traces)
    suffix_lens = _uniform(rng, spec.suffix_len, int(forks.sum()))
    return prefix_lens, forks, suffix_lens


def workload_lengths(spec: WorkloadSpec | str, seed: int | None = None):
    """(prefix_lens, fork_offsets, suffix_lens) of make_workload(spec, seed), as int32,
    without drawing the KV pools and queries."""
    if isinstance(spec, str):
        spec = spec_of(spec)
    rng = np.random.default_rng(spec.seed if seed is None else seed)
    prefix_lens, forks, suffix_lens = _draw_lengths(rng, spec)
    fork_offsets = np.concatenate([[0], np.cumsum(forks)])
    return (prefix_lens.astype(np.int32), fork_offsets.astype(np.int32),
            suffix_lens.astype(np.int32))


def make_workload(spec: WorkloadSpec | str, seed: int | None = None,
                  fill_unused: str = "nan", **overrides) -> dict:
    """Build the host-side workload dict (numpy arrays; bf16 as uint16 bits).

    Keys: q, k_pages, v_pages (None for latent KV), prefix_table,
    prefix_bt_offsets, prefix_lens, fork_offsets, suffix_table,
    suffix_bt_offsets, suffix_lens, num_traces, total_forks, num_pages,
    hq, hkv, dqk, dv, page_size, scale, name, sentinel_ids.
    """
    if isinstance(spec, str):
        spec = spec_of(spec)
    if overrides:
        spec = WorkloadSpec(**{**asdict(spec), **overrides})
    rng = np.random.default_rng(spec.seed if seed is None else seed)
    T, B = spec.num_traces, spec.page_size
    prefix_lens, forks, suffix_lens = _draw_lengths(rng, spec)
    F = int(forks.sum())
    fork_offsets = np.concatenate([[0], np.cumsum(forks)]).astype(np.int64)

    p_pages = -(-prefix_lens // B)
    s_pages = -(-suffix_lens // B)
    n_logical = int(p_pages.sum() + s_pages.sum())
    num_pages = n_logical + spec.sentinel_pages
    phys = rng.permutation(num_pages) if spec.shuffle else np.arange(num_pages)
    phys = phys.astype(np.int32)
    prefix_bt_offsets = np.concatenate([[0], np.cumsum(p_pages)]).astype(np.int32)
    suffix_bt_offsets = np.concatenate([[0], np.cumsum(s_pages)]).astype(np.int32)
    prefix_table = phys[: int(p_pages.sum())].copy()
    suffix_table = phys[int(p_pages.sum()): n_logical].copy()
    sentinel_ids = phys[n_logical:].copy()

    k_pages = bf16_normal(rng, (num_pages, spec.hkv, B, spec.dqk))
    v_pages = bf16_normal(rng, (num_pages, spec.hkv, B, spec.dv)) if spec.separate_v else None
    q = bf16_normal(rng, (F, spec.hq, spec.dqk))

    if fill_unused == "nan":
        pools = [k_pages] + ([v_pages] if v_pages is not None else [])
        for pool in pools:
            pool[sentinel_ids] = BF16_QNAN
            for lens, offs, table in ((prefix_lens, prefix_bt_offsets, prefix_table),
                                      (suffix_lens, suffix_bt_offsets, suffix_table)):
                for i, n in enumerate(lens):
                    used = int(n) % B
                    if used:
                        last = table[offs[i + 1] - 1]
                        pool[last, :, used:, :] = BF16_QNAN
    return dict(
        name=spec.name, q=q, k_pages=k_pages, v_pages=v_pages,
        prefix_table=prefix_table, prefix_bt_offsets=prefix_bt_offsets,
        prefix_lens=prefix_lens.astype(np.int32), fork_offsets=fork_offsets.astype(np.int32),
        suffix_table=suffix_table, suffix_bt_offsets=suffix_bt_offsets,
        suffix_lens=suffix_lens.astype(np.int32), num_traces=T, total_forks=F,
        num_pages=num_pages, hq=spec.hq, hkv=spec.hkv, dqk=spec.dqk, dv=spec.dv,
        page_size=B, scale=spec.scale, sentinel_ids=sentinel_ids,
    )


def algorithmic_bytes(w: dict) -> dict:
    """Unique bytes one fork-decode call must move (counting only).

    Prefix KV read once per trace, every suffix KV read once, Q read, O (bf16)
    and LSE (fp32) written.  A latent KV pool (no separate V) reads each key
    row once.  The F-fold prefix re-read a naive per-fork decode would make is
    deliberately not counted.
    """
    kv_row = w["hkv"] * 2 * (w["dqk"] + (w["dv"] if w["v_pages"] is not None else 0))
    prefix = int(np.sum(w["prefix_lens"])) * kv_row
    suffix = int(np.sum(w["suffix_lens"])) * kv_row
    q = w["total_forks"] * w["hq"] * w["dqk"] * 2
    out = w["total_forks"] * w["hq"] * (w["dv"] * 2 + 4)
    return dict(prefix=prefix, suffix=suffix, q=q, out=out, total=prefix + suffix + q + out)


def algorithmic_flops(w: dict) -> dict:
    """2 flops per multiply-add: QK^T over dqk plus PV over dv, per (row, key)."""
    g = w["hq"] // w["hkv"]
    fo = w["fork_offsets"]
    prefix = sum(int(w["prefix_lens"][t]) * int(fo[t + 1] - fo[t]) for t in range(w["num_traces"]))
    prefix *= w["hkv"] * g * 2 * (w["dqk"] + w["dv"])
    suffix = int(np.sum(w["suffix_lens"])) * w["hkv"] * g * 2 * (w["dqk"] + w["dv"])
    return dict(prefix=prefix, suffix=suffix, total=prefix + suffix)


def shard_traces(w: dict, rank: int, world: int) -> dict:
    """The traces ``t`` with ``t % world == rank`` of a workload, re-indexed.

    Fork decode has no exchange between traces (each trace's forks read only
    that trace's prefix and their own suffixes), so ranks can take disjoint
    sets of traces and run them with no collective.  The KV pools are shared
    by reference: page ids keep pointing into the same pool.  Returns a
    workload dict of the same form (possibly with zero traces).
    """
    traces = [t for t in range(w["num_traces"]) if t % world == rank]
    fo, pbo, sbo = w["fork_offsets"], w["prefix_bt_offsets"], w["suffix_bt_offsets"]
    forks = [f for t in traces for f in range(fo[t], fo[t + 1])]
    pt = [w["prefix_table"][pbo[t]:pbo[t + 1]] for t in traces]
    st = [w["suffix_table"][sbo[f]:sbo[f + 1]] for f in forks]
    cat = lambda parts: (np.concatenate(parts).astype(np.int32) if parts
                         else np.zeros(0, dtype=np.int32))
    offs = lambda parts: np.concatenate([[0], np.cumsum([len(x) for x in parts])]).astype(np.int32)
    out = dict(w)
    out.update(
        q=w["q"][forks] if forks else w["q"][:0],
        prefix_table=cat(pt), prefix_bt_offsets=offs(pt),
        prefix_lens=w["prefix_lens"][traces].astype(np.int32),
        fork_offsets=offs([range(fo[t], fo[t + 1]) for t in traces]),
        suffix_table=cat(st), suffix_bt_offsets=offs(st),
        suffix_lens=w["suffix_lens"][forks].astype(np.int32),
        num_traces=len(traces), total_forks=len(forks),
        global_forks=np.array(forks, dtype=np.int64),
    )
    return out


def tile_kv_pool(pool: np.ndarray) -> np.ndarray:
    """Re-lay a [pages][hkv][B][D] pool into 8 x 8 tiles (the SPECGEN_KV_TILED order).

    Element (t, d) of a (page, head) block moves to
    ((t/8) * (D/8) + d/8) * 64 + (t%8) * 8 + d%8 -- a pure permutation of the
    block, no arithmetic.
    """
    P, H, B, D = pool.shape
    t = pool.reshape(P, H, B // 8, 8, D // 8, 8)           # [.., tg, t8, dc, d8]
    return np.ascontiguousarray(t.transpose(0, 1, 2, 4, 3, 5)).reshape(P, H, B, D)


def make_decode_state(w: dict, steps: int, seed: int = 12345) -> dict:
    """A workload prepared for `steps` decode steps that append to the suffixes.

    Adds spare pages to the pools (NaN-filled, ids appended at the end of the
    pool and handed out through a shuffled free list), widens every fork's
    suffix block table to hold ``suffix_lens + steps`` tokens (unallocated
    entries are -1), and draws the new key/value rows of every step
    (``k_new``: [steps, F, Hkv, dqk], ``v_new``: [steps, F, Hkv, dv] or None).
    Inputs only: no arithmetic of the method.  Returns a new dict.
    """
    B, F = w["page_size"], w["total_forks"]
    rng = np.random.default_rng(seed)
    lens = w["suffix_lens"].astype(np.int64)
    used = -(-lens // B)
    cap = -(-(lens + steps) // B)
    spare = int((cap - used).sum())
    n_old = w["num_pages"]
    offs = np.concatenate([[0], np.cumsum(cap)]).astype(np.int32)
    table = np.full(int(cap.sum()), -1, dtype=np.int32)
    old_offs = w["suffix_bt_offsets"]
    for f in range(F):
        table[offs[f]: offs[f] + used[f]] = w["suffix_table"][old_offs[f]: old_offs[f + 1]]
    free = (n_old + rng.permutation(spare)).astype(np.int32)

    def grow(pool):
        if pool is None:
            return None
        extra = np.full((spare,) + pool.shape[1:], BF16_QNAN, dtype=np.uint16)
        return np.concatenate([pool, extra], axis=0)

    out = dict(w)
    out.update(
        k_pages=grow(w["k_pages"]), v_pages=grow(w["v_pages"]), num_pages=n_old + spare,
        suffix_table=table, suffix_bt_offsets=offs, free_pages=free, steps=steps,
        k_new=bf16_normal(rng, (steps, F, w["hkv"], w["dqk"])),
        v_new=(bf16_normal(rng, (steps, F, w["hkv"], w["dv"])) if w["v_pages"] is not None
               else None))
    return out


def make_prefill(w: dict, chunk: int, seed: int = 777) -> dict:
    """Prefill inputs over a workload: fork f's chunk is its last
    min(chunk, S_f) suffix tokens (their K/V are already in the pools) and each
    chunk token gets its own query row (``q_rows`` [R, hq, dqk], fork by fork).
    Inputs only.  Returns a new dict with ``chunk_lens``, ``q_rows``, ``rows``."""
    rng = np.random.default_rng(seed)
    chunk_lens = np.minimum(w["suffix_lens"], chunk).astype(np.int32)
    rows = int(chunk_lens.sum())
    out = dict(w)
    out.update(chunk_lens=chunk_lens, rows=rows,
               q_rows=bf16_normal(rng, (rows, w["hq"], w["dqk"])))
    return out


def make_cascade(fork_points, forks, suffix_len=(64, 512), hq=64, hkv=8, dqk=128, dv=128,
                 page_size=16, separate_v=True, seed=9) -> dict:
    """A reasoning trace forked repeatedly at growing, page-aligned points.

    ``fork_points[i]`` is the prefix length of fork event i (increasing,
    multiples of page_size) and ``forks[i]`` its number of forks.  Segment s
    holds the trace's tokens [fork_points[s-1], fork_points[s]) (fork_points[-1]
    read as 0) in its own pages and serves every fork of events >= s; forks are
    listed deepest event first, so each segment serves a contiguous range of
    forks (``segment_rows``, flattened [begin, end) pairs).  Suffixes, pools,
    NaN fill and Q follow ``make_workload``.  Also returns ``flat``: the same
    forks as an ordinary workload with one trace per event (prefix = the
    concatenated pages of its segments) for comparisons.  Inputs only.
    """
    rng = np.random.default_rng(seed)
    B = page_size
    pts = [int(p) for p in fork_points]
    if any(p % B or p <= 0 for p in pts) or any(b <= a for a, b in zip(pts, pts[1:])):
        raise ValueError("fork points must be increasing positive multiples of page_size")
    L = len(pts)
    order = list(range(L - 1, -1, -1))                   # deepest event first
    n_forks = [int(forks[i]) for i in order]
    F = sum(n_forks)
    suffix_lens = _uniform(rng, suffix_len, F)
    s_pages = -(-suffix_lens // B)
    n_trace = pts[-1] // B
    num_pages = n_trace + int(s_pages.sum()) + 2
    phys = rng.permutation(num_pages).astype(np.int32)
    trace_pages = phys[:n_trace].copy()
    suffix_bt_offsets = np.concatenate([[0], np.cumsum(s_pages)]).astype(np.int32)
    suffix_table = phys[n_trace: n_trace + int(s_pages.sum())].copy()
    sentinel_ids = phys[n_trace + int(s_pages.sum()):].copy()
    bounds = [0] + pts
    seg_lens = np.diff(bounds).astype(np.int32)
    seg_bt_offsets = (np.array(bounds) // B).astype(np.int32)
    seg_rows = []
    for s in range(L):   # segment s serves events s..L-1, which come first in the fork order
        seg_rows += [0, sum(int(forks[i]) for i in range(s, L))]
    k_pages = bf16_normal(rng, (num_pages, hkv, B, dqk))
    v_pages = bf16_normal(rng, (num_pages, hkv, B, dv)) if separate_v else None
    q = bf16_normal(rng, (F, hq, dqk))
    for pool in [k_pages] + ([v_pages] if v_pages is not None else []):
        pool[sentinel_ids] = BF16_QNAN
        for f, n in enumerate(suffix_lens):
            used = int(n) % B
            if used:
                pool[suffix_table[suffix_bt_offsets[f + 1] - 1], :, used:, :] = BF16_QNAN
    common = dict(q=q, k_pages=k_pages, v_pages=v_pages, suffix_table=suffix_table,
                  suffix_bt_offsets=suffix_bt_offsets, suffix_lens=suffix_lens.astype(np.int32),
                  total_forks=F, num_pages=num_pages, hq=hq, hkv=hkv, dqk=dqk, dv=dv,
                  page_size=B, scale=1.0 / float(np.sqrt(dqk)), sentinel_ids=sentinel_ids)
    cascade = dict(common, name="cascade", num_traces=L, prefix_table=trace_pages,
                   prefix_bt_offsets=seg_bt_offsets, prefix_lens=seg_lens,
                   fork_offsets=np.array([0, F], dtype=np.int32),
                   segment_rows=np.array(seg_rows, dtype=np.int32))
    flat_tables = [trace_pages[: pts[i] // B] for i in order]
    flat = dict(common, name="cascade_flat", num_traces=L,
                prefix_table=np.concatenate(flat_tables).astype(np.int32),
                prefix_bt_offsets=np.concatenate(
                    [[0], np.cumsum([len(t) for t in flat_tables])]).astype(np.int32),
                prefix_lens=np.array([pts[i] for i in order], dtype=np.int32),
                fork_offsets=np.concatenate([[0], np.cumsum(n_forks)]).astype(np.int32))
    cascade["flat"] = flat
    return cascade
