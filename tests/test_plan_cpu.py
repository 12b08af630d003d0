"""Host planner invariants, on the CPU (specgen_fork_attn_plan_host).

A fork-decode plan is correct when, for every query row and every kv head,
its work items cover the row's keys -- the trace's shared prefix, then the
fork's own suffix -- exactly once, each item writes a distinct partial slot
inside the row's slot range, and the merge reads exactly those slots.  These
tests parse the plan bytes the library would upload and check that, with
fake device pointers, over the benchmark workloads and random ragged shapes
on all three kernel paths (tensor-core GQA, latent tensor-core, split-K).
"""

import ctypes as C

import numpy as np
import pytest

from paper_2606_17518_gb300 import _lib, workloads as wl

FAKE = 0x10000
TC_WORDS = 11      # TcItem: int32 fields
SPLIT_WORDS = 10   # SplitItem: int32 fields
SUFFIX_WARPS = 8   # worker warps per suffix-stage CTA


def _args(T, F, hq, hkv, dqk, dv, B, latent, **kw):
    a = _lib.make_args(num_traces=T, total_forks=F, hq=hq, hkv=hkv, head_dim_qk=dqk,
                       head_dim_v=dv, page_size=B, num_pages=1 << 20, scale=0.1, q=FAKE,
                       k_pages=FAKE, v_pages=None if latent else FAKE,
                       prefix_block_table=FAKE, prefix_bt_offsets=FAKE,
                       suffix_block_table=FAKE, suffix_bt_offsets=FAKE, out=FAKE, lse=FAKE,
                       workspace=FAKE, workspace_bytes=1 << 40, kv_layout=_lib.KV_ROWS,
                       suffix_lens=None)
    for k, v in kw.items():
        setattr(a, k, v)
    return a


def _plan(shape, pl, fo, sl, host_offsets=True):
    T, F = len(pl), int(fo[-1])
    B = shape["B"]
    pbo = np.concatenate([[0], np.cumsum((pl + B - 1) // B)]).astype(np.int32)
    sbo = np.concatenate([[0], np.cumsum((sl + B - 1) // B)]).astype(np.int32)
    if host_offsets:
        lens, keep = _lib.make_host_lens(pl, fo, sl, pbo, sbo)
    else:
        lens, keep = _lib.make_host_lens(pl, fo, sl)
    args = _args(T, F, **shape)
    need = _lib.specgen_fork_attn_workspace_size(args, lens)
    assert need > 0
    buf = np.zeros(need, dtype=np.uint8)
    plan = _lib.specgen_fork_attn_plan_host(args, lens, buf)
    return plan, buf, pbo, sbo


def _parse(plan, buf):
    assert plan.valid == 1
    assert not buf[:plan.ws_plan_off].any()  # the status header goes up zeroed
    region = buf[plan.ws_plan_off:plan.ws_plan_off + plan.plan_bytes]
    w = region.view(np.int32)
    (n_split, n_tc, n_ctas, n_forks, so, to, _, coo, pbo_, npo,
     n_sfx, n_sfx_ctas, sfo, sfoo) = (int(x) for x in w[:14])
    words = lambda off, n: w[off // 4: off // 4 + n]
    tc_only = words(to, n_tc * TC_WORDS).reshape(n_tc, TC_WORDS)
    sfx = words(sfo, n_sfx * TC_WORDS).reshape(n_sfx, TC_WORDS)
    n_workers = n_sfx_ctas * SUFFIX_WARPS
    sfx_offsets = words(sfoo, n_workers + 1)
    # the suffix-stage workers: every item in exactly one worker's range, in order
    assert plan.n_sfx_items == n_sfx and plan.n_sfx_ctas == n_sfx_ctas
    assert sfx_offsets[0] == 0 and sfx_offsets[-1] == n_sfx and np.all(np.diff(sfx_offsets) >= 0)
    for kind, seq, g, f0, nf, tb, te, part, dv0, toff, rl in sfx:
        assert kind == 1 and nf == 1 and rl == 0 and dv0 == 0
    return dict(
        split=words(so, n_split * SPLIT_WORDS).reshape(n_split, SPLIT_WORDS),
        tc=np.concatenate([tc_only, sfx]) if n_sfx else tc_only,
        tc_only=tc_only, sfx=sfx, sfx_offsets=sfx_offsets,
        cta_offsets=words(coo, n_ctas + 1) if n_tc else np.zeros(1, np.int32),
        part_base=words(pbo_, n_forks),
        n_parts=words(npo, n_forks * plan.n_part_groups).reshape(n_forks, plan.n_part_groups),
        n_ctas=n_ctas)


def _covers(ranges, length, what):
    """Half-open ranges tile [0, length) exactly once."""
    ranges = sorted(ranges)
    pos = 0
    for b, e in ranges:
        assert b == pos and e > b, (what, ranges, length)
        pos = e
    assert pos == length, (what, ranges, length)


def _check_slots(p, plan, F):
    base = p["part_base"]
    most = p["n_parts"].max(axis=1) if F else np.zeros(0)
    assert base[0] == 0
    ends = base + most
    assert np.all(ends[:-1] <= base[1:])
    assert int(ends[-1]) <= plan.total_slots


def _check_tc(shape, pl, fo, sl, plan, p, pbo, sbo, host_offsets):
    G = shape["hq"] // shape["hkv"]
    F = int(fo[-1])
    tc = p["tc"]
    co = p["cta_offsets"]
    assert co[0] == 0 and co[-1] == len(p["tc_only"]) and np.all(np.diff(co) > 0)
    assert plan.n_tc_ctas + plan.n_sfx_ctas <= 148  # the grids share the SMs (148: no device)
    fork_trace = np.repeat(np.arange(len(pl)), np.diff(fo))
    cover = {}
    parts = {}
    for kind, seq, g, f0, nf, tb, te, part, dv0, toff, rl in tc:
        assert te > tb >= 0 and dv0 == 0 and rl == 0
        assert 1 <= nf and nf * G <= 128 and 0 <= g < shape["hkv"]
        if kind == 0:
            assert np.all(fork_trace[f0:f0 + nf] == seq) and te <= pl[seq]
            assert toff == (pbo[seq] if host_offsets else -1)
        else:
            assert nf == 1 and seq == f0 and te <= sl[seq]
            assert toff == (sbo[seq] if host_offsets else -1)
        for f in range(f0, f0 + nf):
            cover.setdefault((f, g, kind), []).append((int(tb), int(te)))
            parts.setdefault((f, g), []).append(int(part))
    for f in range(F):
        for g in range(shape["hkv"]):
            _covers(cover.get((f, g, 0), []), int(pl[fork_trace[f]]), ("prefix", f, g))
            _covers(cover.get((f, g, 1), []), int(sl[f]), ("suffix", f, g))
            got = sorted(parts.get((f, g), []))
            assert got == list(range(p["n_parts"][f, g])), (f, g, got)
    _check_slots(p, plan, F)


def _check_latent(pl, fo, sl, plan, p):
    F = int(fo[-1])
    fork_trace = np.repeat(np.arange(len(pl)), np.diff(fo))
    cover, parts = {}, {}
    for kind, seq, g, f0, nf, tb, te, part, dv0, toff, rl in p["tc"]:
        assert g == 0 and nf == 1 and dv0 in (0, 256) and te > tb >= 0
        key = (f0, dv0)
        cover.setdefault(key + (kind,), []).append((int(tb), int(te)))
        parts.setdefault(key, []).append(int(part))
        if kind == 0:
            assert seq == fork_trace[f0]
        else:
            assert seq == f0
    for f in range(F):
        for dv0 in (0, 256):
            _covers(cover.get((f, dv0, 0), []), int(pl[fork_trace[f]]), ("prefix", f, dv0))
            _covers(cover.get((f, dv0, 1), []), int(sl[f]), ("suffix", f, dv0))
            assert sorted(parts.get((f, dv0), [])) == list(range(p["n_parts"][f, 0]))
    _check_slots(p, plan, F)


def _check_split(shape, pl, fo, sl, plan, p):
    F = int(fo[-1])
    fork_trace = np.repeat(np.arange(len(pl)), np.diff(fo))
    cover, slots = {}, {}
    for f, kind, seq, g, h0, nrows, dv0, tb, te, slot in p["split"]:
        assert te > tb >= 0 and nrows >= 1 and 0 <= g < shape["hkv"]
        assert seq == (fork_trace[f] if kind == 0 else f)
        key = (f, h0, dv0)
        cover.setdefault(key + (kind,), []).append((int(tb), int(te)))
        slots.setdefault(key, []).append(int(slot) - int(p["part_base"][f]))
    # every fork with keys has items for every (row block, value block), and
    # the row blocks tile the query heads
    blocks = sorted({(int(h0), int(nr), int(dv0)) for _, _, _, _, h0, nr, dv0, _, _, _ in p["split"]})
    heads = sorted({(h0, nr) for h0, nr, _ in blocks})
    _covers([(h0, h0 + nr) for h0, nr in heads], shape["hq"], "row blocks")
    for f in range(F):
        if pl[fork_trace[f]] + sl[f] == 0:
            continue
        for h0, _, dv0 in blocks:
            _covers(cover.get((f, h0, dv0, 0), []), int(pl[fork_trace[f]]), ("prefix", f, h0))
            _covers(cover.get((f, h0, dv0, 1), []), int(sl[f]), ("suffix", f, h0))
            assert sorted(slots[(f, h0, dv0)]) == list(range(p["n_parts"][f, 0]))
    _check_slots(p, plan, F)


SHAPES = {
    "gqa128": dict(hq=64, hkv=8, dqk=128, dv=128, B=16, latent=False),
    "gqa64": dict(hq=8, hkv=2, dqk=64, dv=64, B=16, latent=False),
    "mha": dict(hq=4, hkv=4, dqk=128, dv=128, B=16, latent=False),
    "g128": dict(hq=128, hkv=1, dqk=128, dv=128, B=16, latent=False),
    "latent": dict(hq=128, hkv=1, dqk=576, dv=512, B=64, latent=True),
    "split_page32": dict(hq=16, hkv=2, dqk=128, dv=128, B=32, latent=False),
    "split_latent_page16": dict(hq=16, hkv=1, dqk=576, dv=512, B=16, latent=True),
}


def _check(name, pl, fo, sl, host_offsets=True):
    shape = SHAPES[name]
    plan, buf, pbo, sbo = _plan(shape, pl, fo, sl, host_offsets)
    p = _parse(plan, buf)
    if plan.n_split_items:
        assert plan.n_tc_items == 0
        _check_split(shape, pl, fo, sl, plan, p)
    elif shape["latent"]:
        _check_latent(pl, fo, sl, plan, p)
    else:
        _check_tc(shape, pl, fo, sl, plan, p, pbo, sbo, host_offsets)
    return plan


@pytest.mark.parametrize("name", list(wl.WORKLOAD_ORDER))
def test_workload_plans_cover_every_key_once(name):
    spec = wl.WORKLOADS[name]
    pl, fo, sl = wl.workload_lengths(name)
    shape = dict(hq=spec.hq, hkv=spec.hkv, dqk=spec.dqk, dv=spec.dv, B=spec.page_size,
                 latent=not spec.separate_v)
    key = next(k for k, v in SHAPES.items() if v == shape)
    plan = _check(key, pl, fo, sl)
    assert plan.n_tc_items > 0 and plan.n_split_items == 0


@pytest.mark.parametrize("case", range(24))
def test_random_plans_cover_every_key_once(case):
    rng = np.random.default_rng(1000 + case)
    name = list(SHAPES)[case % len(SHAPES)]
    T = int(rng.integers(1, 6))
    fk = rng.integers(1, 11, T)
    fo = np.concatenate([[0], np.cumsum(fk)]).astype(np.int32)
    F = int(fo[-1])
    pl = rng.integers(0, 6000, T).astype(np.int32)
    sl = rng.integers(0, 800, F).astype(np.int32)
    # degenerate rows: empty prefixes and suffixes, one-token sequences
    pl[rng.random(T) < 0.2] = 0
    sl[rng.random(F) < 0.2] = 0
    sl[rng.random(F) < 0.1] = 1
    _check(name, pl, fo, sl, host_offsets=bool(case % 2))


def test_plan_host_errors():
    shape = SHAPES["gqa128"]
    pl = np.array([100], np.int32)
    fo = np.array([0, 2], np.int32)
    sl = np.array([5, 7], np.int32)
    lens, keep = _lib.make_host_lens(pl, fo, sl)
    args = _args(1, 2, **shape)
    lib = _lib.load()
    plan = _lib.Plan()
    small = np.zeros(8, np.uint8)
    assert lib.specgen_fork_attn_plan_host(C.byref(args), C.byref(lens), small.ctypes.data,
                                           small.nbytes, C.byref(plan)) == \
        _lib.SPECGEN_ERR_WORKSPACE
    assert lib.specgen_fork_attn_plan_host(C.byref(args), C.byref(lens), None, 0,
                                           C.byref(plan)) == _lib.SPECGEN_ERR_NULL
    bad = _args(1, 2, **dict(shape, hq=63))
    buf = np.zeros(1 << 16, np.uint8)
    assert lib.specgen_fork_attn_plan_host(C.byref(bad), C.byref(lens), buf.ctypes.data,
                                           buf.nbytes, C.byref(plan)) == _lib.SPECGEN_ERR_SHAPE


# ---- fork prefill: one query row per chunk token, causal suffix lengths ------

def _prefill_plan(shape, pl, fo, sl, cl):
    B = shape["B"]
    pbo = np.concatenate([[0], np.cumsum((pl + B - 1) // B)]).astype(np.int32)
    sbo = np.concatenate([[0], np.cumsum((sl + cl + B - 1) // B)]).astype(np.int32)
    lens, keep = _lib.make_prefill_lens(pl, fo, sl, cl, pbo, sbo)
    args = _args(len(pl), int(cl.sum()), **shape)
    need = _lib.specgen_fork_prefill_workspace_size(args, lens)
    assert need > 0
    buf = np.zeros(need, dtype=np.uint8)
    plan = _lib.specgen_fork_prefill_plan_host(args, lens, buf)
    return plan, _parse(plan, buf), pbo, sbo


@pytest.mark.parametrize("case", range(10))
def test_prefill_plans_cover_every_causal_key_once(case):
    """Row r (chunk token j of fork f) must see the trace's prefix and suffix keys
    [0, S_f + j + 1) exactly once; a suffix item of several rows masks row i of
    the item at row_limit0 + i keys."""
    rng = np.random.default_rng(2000 + case)
    shape = [SHAPES["gqa128"], SHAPES["gqa64"], SHAPES["g128"], SHAPES["mha"]][case % 4]
    G = shape["hq"] // shape["hkv"]
    T = int(rng.integers(1, 4))
    fk = rng.integers(1, 5, T)
    fo = np.concatenate([[0], np.cumsum(fk)]).astype(np.int32)
    nf = int(fo[-1])
    pl = rng.integers(0, 3000, T).astype(np.int32)
    sl = rng.integers(0, 400, nf).astype(np.int32)
    cl = rng.integers(0, 90, nf).astype(np.int32)
    cl[0] = max(int(cl[0]), 1)
    plan, p, pbo, sbo = _prefill_plan(shape, pl, fo, sl, cl)
    assert plan.n_split_items == 0
    # the query rows: fork by fork, one per chunk token
    row_fork = np.repeat(np.arange(nf), cl)
    row_len = np.concatenate([sl[f] + np.arange(1, cl[f] + 1) for f in range(nf)]).astype(int)
    fork_trace = np.repeat(np.arange(T), np.diff(fo))
    R = len(row_fork)
    cover, parts = {}, {}
    for kind, seq, g, f0, n, tb, te, part, dv0, toff, rl in p["tc"]:
        assert te > tb >= 0 and 1 <= n and n * G <= 128
        rows = range(f0, f0 + n)
        if kind == 0:
            assert all(fork_trace[row_fork[r]] == seq for r in rows) and te <= pl[seq]
            assert rl == 0 and toff == pbo[seq]
            for r in rows:
                cover.setdefault((r, g, 0), []).append((int(tb), int(te)))
        else:
            assert all(row_fork[r] == seq for r in rows) and toff == sbo[seq]
            assert (rl > 0) == (n > 1)
            if n > 1:
                assert rl == row_len[f0] and all(row_len[r] == rl + (r - f0) for r in rows)
            for i, r in enumerate(rows):
                end = min(int(te), int(rl) + i) if n > 1 else int(te)
                assert end <= row_len[r]
                if end > tb:
                    cover.setdefault((r, g, 1), []).append((int(tb), end))
        for r in rows:
            parts.setdefault((r, g), []).append(int(part))
    for r in range(R):
        for g in range(shape["hkv"]):
            _covers(cover.get((r, g, 0), []), int(pl[fork_trace[row_fork[r]]]), ("prefix", r, g))
            _covers(cover.get((r, g, 1), []), int(row_len[r]), ("suffix", r, g))
            assert sorted(parts.get((r, g), [])) == list(range(p["n_parts"][r, g]))
    _check_slots(p, plan, R)


# ---- nested-prefix cascade: laminar shared segments --------------------------

def _laminar(rng, b, e, depth, out):
    """Random laminar segments over forks [b, e): this range, then children that
    partition parts of it."""
    out.append((b, e))
    if depth == 0 or e - b < 2:
        return
    cuts = np.sort(rng.choice(np.arange(b + 1, e), size=min(e - b - 1, int(rng.integers(1, 3))),
                              replace=False))
    edges = [b] + [int(c) for c in cuts] + [e]
    for lo, hi in zip(edges[:-1], edges[1:]):
        if rng.random() < 0.7:
            _laminar(rng, lo, hi, depth - 1, out)


@pytest.mark.parametrize("case", range(10))
def test_cascade_plans_cover_every_segment_once(case):
    """Fork f must see every segment that serves it, each exactly once, then its
    suffix; the slots of its items are distinct and dense."""
    rng = np.random.default_rng(3000 + case)
    shape = [SHAPES["gqa128"], SHAPES["gqa64"], SHAPES["mha"], SHAPES["latent"]][case % 4]
    F = int(rng.integers(2, 24))
    segs = []
    _laminar(rng, 0, F, 3, segs)
    seg_lens = rng.integers(0, 2500, len(segs)).astype(np.int32)
    seg_rows = np.array([x for s in segs for x in s], np.int32)
    sl = rng.integers(0, 500, F).astype(np.int32)
    B = shape["B"]
    sgbo = np.concatenate([[0], np.cumsum((seg_lens + B - 1) // B)]).astype(np.int32)
    sbo = np.concatenate([[0], np.cumsum((sl + B - 1) // B)]).astype(np.int32)
    lens, keep = _lib.make_cascade_lens(seg_lens, seg_rows, sl, sgbo, sbo)
    args = _args(len(segs), F, **shape)
    need = _lib.specgen_fork_cascade_workspace_size(args, lens)
    assert need > 0
    buf = np.zeros(need, dtype=np.uint8)
    plan = _lib.specgen_fork_cascade_plan_host(args, lens, buf)
    p = _parse(plan, buf)
    groups = shape["hkv"] if not shape["latent"] else 1
    cover, parts = {}, {}
    for kind, seq, g, f0, n, tb, te, part, dv0, toff, rl in p["tc"]:
        assert te > tb >= 0 and rl == 0
        key_g = dv0 if shape["latent"] else g
        for f in range(f0, f0 + n):
            if kind == 0:
                assert segs[seq][0] <= f < segs[seq][1] and te <= seg_lens[seq]
                assert toff == sgbo[seq]
            else:
                assert seq == f and te <= sl[f] and toff == sbo[seq]
            cover.setdefault((f, key_g, kind, int(seq) if kind == 0 else -1), []).append(
                (int(tb), int(te)))
            parts.setdefault((f, key_g), []).append(int(part))
    keys_g = (0, 256) if shape["latent"] else range(groups)
    for f in range(F):
        for g in keys_g:
            for si, (b, e) in enumerate(segs):
                want = int(seg_lens[si]) if b <= f < e else 0
                _covers(cover.get((f, g, 0, si), []), want, ("segment", f, g, si))
            _covers(cover.get((f, g, 1, -1), []), int(sl[f]), ("suffix", f, g))
            n_parts = p["n_parts"][f, 0 if shape["latent"] else g]
            assert sorted(parts.get((f, g), [])) == list(range(n_parts)), (f, g)
    _check_slots(p, plan, F)


@pytest.mark.parametrize("name", ["tiny_p512_f4", "fork_p8k_f8", "mla_p16k_f8"])
def test_workload_lengths_match_the_workload(name):
    """The lengths the planner tests draw are the ones the full workload uses."""
    w = wl.make_workload(name)
    pl, fo, sl = wl.workload_lengths(name)
    assert np.array_equal(pl, w["prefix_lens"]) and np.array_equal(fo, w["fork_offsets"])
    assert np.array_equal(sl, w["suffix_lens"])


# ---- suffix stage: per-fork suffix pages on the split-K worker warps ---------

def _sfx_pieces(p):
    """(fork, kv head) -> sorted token ranges of its suffix-stage items, and the
    per-worker page loads."""
    pieces, loads = {}, []
    so = p["sfx_offsets"]
    for w in range(len(so) - 1):
        load = 0
        for it in p["sfx"][so[w]:so[w + 1]]:
            kind, seq, g, f0, nf, tb, te = (int(x) for x in it[:7])
            pieces.setdefault((f0, g), []).append((tb, te))
            load += (te - tb + 15) // 16
        loads.append(load)
    return pieces, np.array(loads)


@pytest.mark.parametrize("case", range(12))
def test_suffix_only_plans_use_the_suffix_stage(case):
    """With no prefix the whole call is the suffix stage: every suffix key is
    covered once (checked with the tensor-core items' rules), items are page
    aligned, no piece is shorter than two pages unless its suffix is, and the
    workers' page loads are within a few pages of each other."""
    rng = np.random.default_rng(4000 + case)
    G = [1, 2, 3, 4, 5, 8, 12, 16][case % 8]
    hkv = [1, 2, 4][case % 3]
    dqk = [64, 128][case % 2]
    shape = dict(hq=G * hkv, hkv=hkv, dqk=dqk, dv=dqk, B=16, latent=False)
    T = int(rng.integers(1, 4))
    fo = np.concatenate([[0], np.cumsum(rng.integers(1, 12, T))]).astype(np.int32)
    F = int(fo[-1])
    pl = np.zeros(T, np.int32)
    sl = rng.integers(0, 3000, F).astype(np.int32)
    sl[rng.random(F) < 0.15] = 0
    sl[rng.random(F) < 0.1] = 1
    if sl.sum() == 0:
        sl[0] = 40
    plan, buf, pbo, sbo = _plan(shape, pl, fo, sl)
    p = _parse(plan, buf)
    assert plan.n_tc_ctas == 0 and plan.n_sfx_ctas > 0 and plan.n_split_items == 0
    _check_tc(shape, pl, fo, sl, plan, p, pbo, sbo, True)
    pieces, loads = _sfx_pieces(p)
    for (f, g), rs in pieces.items():
        rs = sorted(rs)
        for tb, te in rs:
            assert tb % 16 == 0                       # page aligned
            # no piece shorter than two pages unless the whole suffix is
            assert (te - tb + 15) // 16 >= min(2, (int(sl[f]) + 15) // 16)
    assert loads.max() - loads.min() <= 3 + 2 * 3, (loads.min(), loads.max())


def test_split_rules():
    """The suffix stage runs beside the prefix only where it pays: many short
    suffixes (the ragged batch) split, long suffixes (32k prefix, 256-2048-token
    suffixes) and small calls (8k prefix, 8 forks) stay on the tensor-core kernel."""
    def plan_of(name):
        spec = wl.WORKLOADS[name]
        pl, fo, sl = wl.workload_lengths(name)
        shape = dict(hq=spec.hq, hkv=spec.hkv, dqk=spec.dqk, dv=spec.dv, B=spec.page_size,
                     latent=not spec.separate_v)
        plan, buf, pbo, sbo = _plan(shape, pl, fo, sl)
        return plan, _parse(plan, buf), (shape, pl, fo, sl, pbo, sbo)
    plan, p, (shape, pl, fo, sl, pbo, sbo) = plan_of("ragged_t8")
    assert plan.n_tc_ctas > 0 and plan.n_sfx_ctas > 0
    assert plan.n_tc_ctas + plan.n_sfx_ctas <= 148
    # the prefix kernel takes no suffix item, the suffix stage every one
    assert np.all(p["tc_only"][:, 0] == 0) and np.all(p["sfx"][:, 0] == 1)
    # SMs split about in proportion to the work (suffix pages weighted 0.8)
    share = plan.n_sfx_ctas / (plan.n_tc_ctas + plan.n_sfx_ctas)
    assert 0.1 < share < 0.3, share
    for name in ("long_p32k_f16", "fork_p8k_f8", "tiny_p512_f4"):
        plan, p, _ = plan_of(name)
        assert plan.n_sfx_ctas == 0, name
