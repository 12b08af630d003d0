"""The suffix-stage kernel (per-fork suffix pages on split-K worker warps beside
the tensor-core prefix kernel) against the fp64 oracle, through the C ABI.

Every case here plans the suffix stage (checked on the plan), with group sizes
that fill one or two 8-head n-tiles partly or fully, head dims 64 and 128, both
pool layouts, ragged suffix lengths around the 16-token page (0, 1, 15, 16, 17,
...), suffix-only calls (the kernel then runs alone and waits for the stream's
previous kernel itself), invalid page ids and items cut by device lengths.
Tolerances as everywhere: max |dO| <= 2e-2 (bf16 O), max |dLSE| <= 1e-3.
"""

import numpy as np
import pytest

import __graft_entry__
import oracle
from paper_2606_17518_gb300 import _lib, workloads as wl

pytestmark = pytest.mark.gpu

TOL_O = 2e-2
TOL_LSE = 1e-3


@pytest.fixture(scope="module", autouse=True)
def built():
    __graft_entry__.build()


def _run(w, kv_layout, **fd_kw):
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    fd = ForkDecode(w, kv_layout=kv_layout, **fd_kw)
    fd.plan()
    assert fd.plan_info.n_sfx_ctas > 0, "the call should plan the suffix stage"
    fd.run()
    o, lse = fd.results()
    return o, lse, fd


def _compare(o, lse, o_ref, lse_ref, what):
    assert np.all(np.isfinite(o)), what
    fin = np.isfinite(lse_ref)
    assert np.array_equal(np.isfinite(lse), fin), what
    assert np.all(lse[~fin] == lse_ref[~fin]), what
    err_o = float(np.max(np.abs(o - o_ref))) if o.size else 0.0
    err_l = float(np.max(np.abs(lse[fin] - lse_ref[fin]))) if fin.any() else 0.0
    assert err_o <= TOL_O, (what, err_o)
    assert err_l <= TOL_LSE, (what, err_l)


def _spec(G, hkv, dqk, seed, traces=3, prefix=(0, 0), suffix=(0, 300), forks=(1, 6)):
    return wl.WorkloadSpec(name=f"sfx_g{G}_d{dqk}", num_traces=traces, prefix_len=prefix,
                           forks=forks, suffix_len=suffix, hq=G * hkv, hkv=hkv, dqk=dqk,
                           dv=dqk, page_size=16, seed=seed)


EDGE_LENS = [0, 1, 15, 16, 17, 31, 33, 160, 161, 257]

CASES = [(G, hkv, dqk) for G, hkv in [(1, 3), (2, 2), (3, 1), (5, 2), (8, 2), (12, 1), (16, 2)]
         for dqk in (64, 128)]


@pytest.mark.parametrize("layout", ["rows", "tiled"])
@pytest.mark.parametrize("G,hkv,dqk", CASES)
def test_suffix_stage_shapes(G, hkv, dqk, layout):
    """Suffixes only (no prefix: the suffix stage takes every key), so every
    shape runs on the suffix-stage kernel however small it is."""
    seed = 100 * G + dqk + (1 if layout == "tiled" else 0)
    w = wl.make_workload(_spec(G, hkv, dqk, seed, prefix=(0, 0), suffix=(0, 300)))
    rng = np.random.default_rng(seed)
    # suffix lengths on and around page boundaries, each at most the drawn length
    # (the keys past a drawn length are NaN)
    sl = w["suffix_lens"].copy()
    for f in range(len(sl)):
        sl[f] = min(int(rng.choice(EDGE_LENS)), int(sl[f]))
    w["suffix_lens"] = sl.astype(np.int32)
    w = _renan(w)
    kv = _lib.KV_TILED if layout == "tiled" else _lib.KV_ROWS
    o, lse, fd = _run(w, kv)
    assert fd.status() == _lib.SPECGEN_OK
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, f"G{G} hkv{hkv} d{dqk} {layout}")


def _renan(w):
    """NaN in every suffix slot past its (possibly shortened) length."""
    w = dict(w)
    B = w["page_size"]
    for key in ("k_pages", "v_pages"):
        pool = w[key].copy()
        for f, n in enumerate(w["suffix_lens"]):
            pages = w["suffix_table"][w["suffix_bt_offsets"][f]:w["suffix_bt_offsets"][f + 1]]
            for i, pg in enumerate(pages):
                first = max(0, int(n) - i * B)
                if first < B:
                    pool[pg, :, first:, :] = wl.BF16_QNAN
        w[key] = pool
    return w


@pytest.mark.parametrize("layout", ["rows", "tiled"])
@pytest.mark.parametrize("G,hkv", [(8, 8), (4, 8), (16, 4)])
def test_suffix_stage_beside_prefix(G, hkv, layout):
    """A call large enough to run the suffix stage beside the prefix kernel
    (the two grids share the SMs; the merge waits for both): two traces with
    8192-token prefixes and 16 forks each with suffixes of 300-900 tokens."""
    w = wl.make_workload(_spec(G, hkv, 128, 500 + G, traces=2, prefix=(8192, 8192),
                               suffix=(300, 900), forks=(16, 16)))
    kv = _lib.KV_TILED if layout == "tiled" else _lib.KV_ROWS
    o, lse, fd = _run(w, kv)
    assert fd.plan_info.n_tc_ctas > 0
    assert fd.status() == _lib.SPECGEN_OK
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, f"beside prefix G{G} {layout}")


@pytest.mark.parametrize("layout", ["rows", "tiled"])
def test_suffix_only_calls(layout):
    """No prefix anywhere: the suffix-stage kernel is the only partial kernel."""
    w = wl.make_workload(_spec(8, 4, 128, 7, traces=2, prefix=(0, 0), suffix=(1, 700),
                               forks=(3, 9)))
    kv = _lib.KV_TILED if layout == "tiled" else _lib.KV_ROWS
    o, lse, fd = _run(w, kv)
    assert fd.plan_info.n_tc_ctas == 0
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, f"suffix only {layout}")
    # and the workload's own suffixes alone, every row
    wf = wl.make_workload("fork_p8k_f8")
    wf = dict(wf, prefix_lens=np.zeros_like(wf["prefix_lens"]))
    o, lse, fd = _run(wf, kv)
    o_ref, lse_ref = oracle.fork_attn_decode(wf)
    _compare(o, lse, o_ref, lse_ref, f"fork_p8k_f8 suffixes only {layout}")


@pytest.mark.parametrize("layout", ["rows", "tiled"])
def test_suffix_stage_invalid_page_is_reported_not_read(layout):
    """A suffix page id outside the pool is skipped (its keys masked, its value
    rows zeroed) and reported; the forks that do not use it are unaffected."""
    w_ok = wl.make_workload(_spec(8, 2, 128, 11, traces=1, prefix=(0, 0), suffix=(40, 90),
                                  forks=(3, 3)))
    w = dict(w_ok)
    w["suffix_table"] = w_ok["suffix_table"].copy()
    w["suffix_table"][int(w["suffix_bt_offsets"][1])] = w["num_pages"] + 11  # fork 1, page 0
    kv = _lib.KV_TILED if layout == "tiled" else _lib.KV_ROWS
    o, lse, fd = _run(w, kv)
    assert fd.status() == _lib.SPECGEN_ERR_INDEX
    assert np.all(np.isfinite(o))
    o_ref, lse_ref = oracle.fork_attn_decode(w_ok)
    keep = [0, 2]
    _compare(o[keep], lse[keep], o_ref[keep], lse_ref[keep], f"bad page {layout}")


@pytest.mark.parametrize("ahead", [5, 40])
def test_suffix_stage_items_cut_by_device_lengths(ahead):
    """A plan made for suffixes `ahead` tokens longer: the suffix-stage items are
    cut by the device lengths (with 40, some to nothing)."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    base = wl.make_workload(_spec(8, 8, 128, 508, traces=2, prefix=(8192, 8192),
                                  suffix=(300, 900), forks=(16, 16)))
    st = wl.make_decode_state(base, ahead)
    fd = ForkDecode(st, kv_layout=_lib.KV_TILED)
    fd.use_device_lens = True
    lens = st["suffix_lens"].copy()
    fd.set_suffix_lens(lens + ahead, update_device=False)
    fd.suffix_lens_dev.copy_(torch.from_numpy(lens))
    fd.plan()
    assert fd.plan_info.n_sfx_ctas > 0
    fd.run()
    o, lse = fd.results()
    assert fd.status() == _lib.SPECGEN_OK
    o_ref, lse_ref = oracle.fork_attn_decode(dict(st, suffix_lens=lens))
    _compare(o, lse, o_ref, lse_ref, f"ahead {ahead}")


@pytest.mark.parametrize("mode", ["alone", "beside"])
@pytest.mark.parametrize("layout", ["rows", "tiled"])
@pytest.mark.parametrize("G,hkv", [(16, 4), (8, 8)])
def test_suffix_stage_repeatable(G, hkv, layout, mode):
    """Twenty runs of one plan give the same bits: every partial of the suffix
    stage is written by one worker from data it waited for.  A buffer refilled
    too early shows up here as run-to-run differences (it did, for the query
    rows of the second n-tile, before the next item's rows were copied in only
    after the current ones had been consumed)."""
    import torch
    if mode == "alone":
        w = wl.make_workload(_spec(G, hkv, 128, 900 + G, traces=2, prefix=(0, 0),
                                   suffix=(20, 700), forks=(4, 8)))
    else:
        w = wl.make_workload(_spec(G, hkv, 128, 500 + G, traces=2, prefix=(8192, 8192),
                                   suffix=(300, 900), forks=(16, 16)))
    kv = _lib.KV_TILED if layout == "tiled" else _lib.KV_ROWS
    o1, l1, fd = _run(w, kv)
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o1, l1, o_ref, lse_ref, f"repeat G{G} {layout}")
    for _ in range(19):
        fd.out.zero_()
        fd.run()
    torch.cuda.synchronize()
    o2, l2 = fd.results()
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2)
    assert fd.status() == _lib.SPECGEN_OK


def _ragged_fuzz_spec(case):
    """Random multi-trace calls large enough that the planner runs the suffix
    stage beside the prefix kernel: 3-4 traces, 12-20 forks each, prefixes of
    0.5k-5k tokens and suffixes of 150-800, G from 1 to 16 (with G = 3, 6 and
    12 filling their n-tiles partly), head dims 64 and 128."""
    rng = np.random.default_rng(4200 + case)
    G = [1, 2, 4, 8, 12, 16, 3, 6][case]
    hkv = [8, 8, 8, 4, 8, 4, 8, 8][case]
    dqk = [64, 128][case % 2]
    return wl.WorkloadSpec(
        name=f"ragged_fuzz{case}", num_traces=int(rng.integers(3, 5)),
        prefix_len=(int(rng.integers(500, 2000)), int(rng.integers(2000, 5000))),
        forks=(int(rng.integers(12, 15)), int(rng.integers(15, 21))),
        suffix_len=(int(rng.integers(150, 400)), int(rng.integers(500, 800))),
        hq=G * hkv, hkv=hkv, dqk=dqk, dv=dqk, page_size=16, seed=int(rng.integers(1 << 30)))


@pytest.mark.parametrize("case", range(8))
def test_ragged_calls_with_the_suffix_stage_every_row(case):
    """Every (fork, head) row of random ragged calls that split the SMs between
    the prefix kernel and the suffix-stage kernel, against the oracle; the pool
    layout alternates between cases."""
    w = wl.make_workload(_ragged_fuzz_spec(case))
    kv = _lib.KV_TILED if case % 2 else _lib.KV_ROWS
    o, lse, fd = _run(w, kv)
    assert fd.plan_info.n_tc_ctas > 0
    assert fd.status() == _lib.SPECGEN_OK
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, f"ragged fuzz {case}")
