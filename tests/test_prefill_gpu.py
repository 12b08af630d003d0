"""Fork prefill on the GPU against the oracle (through the C ABI)."""

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


def _check(w, chunk, kv_layout=_lib.KV_ROWS, sample=None):
    from paper_2606_17518_gb300.fork_attn import ForkPrefill
    pf = wl.make_prefill(w, chunk)
    fp = ForkPrefill(pf, kv_layout=kv_layout)
    fp.run()
    o, lse = fp.results()
    assert fp.status() == _lib.SPECGEN_OK
    o_ref, lse_ref = oracle.fork_prefill(pf, pf["chunk_lens"], pf["q_rows"])
    assert np.all(np.isfinite(o))
    err_o = float(np.max(np.abs(o - o_ref)))
    fin = np.isfinite(lse_ref)
    assert np.array_equal(np.isfinite(lse), fin)
    err_l = float(np.max(np.abs(lse[fin] - lse_ref[fin])))
    assert err_o <= TOL_O and err_l <= TOL_LSE, (err_o, err_l)


@pytest.mark.parametrize("name,chunk", [("tiny_p512_f4", 32), ("fork_p8k_f8", 16),
                                        ("mla_p16k_f8", 8)])
def test_prefill_workloads(name, chunk):
    _check(wl.make_workload(name), chunk)


def test_prefill_tiled_layout():
    _check(wl.make_workload("tiny_p512_f4"), 17, kv_layout=_lib.KV_TILED)


@pytest.mark.parametrize("case", range(4))
def test_prefill_fuzz(case):
    """Ragged chunks (0..S_f tokens), page 16 and 64 (tensor-core and split
    paths), G 1..16."""
    rng = np.random.default_rng(50 + case)
    B = [16, 64][case % 2]
    G = [1, 4, 8, 16][case]
    spec = wl.WorkloadSpec(name="pf", num_traces=int(rng.integers(1, 3)),
                           prefix_len=(0, 300), forks=(1, 4), suffix_len=(0, 90), hq=G * 2,
                           hkv=2, dqk=128 if case % 2 else 64, dv=128 if case % 2 else 64,
                           page_size=B, seed=int(rng.integers(1 << 30)))
    w = wl.make_workload(spec)
    if w["suffix_lens"].sum() == 0:
        pytest.skip("no suffix tokens to prefill in this draw")
    _check(w, int(rng.integers(1, 40)))


@pytest.mark.parametrize("dqk,G", [(128, 4), (64, 8)])
def test_prefill_long_suffix_groups_cut(dqk, G):
    """Long suffixes behind a short prefix: a fork's chunk tokens share causal
    suffix items (up to 128/G rows each, split where the rows leave a prefix row
    group), and the small total work makes the planner cut those items into
    several token pieces, so rows see pieces that end before, inside and after
    their own causal limit."""
    spec = wl.WorkloadSpec(name="pf_long", num_traces=1, prefix_len=(64, 64), forks=(2, 2),
                           suffix_len=(1200, 1400), hq=G * 2, hkv=2, dqk=dqk, dv=dqk,
                           page_size=16, seed=91 + G)
    _check(wl.make_workload(spec), 48)
