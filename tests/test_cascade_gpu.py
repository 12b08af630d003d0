"""Decode over nested shared prefix segments on the GPU against the oracle."""

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


def _compare(w):
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    fd = ForkDecode(w)
    fd.decode()
    o, lse = fd.results()
    assert fd.status() == _lib.SPECGEN_OK
    o_ref, lse_ref = oracle.fork_cascade_decode(w)
    assert np.all(np.isfinite(o))
    assert float(np.max(np.abs(o - o_ref))) <= TOL_O
    fin = np.isfinite(lse_ref)
    assert np.array_equal(np.isfinite(lse), fin)
    assert float(np.max(np.abs(lse[fin] - lse_ref[fin]))) <= TOL_LSE
    return fd


@pytest.mark.parametrize("points,forks", [((4096, 8192), (8, 8)), ((2048, 4096, 8192), (4, 8, 4)),
                                          ((8192,), (8,))])
def test_cascade_gqa(points, forks):
    _compare(wl.make_cascade(points, forks, seed=len(points)))


def test_cascade_many_forks_per_group():
    """24 forks (G = 8): three row groups; the deeper segment's groups sit on
    the outer segment's grid."""
    _compare(wl.make_cascade((1024, 3072), (10, 14), suffix_len=(1, 200), seed=4))


@pytest.mark.parametrize("page,dqk", [(64, 128), (16, 64)])
def test_cascade_split_path_and_small_heads(page, dqk):
    _compare(wl.make_cascade((page * 4, page * 9), (3, 2), suffix_len=(0, 100), hq=16, hkv=2,
                             dqk=dqk, dv=dqk, page_size=page, seed=page))


def test_cascade_latent():
    _compare(wl.make_cascade((1024, 4096), (3, 2), suffix_len=(64, 300), hq=128, hkv=1,
                             dqk=576, dv=512, page_size=64, separate_v=False, seed=7))


def test_cascade_tree_not_chain():
    """Two sibling segments under one root: forks 0-3 take segment 1, forks
    4-6 segment 2, all take segment 0 (depth-first numbering)."""
    w = wl.make_cascade((2048, 4096), (3, 4), seed=11)
    # segment 1 of the chain serves forks [0, 4); add a sibling over [4, 7) that
    # reuses segment 1's pages (any pages serve; the ranges are what is tested)
    w = dict(w)
    w["prefix_lens"] = np.concatenate([w["prefix_lens"], w["prefix_lens"][1:2]]).astype(np.int32)
    w["prefix_bt_offsets"] = np.concatenate(
        [w["prefix_bt_offsets"], [w["prefix_bt_offsets"][-1] + 128]]).astype(np.int32)
    w["prefix_table"] = np.concatenate([w["prefix_table"], w["prefix_table"][128:256]]).astype(np.int32)
    w["segment_rows"] = np.array([0, 7, 0, 4, 4, 7], dtype=np.int32)
    w["num_traces"] = 3
    _compare(w)


def test_cascade_rejects_crossing_segments():
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = wl.make_cascade((2048, 4096), (3, 4), seed=11)
    w = dict(w, segment_rows=np.array([0, 5, 2, 7], dtype=np.int32))   # neither nested nor disjoint
    with pytest.raises(_lib.SpecgenError):
        ForkDecode(w)
