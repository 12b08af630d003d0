"""The allocation-free entry point, specgen_fork_attn_decode_static.

It serves callers that cannot allocate device memory (a plugin inside an
engine that owns the device memory pool, or a latency-critical path where an
allocation is not allowed): it takes no workspace and uses the library's
fixed 16 MiB scratch array instead.  Its output must match the ordinary entry
point's, call after call, and its status word (kept in that array) must be
readable.  The refusal of oversized calls happens on the host and is checked
by the CPU tests.  This file is collected last on purpose, so that a
run that stops at the first failure has already run every other test.
"""

import numpy as np
import pytest

import __graft_entry__
from paper_2606_17518_gb300 import _lib, workloads as wl

pytestmark = pytest.mark.gpu

TOL_O = 2e-2
TOL_LSE = 1e-3


@pytest.fixture(scope="module", autouse=True)
def built():
    __graft_entry__.build()


@pytest.mark.parametrize("name", ["tiny_p512_f4", "fork_p8k_f8"])
def test_static_matches_workspace_entry_point_twice(name):
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = wl.make_workload(name)
    fd = ForkDecode(w)
    fd.decode()
    o_ref, l_ref = fd.results()
    for _ in range(2):  # two calls in a row share the same scratch array
        fd.out.zero_()
        fd.lse.zero_()
        args = fd.args(with_ws=False)
        _lib.specgen_fork_attn_decode_static(args, fd.lens)
        torch.cuda.synchronize()
        o, lse = fd.results()
        assert np.all(np.isfinite(o))
        assert np.max(np.abs(o - o_ref)) <= TOL_O
        fin = np.isfinite(l_ref)
        assert np.array_equal(np.isfinite(lse), fin)
        assert np.max(np.abs(lse[fin] - l_ref[fin])) <= TOL_LSE
        # the status word lives in the library's array: readable, and clean
        assert _lib.specgen_static_workspace_status() == _lib.SPECGEN_OK


def test_static_with_the_suffix_stage_and_the_largest_workload():
    """Plans that run the suffix-stage kernel beside the prefix kernel (ragged_t8,
    the largest workload, 9.5 MB of scratch, and a 16-fork call with G = 16)
    through the scratch array: the same bits as the workspace entry point."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    spec = wl.WorkloadSpec(name="static_sfx_g16", num_traces=2, prefix_len=(8192, 8192),
                           forks=(16, 16), suffix_len=(300, 900), hq=64, hkv=4, dqk=128,
                           dv=128, page_size=16, seed=516)
    for w in (wl.make_workload("ragged_t8"), wl.make_workload(spec)):
        fd = ForkDecode(w, kv_layout=_lib.KV_TILED)
        fd.plan()
        assert fd.plan_info.n_sfx_ctas > 0 and fd.plan_info.ws_end <= (16 << 20)
        fd.run()
        torch.cuda.synchronize()
        o_ref, l_ref = fd.results()
        fd.out.zero_()
        fd.lse.zero_()
        _lib.specgen_fork_attn_decode_static(fd.args(with_ws=False), fd.lens)
        torch.cuda.synchronize()
        assert _lib.specgen_static_workspace_status() == _lib.SPECGEN_OK
        o, lse = fd.results()
        assert np.array_equal(o, o_ref) and np.array_equal(lse, l_ref)


def test_static_status_reports_a_bad_page_id():
    """A page id outside the pool is skipped by the kernels and reported in the
    scratch array's status word; the next clean call resets it."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = dict(wl.make_workload("tiny_p512_f4"))
    good = ForkDecode(w)
    w["suffix_table"] = w["suffix_table"].copy()
    w["suffix_table"][0] = w["num_pages"] + 5
    bad = ForkDecode(w)
    _lib.specgen_fork_attn_decode_static(bad.args(with_ws=False), bad.lens)
    torch.cuda.synchronize()
    assert _lib.specgen_static_workspace_status() == _lib.SPECGEN_ERR_INDEX
    o, _ = bad.results()
    assert np.all(np.isfinite(o))
    _lib.specgen_fork_attn_decode_static(good.args(with_ws=False), good.lens)
    torch.cuda.synchronize()
    assert _lib.specgen_static_workspace_status() == _lib.SPECGEN_OK
