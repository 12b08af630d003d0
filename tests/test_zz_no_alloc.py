"""The allocation-free entry point, specgen_fork_attn_decode_static.

It serves callers that cannot allocate device memory (a plugin inside an
engine that owns the device memory pool, or a latency-critical path where an
allocation is not allowed): it takes no workspace and uses the library's
fixed 16 MiB scratch array instead.  Its output must match the ordinary entry
point's, call after call.  This file is collected last on purpose, so that a
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


def test_static_rejects_oversized_calls():
    """A consistent workload whose workspace exceeds 16 MiB is refused on the host."""
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    spec = wl.WorkloadSpec(name="many_forks", num_traces=1, prefix_len=(64, 64),
                           forks=(2000, 2000), suffix_len=(1, 1), hq=64, hkv=8, dqk=128,
                           dv=128, page_size=16, seed=7)
    w = wl.make_workload(spec)
    fd = ForkDecode(w)
    assert fd.ws_bytes > (16 << 20)
    with pytest.raises(_lib.SpecgenError) as err:
        _lib.specgen_fork_attn_decode_static(fd.args(with_ws=False), fd.lens)
    assert err.value.status == _lib.SPECGEN_ERR_WORKSPACE
