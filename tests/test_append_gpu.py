"""Decode-step append on the GPU against the oracle (through the C ABI).

Bit-exact: the pools (every byte, NaN fill included), the block tables and the
number of pages taken must equal the oracle's after every step.  The attention
of each step then reads the grown suffixes (tolerance as in test_parity_gpu).
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


def _pools(fd, state):
    import torch
    torch.cuda.synchronize()
    view = lambda t: t.view(torch.int16).cpu().numpy().view(np.uint16)
    k = view(fd.k_pages)
    v = None if fd.v_pages is None else view(fd.v_pages)
    if fd.kv_layout == _lib.KV_TILED:   # compare in the oracle's row layout
        inv = lambda a: untile(a)
        k, v = inv(k), (None if v is None else inv(v))
    return k, v, fd.suffix_table.cpu().numpy()


def untile(pool):
    P, H, B, D = pool.shape
    t = pool.reshape(P, H, B // 8, D // 8, 8, 8)
    return np.ascontiguousarray(t.transpose(0, 1, 2, 4, 3, 5)).reshape(P, H, B, D)


def _run_steps(name, steps, kv_layout=_lib.KV_ROWS, attend_every=0):
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    st = wl.make_decode_state(wl.make_workload(name), steps)
    fd = ForkDecode(st, kv_layout=kv_layout)
    free = torch.from_numpy(st["free_pages"]).cuda()
    k_new = [torch.from_numpy(st["k_new"][s].view(np.int16)).cuda().view(torch.bfloat16)
             for s in range(steps)]
    v_new = [None if st["v_new"] is None else
             torch.from_numpy(st["v_new"][s].view(np.int16)).cuda().view(torch.bfloat16)
             for s in range(steps)]
    ref_k, ref_v, ref_t = st["k_pages"], st["v_pages"], st["suffix_table"]
    lens = st["suffix_lens"].copy()
    used = 0
    for s in range(steps):
        fd.append_kv(k_new[s], v_new[s], free[used:], len(st["free_pages"]) - used)
        ref_k, ref_v, ref_t, taken = oracle.append_kv(
            ref_k, ref_v, ref_t, st["suffix_bt_offsets"], lens, st["k_new"][s],
            None if st["v_new"] is None else st["v_new"][s], st["free_pages"][used:],
            st["page_size"])
        used += taken
        lens = lens + 1
        fd.set_suffix_lens(lens)
        if attend_every and (s + 1) % attend_every == 0:
            fd.decode()
            o, lse = fd.results()
            w_ref = dict(st, k_pages=ref_k, v_pages=ref_v, suffix_table=ref_t, suffix_lens=lens)
            o_ref, lse_ref = oracle.fork_attn_decode(w_ref)
            assert np.all(np.isfinite(o))
            assert float(np.max(np.abs(o - o_ref))) <= TOL_O
            fin = np.isfinite(lse_ref)
            assert float(np.max(np.abs(lse[fin] - lse_ref[fin]))) <= TOL_LSE
    k, v, t = _pools(fd, st)
    assert np.array_equal(t, ref_t)
    assert np.array_equal(k, ref_k)
    if ref_v is not None:
        assert np.array_equal(v, ref_v)
    assert fd.status() == _lib.SPECGEN_OK
    return st, used


@pytest.mark.parametrize("name,steps", [("tiny_p512_f4", 40), ("fork_p8k_f8", 20),
                                        ("mla_p16k_f8", 70)])
def test_append_bit_exact(name, steps):
    st, used = _run_steps(name, steps)
    assert used > 0  # page boundaries were crossed


def test_append_bit_exact_tiled_layout():
    _run_steps("tiny_p512_f4", 40, kv_layout=_lib.KV_TILED)


@pytest.mark.parametrize("name", ["tiny_p512_f4", "mla_p16k_f8"])
def test_multi_step_decode_matches_oracle(name):
    """append + attention for several steps; every 7th step's outputs checked."""
    _run_steps(name, 21, attend_every=7)


def test_append_reports_exhausted_free_list_and_full_table():
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    st = wl.make_decode_state(wl.make_workload("tiny_p512_f4"), 16)
    # suffix length 32 with page 16: every fork starts a new page this step
    fd = ForkDecode(st)
    k_new = torch.from_numpy(st["k_new"][0].view(np.int16)).cuda().view(torch.bfloat16)
    v_new = torch.from_numpy(st["v_new"][0].view(np.int16)).cuda().view(torch.bfloat16)
    free = torch.from_numpy(st["free_pages"]).cuda()
    before = fd.suffix_table.cpu().numpy().copy()
    fd.append_kv(k_new, v_new, free, 2)          # four forks need a page, two exist
    assert fd.status() == _lib.SPECGEN_ERR_INDEX
    t = fd.suffix_table.cpu().numpy()
    changed = np.nonzero(t != before)[0]
    assert len(changed) == 2                      # forks 0 and 1 got pages, 2 and 3 wrote nothing
    assert sorted(t[changed].tolist()) == sorted(st["free_pages"][:2].tolist())
    # a table with no room: length already at capacity
    st2 = dict(st)
    st2["suffix_lens"] = (st["suffix_bt_offsets"][1:] - st["suffix_bt_offsets"][:-1]) * 16
    fd2 = ForkDecode(wl.make_workload("tiny_p512_f4"))
    fd2.set_suffix_lens(np.full(4, 32, np.int32))   # exactly 2 pages each: no room for a third
    fd2.append_kv(k_new, v_new, free, 4)
    assert fd2.status() == _lib.SPECGEN_ERR_INDEX
