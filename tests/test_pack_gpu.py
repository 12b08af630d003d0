"""Prefix page pack / unpack on the GPU against the oracle (bit-exact, through the C ABI)."""

import numpy as np
import pytest

import __graft_entry__
import oracle
from paper_2606_17518_gb300 import _lib, workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    __graft_entry__.build()


def _dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()


def _host(t):
    import torch
    torch.cuda.synchronize()
    return t.cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("name,layout", [("fork_p8k_f8", "rows"), ("tiny_p512_f4", "tiled"),
                                         ("mla_p16k_f8", "rows")])
def test_pack_unpack_bit_exact(name, layout):
    import torch
    w = wl.make_workload(name)
    k, v = w["k_pages"], w["v_pages"]
    if layout == "tiled":
        k, v = wl.tile_kv_pool(k), wl.tile_kv_pool(v)
    dk, dv = _dev(k), (None if v is None else _dev(v))
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    desc = _lib.make_pool_desc(hkv=w["hkv"], head_dim_qk=w["dqk"], head_dim_v=w["dv"],
                               page_size=w["page_size"], num_pages=w["num_pages"], k_pages=dk,
                               v_pages=dv, status=status)
    table = w["prefix_table"][w["prefix_bt_offsets"][0]: w["prefix_bt_offsets"][1]]
    n = len(table)
    nbytes = _lib.specgen_packed_bytes(desc, n)
    packed = torch.empty(nbytes // 2, dtype=torch.int16, device="cuda")
    _lib.specgen_pack_pages(desc, torch.from_numpy(table).cuda(), n, packed)
    ref = oracle.pack_pages(k, v, table)
    assert np.array_equal(_host(packed), ref)
    # unpack under a new table: the prefix's pages in reverse order
    new = table[::-1].copy()
    _lib.specgen_unpack_pages(desc, torch.from_numpy(new).cuda(), n, packed)
    rk, rv = oracle.unpack_pages(k, v, new, ref)
    assert np.array_equal(_host(dk), rk)
    if v is not None:
        assert np.array_equal(_host(dv), rv)
    assert int(status.item()) == 0


def test_pack_skips_and_reports_bad_page_ids():
    import torch
    w = wl.make_workload("tiny_p512_f4")
    dk, dv = _dev(w["k_pages"]), _dev(w["v_pages"])
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    desc = _lib.make_pool_desc(hkv=w["hkv"], head_dim_qk=w["dqk"], head_dim_v=w["dv"],
                               page_size=w["page_size"], num_pages=w["num_pages"], k_pages=dk,
                               v_pages=dv, status=status)
    table = np.array([3, w["num_pages"] + 5, -1, 7], dtype=np.int32)
    nbytes = _lib.specgen_packed_bytes(desc, 4)
    packed = torch.full((nbytes // 2,), 0x1234, dtype=torch.int16, device="cuda")
    _lib.specgen_pack_pages(desc, torch.from_numpy(table).cuda(), 4, packed)
    got = _host(packed)
    assert int(status.item()) == 1
    blk = w["hkv"] * w["page_size"] * w["dqk"]
    ok = oracle.pack_pages(w["k_pages"], w["v_pages"], [3, 3, 3, 7])
    for sec in range(2):
        for i in (0, 3):      # valid pages copied
            sl = slice(sec * 4 * blk + i * blk, sec * 4 * blk + (i + 1) * blk)
            assert np.array_equal(got[sl], ok[sl])
        for i in (1, 2):      # invalid ids: the buffer is left as it was
            sl = slice(sec * 4 * blk + i * blk, sec * 4 * blk + (i + 1) * blk)
            assert np.all(got[sl] == 0x1234)
