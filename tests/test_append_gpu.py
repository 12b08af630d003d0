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
    lens0 = fd.suffix_lens_dev.cpu().numpy().copy()
    fd.append_kv(k_new, v_new, free, 2, advance=True)  # four forks need a page, two exist
    assert fd.status() == _lib.SPECGEN_ERR_INDEX
    t = fd.suffix_table.cpu().numpy()
    changed = np.nonzero(t != before)[0]
    assert len(changed) == 2                      # forks 0 and 1 got pages, 2 and 3 wrote nothing
    assert sorted(t[changed].tolist()) == sorted(st["free_pages"][:2].tolist())
    # the advanced lengths: +1 only where the fork appended
    assert np.array_equal(fd.suffix_lens_dev.cpu().numpy(), lens0 + np.array([1, 1, 0, 0]))
    # a table with no room: length already at capacity
    st2 = dict(st)
    st2["suffix_lens"] = (st["suffix_bt_offsets"][1:] - st["suffix_bt_offsets"][:-1]) * 16
    fd2 = ForkDecode(wl.make_workload("tiny_p512_f4"))
    fd2.set_suffix_lens(np.full(4, 32, np.int32))   # exactly 2 pages each: no room for a third
    fd2.append_kv(k_new, v_new, free, 4)
    assert fd2.status() == _lib.SPECGEN_ERR_INDEX


def _fuzz_page64(seed):
    return wl.WorkloadSpec(name="split64", num_traces=2, prefix_len=(100, 300), forks=(2, 3),
                           suffix_len=(1, 70), hq=8, hkv=2, dqk=128, dv=128, page_size=64,
                           seed=seed)


@pytest.mark.parametrize("name", ["tiny_p512_f4", "fork_p8k_f8", "mla_p16k_f8", "split64"])
@pytest.mark.parametrize("ahead", [0, 7, 40])
def test_plan_ahead_cut_to_device_lengths(name, ahead):
    """A plan made for suffixes `ahead` tokens longer, run with the actual
    lengths in the device array: the oracle's result at the actual lengths.
    Slots past the actual lengths hold NaN, so any read there would show; with
    ahead = 40 whole suffix items are cut to nothing."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    base = wl.make_workload(_fuzz_page64(3) if name == "split64" else name)
    st = wl.make_decode_state(base, ahead)
    fd = ForkDecode(st)
    fd.use_device_lens = True
    lens = st["suffix_lens"].copy()
    fd.set_suffix_lens(lens + ahead, update_device=False)   # plan for the longer lengths
    fd.suffix_lens_dev.copy_(torch.from_numpy(lens))         # run with the actual ones
    fd.decode()
    o, lse = fd.results()
    assert fd.status() == _lib.SPECGEN_OK
    o_ref, lse_ref = oracle.fork_attn_decode(dict(st, suffix_lens=lens))
    assert np.all(np.isfinite(o))
    assert float(np.max(np.abs(o - o_ref))) <= TOL_O
    fin = np.isfinite(lse_ref)
    assert np.array_equal(np.isfinite(lse), fin)
    assert float(np.max(np.abs(lse[fin] - lse_ref[fin]))) <= TOL_LSE


# a ragged call whose plan runs the suffix-stage kernel beside the prefix kernel
SPLIT_SPEC = wl.WorkloadSpec(name="split_g8", num_traces=3, prefix_len=(800, 4000),
                             forks=(14, 20), suffix_len=(200, 700), hq=32, hkv=4, dqk=128,
                             dv=128, page_size=16, seed=4321)


@pytest.mark.parametrize("advance", ["torch", "append"])
@pytest.mark.parametrize("name", ["fork_p8k_f8", "mla_p16k_f8", "split_g8"])
def test_one_plan_many_decode_steps_in_a_graph(name, advance):
    """One plan for 12 steps ahead; 12 steps of (append, advance the device
    lengths, attention) captured in one CUDA graph; the last step's output and
    the pools match the oracle.  The lengths advance either by a torch add on
    the device or by the append itself (into the other of two arrays).  With
    split_g8 the plan runs the suffix-stage kernel, whose items the device
    lengths cut every step."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    steps = 12
    base = wl.make_workload(SPLIT_SPEC if name == "split_g8" else name)
    st = wl.make_decode_state(base, steps)
    fd = ForkDecode(st)
    fd.use_device_lens = True
    lens0 = st["suffix_lens"].copy()
    fd.set_suffix_lens(lens0 + steps, update_device=False)
    fd.suffix_lens_dev.copy_(torch.from_numpy(lens0))
    stream = torch.cuda.Stream()
    sp = stream.cuda_stream
    fd.plan(sp)
    torch.cuda.synchronize()
    if name == "split_g8":
        assert fd.plan_info.n_sfx_ctas > 0 and fd.plan_info.n_tc_ctas > 0
    free = torch.from_numpy(st["free_pages"]).cuda()
    k_new = torch.from_numpy(st["k_new"].view(np.int16)).cuda().view(torch.bfloat16)
    v_new = (None if st["v_new"] is None else
             torch.from_numpy(st["v_new"].view(np.int16)).cuda().view(torch.bfloat16))
    # pages each step takes: known on the host from the lengths
    offs, lens = [], lens0.copy()
    used = 0
    for s in range(steps):
        offs.append(used)
        used += int(np.sum(lens % st["page_size"] == 0))
        lens = lens + 1
    fd.run(sp)                      # first launches configure the kernels outside the capture
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for s in range(steps):
            fd.append_kv(k_new[s], None if v_new is None else v_new[s], free[offs[s]:],
                         len(st["free_pages"]) - offs[s], sp, advance=advance == "append")
            if advance == "torch":
                fd.suffix_lens_dev.add_(1)
            fd.run(sp)
    graph.replay()
    torch.cuda.synchronize()
    o, lse = fd.results()
    assert fd.status() == _lib.SPECGEN_OK
    assert np.array_equal(fd.suffix_lens_dev.cpu().numpy(), lens0 + steps)
    ref_k, ref_v, ref_t, lens = st["k_pages"], st["v_pages"], st["suffix_table"], lens0.copy()
    used = 0
    for s in range(steps):
        ref_k, ref_v, ref_t, taken = oracle.append_kv(
            ref_k, ref_v, ref_t, st["suffix_bt_offsets"], lens, st["k_new"][s],
            None if st["v_new"] is None else st["v_new"][s], st["free_pages"][used:],
            st["page_size"])
        used += taken
        lens = lens + 1
    k, v, t = _pools(fd, st)
    assert np.array_equal(t, ref_t) and np.array_equal(k, ref_k)
    if ref_v is not None:
        assert np.array_equal(v, ref_v)
    o_ref, lse_ref = oracle.fork_attn_decode(
        dict(st, k_pages=ref_k, v_pages=ref_v, suffix_table=ref_t, suffix_lens=lens))
    assert float(np.max(np.abs(o - o_ref))) <= TOL_O
    fin = np.isfinite(lse_ref)
    assert float(np.max(np.abs(lse[fin] - lse_ref[fin]))) <= TOL_LSE
