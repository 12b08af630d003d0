"""GPU vs fp64 oracle parity, through the C ABI (libspecgen.so).

Tolerances (from the fork-decode target): max |dO| <= 2e-2 on bf16 outputs
and max |dLSE| <= 1e-3 on fp32 LSE.  Index handling is bit-exact: the same
logical KV at a different physical page placement gives identical bits, and a
page id outside the pool is reported, never read.  Every pool holds NaN in
unused slots and sentinel pages, so any read past a length shows up.
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


def _gpu(w, kv_layout=_lib.KV_ROWS):
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    fd = ForkDecode(w, kv_layout=kv_layout)
    fd.decode()
    o, lse = fd.results()
    assert fd.status() == _lib.SPECGEN_OK
    return o, lse, fd


def _compare(o, lse, o_ref, lse_ref, what=""):
    assert np.all(np.isfinite(o)), what
    fin = np.isfinite(lse_ref)
    assert np.array_equal(np.isfinite(lse), fin), what
    assert np.all(lse[~fin] == lse_ref[~fin]), what
    err_o = float(np.max(np.abs(o - o_ref))) if o.size else 0.0
    err_l = float(np.max(np.abs(lse[fin] - lse_ref[fin]))) if fin.any() else 0.0
    assert err_o <= TOL_O, (what, err_o)
    assert err_l <= TOL_LSE, (what, err_l)
    return err_o, err_l


@pytest.mark.parametrize("name", ["tiny_p512_f4", "fork_p8k_f8", "mla_p16k_f8"])
def test_workload_full(name):
    w = wl.make_workload(name)
    o, lse, _ = _gpu(w)
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, name)


# The two large workloads are generated and run through the oracle once per
# module (every row, both pool layouts compare against the same reference).
_LARGE = {}


def _large(name):
    if name not in _LARGE:
        w = wl.make_workload(name)
        _LARGE[name] = (w, oracle.fork_attn_decode(w))
    return _LARGE[name]


@pytest.mark.parametrize("layout", ["rows", "tiled"])
@pytest.mark.parametrize("name", ["long_p32k_f16", "ragged_t8"])
def test_large_workload_every_row(name, layout):
    """The long trace (16 forks of a 32k prefix: 1,024 rows) and the ragged
    multi-trace batch (8 traces, 61 forks: 3,904 rows) compared element by
    element on every (fork, head) row, in both pool layouts.  These are the
    plans where the prefix of a trace is cut over many CTAs and the suffixes
    of many forks are packed beside it."""
    w, (o_ref, lse_ref) = _large(name)
    kv = _lib.KV_TILED if layout == "tiled" else _lib.KV_ROWS
    o, lse, _ = _gpu(w, kv)
    assert o.shape == o_ref.shape
    _compare(o, lse, o_ref, lse_ref, f"{name}/{layout}")


def _fuzz_spec(rng, page_size, dqk, G, hkv):
    B = page_size
    edge = [0, 1, B - 1, B, B + 1, 3 * B + 5]
    return wl.WorkloadSpec(
        name="fuzz", num_traces=int(rng.integers(1, 4)),
        prefix_len=tuple(sorted(int(x) for x in rng.choice(edge + [200, 700], 2))),
        forks=(1, int(rng.integers(1, 6))),
        suffix_len=tuple(sorted(int(x) for x in rng.choice(edge + [130], 2))),
        hq=G * hkv, hkv=hkv, dqk=dqk, dv=dqk, page_size=B, seed=int(rng.integers(1 << 30)))


@pytest.mark.parametrize("case", range(12))
def test_fuzz_small_shapes(case):
    rng = np.random.default_rng(1000 + case)
    page_size = [16, 64][case % 2]
    dqk = [64, 128][(case // 2) % 2]
    G = [1, 4, 8, 16][case % 4]
    hkv = [1, 2, 3][case % 3]
    w = wl.make_workload(_fuzz_spec(rng, page_size, dqk, G, hkv))
    o, lse, _ = _gpu(w)
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, f"fuzz{case}")


EDGE_SPECS = {
    # the largest row tile: one fork's 128 query heads on one kv head
    "g128_d128": dict(num_traces=1, prefix_len=(3001, 3001), forks=(3, 3), suffix_len=(0, 700),
                      hq=128, hkv=1, dqk=128, dv=128),
    "g64_d64": dict(num_traces=2, prefix_len=(17, 1500), forks=(1, 4), suffix_len=(1, 300),
                    hq=128, hkv=2, dqk=64, dv=64),
    # many forks of one trace: three prefix row groups of 16, 16 and 8 forks
    "forks40": dict(num_traces=1, prefix_len=(2000, 2000), forks=(40, 40), suffix_len=(0, 200),
                    hq=8, hkv=1, dqk=128, dv=128),
    # G = 2: 64 forks per prefix item, 70 forks
    "g2_forks70": dict(num_traces=1, prefix_len=(900, 900), forks=(70, 70), suffix_len=(5, 60),
                       hq=4, hkv=2, dqk=128, dv=128),
    # a 64k-token prefix (512 tiles per kv head, cut over many CTAs)
    "prefix64k": dict(num_traces=1, prefix_len=(65543, 65543), forks=(2, 2), suffix_len=(1, 33),
                      hq=16, hkv=2, dqk=128, dv=128),
}


@pytest.mark.parametrize("name", list(EDGE_SPECS))
def test_edge_sizes_against_oracle(name):
    """Row tiles of 128 heads, many forks per trace and long prefixes, every row."""
    spec = wl.WorkloadSpec(name=name, page_size=16, seed=77, **EDGE_SPECS[name])
    w = wl.make_workload(spec)
    o, lse, _ = _gpu(w)
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, name)


@pytest.mark.parametrize("name", ["tiny_p512_f4", "fork_p8k_f8"])
def test_tiled_layout_workload_full(name):
    """K/V pools in the 8x8-tiled layout (one bulk copy per page and head)."""
    w = wl.make_workload(name)
    o, lse, _ = _gpu(w, _lib.KV_TILED)
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, name + "/tiled")


@pytest.mark.parametrize("case", [0, 2, 4, 6, 8, 10])
def test_tiled_layout_fuzz(case):
    """The page-16 fuzz shapes (ragged tails, empty sequences, G 1..16) in the tiled layout."""
    rng = np.random.default_rng(1000 + case)
    dqk = [64, 128][(case // 2) % 2]
    G = [1, 4, 8, 16][case % 4]
    hkv = [1, 2, 3][case % 3]
    w = wl.make_workload(_fuzz_spec(rng, 16, dqk, G, hkv))
    o, lse, _ = _gpu(w, _lib.KV_TILED)
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, f"tiled fuzz{case}")


def test_tiled_invalid_page_id_is_reported_not_read():
    w = dict(wl.make_workload("tiny_p512_f4"))
    w["prefix_table"] = w["prefix_table"].copy()
    w["prefix_table"][5] = w["num_pages"] + 3
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    fd = ForkDecode(w, kv_layout=_lib.KV_TILED)
    fd.decode()
    o, lse = fd.results()
    assert fd.status() == _lib.SPECGEN_ERR_INDEX
    assert np.all(np.isfinite(o))


def test_empty_prefix_and_suffix_edges():
    spec = wl.WorkloadSpec(name="edges", num_traces=3, prefix_len=(0, 40), forks=(2, 4),
                           suffix_len=(0, 2), hq=8, hkv=2, dqk=128, dv=128, page_size=16,
                           seed=77)
    w = wl.make_workload(spec)
    w["prefix_lens"][0] = 0          # trace 0: no prefix (its forks see only their suffix)
    w["suffix_lens"][:] = [0 if i % 2 == 0 else x for i, x in enumerate(w["suffix_lens"])]
    w["suffix_lens"][w["fork_offsets"][0]] = 0   # a fork with nothing at all: O = 0, LSE = -inf
    o, lse, _ = _gpu(w)
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, "edges")
    assert np.all(lse[0] == -np.inf) and np.all(o[0] == 0)


def test_latent_small_against_oracle():
    spec = wl.WorkloadSpec(name="mla_small", num_traces=2, prefix_len=(60, 300), forks=(1, 3),
                           suffix_len=(0, 130), hq=128, hkv=1, dqk=576, dv=512, page_size=64,
                           separate_v=False, seed=5)
    w = wl.make_workload(spec)
    o, lse, _ = _gpu(w)
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(o, lse, o_ref, lse_ref, "mla_small")


def test_page_placement_is_bit_exact():
    w = wl.make_workload("fork_p8k_f8")
    o1, l1, _ = _gpu(w)
    perm = np.random.default_rng(9).permutation(w["num_pages"]).astype(np.int32)
    w2 = dict(w)
    for key in ("k_pages", "v_pages"):
        pool = np.empty_like(w[key])
        pool[perm] = w[key]
        w2[key] = pool
    w2["prefix_table"] = perm[w["prefix_table"]]
    w2["suffix_table"] = perm[w["suffix_table"]]
    o2, l2, _ = _gpu(w2)
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2)


def test_invalid_page_id_is_reported_not_read():
    w = wl.make_workload("tiny_p512_f4")
    w = dict(w)
    w["suffix_table"] = w["suffix_table"].copy()
    w["suffix_table"][0] = w["num_pages"] + 7
    w["prefix_table"] = w["prefix_table"].copy()
    w["prefix_table"][3] = -2
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    fd = ForkDecode(w)
    fd.decode()
    o, lse = fd.results()
    assert fd.status() == _lib.SPECGEN_ERR_INDEX
    assert np.all(np.isfinite(o))


def _pack_device(tensors):
    """One device buffer holding copies of `tensors` (256-byte aligned views) and
    a pinned host twin: (device bytes, host bytes, views)."""
    import torch
    offs, n = [], 0
    for t in tensors:
        offs.append(n)
        n = (n + t.numel() * t.element_size() + 255) // 256 * 256
    dbuf = torch.empty(n, dtype=torch.uint8, device="cuda")
    views = []
    for t, o in zip(tensors, offs):
        v = dbuf[o:o + t.numel() * t.element_size()].view(t.dtype).view(t.shape)
        v.copy_(t)
        views.append(v)
    hbuf = torch.empty(n, dtype=torch.uint8).pin_memory()
    hbuf.copy_(dbuf)
    return dbuf, hbuf, views, offs


@pytest.mark.parametrize("name", ["tiny_p512_f4", "fork_p8k_f8"])
def test_staged_decode_from_host_buffers(name):
    """specgen_fork_attn_decode_staged: the step's inputs arrive only through its
    host->device copy (the device copy is wiped first), and its outputs, read
    from the pinned host buffer, equal the plain call's bits, call after call."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = wl.make_workload(name)
    fd = ForkDecode(w)
    fd.decode()
    o_ref, l_ref = fd.results()
    din, hin, (fd.q, fd.prefix_table, fd.prefix_off, fd.suffix_table, fd.suffix_off), _ = \
        _pack_device([fd.q, fd.prefix_table, fd.prefix_off, fd.suffix_table, fd.suffix_off])
    dout, hout, (fd.out, fd.lse), ooff = _pack_device([fd.out, fd.lse])
    F, hq, dv = w["total_forks"], w["hq"], w["dv"]
    for _ in range(2):
        din.zero_()
        dout.zero_()
        hout.zero_()
        torch.cuda.synchronize()
        _lib.specgen_fork_attn_decode_staged(fd.args(), fd.lens, hin, din, din.numel(), dout, hout,
                                             dout.numel())
        torch.cuda.synchronize()
        o = hout[ooff[0]:ooff[0] + F * hq * dv * 2].view(torch.bfloat16).float().numpy()
        lse = hout[ooff[1]:ooff[1] + F * hq * 4].view(torch.float32).numpy()
        assert np.array_equal(o.astype(np.float64).reshape(F, hq, dv), o_ref)
        assert np.array_equal(lse.astype(np.float64).reshape(F, hq), l_ref)
    assert fd.status() == _lib.SPECGEN_OK


def test_staged_calls_queued_back_to_back():
    """Ten staged calls on one stream with no host synchronisation in between,
    each with other suffix lengths and its own pinned output buffer.  That is
    more calls than the library's page-locked plan staging ring has slots, so
    slots are written again behind queued copies; every call must still see
    its own plan (element-wise against the oracle at its lengths)."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = wl.make_workload("tiny_p512_f4")
    fd = ForkDecode(w)
    base = np.asarray(w["suffix_lens"], dtype=np.int32)
    din, hin, (fd.q, fd.prefix_table, fd.prefix_off, fd.suffix_table, fd.suffix_off), _ = \
        _pack_device([fd.q, fd.prefix_table, fd.prefix_off, fd.suffix_table, fd.suffix_off])
    dout, _, (fd.out, fd.lse), ooff = _pack_device([fd.out, fd.lse])
    F, hq, dv = w["total_forks"], w["hq"], w["dv"]
    stream = torch.cuda.current_stream().cuda_stream
    torch.cuda.synchronize()
    houts, cuts = [], []
    for i in range(10):
        cut = np.maximum(base - (i * 7) % 19 - np.arange(len(base)) * (i % 4), 0).astype(np.int32)
        fd.set_suffix_lens(cut)
        hout = torch.zeros(dout.numel(), dtype=torch.uint8).pin_memory()
        _lib.specgen_fork_attn_decode_staged(fd.args(), fd.lens, hin, din, din.numel(), dout,
                                             hout, dout.numel(), stream)
        houts.append(hout)
        cuts.append(cut)
    torch.cuda.synchronize()
    assert fd.status() == _lib.SPECGEN_OK
    for cut, hout in zip(cuts, houts):
        o = hout[ooff[0]:ooff[0] + F * hq * dv * 2].view(torch.bfloat16).float().numpy()
        lse = hout[ooff[1]:ooff[1] + F * hq * 4].view(torch.float32).numpy()
        wc = dict(w)
        wc["suffix_lens"] = cut
        o_ref, lse_ref = oracle.fork_attn_decode(wc)
        _compare(o.astype(np.float64).reshape(F, hq, dv), lse.astype(np.float64).reshape(F, hq),
                 o_ref, lse_ref, f"staged cut {cut.tolist()}")


def _inline_buffers(fd, extra):
    """The step's packed inputs with `extra` bytes of room after them (for the
    plan region), on the device and in a pinned host twin."""
    import torch
    din, hin, views, _ = _pack_device([fd.q, fd.prefix_table, fd.prefix_off, fd.suffix_table,
                                       fd.suffix_off])
    in_bytes = din.numel()
    r = (in_bytes + 255) // 256 * 256
    d2 = torch.zeros(r + extra, dtype=torch.uint8, device="cuda")
    d2[:in_bytes].copy_(din)
    h2 = torch.zeros(r + extra, dtype=torch.uint8).pin_memory()
    h2[:in_bytes].copy_(hin)
    # views into the new device buffer at the same offsets
    out = []
    for v in views:
        o = v.data_ptr() - din.data_ptr()
        n = v.numel() * v.element_size()
        out.append(d2[o:o + n].view(v.dtype).view(v.shape))
    return d2, h2, in_bytes, r, out


@pytest.mark.parametrize("name", ["tiny_p512_f4", "fork_p8k_f8", "ragged_t8"])
def test_staged_inline_decode_from_host_buffers(name):
    """specgen_fork_attn_decode_staged_inline on an idle stream (the inputs go up
    at once, the plan region after the planning): its outputs equal the plain
    call's bits, call after call, and its status word sits after the inputs."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = wl.make_workload(name)
    fd = ForkDecode(w)
    fd.plan()
    fd.run()
    o_ref, l_ref = fd.results()
    region = int(fd.plan_info.ws_plan_off + fd.plan_info.plan_bytes)
    din, hin, in_bytes, r, views = _inline_buffers(fd, region + 4096)
    fd.q, fd.prefix_table, fd.prefix_off, fd.suffix_table, fd.suffix_off = views
    dout, hout, (fd.out, fd.lse), ooff = _pack_device([fd.out, fd.lse])
    F, hq, dv = w["total_forks"], w["hq"], w["dv"]
    for _ in range(2):
        din.zero_()
        dout.zero_()
        hout.zero_()
        torch.cuda.synchronize()
        _lib.specgen_fork_attn_decode_staged_inline(fd.args(), fd.lens, hin, din, in_bytes,
                                                    din.numel(), dout, hout, dout.numel())
        torch.cuda.synchronize()
        o = hout[ooff[0]:ooff[0] + F * hq * dv * 2].view(torch.bfloat16).float().numpy()
        lse = hout[ooff[1]:ooff[1] + F * hq * 4].view(torch.float32).numpy()
        assert np.array_equal(o.astype(np.float64).reshape(F, hq, dv), o_ref)
        assert np.array_equal(lse.astype(np.float64).reshape(F, hq), l_ref)
        assert _lib.specgen_workspace_status(din[r:]) == _lib.SPECGEN_OK
        # the plan region went up with the inputs
        assert np.array_equal(din[r:r + region].cpu().numpy(), hin[r:r + region].numpy())


def test_staged_inline_calls_queued_back_to_back():
    """Ten staged calls with the plan in the input buffers, queued without a host
    synchronisation (the stream is busy, so inputs and plan go up in one copy),
    each with other suffix lengths, its own pinned input buffer (the call writes
    its plan there) and its own output buffer: every call sees its own plan."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = wl.make_workload("tiny_p512_f4")
    fd = ForkDecode(w)
    fd.plan()
    region = int(fd.plan_info.ws_plan_off + fd.plan_info.plan_bytes)
    din, hin0, in_bytes, r, views = _inline_buffers(fd, region + 4096)
    fd.q, fd.prefix_table, fd.prefix_off, fd.suffix_table, fd.suffix_off = views
    dout, _, (fd.out, fd.lse), ooff = _pack_device([fd.out, fd.lse])
    F, hq, dv = w["total_forks"], w["hq"], w["dv"]
    base = np.asarray(w["suffix_lens"], dtype=np.int32)
    stream = torch.cuda.current_stream().cuda_stream
    torch.cuda.synchronize()
    houts, cuts, hins = [], [], []
    for i in range(10):
        cut = np.maximum(base - (i * 5) % 13 - np.arange(len(base)) * (i % 3), 0).astype(np.int32)
        fd.set_suffix_lens(cut)
        hin = torch.zeros_like(hin0).pin_memory()
        hin[:in_bytes].copy_(hin0[:in_bytes])
        hout = torch.zeros(dout.numel(), dtype=torch.uint8).pin_memory()
        _lib.specgen_fork_attn_decode_staged_inline(fd.args(), fd.lens, hin, din, in_bytes,
                                                    din.numel(), dout, hout, dout.numel(), stream)
        hins.append(hin)
        houts.append(hout)
        cuts.append(cut)
    torch.cuda.synchronize()
    assert _lib.specgen_workspace_status(din[r:]) == _lib.SPECGEN_OK
    for cut, hout in zip(cuts, houts):
        o = hout[ooff[0]:ooff[0] + F * hq * dv * 2].view(torch.bfloat16).float().numpy()
        lse = hout[ooff[1]:ooff[1] + F * hq * 4].view(torch.float32).numpy()
        wc = dict(w)
        wc["suffix_lens"] = cut
        o_ref, lse_ref = oracle.fork_attn_decode(wc)
        _compare(o.astype(np.float64).reshape(F, hq, dv), lse.astype(np.float64).reshape(F, hq),
                 o_ref, lse_ref, f"inline cut {cut.tolist()}")


def test_plan_once_run_many_is_deterministic():
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = wl.make_workload("fork_p8k_f8")
    fd = ForkDecode(w)
    fd.plan()
    fd.run()
    o1, l1 = fd.results()
    fd.out.zero_()
    fd.run()
    fd.run()
    o2, l2 = fd.results()
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2)


@pytest.mark.parametrize("dtype", [0, 1])
def test_lse_merge_standalone(dtype):
    import torch
    rng = np.random.default_rng(4 + dtype)
    rows, dv = 777, 128
    oa, ob = rng.standard_normal((rows, dv)), rng.standard_normal((rows, dv))
    la, lb = rng.standard_normal(rows) * 3, rng.standard_normal(rows) * 3
    la[::7] = -np.inf
    lb[::11] = -np.inf
    tdt = torch.bfloat16 if dtype == 0 else torch.float32
    t = lambda a, dt: torch.tensor(a, dtype=dt, device="cuda")
    d_oa, d_ob = t(oa, tdt), t(ob, tdt)
    d_la, d_lb = t(la, torch.float32), t(lb, torch.float32)
    d_o = torch.empty_like(d_oa)
    d_l = torch.empty_like(d_la)
    _lib.specgen_lse_merge(d_oa, d_la, d_ob, d_lb, d_o, d_l, rows, dv, dtype)
    torch.cuda.synchronize()
    # the oracle merges the same (rounded) inputs the GPU saw
    oa_in = d_oa.float().cpu().numpy().astype(np.float64)
    ob_in = d_ob.float().cpu().numpy().astype(np.float64)
    o_ref, l_ref = oracle.lse_merge(oa_in, la.astype(np.float32).astype(np.float64),
                                    ob_in, lb.astype(np.float32).astype(np.float64))
    o = d_o.float().cpu().numpy().astype(np.float64)
    lse = d_l.cpu().numpy().astype(np.float64)
    tol = TOL_O if dtype == 0 else 1e-5
    _compare(o, lse, o_ref, l_ref, "merge")
    assert np.max(np.abs(o - o_ref)) <= tol
    # in place: out aliases the a-side
    _lib.specgen_lse_merge(d_oa, d_la, d_ob, d_lb, d_oa, d_la, rows, dv, dtype)
    torch.cuda.synchronize()
    assert torch.equal(d_oa, d_o) and torch.equal(d_la, d_l)


def test_without_host_table_offsets():
    """The host copies of the block-table offsets are optional (device lookup)."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    for name in ["fork_p8k_f8", "mla_p16k_f8"]:
        w = wl.make_workload(name)
        fd = ForkDecode(w)
        lens, keep = _lib.make_host_lens(w["prefix_lens"], w["fork_offsets"], w["suffix_lens"])
        _lib.specgen_fork_attn_decode(fd.args(), lens)
        torch.cuda.synchronize()
        o, lse = fd.results()
        fd.decode()
        o2, l2 = fd.results()
        assert np.array_equal(o, o2) and np.array_equal(lse, l2)


@pytest.mark.parametrize("name", ["fork_p8k_f8", "mla_p16k_f8"])
def test_stages_equal_one_run(name):
    """run_partials then run_merge on one stream gives the bits of one run."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = wl.make_workload(name)
    fd = ForkDecode(w)
    fd.plan()
    fd.run()
    o1, l1 = fd.results()
    fd.out.zero_()
    fd.lse.zero_()
    _lib.specgen_fork_attn_run_partials(fd.args(), fd.plan_info)
    _lib.specgen_fork_attn_run_merge(fd.args(), fd.plan_info)
    torch.cuda.synchronize()
    o2, l2 = fd.results()
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2)


def test_back_to_back_plans_with_changing_lengths():
    """Twelve plan + run calls on one stream with no host synchronisation in
    between, each with different suffix lengths.  Every plan is uploaded from
    the same reused pageable host buffer (cudaMemcpyAsync stages a pageable
    source before it returns, so the next plan may overwrite it while earlier
    copies are still queued), and every call must still see its own plan."""
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = wl.make_workload("tiny_p512_f4")
    fd = ForkDecode(w)
    base = np.asarray(w["suffix_lens"], dtype=np.int32)
    outs, cuts = [], []
    stream = torch.cuda.current_stream().cuda_stream
    for i in range(12):
        cut = np.maximum(base - (i * 5) % 17 - np.arange(len(base)) * (i % 3), 0).astype(np.int32)
        fd.set_suffix_lens(cut)
        fd.plan(stream)
        fd.run(stream)
        outs.append((fd.out.clone(), fd.lse.clone()))
        cuts.append(cut)
    torch.cuda.synchronize()
    assert fd.status() == _lib.SPECGEN_OK
    for cut, (o, lse) in zip(cuts, outs):
        wc = dict(w)
        wc["suffix_lens"] = cut
        o_ref, lse_ref = oracle.fork_attn_decode(wc)
        _compare(o.float().cpu().numpy().astype(np.float64), lse.cpu().numpy().astype(np.float64),
                 o_ref, lse_ref, f"cut {cut.tolist()}")


@pytest.mark.parametrize("name,layout", [("ragged_t8", "tiled"), ("fork_p8k_f8", "rows"),
                                         ("mla_p16k_f8", "rows")])
def test_alternating_calls_sharing_a_workspace(name, layout):
    """Two calls with different queries share one workspace (plan and partials)
    and are queued back to back, five pairs between host synchronisations: each
    call's own output keeps its single-call bits.  A call whose kernels wrote
    partials while the previous call's merge still read them (the
    grid-dependency waits of the chained launches) would show here."""
    import copy
    import torch
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    w = wl.make_workload(name)
    kv = _lib.KV_TILED if layout == "tiled" else _lib.KV_ROWS
    a = ForkDecode(w, kv_layout=kv)
    b = copy.copy(a)  # the same pools, tables and workspace
    b.q = a.q.flip(0).contiguous()  # other queries: the forks' rows in reverse order
    b.out, b.lse = torch.empty_like(a.out), torch.empty_like(a.lse)
    a.plan()
    b.plan_info = a.plan_info  # the same plan, in the same workspace
    a.run()
    torch.cuda.synchronize()
    ra = (a.out.clone(), a.lse.clone())
    b.run()
    torch.cuda.synchronize()
    rb = (b.out.clone(), b.lse.clone())
    a.out.zero_()
    b.out.zero_()
    for i in range(100):
        a.run()
        b.run()
        if i % 5 == 4:
            assert torch.equal(a.out, ra[0]) and torch.equal(a.lse, ra[1]), i
            assert torch.equal(b.out, rb[0]) and torch.equal(b.lse, rb[1]), i
            a.out.zero_()
            b.out.zero_()
    assert a.status() == _lib.SPECGEN_OK
    # and the references themselves are right
    o_ref, lse_ref = oracle.fork_attn_decode(w)
    _compare(ra[0].float().cpu().numpy().astype(np.float64),
             ra[1].cpu().numpy().astype(np.float64), o_ref, lse_ref, name)
