"""C-ABI checks that need no GPU: the library loads, exports every entry point
declared in include/specgen.h, and rejects bad arguments with status codes
before touching the device."""

import ctypes as C
import os
import re

import numpy as np
import pytest

import __graft_entry__
from paper_2606_17518_gb300 import _lib, workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    __graft_entry__.build()


def _declared():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(specgen_\w+)\s*\(", src))
    return names


def test_exports_every_declared_symbol():
    lib = _lib.load()
    declared = _declared()
    assert declared >= set(_lib.EXPORTED), declared
    for name in declared:
        assert hasattr(lib, name), name


def test_status_strings():
    for code in range(0, -8, -1):
        s = _lib.status_string(code)
        assert s and s != "unknown status"
    assert _lib.status_string(-99) == "unknown status"
    assert _lib.specgen_version() >= 100


def _fake_args(w, **kw):
    # non-null fake device pointers: the checks below fail before any CUDA call
    fake = 0x10000
    base = dict(num_traces=w["num_traces"], total_forks=w["total_forks"], hq=w["hq"],
                hkv=w["hkv"], head_dim_qk=w["dqk"], head_dim_v=w["dv"],
                page_size=w["page_size"], num_pages=w["num_pages"], scale=w["scale"])
    args = _lib.ForkAttnArgs(*[int(base[k]) if k != "scale" else float(base[k])
                               for k in ("num_traces", "total_forks", "hq", "hkv",
                                         "head_dim_qk", "head_dim_v", "page_size",
                                         "num_pages", "scale")])
    for name in ("q", "k_pages", "v_pages", "prefix_block_table", "prefix_bt_offsets",
                 "suffix_block_table", "suffix_bt_offsets", "out", "lse", "workspace"):
        setattr(args, name, fake)
    if w["v_pages"] is None:
        args.v_pages = None
    args.workspace_bytes = 1 << 40
    for k, v in kw.items():
        setattr(args, k, v)
    return args


def _lens(w, **kw):
    arrs = dict(prefix_lens=w["prefix_lens"], fork_offsets=w["fork_offsets"],
                suffix_lens=w["suffix_lens"])
    arrs.update(kw)
    return _lib.make_host_lens(arrs["prefix_lens"], arrs["fork_offsets"], arrs["suffix_lens"])


def _plan_status(args, lens):
    plan = _lib.Plan()
    return _lib.load().specgen_fork_attn_plan(C.byref(args), C.byref(lens), C.byref(plan), None)


@pytest.fixture(scope="module")
def w():
    return wl.make_workload("tiny_p512_f4")


def test_workspace_size_positive_and_monotone(w):
    lens, keep = _lens(w)
    n = _lib.specgen_fork_attn_workspace_size(_fake_args(w), lens)
    assert n > 0 and n % 256 == 0
    lens2, keep2 = _lens(w, suffix_lens=w["suffix_lens"] * 40)
    assert _lib.specgen_fork_attn_workspace_size(_fake_args(w), lens2) >= n


@pytest.mark.parametrize("name", wl.WORKLOAD_ORDER)
def test_workspace_size_all_workloads(name):
    spec = wl.WORKLOADS[name]
    # sizes only: build a length-only workload without drawing the pools
    rng = np.random.default_rng(0)
    T = spec.num_traces
    pl = rng.integers(spec.prefix_len[0], spec.prefix_len[1] + 1, T).astype(np.int32)
    fk = rng.integers(spec.forks[0], spec.forks[1] + 1, T)
    fo = np.concatenate([[0], np.cumsum(fk)]).astype(np.int32)
    sl = rng.integers(spec.suffix_len[0], spec.suffix_len[1] + 1, int(fo[-1])).astype(np.int32)
    w = dict(num_traces=T, total_forks=int(fo[-1]), hq=spec.hq, hkv=spec.hkv, dqk=spec.dqk,
             dv=spec.dv, page_size=spec.page_size, num_pages=1000, scale=spec.scale,
             v_pages=(None if not spec.separate_v else 1), prefix_lens=pl, fork_offsets=fo,
             suffix_lens=sl)
    lens, keep = _lens(w)
    n = _lib.specgen_fork_attn_workspace_size(_fake_args(w), lens)
    assert 0 < n < (1 << 31)


def test_shape_errors(w):
    lens, keep = _lens(w)
    S = _lib
    assert _plan_status(_fake_args(w, hq=7), lens) == S.SPECGEN_ERR_SHAPE          # hq % hkv
    assert _plan_status(_fake_args(w, num_traces=0), lens) == S.SPECGEN_ERR_SHAPE
    assert _plan_status(_fake_args(w, head_dim_qk=96, head_dim_v=96), lens) == \
        S.SPECGEN_ERR_UNSUPPORTED
    assert _plan_status(_fake_args(w, page_size=12), lens) == S.SPECGEN_ERR_UNSUPPORTED
    assert _plan_status(_fake_args(w, scale=float("nan")), lens) == S.SPECGEN_ERR_SHAPE
    assert _plan_status(_fake_args(w, scale=-0.125), lens) == S.SPECGEN_ERR_SHAPE
    bad, k1 = _lens(w, suffix_lens=np.array([1, -1, 2, 3], dtype=np.int32))
    assert _plan_status(_fake_args(w), bad) == S.SPECGEN_ERR_SHAPE
    bad, k2 = _lens(w, fork_offsets=np.array([0, 3], dtype=np.int32))              # != F
    assert _plan_status(_fake_args(w), bad) == S.SPECGEN_ERR_SHAPE
    assert _lib.specgen_fork_attn_workspace_size(_fake_args(w, hq=7), lens) == 0


def test_kv_layout_checks(w):
    lens, keep = _lens(w)
    S = _lib
    assert _plan_status(_fake_args(w, kv_layout=2), lens) == S.SPECGEN_ERR_SHAPE
    assert _plan_status(_fake_args(w, kv_layout=-1), lens) == S.SPECGEN_ERR_SHAPE
    # the tiled layout exists only on the tensor-core shapes (page 16, head dim 64/128)
    assert _plan_status(_fake_args(w, kv_layout=S.KV_TILED, page_size=64), lens) == \
        S.SPECGEN_ERR_UNSUPPORTED
    assert _plan_status(_fake_args(w, kv_layout=S.KV_TILED, head_dim_qk=256, head_dim_v=256),
                        lens) == S.SPECGEN_ERR_UNSUPPORTED
    wm = wl.make_workload(wl.WorkloadSpec(
        name="m", num_traces=1, prefix_len=(64, 64), forks=(1, 1), suffix_len=(0, 0), hq=128,
        hkv=1, dqk=576, dv=512, page_size=64, separate_v=False, seed=1))
    lm, km = _lens(wm)
    assert _plan_status(_fake_args(wm, kv_layout=S.KV_TILED), lm) == S.SPECGEN_ERR_UNSUPPORTED
    assert _lib.specgen_fork_attn_workspace_size(_fake_args(w, kv_layout=S.KV_TILED), lens) > 0


def test_tile_kv_pool_mapping():
    """The tiled pool puts (t, d) of every (page, head) block at
    ((t/8)*(D/8) + d/8)*64 + (t%8)*8 + d%8 and keeps the block in place."""
    rng = np.random.default_rng(3)
    pool = rng.integers(0, 1 << 15, (3, 2, 16, 64)).astype(np.uint16)
    tiled = wl.tile_kv_pool(pool).reshape(3, 2, -1)
    for t in range(16):
        for d in range(64):
            assert np.array_equal(tiled[:, :, ((t // 8) * 8 + d // 8) * 64 + (t % 8) * 8 + d % 8],
                                  pool[:, :, t, d])


def test_null_and_workspace_errors(w):
    lens, keep = _lens(w)
    S = _lib
    assert _plan_status(_fake_args(w, q=None), lens) == S.SPECGEN_ERR_NULL
    assert _plan_status(_fake_args(w, out=None), lens) == S.SPECGEN_ERR_NULL
    assert _plan_status(_fake_args(w, workspace=0x10010), lens) == S.SPECGEN_ERR_WORKSPACE
    # queries and pools move in 16-byte pieces and bulk copies
    assert _plan_status(_fake_args(w, q=0x10008), lens) == S.SPECGEN_ERR_SHAPE
    assert _plan_status(_fake_args(w, k_pages=0x10004), lens) == S.SPECGEN_ERR_SHAPE
    assert _plan_status(_fake_args(w, v_pages=0x10002), lens) == S.SPECGEN_ERR_SHAPE
    assert _plan_status(_fake_args(w, workspace_bytes=1024), lens) == S.SPECGEN_ERR_WORKSPACE
    plan = _lib.Plan()
    lib = _lib.load()
    assert lib.specgen_fork_attn_plan(None, C.byref(lens), C.byref(plan), None) == \
        S.SPECGEN_ERR_NULL
    assert lib.specgen_fork_attn_plan(C.byref(_fake_args(w)), C.byref(lens), None, None) == \
        S.SPECGEN_ERR_NULL
    # run with an invalid (zeroed) plan is rejected on the host
    assert lib.specgen_fork_attn_run(C.byref(_fake_args(w)), C.byref(plan), None) == \
        S.SPECGEN_ERR_SHAPE
    # the staged decode rejects a missing buffer of a non-empty copy before any copy
    staged = lib.specgen_fork_attn_decode_staged
    args = _fake_args(w)
    assert staged(C.byref(args), C.byref(lens), None, 0x10000, 64, None, None, 0, None) == \
        S.SPECGEN_ERR_NULL
    assert staged(C.byref(args), C.byref(lens), None, None, 0, 0x10000, None, 64, None) == \
        S.SPECGEN_ERR_NULL
    assert staged(None, C.byref(lens), None, None, 0, None, None, 0, None) == S.SPECGEN_ERR_NULL


def test_lse_merge_host_checks():
    lib = _lib.load()
    S = _lib
    fake = C.c_void_p(0x10000)
    assert lib.specgen_lse_merge(fake, fake, fake, fake, fake, fake, 0, 128, 0, None) == S.SPECGEN_OK
    assert lib.specgen_lse_merge(fake, fake, fake, fake, fake, fake, 4, 128, 3, None) == \
        S.SPECGEN_ERR_UNSUPPORTED
    assert lib.specgen_lse_merge(None, fake, fake, fake, fake, fake, 4, 128, 0, None) == \
        S.SPECGEN_ERR_NULL
    assert lib.specgen_lse_merge(fake, fake, fake, fake, fake, fake, -1, 128, 0, None) == \
        S.SPECGEN_ERR_SHAPE


def test_product_path_has_no_oracle_import():
    """The package never imports the oracle (it is test infrastructure)."""
    pkg = os.path.join(ROOT, "paper_2606_17518_gb300")
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if fn.endswith((".py", ".cu", ".cuh", ".h")):
                src = open(os.path.join(dirpath, fn)).read()
                assert not re.search(r"^\s*(import|from)\s+oracle\b", src, re.M), fn
                assert "oracle/" not in src, fn


def test_append_host_checks():
    S = _lib
    lib = _lib.load()
    fake = 0x10000
    base = dict(total_forks=4, hkv=2, head_dim_qk=64, head_dim_v=64, page_size=16, num_pages=10,
                k_new=fake, v_new=fake, k_pages=fake, v_pages=fake, suffix_block_table=fake,
                suffix_bt_offsets=fake, suffix_lens=fake, free_pages=fake, num_free=3)
    st = lambda **kw: lib.specgen_append_kv(C.byref(_lib.make_append_args(**{**base, **kw})), None)
    assert lib.specgen_append_kv(None, None) == S.SPECGEN_ERR_NULL
    assert st(total_forks=0) == S.SPECGEN_OK                    # nothing to do, nothing launched
    assert st(total_forks=-1) == S.SPECGEN_ERR_SHAPE
    assert st(hkv=0) == S.SPECGEN_ERR_SHAPE
    assert st(head_dim_qk=60) == S.SPECGEN_ERR_UNSUPPORTED      # rows move in 16-byte pieces
    assert st(page_size=12) == S.SPECGEN_ERR_UNSUPPORTED
    assert st(v_new=None) == S.SPECGEN_ERR_SHAPE                # value rows without a value pool
    assert st(kv_layout=7) == S.SPECGEN_ERR_SHAPE
    assert st(kv_layout=S.KV_TILED, v_pages=None, v_new=None) == S.SPECGEN_ERR_UNSUPPORTED
    assert st(suffix_lens=None) == S.SPECGEN_ERR_NULL
    assert st(free_pages=None) == S.SPECGEN_ERR_NULL
    assert st(k_new=fake + 8) == S.SPECGEN_ERR_SHAPE            # not 16-byte aligned
    assert st(suffix_lens_next=fake) == S.SPECGEN_ERR_UNSUPPORTED  # in place: races


def test_pack_host_checks():
    S = _lib
    lib = _lib.load()
    fake = 0x10000
    base = dict(hkv=8, head_dim_qk=128, head_dim_v=128, page_size=16, num_pages=100,
                k_pages=fake, v_pages=fake)
    d = lambda **kw: _lib.make_pool_desc(**{**base, **kw})
    assert _lib.specgen_packed_bytes(d(), 3) == 3 * 2 * 8 * 16 * 128 * 2
    assert _lib.specgen_packed_bytes(d(v_pages=None), 3) == 3 * 8 * 16 * 128 * 2
    assert _lib.specgen_packed_bytes(d(hkv=1, page_size=1, head_dim_qk=3, v_pages=None), 1) == 0
    assert _lib.specgen_packed_bytes(d(hkv=0), 1) == 0
    pk = lambda desc, n, table=fake, packed=fake: lib.specgen_pack_pages(
        C.byref(desc), table, n, packed, None)
    assert pk(d(), 0) == S.SPECGEN_OK                           # nothing to copy
    assert pk(d(), -1) == S.SPECGEN_ERR_SHAPE
    assert pk(d(), 2, table=None) == S.SPECGEN_ERR_NULL
    assert pk(d(), 2, packed=None) == S.SPECGEN_ERR_NULL
    assert pk(d(), 2, packed=fake + 4) == S.SPECGEN_ERR_SHAPE    # not 16-byte aligned
    assert pk(d(hkv=1, page_size=1, head_dim_qk=4, v_pages=None), 2) == S.SPECGEN_ERR_UNSUPPORTED
    assert lib.specgen_pack_pages(None, fake, 1, fake, None) == S.SPECGEN_ERR_NULL


def test_header_is_plain_c_and_links(tmp_path):
    """include/specgen.h compiles as C99 and a C program links against the
    library and calls it (host-side checks only: no device work)."""
    import os
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not found")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    src = tmp_path / "abi.c"
    src.write_text(
        '#include <stdio.h>\n#include <string.h>\n#include "specgen.h"\n'
        "int main(void) {\n"
        "  specgen_plan plan;\n"
        "  memset(&plan, 0, sizeof(plan));\n"
        "  if (specgen_fork_attn_plan(NULL, NULL, &plan, NULL) != SPECGEN_ERR_NULL) return 1;\n"
        "  if (specgen_fork_attn_decode_staged(NULL, NULL, NULL, NULL, 0, NULL, NULL, 0, NULL)\n"
        "      != SPECGEN_ERR_NULL) return 2;\n"
        '  printf("%d %s\\n", specgen_version(), specgen_status_string(SPECGEN_ERR_SHAPE));\n'
        "  return 0;\n}\n")
    exe = tmp_path / "abi"
    lib_dir = os.path.dirname(_lib.LIB_PATH)
    cmd = [gcc, "-std=c99", "-Wall", "-Werror", "-I", os.path.join(root, "include"), str(src),
           "-o", str(exe), "-L", lib_dir, "-lspecgen", "-Wl,-rpath," + lib_dir]
    res = subprocess.run(cmd, capture_output=True, text=True)
    assert res.returncode == 0, res.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert run.returncode == 0, (run.returncode, run.stderr)
    assert run.stdout.split()[0].isdigit()


def test_static_decode_refuses_oversized_calls_on_the_host():
    """The allocation-free decode refuses a call whose workspace would exceed its
    fixed scratch array before it touches the device."""
    lib = _lib.load()
    F = 2000
    pl = np.array([64], np.int32)
    fo = np.array([0, F], np.int32)
    sl = np.ones(F, np.int32)
    lens, keep = _lib.make_host_lens(pl, fo, sl)
    w = dict(num_traces=1, total_forks=F, hq=64, hkv=8, dqk=128, dv=128, page_size=16,
             num_pages=1 << 16, scale=0.088, v_pages=1, prefix_lens=pl, fork_offsets=fo,
             suffix_lens=sl)
    args = _fake_args(w)
    assert _lib.specgen_fork_attn_workspace_size(args, lens) > (16 << 20)
    assert lib.specgen_fork_attn_decode_static(C.byref(args), C.byref(lens), None) == \
        _lib.SPECGEN_ERR_WORKSPACE
    assert lib.specgen_fork_attn_decode_static(None, C.byref(lens), None) == _lib.SPECGEN_ERR_NULL


def test_static_decode_plans_once():
    """The allocation-free decode plans a call once: on a host without a GPU it
    stops at its first CUDA call (the scratch array's address), after planning,
    and takes about the host time of one plan -- not the two plans of a size
    query followed by a planning decode."""
    from conftest import cuda_available
    if cuda_available():
        pytest.skip("with a GPU the call would go on to launch kernels on the fake pointers")
    import time
    lib = _lib.load()
    rng = np.random.default_rng(0)
    T = 8  # a ragged batch: 8 traces of 4-16 forks, planning takes ~0.1 ms
    pl = rng.integers(4096, 32769, T).astype(np.int32)
    fo = np.concatenate([[0], np.cumsum(rng.integers(4, 17, T))]).astype(np.int32)
    F = int(fo[-1])
    sl = rng.integers(32, 1025, F).astype(np.int32)
    lens, keep = _lib.make_host_lens(pl, fo, sl)
    w = dict(num_traces=T, total_forks=F, hq=64, hkv=8, dqk=128, dv=128, page_size=16,
             num_pages=1 << 20, scale=0.088, v_pages=1, prefix_lens=pl, fork_offsets=fo,
             suffix_lens=sl)
    args = _fake_args(w)
    assert _lib.specgen_fork_attn_workspace_size(args, lens) <= (16 << 20)
    dst = np.zeros(1 << 22, np.uint8)
    plan = _lib.Plan()

    def one_plan():
        t = time.perf_counter()
        st = lib.specgen_fork_attn_plan_host(C.byref(args), C.byref(lens), dst.ctypes.data,
                                             dst.nbytes, C.byref(plan))
        assert st == _lib.SPECGEN_OK
        return time.perf_counter() - t

    def static_call():
        t = time.perf_counter()
        st = lib.specgen_fork_attn_decode_static(C.byref(args), C.byref(lens), None)
        assert st == _lib.SPECGEN_ERR_CUDA  # planned, then no device
        return time.perf_counter() - t

    static_call()
    t_plan = np.median([one_plan() for _ in range(300)])
    t_static = np.median([static_call() for _ in range(300)])
    assert t_static < 1.5 * t_plan, (t_static, t_plan)


def test_staged_inline_refuses_on_the_host():
    """The one-copy staged decode checks everything that can refuse the call
    (buffers, alignment, shapes, the room left for the plan region after the
    inputs) on the host, before anything is queued, and writes the plan region
    into the host buffer at the 256-byte boundary after the inputs only then."""
    lib = _lib.load()
    w = wl.make_workload("tiny_p512_f4")
    args = _fake_args(w)
    lens, keep = _lens(w)
    plan_buf = np.zeros(1 << 20, np.uint8)
    plan = _lib.specgen_fork_attn_plan_host(args, lens, plan_buf)
    region = int(plan.ws_plan_off + plan.plan_bytes)
    in_bytes = 1000
    off = 1024
    host = np.full(off + region, 7, np.uint8)
    dev = 0x100000
    call = lambda h, d, cap, **kw: lib.specgen_fork_attn_decode_staged_inline(
        C.byref(kw.get("args", args)), C.byref(lens), h, C.c_void_p(d), C.c_size_t(in_bytes),
        C.c_size_t(cap), None, None, C.c_size_t(0), None)
    hp = host.ctypes.data_as(C.c_void_p)
    assert call(None, dev, len(host)) == _lib.SPECGEN_ERR_NULL
    assert call(hp, dev + 16, len(host)) == _lib.SPECGEN_ERR_SHAPE       # dev_in not 256-aligned
    assert call(hp, dev, off + region - 1) == _lib.SPECGEN_ERR_WORKSPACE  # no room for the plan
    bad = _fake_args(w, hkv=3)
    assert call(hp, dev, len(host), args=bad) == _lib.SPECGEN_ERR_SHAPE
    assert np.all(host == 7)                                              # nothing written
