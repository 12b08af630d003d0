"""ctypes binding of the fork-decode C ABI (``include/specgen.h``).

Argument marshalling only: every step of the computation runs in the CUDA
kernels of ``libspecgen.so``.  The function names match the C entry points.
The library is built in-tree (``paper_2606_17518_gb300/build.py``); if it is
missing, loading fails loudly -- there is no fallback implementation.
"""

from __future__ import annotations

import ctypes as C
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libspecgen.so")

SPECGEN_OK = 0
SPECGEN_ERR_NULL = -1
SPECGEN_ERR_SHAPE = -2
SPECGEN_ERR_UNSUPPORTED = -3
SPECGEN_ERR_WORKSPACE = -4
SPECGEN_ERR_INDEX = -5
SPECGEN_ERR_CUDA = -6
SPECGEN_ERR_TIMEOUT = -7

EXPORTED = [
    "specgen_fork_attn_workspace_size",
    "specgen_fork_attn_plan",
    "specgen_fork_attn_plan_host",
    "specgen_fork_attn_run",
    "specgen_fork_attn_run_profiled",
    "specgen_fork_attn_run_partials",
    "specgen_fork_attn_run_merge",
    "specgen_fork_cascade_workspace_size",
    "specgen_fork_cascade_plan",
    "specgen_fork_cascade_plan_host",
    "specgen_fork_prefill_workspace_size",
    "specgen_fork_prefill_plan",
    "specgen_fork_prefill_plan_host",
    "specgen_fork_attn_decode",
    "specgen_fork_attn_decode_staged",
    "specgen_fork_attn_decode_staged_inline",
    "specgen_fork_attn_decode_static",
    "specgen_lse_merge",
    "specgen_append_kv",
    "specgen_packed_bytes",
    "specgen_pack_pages",
    "specgen_unpack_pages",
    "specgen_workspace_status",
    "specgen_static_workspace_status",
    "specgen_status_string",
    "specgen_version",
]


class ForkAttnArgs(C.Structure):
    _fields_ = [
        ("num_traces", C.c_int), ("total_forks", C.c_int), ("hq", C.c_int), ("hkv", C.c_int),
        ("head_dim_qk", C.c_int), ("head_dim_v", C.c_int), ("page_size", C.c_int),
        ("num_pages", C.c_int), ("scale", C.c_float),
        ("q", C.c_void_p), ("k_pages", C.c_void_p), ("v_pages", C.c_void_p),
        ("prefix_block_table", C.c_void_p), ("prefix_bt_offsets", C.c_void_p),
        ("suffix_block_table", C.c_void_p), ("suffix_bt_offsets", C.c_void_p),
        ("out", C.c_void_p), ("lse", C.c_void_p),
        ("workspace", C.c_void_p), ("workspace_bytes", C.c_size_t), ("kv_layout", C.c_int),
        ("suffix_lens", C.c_void_p),
    ]


KV_ROWS = 0
KV_TILED = 1


class AppendArgs(C.Structure):
    _fields_ = [
        ("total_forks", C.c_int), ("hkv", C.c_int), ("head_dim_qk", C.c_int),
        ("head_dim_v", C.c_int), ("page_size", C.c_int), ("num_pages", C.c_int),
        ("kv_layout", C.c_int),
        ("k_new", C.c_void_p), ("v_new", C.c_void_p), ("k_pages", C.c_void_p),
        ("v_pages", C.c_void_p), ("suffix_block_table", C.c_void_p),
        ("suffix_bt_offsets", C.c_void_p), ("suffix_lens", C.c_void_p),
        ("free_pages", C.c_void_p), ("num_free", C.c_int), ("status", C.c_void_p),
        ("suffix_lens_next", C.c_void_p),
    ]


class PoolDesc(C.Structure):
    _fields_ = [
        ("hkv", C.c_int), ("head_dim_qk", C.c_int), ("head_dim_v", C.c_int),
        ("page_size", C.c_int), ("num_pages", C.c_int), ("k_pages", C.c_void_p),
        ("v_pages", C.c_void_p), ("status", C.c_void_p),
    ]


class HostLens(C.Structure):
    _fields_ = [("prefix_lens", C.c_void_p), ("fork_offsets", C.c_void_p),
                ("suffix_lens", C.c_void_p), ("prefix_bt_offsets", C.c_void_p),
                ("suffix_bt_offsets", C.c_void_p)]


class PrefillLens(C.Structure):
    _fields_ = [("prefix_lens", C.c_void_p), ("fork_offsets", C.c_void_p),
                ("suffix_lens", C.c_void_p), ("chunk_lens", C.c_void_p),
                ("prefix_bt_offsets", C.c_void_p), ("suffix_bt_offsets", C.c_void_p)]


class CascadeLens(C.Structure):
    _fields_ = [("num_segments", C.c_int), ("segment_lens", C.c_void_p),
                ("segment_rows", C.c_void_p), ("suffix_lens", C.c_void_p),
                ("segment_bt_offsets", C.c_void_p), ("suffix_bt_offsets", C.c_void_p)]


class Plan(C.Structure):
    _fields_ = [
        ("valid", C.c_int32), ("n_tc_items", C.c_int32), ("n_tc_ctas", C.c_int32),
        ("n_split_items", C.c_int32), ("n_rows", C.c_int32), ("total_slots", C.c_int32),
        ("flags", C.c_int32), ("n_part_groups", C.c_int32),
        ("plan_bytes", C.c_int64), ("ws_plan_off", C.c_int64), ("ws_part_o_off", C.c_int64),
        ("ws_part_lse_off", C.c_int64), ("ws_end", C.c_int64), ("offsets", C.c_int64 * 8),
        ("n_sfx_items", C.c_int32), ("n_sfx_ctas", C.c_int32), ("sfx_offsets", C.c_int64 * 2),
    ]


class SpecgenError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} ({status})")


_lib = None


def load() -> C.CDLL:
    """Load libspecgen.so (built in-tree); raise if it is absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: run paper_2606_17518_gb300.build.build() "
                           "first (no CPU fallback exists)")
    lib = C.CDLL(LIB_PATH)
    P = C.POINTER
    lib.specgen_fork_attn_workspace_size.restype = C.c_size_t
    lib.specgen_fork_attn_workspace_size.argtypes = [P(ForkAttnArgs), P(HostLens)]
    lib.specgen_fork_attn_plan.restype = C.c_int
    lib.specgen_fork_attn_plan.argtypes = [P(ForkAttnArgs), P(HostLens), P(Plan), C.c_void_p]
    lib.specgen_fork_attn_plan_host.restype = C.c_int
    lib.specgen_fork_attn_plan_host.argtypes = [P(ForkAttnArgs), P(HostLens), C.c_void_p,
                                                C.c_size_t, P(Plan)]
    lib.specgen_fork_attn_run.restype = C.c_int
    lib.specgen_fork_attn_run.argtypes = [P(ForkAttnArgs), P(Plan), C.c_void_p]
    lib.specgen_fork_cascade_workspace_size.restype = C.c_size_t
    lib.specgen_fork_cascade_workspace_size.argtypes = [P(ForkAttnArgs), P(CascadeLens)]
    lib.specgen_fork_cascade_plan.restype = C.c_int
    lib.specgen_fork_cascade_plan.argtypes = [P(ForkAttnArgs), P(CascadeLens), P(Plan),
                                              C.c_void_p]
    lib.specgen_fork_prefill_workspace_size.restype = C.c_size_t
    lib.specgen_fork_prefill_workspace_size.argtypes = [P(ForkAttnArgs), P(PrefillLens)]
    lib.specgen_fork_prefill_plan.restype = C.c_int
    lib.specgen_fork_prefill_plan.argtypes = [P(ForkAttnArgs), P(PrefillLens), P(Plan),
                                              C.c_void_p]
    for name, lens_t in (("specgen_fork_prefill_plan_host", PrefillLens),
                         ("specgen_fork_cascade_plan_host", CascadeLens)):
        fn = getattr(lib, name)
        fn.restype = C.c_int
        fn.argtypes = [P(ForkAttnArgs), P(lens_t), C.c_void_p, C.c_size_t, P(Plan)]
    lib.specgen_append_kv.restype = C.c_int
    lib.specgen_append_kv.argtypes = [P(AppendArgs), C.c_void_p]
    lib.specgen_packed_bytes.restype = C.c_size_t
    lib.specgen_packed_bytes.argtypes = [P(PoolDesc), C.c_int]
    for name in ("specgen_pack_pages", "specgen_unpack_pages"):
        getattr(lib, name).restype = C.c_int
        getattr(lib, name).argtypes = [P(PoolDesc), C.c_void_p, C.c_int, C.c_void_p, C.c_void_p]
    for stage in ("specgen_fork_attn_run_partials", "specgen_fork_attn_run_merge"):
        getattr(lib, stage).restype = C.c_int
        getattr(lib, stage).argtypes = [P(ForkAttnArgs), P(Plan), C.c_void_p]
    lib.specgen_fork_attn_run_profiled.restype = C.c_int
    lib.specgen_fork_attn_run_profiled.argtypes = [P(ForkAttnArgs), P(Plan), C.c_void_p,
                                                   C.c_void_p, C.c_int, P(C.c_int)]
    lib.specgen_fork_attn_decode.restype = C.c_int
    lib.specgen_fork_attn_decode.argtypes = [P(ForkAttnArgs), P(HostLens), C.c_void_p]
    lib.specgen_fork_attn_decode_staged.restype = C.c_int
    lib.specgen_fork_attn_decode_staged.argtypes = [
        P(ForkAttnArgs), P(HostLens), C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p,
        C.c_void_p, C.c_size_t, C.c_void_p]
    lib.specgen_fork_attn_decode_staged_inline.restype = C.c_int
    lib.specgen_fork_attn_decode_staged_inline.argtypes = [
        P(ForkAttnArgs), P(HostLens), C.c_void_p, C.c_void_p, C.c_size_t, C.c_size_t,
        C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p]
    lib.specgen_fork_attn_decode_static.restype = C.c_int
    lib.specgen_fork_attn_decode_static.argtypes = [P(ForkAttnArgs), P(HostLens), C.c_void_p]
    lib.specgen_lse_merge.restype = C.c_int
    lib.specgen_lse_merge.argtypes = [C.c_void_p] * 6 + [C.c_int, C.c_int, C.c_int, C.c_void_p]
    lib.specgen_workspace_status.restype = C.c_int
    lib.specgen_workspace_status.argtypes = [C.c_void_p, C.c_void_p]
    lib.specgen_static_workspace_status.restype = C.c_int
    lib.specgen_static_workspace_status.argtypes = [C.c_void_p]
    lib.specgen_status_string.restype = C.c_char_p
    lib.specgen_status_string.argtypes = [C.c_int]
    lib.specgen_version.restype = C.c_int
    lib.specgen_version.argtypes = []
    _lib = lib
    return lib


def status_string(status: int) -> str:
    return load().specgen_status_string(int(status)).decode()


def _check(status: int, what: str):
    if status != SPECGEN_OK:
        raise SpecgenError(status, what)


def _ptr(t) -> int | None:
    """Data pointer of a torch tensor / numpy array (or a raw address), or None."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def make_host_lens(prefix_lens, fork_offsets, suffix_lens, prefix_bt_offsets=None,
                   suffix_bt_offsets=None):
    """HostLens over int32 numpy arrays (kept alive by the returned tuple)."""
    arrs = tuple(None if a is None else np.ascontiguousarray(a, dtype=np.int32) for a in
                 (prefix_lens, fork_offsets, suffix_lens, prefix_bt_offsets, suffix_bt_offsets))
    return HostLens(*(None if a is None else a.ctypes.data for a in arrs)), arrs


def make_args(*, num_traces, total_forks, hq, hkv, head_dim_qk, head_dim_v, page_size,
              num_pages, scale, q, k_pages, v_pages, prefix_block_table, prefix_bt_offsets,
              suffix_block_table, suffix_bt_offsets, out, lse, workspace=None,
              workspace_bytes=0, kv_layout=KV_ROWS, suffix_lens=None) -> ForkAttnArgs:
    return ForkAttnArgs(
        int(num_traces), int(total_forks), int(hq), int(hkv), int(head_dim_qk),
        int(head_dim_v), int(page_size), int(num_pages), float(scale),
        _ptr(q), _ptr(k_pages), _ptr(v_pages), _ptr(prefix_block_table),
        _ptr(prefix_bt_offsets), _ptr(suffix_block_table), _ptr(suffix_bt_offsets),
        _ptr(out), _ptr(lse), _ptr(workspace), int(workspace_bytes), int(kv_layout),
        _ptr(suffix_lens))


def make_append_args(*, total_forks, hkv, head_dim_qk, head_dim_v, page_size, num_pages,
                     k_new, v_new, k_pages, v_pages, suffix_block_table, suffix_bt_offsets,
                     suffix_lens, free_pages, num_free, status=None,
                     kv_layout=KV_ROWS, suffix_lens_next=None) -> AppendArgs:
    return AppendArgs(
        int(total_forks), int(hkv), int(head_dim_qk), int(head_dim_v), int(page_size),
        int(num_pages), int(kv_layout), _ptr(k_new), _ptr(v_new), _ptr(k_pages), _ptr(v_pages),
        _ptr(suffix_block_table), _ptr(suffix_bt_offsets), _ptr(suffix_lens), _ptr(free_pages),
        int(num_free), _ptr(status), _ptr(suffix_lens_next))


def specgen_append_kv(args: AppendArgs, stream: int = 0) -> None:
    _check(load().specgen_append_kv(C.byref(args), C.c_void_p(stream)), "specgen_append_kv")


def make_pool_desc(*, hkv, head_dim_qk, head_dim_v, page_size, num_pages, k_pages, v_pages,
                   status=None) -> PoolDesc:
    return PoolDesc(int(hkv), int(head_dim_qk), int(head_dim_v), int(page_size),
                    int(num_pages), _ptr(k_pages), _ptr(v_pages), _ptr(status))


def specgen_packed_bytes(pool: PoolDesc, n_pages: int) -> int:
    return int(load().specgen_packed_bytes(C.byref(pool), int(n_pages)))


def specgen_pack_pages(pool: PoolDesc, table, n_pages: int, packed, stream: int = 0) -> None:
    _check(load().specgen_pack_pages(C.byref(pool), _ptr(table), int(n_pages), _ptr(packed),
                                     C.c_void_p(stream)), "specgen_pack_pages")


def specgen_unpack_pages(pool: PoolDesc, table, n_pages: int, packed, stream: int = 0) -> None:
    _check(load().specgen_unpack_pages(C.byref(pool), _ptr(table), int(n_pages), _ptr(packed),
                                       C.c_void_p(stream)), "specgen_unpack_pages")


def make_prefill_lens(prefix_lens, fork_offsets, suffix_lens, chunk_lens,
                      prefix_bt_offsets=None, suffix_bt_offsets=None):
    """PrefillLens over host int32 copies; returns (struct, keepalive)."""
    keep = [np.ascontiguousarray(a, dtype=np.int32)
            for a in (prefix_lens, fork_offsets, suffix_lens, chunk_lens)]
    opt = [None if a is None else np.ascontiguousarray(a, dtype=np.int32)
           for a in (prefix_bt_offsets, suffix_bt_offsets)]
    ptrs = [a.ctypes.data for a in keep] + [None if a is None else a.ctypes.data for a in opt]
    return PrefillLens(*ptrs), keep + opt


def make_cascade_lens(segment_lens, segment_rows, suffix_lens, segment_bt_offsets=None,
                      suffix_bt_offsets=None):
    """CascadeLens over host int32 copies; returns (struct, keepalive)."""
    keep = [np.ascontiguousarray(a, dtype=np.int32)
            for a in (segment_lens, segment_rows, suffix_lens)]
    opt = [None if a is None else np.ascontiguousarray(a, dtype=np.int32)
           for a in (segment_bt_offsets, suffix_bt_offsets)]
    return CascadeLens(len(keep[0]), keep[0].ctypes.data, keep[1].ctypes.data,
                       keep[2].ctypes.data, *[None if a is None else a.ctypes.data
                                              for a in opt]), keep + opt


def specgen_fork_cascade_workspace_size(args: ForkAttnArgs, lens: CascadeLens) -> int:
    return int(load().specgen_fork_cascade_workspace_size(C.byref(args), C.byref(lens)))


def specgen_fork_cascade_plan(args: ForkAttnArgs, lens: CascadeLens, stream: int = 0) -> Plan:
    plan = Plan()
    _check(load().specgen_fork_cascade_plan(C.byref(args), C.byref(lens), C.byref(plan),
                                            C.c_void_p(stream)), "specgen_fork_cascade_plan")
    return plan


def specgen_fork_prefill_workspace_size(args: ForkAttnArgs, lens: PrefillLens) -> int:
    return int(load().specgen_fork_prefill_workspace_size(C.byref(args), C.byref(lens)))


def specgen_fork_prefill_plan(args: ForkAttnArgs, lens: PrefillLens, stream: int = 0) -> Plan:
    plan = Plan()
    _check(load().specgen_fork_prefill_plan(C.byref(args), C.byref(lens), C.byref(plan),
                                            C.c_void_p(stream)), "specgen_fork_prefill_plan")
    return plan


def specgen_fork_attn_workspace_size(args: ForkAttnArgs, lens: HostLens) -> int:
    return int(load().specgen_fork_attn_workspace_size(C.byref(args), C.byref(lens)))


def specgen_fork_attn_plan(args: ForkAttnArgs, lens: HostLens, stream: int = 0) -> Plan:
    plan = Plan()
    _check(load().specgen_fork_attn_plan(C.byref(args), C.byref(lens), C.byref(plan),
                                         C.c_void_p(stream)), "specgen_fork_attn_plan")
    return plan


def specgen_fork_attn_run(args: ForkAttnArgs, plan: Plan, stream: int = 0) -> None:
    _check(load().specgen_fork_attn_run(C.byref(args), C.byref(plan), C.c_void_p(stream)),
           "specgen_fork_attn_run")


def specgen_fork_attn_run_partials(args: ForkAttnArgs, plan: Plan, stream: int = 0) -> None:
    _check(load().specgen_fork_attn_run_partials(C.byref(args), C.byref(plan),
                                                 C.c_void_p(stream)),
           "specgen_fork_attn_run_partials")


def specgen_fork_attn_run_merge(args: ForkAttnArgs, plan: Plan, stream: int = 0) -> None:
    _check(load().specgen_fork_attn_run_merge(C.byref(args), C.byref(plan), C.c_void_p(stream)),
           "specgen_fork_attn_run_merge")


def specgen_fork_attn_run_profiled(args: ForkAttnArgs, plan: Plan, stream: int, events,
                                   n_events: int) -> int:
    """Run with timing marks; ``events`` is a ctypes void* array (or a byref into one)."""
    n = C.c_int(0)
    _check(load().specgen_fork_attn_run_profiled(C.byref(args), C.byref(plan),
                                                 C.c_void_p(stream), events, int(n_events),
                                                 C.byref(n)), "specgen_fork_attn_run_profiled")
    return n.value


def specgen_fork_attn_decode(args: ForkAttnArgs, lens: HostLens, stream: int = 0) -> None:
    _check(load().specgen_fork_attn_decode(C.byref(args), C.byref(lens), C.c_void_p(stream)),
           "specgen_fork_attn_decode")


def specgen_fork_attn_plan_host(args: ForkAttnArgs, lens: HostLens, host_dst: np.ndarray) -> Plan:
    """Plan into host memory: the plan region's bytes go to ``host_dst`` (uint8)."""
    plan = Plan()
    _check(load().specgen_fork_attn_plan_host(C.byref(args), C.byref(lens),
                                              host_dst.ctypes.data, host_dst.nbytes,
                                              C.byref(plan)),
           "specgen_fork_attn_plan_host")
    return plan


def specgen_fork_prefill_plan_host(args: ForkAttnArgs, lens, host_dst: np.ndarray) -> Plan:
    """Prefill plan into host memory (``host_dst``, uint8)."""
    plan = Plan()
    _check(load().specgen_fork_prefill_plan_host(C.byref(args), C.byref(lens),
                                                 host_dst.ctypes.data, host_dst.nbytes,
                                                 C.byref(plan)),
           "specgen_fork_prefill_plan_host")
    return plan


def specgen_fork_cascade_plan_host(args: ForkAttnArgs, lens, host_dst: np.ndarray) -> Plan:
    """Cascade plan into host memory (``host_dst``, uint8)."""
    plan = Plan()
    _check(load().specgen_fork_cascade_plan_host(C.byref(args), C.byref(lens),
                                                 host_dst.ctypes.data, host_dst.nbytes,
                                                 C.byref(plan)),
           "specgen_fork_cascade_plan_host")
    return plan


def specgen_fork_attn_decode_staged(args: ForkAttnArgs, lens: HostLens, host_in, dev_in,
                                    in_bytes: int, dev_out, host_out, out_bytes: int,
                                    stream: int = 0) -> None:
    """One decode step from host memory: copy in, plan + run, copy out (one call)."""
    _check(load().specgen_fork_attn_decode_staged(
        C.byref(args), C.byref(lens), _ptr(host_in), _ptr(dev_in), C.c_size_t(in_bytes),
        _ptr(dev_out), _ptr(host_out), C.c_size_t(out_bytes), C.c_void_p(stream)),
        "specgen_fork_attn_decode_staged")


def specgen_fork_attn_decode_staged_inline(args: ForkAttnArgs, lens: HostLens, host_in, dev_in,
                                           in_bytes: int, in_capacity: int, dev_out, host_out,
                                           out_bytes: int, stream: int = 0) -> None:
    """One decode step from host memory with the plan in the same host-to-device copy."""
    _check(load().specgen_fork_attn_decode_staged_inline(
        C.byref(args), C.byref(lens), _ptr(host_in), _ptr(dev_in), C.c_size_t(in_bytes),
        C.c_size_t(in_capacity), _ptr(dev_out), _ptr(host_out), C.c_size_t(out_bytes),
        C.c_void_p(stream)), "specgen_fork_attn_decode_staged_inline")


def specgen_fork_attn_decode_static(args: ForkAttnArgs, lens: HostLens, stream: int = 0) -> None:
    """Fork decode using the library's fixed scratch array (no workspace, no allocation)."""
    _check(load().specgen_fork_attn_decode_static(C.byref(args), C.byref(lens),
                                                  C.c_void_p(stream)),
           "specgen_fork_attn_decode_static")


def specgen_lse_merge(out_a, lse_a, out_b, lse_b, out, lse, rows: int, dv: int, dtype: int,
                      stream: int = 0) -> None:
    _check(load().specgen_lse_merge(_ptr(out_a), _ptr(lse_a), _ptr(out_b), _ptr(lse_b),
                                    _ptr(out), _ptr(lse), int(rows), int(dv), int(dtype),
                                    C.c_void_p(stream)), "specgen_lse_merge")


def specgen_workspace_status(workspace, stream: int = 0) -> int:
    return int(load().specgen_workspace_status(_ptr(workspace), C.c_void_p(stream)))


def specgen_static_workspace_status(stream: int = 0) -> int:
    """Status word of the scratch array used by specgen_fork_attn_decode_static."""
    return int(load().specgen_static_workspace_status(C.c_void_p(stream)))


def specgen_version() -> int:
    return int(load().specgen_version())
