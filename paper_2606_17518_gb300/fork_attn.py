"""Device-side fork-decode call over torch-allocated buffers.

``ForkDecode`` owns the device copies of one workload (PyTorch is used only
to allocate device memory and provide streams), builds the C-ABI argument
structs and calls ``specgen_fork_attn_plan`` / ``specgen_fork_attn_run`` /
``specgen_fork_attn_decode`` and, for multi-step decode, ``specgen_append_kv``.
It does no arithmetic of its own.
"""

from __future__ import annotations

import numpy as np

from . import _lib


def _bf16(a, device):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(device).view(torch.bfloat16)


def _i32(a, device):
    import torch
    a = np.ascontiguousarray(a, dtype=np.int32)
    if a.size == 0:                      # keep a valid (never read) pointer for empty tables
        a = np.zeros(1, dtype=np.int32)
    return torch.from_numpy(a).to(device)


class ForkDecode:
    """One workload resident on the GPU plus its output and workspace buffers."""

    def __init__(self, w: dict, device="cuda", upload_kv: bool = True,
                 kv_layout: int = _lib.KV_ROWS):
        import torch
        from . import workloads
        self.w = dict(w)  # lengths change under multi-step decode; the caller's dict does not
        self.device = torch.device(device)
        self.latent = w["v_pages"] is None
        self.kv_layout = kv_layout
        lay = (lambda a: workloads.tile_kv_pool(a)) if kv_layout == _lib.KV_TILED else (lambda a: a)
        self.q = _bf16(w["q"], device)
        self.k_pages = _bf16(lay(w["k_pages"]), device) if upload_kv else None
        self.v_pages = (None if self.latent else _bf16(lay(w["v_pages"]), device)) if upload_kv else None
        self.prefix_table = _i32(w["prefix_table"], device)
        self.prefix_off = _i32(w["prefix_bt_offsets"], device)
        self.suffix_table = _i32(w["suffix_table"], device)
        self.suffix_off = _i32(w["suffix_bt_offsets"], device)
        self.suffix_lens_dev = _i32(w["suffix_lens"], device)  # read by specgen_append_kv
        # the other device length array of an advancing append (made here, not
        # inside a graph capture)
        self._lens_alt = torch.empty_like(self.suffix_lens_dev)
        F, hq, dv = w["total_forks"], w["hq"], w["dv"]
        self.out = torch.empty((F, hq, dv), dtype=torch.bfloat16, device=device)
        self.lse = torch.empty((F, hq), dtype=torch.float32, device=device)
        self.workspace = None
        self.ws_bytes = 0
        # when True the kernels cut suffix items to suffix_lens_dev (a plan made
        # for longer host lengths then serves several decode steps)
        self.use_device_lens = False
        self.cascade = "segment_rows" in w
        self.set_suffix_lens(w["suffix_lens"])

    def set_suffix_lens(self, suffix_lens, update_device: bool = True):
        """Host suffix lengths for the next plan (the device copy is updated too,
        unless the caller advanced it on the device itself); the workspace grows
        if the new lengths need more."""
        import torch
        w = self.w
        w["suffix_lens"] = np.ascontiguousarray(suffix_lens, dtype=np.int32)
        if self.cascade:   # prefix tables are nested segments serving ranges of forks
            self.lens, self._lens_keep = _lib.make_cascade_lens(
                w["prefix_lens"], w["segment_rows"], w["suffix_lens"], w["prefix_bt_offsets"],
                w["suffix_bt_offsets"])
            need = _lib.specgen_fork_cascade_workspace_size(self.args(with_ws=False), self.lens)
        else:
            self.lens, self._lens_keep = _lib.make_host_lens(
                w["prefix_lens"], w["fork_offsets"], w["suffix_lens"], w["prefix_bt_offsets"],
                w["suffix_bt_offsets"])
            need = _lib.specgen_fork_attn_workspace_size(self.args(with_ws=False), self.lens)
        if need == 0:
            raise _lib.SpecgenError(_lib.SPECGEN_ERR_SHAPE, "specgen_fork_attn_workspace_size")
        if need > self.ws_bytes:
            self.ws_bytes = need
            self.workspace = torch.zeros(need, dtype=torch.uint8, device=self.device)
        if update_device and self.suffix_lens_dev is not None and w["total_forks"] > 0:
            self.suffix_lens_dev.copy_(torch.from_numpy(w["suffix_lens"]))
        self.plan_info = None

    def append_kv(self, k_new, v_new, free_pages, num_free: int, stream: int = 0,
                  advance: bool = False):
        """One decode step's K/V rows (device bf16 [F][Hkv][D]) into the suffixes,
        taking pages from ``free_pages`` (device int32); status bits go to the
        workspace status word.  Without ``advance`` the caller then advances the
        device lengths; with it the kernel writes them into a second device
        array, which becomes ``suffix_lens_dev`` (the two swap every step)."""
        w = self.w
        nxt = self._lens_alt if advance else None
        args = _lib.make_append_args(
            total_forks=w["total_forks"], hkv=w["hkv"], head_dim_qk=w["dqk"],
            head_dim_v=w["dv"], page_size=w["page_size"], num_pages=w["num_pages"],
            k_new=k_new, v_new=v_new, k_pages=self.k_pages, v_pages=self.v_pages,
            suffix_block_table=self.suffix_table, suffix_bt_offsets=self.suffix_off,
            suffix_lens=self.suffix_lens_dev, free_pages=free_pages, num_free=num_free,
            status=self.workspace, kv_layout=self.kv_layout, suffix_lens_next=nxt)
        _lib.specgen_append_kv(args, stream)
        if advance:
            self.suffix_lens_dev, self._lens_alt = self._lens_alt, self.suffix_lens_dev

    def args(self, with_ws: bool = True, **override) -> _lib.ForkAttnArgs:
        w = self.w
        kw = dict(
            num_traces=w["num_traces"], total_forks=w["total_forks"], hq=w["hq"], hkv=w["hkv"],
            head_dim_qk=w["dqk"], head_dim_v=w["dv"], page_size=w["page_size"],
            num_pages=w["num_pages"], scale=w["scale"], q=self.q, k_pages=self.k_pages,
            v_pages=self.v_pages, prefix_block_table=self.prefix_table,
            prefix_bt_offsets=self.prefix_off, suffix_block_table=self.suffix_table,
            suffix_bt_offsets=self.suffix_off, out=self.out, lse=self.lse,
            workspace=self.workspace if with_ws else None,
            workspace_bytes=self.ws_bytes if with_ws else 0, kv_layout=self.kv_layout,
            suffix_lens=self.suffix_lens_dev if self.use_device_lens else None)
        kw.update(override)
        return _lib.make_args(**kw)

    def plan(self, stream: int = 0):
        planner = _lib.specgen_fork_cascade_plan if self.cascade else _lib.specgen_fork_attn_plan
        self.plan_info = planner(self.args(), self.lens, stream)
        return self.plan_info

    def run(self, stream: int = 0):
        if self.plan_info is None:
            self.plan(stream)
        _lib.specgen_fork_attn_run(self.args(), self.plan_info, stream)

    def decode(self, stream: int = 0):
        if self.cascade:
            self.plan(stream)
            self.run(stream)
            return
        _lib.specgen_fork_attn_decode(self.args(), self.lens, stream)

    def status(self, stream: int = 0) -> int:
        return _lib.specgen_workspace_status(self.workspace, stream)

    def results(self):
        """(O as float64 numpy [F, hq, dv], LSE as float64 numpy [F, hq])."""
        import torch
        torch.cuda.synchronize(self.device)
        return (self.out.float().cpu().numpy().astype(np.float64),
                self.lse.cpu().numpy().astype(np.float64))


class ForkPrefill:
    """Causal prefill of every fork's newest suffix tokens (one query row per
    chunk token) through ``specgen_fork_prefill_plan`` + ``specgen_fork_attn_run``.

    ``w`` is a workload whose suffix lengths already count the chunk, plus
    ``chunk_lens`` and ``q_rows`` (see ``workloads.make_prefill``).
    """

    def __init__(self, w: dict, device="cuda", kv_layout: int = _lib.KV_ROWS):
        import torch
        from . import workloads
        self.w = w
        self.device = torch.device(device)
        self.kv_layout = kv_layout
        lay = (lambda a: workloads.tile_kv_pool(a)) if kv_layout == _lib.KV_TILED else (lambda a: a)
        self.latent = w["v_pages"] is None
        self.q = _bf16(w["q_rows"], device)
        self.k_pages = _bf16(lay(w["k_pages"]), device)
        self.v_pages = None if self.latent else _bf16(lay(w["v_pages"]), device)
        self.prefix_table = _i32(w["prefix_table"], device)
        self.prefix_off = _i32(w["prefix_bt_offsets"], device)
        self.suffix_table = _i32(w["suffix_table"], device)
        self.suffix_off = _i32(w["suffix_bt_offsets"], device)
        R, hq, dv = w["rows"], w["hq"], w["dv"]
        self.out = torch.empty((R, hq, dv), dtype=torch.bfloat16, device=device)
        self.lse = torch.empty((R, hq), dtype=torch.float32, device=device)
        before = (w["suffix_lens"] - w["chunk_lens"]).astype(np.int32)
        self.lens, self._keep = _lib.make_prefill_lens(
            w["prefix_lens"], w["fork_offsets"], before, w["chunk_lens"],
            w["prefix_bt_offsets"], w["suffix_bt_offsets"])
        self.workspace, self.ws_bytes = None, 0
        self.ws_bytes = _lib.specgen_fork_prefill_workspace_size(self.args(with_ws=False),
                                                                 self.lens)
        if self.ws_bytes == 0:
            raise _lib.SpecgenError(_lib.SPECGEN_ERR_SHAPE, "specgen_fork_prefill_workspace_size")
        self.workspace = torch.zeros(self.ws_bytes, dtype=torch.uint8, device=device)
        self.plan_info = None

    def args(self, with_ws: bool = True) -> _lib.ForkAttnArgs:
        w = self.w
        return _lib.make_args(
            num_traces=w["num_traces"], total_forks=w["rows"], hq=w["hq"], hkv=w["hkv"],
            head_dim_qk=w["dqk"], head_dim_v=w["dv"], page_size=w["page_size"],
            num_pages=w["num_pages"], scale=w["scale"], q=self.q, k_pages=self.k_pages,
            v_pages=self.v_pages, prefix_block_table=self.prefix_table,
            prefix_bt_offsets=self.prefix_off, suffix_block_table=self.suffix_table,
            suffix_bt_offsets=self.suffix_off, out=self.out, lse=self.lse,
            workspace=self.workspace if with_ws else None,
            workspace_bytes=self.ws_bytes if with_ws else 0, kv_layout=self.kv_layout)

    def plan(self, stream: int = 0):
        self.plan_info = _lib.specgen_fork_prefill_plan(self.args(), self.lens, stream)
        return self.plan_info

    def run(self, stream: int = 0):
        if self.plan_info is None:
            self.plan(stream)
        _lib.specgen_fork_attn_run(self.args(), self.plan_info, stream)

    def status(self, stream: int = 0) -> int:
        return _lib.specgen_workspace_status(self.workspace, stream)

    def results(self):
        import torch
        torch.cuda.synchronize(self.device)
        return (self.out.float().cpu().numpy().astype(np.float64),
                self.lse.cpu().numpy().astype(np.float64))
