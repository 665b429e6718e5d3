"""Thin Python binding of ``include/mpt.h`` (the exact MPT solver on GB300).

Argument marshalling only: every step of a solve runs in the CUDA kernels of
``libmpt.so``.  PyTorch supplies device memory (the workspace) and the
current stream.  The functions carry the C names; :func:`solve` strings them
together for the common case.

The library must have been built (``paper_2609_13692_gb300.build.build()``);
there is no fallback: loading fails loudly if it is missing.
"""

from __future__ import annotations

import ctypes
import os
import itertools
from dataclasses import dataclass
from pathlib import Path
from typing import Optional

import numpy as np

from . import build as _build

MPT_OK = 0
MPT_DP_AUTO, MPT_DP_BLOCKED, MPT_DP_GENERAL, MPT_DP_WIDE = 0, 1, 2, 3
_MODES = {"auto": MPT_DP_AUTO, "blocked": MPT_DP_BLOCKED, "general": MPT_DP_GENERAL, "wide": MPT_DP_WIDE}

STATUS_NAMES = {
    0: "MPT_OK",
    1: "MPT_ERR_INVALID_ARG",
    2: "MPT_ERR_TOO_LARGE",
    3: "MPT_ERR_OVERFLOW",
    4: "MPT_ERR_OUT_OF_MEMORY",
    5: "MPT_ERR_WORKSPACE_TOO_SMALL",
    6: "MPT_ERR_CUDA",
    7: "MPT_ERR_NOT_SOLVED",
    8: "MPT_ERR_TIMEOUT",
    9: "MPT_ERR_INTERNAL",
}

EXPORTED = [
    "mpt_create", "mpt_workspace_bytes", "mpt_set_dp_mode", "mpt_solve", "mpt_tables", "mpt_layout_size",
    "mpt_layout", "mpt_trie_cost", "mpt_set_profiling", "mpt_get_profile", "mpt_destroy", "mpt_status_string",
    "mpt_last_error", "mpt_solve_noalloc", "mpt_batch_create", "mpt_batch_workspace_bytes", "mpt_batch_solve",
    "mpt_batch_results", "mpt_batch_tables", "mpt_batch_destroy", "mpt_greedy", "mpt_serve_order",
    "mpt_cache_costs", "mpt_layout_pinned", "mpt_solve_steps", "mpt_solve_begin", "mpt_solve_layers",
    "mpt_solve_end", "mpt_solve_resume", "mpt_set_tables", "mpt_tables32", "mpt_gather_bandwidth",
    "mpt_alu_addmin_peak", "mpt_build_info",
]


class MPTError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str = ""):
        self.status = status
        name = STATUS_NAMES.get(status, str(status))
        super().__init__(f"{where}: {name}" + (f" ({detail})" if detail else ""))


class mpt_profile(ctypes.Structure):
    _fields_ = [
        ("ms_h2d", ctypes.c_double),
        ("ms_scatter", ctypes.c_double),
        ("ms_zeta", ctypes.c_double),
        ("ms_dp_pairs", ctypes.c_double),
        ("ms_dp_tiles", ctypes.c_double),
        ("ms_dp_general", ctypes.c_double),
        ("ms_walk", ctypes.c_double),
        ("ms_d2h", ctypes.c_double),
        ("splits_pairs", ctypes.c_double),
        ("splits_total", ctypes.c_double),
        ("launches_pairs", ctypes.c_int64),
        ("launches_total", ctypes.c_int64),
        ("dp_mode", ctypes.c_int32),
        ("tile_bits", ctypes.c_int32),
    ]

    def as_dict(self) -> dict:
        return {name: getattr(self, name) for name, _ in self._fields_}


_LIB = None


def library_path() -> str:
    """The in-tree libmpt.so, or the build named by MPT_LIBRARY (for instance
    the bounds-checked one from build(bounds=True))."""
    return os.environ.get("MPT_LIBRARY") or str(_build.LIB)


def load() -> ctypes.CDLL:
    """Load libmpt.so (built in-tree); raises if it has not been built."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = Path(library_path())
    if not path.exists():
        raise RuntimeError(f"{path} is missing: build the CUDA library first "
                           "(python -c 'import __graft_entry__ as g; g.build()')")
    lib = ctypes.CDLL(str(path))
    vp, i64, i32, sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_size_t
    i64p = ctypes.POINTER(ctypes.c_int64)
    u64p = ctypes.POINTER(ctypes.c_uint64)
    i32p = ctypes.POINTER(ctypes.c_int32)
    sig = {
        "mpt_create": ([i64p, i64, u64p, i32, ctypes.POINTER(vp)], ctypes.c_int),
        "mpt_workspace_bytes": ([vp, ctypes.POINTER(sz)], ctypes.c_int),
        "mpt_set_dp_mode": ([vp, i32], ctypes.c_int),
        "mpt_solve": ([vp, vp, sz, vp, i64p], ctypes.c_int),
        "mpt_tables": ([vp, ctypes.POINTER(vp), ctypes.POINTER(vp), ctypes.POINTER(vp)], ctypes.c_int),
        "mpt_layout_size": ([vp, i64p], ctypes.c_int),
        "mpt_layout": ([vp, i64p, i64p, i32p], ctypes.c_int),
        "mpt_trie_cost": ([i64p, i64, i32, i64p, i64p, i64p], ctypes.c_int),
        "mpt_set_profiling": ([vp, i32], ctypes.c_int),
        "mpt_get_profile": ([vp, ctypes.POINTER(mpt_profile)], ctypes.c_int),
        "mpt_destroy": ([vp], None),
        "mpt_status_string": ([ctypes.c_int], ctypes.c_char_p),
        "mpt_last_error": ([vp], ctypes.c_char_p),
        "mpt_solve_noalloc": ([vp, i64, vp, i32, vp, vp, vp, vp, vp], ctypes.c_int),
        "mpt_batch_create": ([i64p, i64, i32, i64p, i64p, i64p, ctypes.POINTER(vp)], ctypes.c_int),
        "mpt_batch_workspace_bytes": ([vp, ctypes.POINTER(sz)], ctypes.c_int),
        "mpt_batch_solve": ([vp, vp, sz, vp], ctypes.c_int),
        "mpt_batch_results": ([vp, i64p, i64p, i32p], ctypes.c_int),
        "mpt_batch_tables": ([vp, ctypes.POINTER(vp), ctypes.POINTER(vp), i64p], ctypes.c_int),
        "mpt_batch_destroy": ([vp], None),
        "mpt_greedy": ([i64p, i64, i32, i64p, i64p, vp, i64p, i64p, i64p, i32p, i64p, i64p, i32p], ctypes.c_int),
        "mpt_serve_order": ([i64, i32, i64p, i64p, i32p, i32, vp, i32p], ctypes.c_int),
        "mpt_cache_costs": ([i64p, i64, i32, i64p, i64p, i32p, i64p, i32, vp, i64p, i64p], ctypes.c_int),
        "mpt_layout_pinned": ([i64p, i64, i32, i64p, i64p, i32, i32, vp, i64p, i32p, i64p], ctypes.c_int),
        "mpt_solve_steps": ([vp, i32p], ctypes.c_int),
        "mpt_solve_begin": ([vp, vp, sz, vp], ctypes.c_int),
        "mpt_solve_layers": ([vp, vp, sz, vp, i32, i32p], ctypes.c_int),
        "mpt_solve_end": ([vp, vp, sz, vp, i64p], ctypes.c_int),
        "mpt_solve_resume": ([vp, vp, sz, i32], ctypes.c_int),
        "mpt_set_tables": ([vp, i32], ctypes.c_int),
        "mpt_tables32": ([vp, ctypes.POINTER(vp), ctypes.POINTER(vp)], ctypes.c_int),
        "mpt_gather_bandwidth": ([i32, i64, vp, ctypes.POINTER(ctypes.c_double)], ctypes.c_int),
        "mpt_alu_addmin_peak": ([i64, vp, ctypes.POINTER(ctypes.c_double)], ctypes.c_int),
        "mpt_build_info": ([i32p], ctypes.c_int),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    _LIB = lib
    return lib


def _ptr(a: np.ndarray, ct):
    return a.ctypes.data_as(ctypes.POINTER(ct))


def _check(status: int, where: str, ctx=None):
    if status != MPT_OK:
        detail = ""
        if ctx is not None and ctx.handle:
            detail = load().mpt_last_error(ctx.handle).decode()
        raise MPTError(status, where, detail)


class Context:
    """Owns one ``mpt_ctx`` (one instance) and, optionally, a torch workspace."""

    def __init__(self, handle: int, m: int, n: int):
        self.handle = ctypes.c_void_p(handle)
        self.m = m
        self.n = n
        self.workspace = None  # torch uint8 tensor, when the binding allocated it

    def __del__(self):
        try:
            mpt_destroy(self)
        except Exception:
            pass


def mpt_create(weights, bits) -> Context:
    """Validate and copy an instance (host arrays); see ``mpt_create`` in mpt.h."""
    lib = load()
    w = np.ascontiguousarray(weights, dtype=np.int64)
    b = np.ascontiguousarray(bits, dtype=np.uint64)
    if b.ndim != 2:
        raise ValueError("bits must be uint64[m, ceil(n/64)]")
    m, n = int(b.shape[0]), int(w.shape[0])
    if b.shape[1] != (n + 63) // 64:
        raise ValueError("bits must have ceil(n/64) words per request")
    h = ctypes.c_void_p()
    _check(lib.mpt_create(_ptr(w, ctypes.c_int64), n, _ptr(b, ctypes.c_uint64), m, ctypes.byref(h)), "mpt_create")
    return Context(h.value, m, n)


def mpt_workspace_bytes(ctx: Context) -> int:
    out = ctypes.c_size_t()
    _check(load().mpt_workspace_bytes(ctx.handle, ctypes.byref(out)), "mpt_workspace_bytes", ctx)
    return int(out.value)


def mpt_set_dp_mode(ctx: Context, mode: str | int) -> None:
    """DP kernels: "auto" (default), "blocked" (32-bit keys), "wide" (64-bit
    keys) or "general"; see ``mpt_set_dp_mode`` in mpt.h."""
    code = _MODES[mode] if isinstance(mode, str) else int(mode)
    _check(load().mpt_set_dp_mode(ctx.handle, code), "mpt_set_dp_mode", ctx)


def mpt_set_profiling(ctx: Context, on: bool) -> None:
    _check(load().mpt_set_profiling(ctx.handle, 1 if on else 0), "mpt_set_profiling", ctx)


def mpt_get_profile(ctx: Context) -> dict:
    p = mpt_profile()
    _check(load().mpt_get_profile(ctx.handle, ctypes.byref(p)), "mpt_get_profile", ctx)
    return p.as_dict()


def _default_stream_ptr() -> int:
    import torch

    return int(torch.cuda.current_stream().cuda_stream)


def mpt_solve(ctx: Context, workspace=None, stream: Optional[int] = None) -> int:
    """Run the solve on ``stream`` (default: torch's current stream) using
    ``workspace`` (a CUDA uint8 tensor of at least mpt_workspace_bytes bytes;
    default: one the binding allocates with torch and keeps on the context).
    Returns OPT."""
    import torch

    need = mpt_workspace_bytes(ctx)
    if workspace is None:
        if ctx.workspace is None or ctx.workspace.numel() < need:
            ctx.workspace = torch.empty(need, dtype=torch.uint8, device="cuda")
        workspace = ctx.workspace
    if not (workspace.is_cuda and workspace.dtype == torch.uint8 and workspace.is_contiguous()):
        raise ValueError("workspace must be a contiguous CUDA uint8 tensor")
    s = _default_stream_ptr() if stream is None else int(stream)
    opt = ctypes.c_int64()
    _check(load().mpt_solve(ctx.handle, ctypes.c_void_p(workspace.data_ptr()), workspace.numel(),
                            ctypes.c_void_p(s), ctypes.byref(opt)), "mpt_solve", ctx)
    ctx._solved_ws = workspace
    return int(opt.value)


def _workspace_for(ctx: Context, workspace):
    import torch

    need = mpt_workspace_bytes(ctx)
    if workspace is None:
        if ctx.workspace is None or ctx.workspace.numel() < need:
            ctx.workspace = torch.empty(need, dtype=torch.uint8, device="cuda")
        workspace = ctx.workspace
    if not (workspace.is_cuda and workspace.dtype == torch.uint8 and workspace.is_contiguous()):
        raise ValueError("workspace must be a contiguous CUDA uint8 tensor")
    return workspace


def mpt_solve_steps(ctx: Context) -> int:
    """Number of steps of the recurrence (see mpt_solve_begin)."""
    n = ctypes.c_int32()
    _check(load().mpt_solve_steps(ctx.handle, ctypes.byref(n)), "mpt_solve_steps", ctx)
    return int(n.value)


def mpt_solve_begin(ctx: Context, workspace=None, stream: Optional[int] = None):
    """Start a staged solve; returns the workspace tensor it runs in."""
    ws = _workspace_for(ctx, workspace)
    s = _default_stream_ptr() if stream is None else int(stream)
    _check(load().mpt_solve_begin(ctx.handle, ctypes.c_void_p(ws.data_ptr()), ws.numel(), ctypes.c_void_p(s)),
           "mpt_solve_begin", ctx)
    return ws


def mpt_solve_layers(ctx: Context, workspace, count: int, stream: Optional[int] = None) -> int:
    """Run the next ``count`` steps in ``workspace``; returns the next step."""
    s = _default_stream_ptr() if stream is None else int(stream)
    nxt = ctypes.c_int32()
    _check(load().mpt_solve_layers(ctx.handle, ctypes.c_void_p(workspace.data_ptr()), workspace.numel(),
                                   ctypes.c_void_p(s), int(count), ctypes.byref(nxt)), "mpt_solve_layers", ctx)
    return int(nxt.value)


def mpt_solve_end(ctx: Context, workspace, stream: Optional[int] = None) -> int:
    """Finish a staged solve (layout walk); returns OPT."""
    s = _default_stream_ptr() if stream is None else int(stream)
    opt = ctypes.c_int64()
    _check(load().mpt_solve_end(ctx.handle, ctypes.c_void_p(workspace.data_ptr()), workspace.numel(),
                                ctypes.c_void_p(s), ctypes.byref(opt)), "mpt_solve_end", ctx)
    ctx._solved_ws = workspace
    return int(opt.value)


def mpt_solve_resume(ctx: Context, workspace, next_step: int) -> None:
    """Continue a staged solve from a checkpoint restored into ``workspace``."""
    _check(load().mpt_solve_resume(ctx.handle, ctypes.c_void_p(workspace.data_ptr()), workspace.numel(),
                                   int(next_step)), "mpt_solve_resume", ctx)


def mpt_tables(ctx: Context):
    """Device views (torch tensors of length 2^m) of F, wI and split."""
    import torch

    pF, pW, pS = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p()
    _check(load().mpt_tables(ctx.handle, ctypes.byref(pF), ctypes.byref(pW), ctypes.byref(pS)), "mpt_tables", ctx)
    ws = ctx._solved_ws
    base = ws.data_ptr()
    N = 1 << ctx.m

    def view(ptr, nbytes, dtype):
        off = ptr.value - base
        if off < 0 or off + nbytes > ws.numel():
            raise RuntimeError("table pointer outside the workspace")
        return ws[off:off + nbytes].view(dtype)

    return view(pF, 8 * N, torch.int64), view(pW, 8 * N, torch.int64), view(pS, 4 * N, torch.int32)


TABLES = {"int64": 0, "lean": 1}


def mpt_set_tables(ctx: Context, kind: str | int) -> None:
    """Table layout: "int64" (default) or "lean" (one int32 table, F over w(I))."""
    k = TABLES[kind] if isinstance(kind, str) else int(kind)
    _check(load().mpt_set_tables(ctx.handle, k), "mpt_set_tables", ctx)


def mpt_tables32(ctx: Context):
    """Device views (torch tensors of length 2^m) of the lean F (int32) and split."""
    import torch

    pF, pS = ctypes.c_void_p(), ctypes.c_void_p()
    _check(load().mpt_tables32(ctx.handle, ctypes.byref(pF), ctypes.byref(pS)), "mpt_tables32", ctx)
    ws = ctx._solved_ws
    base = ws.data_ptr()
    N = 1 << ctx.m

    def view(ptr, nbytes, dtype):
        off = ptr.value - base
        if off < 0 or off + nbytes > ws.numel():
            raise RuntimeError("table pointer outside the workspace")
        return ws[off:off + nbytes].view(dtype)

    return view(pF, 4 * N, torch.int32), view(pS, 4 * N, torch.int32)


def mpt_layout(ctx: Context):
    """(perm_offsets int64[m+1], perm_chunks int64[sum |R_i|], dfs_order int32[m])."""
    lib = load()
    total = ctypes.c_int64()
    _check(lib.mpt_layout_size(ctx.handle, ctypes.byref(total)), "mpt_layout_size", ctx)
    offs = np.zeros(ctx.m + 1, dtype=np.int64)
    chunks = np.zeros(max(1, total.value), dtype=np.int64)
    dfs = np.zeros(ctx.m, dtype=np.int32)
    _check(lib.mpt_layout(ctx.handle, _ptr(offs, ctypes.c_int64), _ptr(chunks, ctypes.c_int64),
                          _ptr(dfs, ctypes.c_int32)), "mpt_layout", ctx)
    return offs, chunks[:total.value], dfs


def mpt_trie_cost(weights, perm_offsets, perm_chunks) -> int:
    """Trie cost (eq. 1) of a layout, computed by the library's kernel."""
    w = np.ascontiguousarray(weights, dtype=np.int64)
    offs = np.ascontiguousarray(perm_offsets, dtype=np.int64)
    ch = np.ascontiguousarray(perm_chunks, dtype=np.int64)
    if ch.size == 0:
        ch = np.zeros(1, dtype=np.int64)
    m = int(offs.shape[0]) - 1
    out = ctypes.c_int64()
    _check(load().mpt_trie_cost(_ptr(w, ctypes.c_int64), int(w.shape[0]), m, _ptr(offs, ctypes.c_int64),
                                _ptr(ch, ctypes.c_int64), ctypes.byref(out)), "mpt_trie_cost")
    return int(out.value)


def mpt_destroy(ctx: Context) -> None:
    if ctx.handle and ctx.handle.value:
        load().mpt_destroy(ctx.handle)
        ctx.handle = ctypes.c_void_p()


def mpt_solve_noalloc(d_weights, d_bits, d_F, d_wI, d_split, d_opt, stream: Optional[int] = None) -> None:
    """Exact solve into caller-owned device tensors without any allocation by
    the library (for callers that cannot allocate device memory; see mpt.h).
    d_weights: CUDA int64[n]; d_bits: CUDA 64-bit [m, ceil(n/64)] (the uint64
    request bitsets, any 64-bit dtype); d_F, d_wI: CUDA int64[2^m];
    d_split: CUDA int32[2^m]; d_opt: CUDA int64[1].  Enqueued on ``stream``
    (default: torch's current stream)."""
    for t in (d_weights, d_bits, d_F, d_wI, d_split, d_opt):
        if not (t.is_cuda and t.is_contiguous()):
            raise ValueError("every argument must be a contiguous CUDA tensor")
    m, n = int(d_bits.shape[0]), int(d_weights.shape[0])
    s = _default_stream_ptr() if stream is None else int(stream)
    _check(load().mpt_solve_noalloc(ctypes.c_void_p(d_weights.data_ptr()), n, ctypes.c_void_p(d_bits.data_ptr()), m,
                                    ctypes.c_void_p(d_F.data_ptr()), ctypes.c_void_p(d_wI.data_ptr()),
                                    ctypes.c_void_p(d_split.data_ptr()), ctypes.c_void_p(d_opt.data_ptr()),
                                    ctypes.c_void_p(s)), "mpt_solve_noalloc")


@dataclass
class Result:
    opt: int
    perm_offsets: np.ndarray
    perm_chunks: np.ndarray
    dfs_order: np.ndarray
    ctx: Context

    def permutations(self) -> list[list[int]]:
        o = self.perm_offsets
        return [self.perm_chunks[o[i]:o[i + 1]].tolist() for i in range(len(o) - 1)]


def solve(weights, bits, mode: str = "auto", workspace=None, stream: Optional[int] = None,
          profile: bool = False, tables: str = "int64") -> Result:
    """Exact MPT solve of one instance: OPT, per-request permutations and the
    DFS serving order.  ``result.ctx`` keeps the device tables alive."""
    ctx = mpt_create(weights, bits)
    if mode != "auto":
        mpt_set_dp_mode(ctx, mode)
    if tables != "int64":
        mpt_set_tables(ctx, tables)
    if profile:
        mpt_set_profiling(ctx, True)
    opt = mpt_solve(ctx, workspace, stream)
    offs, chunks, dfs = mpt_layout(ctx)
    return Result(opt, offs, chunks, dfs, ctx)


# ---------------------------------------------------------------------------
# Batched small instances (mpt_batch_*)
# ---------------------------------------------------------------------------

class Batch:
    """Owns one ``mpt_batch`` (many instances of at most 16 requests)."""

    def __init__(self, handle: int, batch: int, inst_requests: np.ndarray, req_offsets: np.ndarray):
        self.handle = ctypes.c_void_p(handle)
        self.batch = batch
        self.inst_requests = inst_requests
        self.req_offsets = req_offsets
        self.workspace = None

    def __del__(self):
        try:
            mpt_batch_destroy(self)
        except Exception:
            pass


def mpt_batch_create(weights, inst_requests, req_offsets, chunk_ids) -> Batch:
    lib = load()
    w = np.ascontiguousarray(weights, dtype=np.int64)
    ir = np.ascontiguousarray(inst_requests, dtype=np.int64)
    ro = np.ascontiguousarray(req_offsets, dtype=np.int64)
    ch = np.ascontiguousarray(chunk_ids, dtype=np.int64)
    if ch.size == 0:
        ch = np.zeros(1, dtype=np.int64)
    h = ctypes.c_void_p()
    _check(lib.mpt_batch_create(_ptr(w, ctypes.c_int64), int(w.shape[0]), int(ir.shape[0]) - 1,
                                _ptr(ir, ctypes.c_int64), _ptr(ro, ctypes.c_int64), _ptr(ch, ctypes.c_int64),
                                ctypes.byref(h)), "mpt_batch_create")
    return Batch(h.value, int(ir.shape[0]) - 1, ir, ro)


def mpt_batch_workspace_bytes(b: Batch) -> int:
    out = ctypes.c_size_t()
    _check(load().mpt_batch_workspace_bytes(b.handle, ctypes.byref(out)), "mpt_batch_workspace_bytes")
    return int(out.value)


def mpt_batch_solve(b: Batch, workspace=None, stream: Optional[int] = None) -> None:
    import torch

    need = mpt_batch_workspace_bytes(b)
    if workspace is None:
        if b.workspace is None or b.workspace.numel() < need:
            b.workspace = torch.empty(need, dtype=torch.uint8, device="cuda")
        workspace = b.workspace
    s = _default_stream_ptr() if stream is None else int(stream)
    _check(load().mpt_batch_solve(b.handle, ctypes.c_void_p(workspace.data_ptr()), workspace.numel(),
                                  ctypes.c_void_p(s)), "mpt_batch_solve")
    b._solved_ws = workspace


def mpt_batch_results(b: Batch):
    """(opt int64[batch], perm_chunks int64[occurrences], dfs_order int32[requests])."""
    opt = np.zeros(b.batch, dtype=np.int64)
    perm = np.zeros(max(1, int(b.req_offsets[-1])), dtype=np.int64)
    dfs = np.zeros(max(1, int(b.inst_requests[-1])), dtype=np.int32)
    _check(load().mpt_batch_results(b.handle, _ptr(opt, ctypes.c_int64), _ptr(perm, ctypes.c_int64),
                                    _ptr(dfs, ctypes.c_int32)), "mpt_batch_results")
    return opt, perm[:int(b.req_offsets[-1])], dfs[:int(b.inst_requests[-1])]


def mpt_batch_tables(b: Batch):
    """Device views of all instances' F (int64) and split (int32) tables and
    the host offsets (instance i's tables start at offsets[i])."""
    import torch

    pF, pS = ctypes.c_void_p(), ctypes.c_void_p()
    offs = np.zeros(b.batch + 1, dtype=np.int64)
    _check(load().mpt_batch_tables(b.handle, ctypes.byref(pF), ctypes.byref(pS), _ptr(offs, ctypes.c_int64)),
           "mpt_batch_tables")
    ws = b._solved_ws
    total = int(offs[-1])

    def view(ptr, nbytes, dtype):
        off = ptr.value - ws.data_ptr()
        return ws[off:off + nbytes].view(dtype)

    return view(pF, 8 * total, torch.int64), view(pS, 4 * total, torch.int32), offs


def mpt_batch_destroy(b: Batch) -> None:
    if b.handle and b.handle.value:
        load().mpt_batch_destroy(b.handle)
        b.handle = ctypes.c_void_p()


def pack_batch(instances):
    """CSR arrays (inst_requests, req_offsets, chunk_ids) from a list of
    instances, each a list of requests, each a list of chunk ids."""
    inst = [0]
    offs = [0]
    ids = []
    for requests in instances:
        for r in requests:
            ids.extend(int(x) for x in r)
            offs.append(len(ids))
        inst.append(len(offs) - 1)
    return (np.asarray(inst, dtype=np.int64), np.asarray(offs, dtype=np.int64),
            np.asarray(ids, dtype=np.int64))


def solve_batch(weights, instances, workspace=None, stream: Optional[int] = None):
    """Exact solves of many small instances.  Returns (opt per instance,
    per-instance list of per-request chunk orders, per-instance DFS order, batch)."""
    ir, ro, ch = pack_batch(instances)
    b = mpt_batch_create(weights, ir, ro, ch)
    mpt_batch_solve(b, workspace, stream)
    opt, perm, dfs = mpt_batch_results(b)
    perms, orders = [], []
    for i in range(b.batch):
        r0, r1 = int(ir[i]), int(ir[i + 1])
        perms.append([perm[ro[r]:ro[r + 1]].tolist() for r in range(r0, r1)])
        orders.append(dfs[r0:r1].tolist())
    return opt, perms, orders, b


# ---------------------------------------------------------------------------
# Agglomerative greedy and spanning-tree bound (mpt_greedy)
# ---------------------------------------------------------------------------

@dataclass
class GreedyResult:
    cost: int
    savings: int
    lower_bound: int
    merges: np.ndarray        # int32[m-1, 2] slot pairs
    merge_values: np.ndarray  # int64[m-1]
    perms: list
    dfs_order: np.ndarray


def mpt_greedy(weights, requests, stream: Optional[int] = None) -> GreedyResult:
    """Greedy hierarchy + layout + lower bound for ``requests`` (a list of
    chunk-id lists) over the universe of ``weights``."""
    lib = load()
    w = np.ascontiguousarray(weights, dtype=np.int64)
    offs, ids = _csr(requests)
    m = _count(requests)
    cost, sav, lb = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    merges = np.zeros(max(1, 2 * (m - 1)), dtype=np.int32)
    vals = np.zeros(max(1, m - 1), dtype=np.int64)
    perm = np.zeros(max(1, int(offs[-1])), dtype=np.int64)
    dfs = np.zeros(m, dtype=np.int32)
    s = 0 if stream is None else int(stream)
    _check(lib.mpt_greedy(_ptr(w, ctypes.c_int64), int(w.shape[0]), m, _ptr(offs, ctypes.c_int64),
                          _ptr(ids, ctypes.c_int64), ctypes.c_void_p(s), ctypes.byref(cost), ctypes.byref(sav),
                          ctypes.byref(lb), _ptr(merges, ctypes.c_int32), _ptr(vals, ctypes.c_int64),
                          _ptr(perm, ctypes.c_int64), _ptr(dfs, ctypes.c_int32)), "mpt_greedy")
    perms = [perm[offs[i]:offs[i + 1]].tolist() for i in range(m)]
    return GreedyResult(int(cost.value), int(sav.value), int(lb.value), merges[:2 * (m - 1)].reshape(-1, 2),
                        vals[:m - 1], perms, dfs)


def _csr(strings):
    """(offsets, ids) int64 arrays of a list of chunk-id lists (or such a pair
    already built: a tuple of two arrays); ids has >= 1 entry."""
    if isinstance(strings, tuple) and len(strings) == 2 and isinstance(strings[0], np.ndarray):
        offs = np.ascontiguousarray(strings[0], dtype=np.int64)
        ids = np.ascontiguousarray(strings[1], dtype=np.int64)
        return offs, (ids if ids.size else np.zeros(1, dtype=np.int64))
    lens = np.fromiter((len(r) for r in strings), dtype=np.int64, count=len(strings))
    offs = np.zeros(len(strings) + 1, dtype=np.int64)
    np.cumsum(lens, out=offs[1:])
    total = int(offs[-1])
    ids = (np.fromiter(itertools.chain.from_iterable(strings), dtype=np.int64, count=total)
           if total else np.zeros(1, dtype=np.int64))
    return offs, ids


def to_csr(strings):
    """(offsets int64[m+1], ids int64) of a list of chunk-id lists, to pass to
    mpt_serve_order / mpt_cache_costs in place of the list (built once)."""
    return _csr(strings)


def _count(strings) -> int:
    """Number of strings in a list or in an (offsets, ids) pair."""
    if isinstance(strings, tuple) and len(strings) == 2 and isinstance(strings[0], np.ndarray):
        return int(strings[0].shape[0]) - 1
    return len(strings)


def mpt_serve_order(n_chunks: int, strings, arrival=None, window: int = 0,
                    stream: Optional[int] = None) -> np.ndarray:
    """Thm 7's serving order of ``strings`` (lists of chunk ids), optionally
    sorted only inside consecutive windows of ``window`` arrivals of ``arrival``."""
    lib = load()
    offs, ids = _csr(strings)
    m = _count(strings)
    arr = None if arrival is None else np.ascontiguousarray(arrival, dtype=np.int32)
    out = np.zeros(max(m, 1), dtype=np.int32)
    s = 0 if stream is None else int(stream)
    _check(lib.mpt_serve_order(int(n_chunks), m, _ptr(offs, ctypes.c_int64), _ptr(ids, ctypes.c_int64),
                               None if arr is None else _ptr(arr, ctypes.c_int32), int(window), ctypes.c_void_p(s),
                               _ptr(out, ctypes.c_int32)), "mpt_serve_order")
    return out[:m]


def mpt_cache_costs(weights, strings, capacities, order=None, stream: Optional[int] = None):
    """Prefill cost of serving ``strings`` in ``order`` through a radix cache
    with LRU leaf eviction, at every capacity in ``capacities``.  Returns
    (costs int64[len(capacities)], unbounded-cache cost)."""
    lib = load()
    w = np.ascontiguousarray(weights, dtype=np.int64)
    offs, ids = _csr(strings)
    m = _count(strings)
    caps = np.ascontiguousarray(capacities, dtype=np.int64)
    if caps.size == 0:
        caps = np.zeros(1, dtype=np.int64)
        n_caps = 0
    else:
        n_caps = int(caps.size)
    ordv = None if order is None else np.ascontiguousarray(order, dtype=np.int32)
    costs = np.zeros(max(n_caps, 1), dtype=np.int64)
    unb = ctypes.c_int64()
    s = 0 if stream is None else int(stream)
    _check(lib.mpt_cache_costs(_ptr(w, ctypes.c_int64), int(w.shape[0]), m, _ptr(offs, ctypes.c_int64),
                               _ptr(ids, ctypes.c_int64), None if ordv is None else _ptr(ordv, ctypes.c_int32),
                               _ptr(caps, ctypes.c_int64), n_caps, ctypes.c_void_p(s), _ptr(costs, ctypes.c_int64),
                               ctypes.byref(unb)), "mpt_cache_costs")
    return costs[:n_caps], int(unb.value)


PIN_METHODS = {"exact": 0, "greedy": 1}


@dataclass
class PinnedResult:
    strings: list  # per request: free layout, then the pinned passages
    serve_order: np.ndarray
    cost: int


def mpt_layout_pinned(weights, ranked, t: int, method: str = "exact",
                      stream: Optional[int] = None) -> PinnedResult:
    """Sec. 7.1 layout: each request's first ``t`` passages of ``ranked[i]``
    (relevance order) pinned at the end, the rest laid out by ``method``."""
    lib = load()
    w = np.ascontiguousarray(weights, dtype=np.int64)
    offs, ids = _csr(ranked)
    m = len(ranked)
    perm = np.zeros(max(1, int(offs[-1])), dtype=np.int64)
    order = np.zeros(max(m, 1), dtype=np.int32)
    cost = ctypes.c_int64()
    s = 0 if stream is None else int(stream)
    _check(lib.mpt_layout_pinned(_ptr(w, ctypes.c_int64), int(w.shape[0]), m, _ptr(offs, ctypes.c_int64),
                                 _ptr(ids, ctypes.c_int64), int(t), PIN_METHODS[method], ctypes.c_void_p(s),
                                 _ptr(perm, ctypes.c_int64), _ptr(order, ctypes.c_int32), ctypes.byref(cost)),
           "mpt_layout_pinned")
    strings = [perm[offs[i]:offs[i + 1]].tolist() for i in range(m)]
    return PinnedResult(strings, order[:m], int(cost.value))


def mpt_gather_bandwidth(log2_entries: int, loads: int = 1 << 28, stream: Optional[int] = None) -> float:
    """Measured GB/s of uniformly random 8-byte loads from a 2^log2_entries int64 table."""
    out = ctypes.c_double()
    s = 0 if stream is None else int(stream)
    _check(load().mpt_gather_bandwidth(int(log2_entries), int(loads), ctypes.c_void_p(s), ctypes.byref(out)),
           "mpt_gather_bandwidth")
    return float(out.value)


def mpt_alu_addmin_peak(ops: int = 1 << 42, stream: Optional[int] = None) -> float:
    """Measured add-min instructions per second of the integer ALU pipe, all SMs busy."""
    out = ctypes.c_double()
    s = 0 if stream is None else int(stream)
    _check(load().mpt_alu_addmin_peak(int(ops), ctypes.c_void_p(s), ctypes.byref(out)), "mpt_alu_addmin_peak")
    return float(out.value)


def mpt_build_info() -> dict:
    """How the loaded library was built: {"bounds_checked": bool}."""
    flags = ctypes.c_int32()
    _check(load().mpt_build_info(ctypes.byref(flags)), "mpt_build_info")
    return {"bounds_checked": bool(flags.value & 1)}
