"""GB300-native TurboQuant search path (rotate, quantise, pack; filtered top-k scan).

Every computation runs in the CUDA library libtq.so built from csrc/ (C ABI in
include/tq.h).  This module only marshals torch tensors and numpy arrays into
that ABI: torch provides device memory and streams.  There is no CPU fallback:
if libtq.so is missing, every call raises.
"""
from __future__ import annotations

import ctypes as C

import numpy as np

from ._lib import (MARGINALS, PATHS, SCALE_MODES, TQ_EUNSUPPORTED, TQError, check, load)  # noqa: F401

__all__ = ["codebook", "rotation", "encode", "encode_plan", "encode_plan_bytes", "encode_check", "calibrate", "Filter", "IdMap", "Index", "search", "search_workspace",
           "search_from_host", "search_host_staging", "search_check", "merge_topk", "set_search_path",
           "profile_events", "row_bytes", "load", "TQError"]


def _torch():
    import torch
    return torch


def _stream_handle(stream) -> int:
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


class _on_stream:
    """Allocations made inside belong to `stream` (None: the current stream).

    Tensors a call creates for work it queues on a side stream must come from
    that stream's pool: the caching allocator recycles a freed block for the
    next allocation on the block's own stream without waiting, so a temporary
    taken from the current stream and freed on return could be handed out
    again while the side stream's kernels still read or write it."""

    def __init__(self, stream):
        self._ctx = _torch().cuda.stream(stream) if stream is not None else None

    def __enter__(self):
        if self._ctx is not None:
            self._ctx.__enter__()
        return self

    def __exit__(self, *exc):
        if self._ctx is not None:
            return self._ctx.__exit__(*exc)
        return False


def _used_on(t, stream) -> None:
    """Marks a tensor allocated elsewhere as used by work queued on `stream`,
    so that its memory is not reused before that work has finished."""
    if stream is not None and t is not None and t.is_cuda:
        t.record_stream(stream)


def _dev_ptr(t, name: str, dtype=None, contiguous: bool = True) -> int:
    if t is None:
        return 0
    if not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype not in (dtype if isinstance(dtype, tuple) else (dtype,)):
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if contiguous and not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return int(t.data_ptr())


def row_bytes(d: int, bits: int) -> int:
    """Bytes of one packed vector: d*bits/8 (768 at d=1536, 4 bits)."""
    return d * bits // 8


def codebook(d: int, bits: int, marginal: str = "beta"):
    """tq_codebook: Lloyd-Max centroids [2^bits], boundaries [2^bits - 1]
    (float32 numpy) and the per-coordinate distortion."""
    lib = load()
    L = 1 << bits
    c = np.zeros(L, np.float32)
    t = np.zeros(max(L - 1, 1), np.float32)
    D = C.c_double()
    check(lib.tq_codebook(d, bits, MARGINALS[marginal], c.ctypes.data, t.ctypes.data, C.byref(D)))
    return c, t[: L - 1], D.value


def rotation(d: int, seed: int) -> np.ndarray:
    """tq_rotation: float32 [d, d] row-major R (y = R x)."""
    R = np.empty((d, d), np.float32)
    check(load().tq_rotation(d, seed, R.ctypes.data))
    return R


def encode(X, R, centroids, boundaries, bits: int, scale_mode: str = "norm",
           codes=None, scale=None, stream=None, calib=None, plan=None):
    """tq_encode (tq_encode_ex with a TQ+ calibration `calib` = (mu, a), CUDA
    float32 tensors [d]) on CUDA tensors: returns (codes uint8 [n, d*bits/8],
    scale f32 [n]).  With `plan` (encode_plan(R)) the rotation runs on the
    tensor cores (tq_encode_planned) and R is not read."""
    torch = _torch()
    n, d = X.shape
    with _on_stream(stream):
        if codes is None:
            codes = torch.empty((n, row_bytes(d, bits)), dtype=torch.uint8, device=X.device)
        if scale is None:
            scale = torch.empty(n, dtype=torch.float32, device=X.device)
    f32 = torch.float32
    mu, a = calib if calib is not None else (None, None)
    tail = (_dev_ptr(centroids, "centroids", f32), _dev_ptr(boundaries, "boundaries", f32), bits,
            SCALE_MODES[scale_mode], _dev_ptr(mu, "mu", f32) or None, _dev_ptr(a, "a", f32) or None,
            _dev_ptr(codes, "codes", torch.uint8), _dev_ptr(scale, "scale", f32), _stream_handle(stream))
    if plan is not None:
        check(load().tq_encode_planned(_dev_ptr(X, "X", f32), n, d, _dev_ptr(plan, "plan", torch.uint8), *tail))
    else:
        check(load().tq_encode_ex(_dev_ptr(X, "X", f32), n, d, _dev_ptr(R, "R", f32), *tail))
    return codes, scale


def encode_plan_bytes(d: int):
    """tq_encode_plan_bytes: device bytes of a tensor-core encode plan for
    dimension d, or None where the tensor-core encoder does not apply."""
    need = C.c_size_t()
    st = load().tq_encode_plan_bytes(d, C.byref(need))
    if st == TQ_EUNSUPPORTED:
        return None
    check(st)
    return need.value


def encode_plan(R, stream=None):
    """tq_encode_plan: R (CUDA float32 [d, d]) split into TF32 parts for the
    tensor-core encoder; returns the plan (CUDA uint8 tensor)."""
    torch = _torch()
    d = R.shape[0]
    need = encode_plan_bytes(d)
    if need is None:
        raise TQError(TQ_EUNSUPPORTED, f"no tensor-core encode for d={d}")
    with _on_stream(stream):
        plan = torch.empty(need, dtype=torch.uint8, device=R.device)
    check(load().tq_encode_plan(_dev_ptr(R, "R", torch.float32), d, _dev_ptr(plan, "plan", torch.uint8), need,
                                _stream_handle(stream)))
    return plan


def encode_check(plan, stream=None) -> None:
    """tq_encode_check: raises TQError(TQ_ETIMEOUT) if an encode with `plan`
    gave up on a bounded wait since the last check."""
    torch = _torch()
    check(load().tq_encode_check(_dev_ptr(plan, "plan", torch.uint8), _stream_handle(stream)))


def calibrate(X, R, stream=None):
    """tq_calibrate: the TQ+ per-coordinate shift and scale (Sec. II-B) of the
    rows of X (CUDA float32 [n, d]): returns (mu, a), CUDA float32 [d] each."""
    torch = _torch()
    n, d = X.shape
    need = C.c_size_t()
    check(load().tq_calibrate_workspace(n, d, C.byref(need)))
    with _on_stream(stream):
        ws = torch.empty(max(need.value, 1), dtype=torch.uint8, device=X.device)
        mu = torch.empty(d, dtype=torch.float32, device=X.device)
        a = torch.empty(d, dtype=torch.float32, device=X.device)
    f32 = torch.float32
    check(load().tq_calibrate(_dev_ptr(X, "X", f32), n, d, _dev_ptr(R, "R", f32), _dev_ptr(mu, "mu"),
                              _dev_ptr(a, "a"), _dev_ptr(ws, "workspace"), ws.numel(), _stream_handle(stream)))
    return mu, a


class Filter:
    """tq_filter handle: per-block tenant bitmaps of a corpus (Sec. III-B)."""

    def __init__(self, tenant_ids, block: int = 64, stream=None):
        torch = _torch()
        self._h = C.c_void_p()
        ptr = _dev_ptr(tenant_ids, "tenant_ids", (torch.int32, getattr(torch, "uint32", torch.int32)))
        check(load().tq_filter_build(ptr, tenant_ids.numel(), block, C.byref(self._h),
                                     _stream_handle(stream)))

    @property
    def handle(self) -> int:
        return self._h.value or 0

    def append(self, tenant_ids, stream=None) -> None:
        """tq_filter_append: tenants of the rows added after the current ones."""
        torch = _torch()
        ptr = _dev_ptr(tenant_ids, "tenant_ids", (torch.int32, getattr(torch, "uint32", torch.int32)))
        check(load().tq_filter_append(self._h, ptr, tenant_ids.numel(), _stream_handle(stream)))

    def info(self):
        n, b, t = C.c_int64(), C.c_int(), C.c_int64()
        check(load().tq_filter_info(self._h, C.byref(n), C.byref(b), C.byref(t)))
        return {"n": n.value, "block": b.value, "n_tenants": t.value}

    def close(self) -> None:
        if self._h and self._h.value:
            load().tq_filter_destroy(self._h)
            self._h = C.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class IdMap:
    """tq_idmap handle: external uint64 ids of rows 0, 1, ... in insertion
    order, O(1) lookup and deletion (Sec. III-A).  Pass it to search() as
    `idmap`: deleted rows are never returned and results come back as
    external ids (int64 bit patterns; -1 marks an empty slot)."""

    def __init__(self, capacity: int):
        self._h = C.c_void_p()
        check(load().tq_idmap_create(int(capacity), C.byref(self._h)))

    @property
    def handle(self) -> int:
        return self._h.value or 0

    @staticmethod
    def _ids(ext_ids) -> np.ndarray:
        a = np.ascontiguousarray(np.asarray(ext_ids).reshape(-1))
        if a.dtype == np.int64:
            a = a.view(np.uint64)
        return np.ascontiguousarray(a, dtype=np.uint64)

    def add(self, ext_ids, stream=None) -> int:
        """Appends rows with these external ids; returns the first new row."""
        a = self._ids(ext_ids)
        first = C.c_int64()
        check(load().tq_idmap_add(self._h, a.ctypes.data, a.size, C.byref(first), _stream_handle(stream)))
        return first.value

    def remove(self, ext_ids, stream=None) -> int:
        """Deletes the rows of these ids (ids that are not live are ignored);
        returns how many were removed."""
        a = self._ids(ext_ids)
        n = C.c_int64()
        check(load().tq_idmap_remove(self._h, a.ctypes.data, a.size, C.byref(n), _stream_handle(stream)))
        return n.value

    def lookup(self, ext_id: int) -> int:
        """Row of a live external id, or -1."""
        row = C.c_int64()
        check(load().tq_idmap_lookup(self._h, C.c_uint64(int(ext_id) & 0xFFFFFFFFFFFFFFFF), C.byref(row)))
        return row.value

    def info(self):
        r, c, l = C.c_int64(), C.c_int64(), C.c_int64()
        check(load().tq_idmap_info(self._h, C.byref(r), C.byref(c), C.byref(l)))
        return {"rows": r.value, "capacity": c.value, "live": l.value}

    def device(self):
        """(tombstone bitmap, external ids) device addresses for tq_search_ex."""
        dd, de = C.c_void_p(), C.c_void_p()
        check(load().tq_idmap_device(self._h, C.byref(dd), C.byref(de)))
        return dd.value or 0, de.value or 0

    def export(self):
        """(external ids uint64 [rows], tombstone bitmap uint32 [ceil(rows/32)])
        as host arrays."""
        rows = self.info()["rows"]
        ext = np.zeros(rows, np.uint64)
        dead = np.zeros((rows + 31) // 32, np.uint32)
        check(load().tq_idmap_export(self._h, ext.ctypes.data, dead.ctypes.data))
        return ext, dead

    def import_(self, ext_ids, deleted, stream=None) -> None:
        """Fills this (empty) map from export()'s arrays."""
        ext = self._ids(ext_ids)
        dead = np.ascontiguousarray(deleted, dtype=np.uint32)
        if dead.size != (ext.size + 31) // 32:
            raise ValueError("the tombstone bitmap needs ceil(rows/32) words")
        check(load().tq_idmap_import(self._h, ext.ctypes.data, dead.ctypes.data, ext.size, _stream_handle(stream)))

    def close(self) -> None:
        if self._h and self._h.value:
            load().tq_idmap_destroy(self._h)
            self._h = C.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def search_workspace(nq: int, n: int, d: int, bits: int, k: int, filter: Filter | None = None) -> int:
    out = C.c_size_t()
    check(load().tq_search_workspace(nq, n, d, bits, k, filter.handle if filter else None, C.byref(out)))
    return out.value


def search(Q, R, centroids, bits: int, codes, scale, k: int, filter: Filter | None = None,
           allow_off=None, allow_tenants=None, workspace=None, out_ids=None, out_scores=None,
           stream=None, idmap: IdMap | None = None, calib=None):
    """tq_search (tq_search_ex with an IdMap) on CUDA tensors: returns
    (ids int64 [nq, k], scores f32 [nq, k]); with an IdMap the ids are
    external ids and deleted rows are skipped; `calib` = (mu, a) searches
    codes encoded with that TQ+ calibration."""
    torch = _torch()
    nq, d = Q.shape
    n = codes.shape[0]
    deleted = ext = 0
    if idmap is not None:
        if idmap.info()["rows"] < n:
            raise ValueError(f"the id map holds {idmap.info()['rows']} rows, the corpus {n}")
        deleted, ext = idmap.device()
    dev = Q.device
    with _on_stream(stream):  # freed temporaries must not be recycled before the search ends
        if out_ids is None:
            out_ids = torch.empty((nq, k), dtype=torch.int64, device=dev)
        if out_scores is None:
            out_scores = torch.empty((nq, k), dtype=torch.float32, device=dev)
        if workspace is None:  # a caller-owned workspace is size-checked by tq_search itself
            need = search_workspace(nq, n, d, bits, k, filter)
            workspace = torch.empty(max(need, 1), dtype=torch.uint8, device=dev)
    f32 = torch.float32
    u32 = (torch.int32, getattr(torch, "uint32", torch.int32))
    check(load().tq_search_ex(
        _dev_ptr(Q, "Q", f32), nq, d, _dev_ptr(R, "R", f32), _dev_ptr(centroids, "centroids", f32), bits,
        _dev_ptr(codes, "codes", torch.uint8), _dev_ptr(scale, "scale", f32), n,
        filter.handle if filter else None, _dev_ptr(allow_off, "allow_off", torch.int64),
        _dev_ptr(allow_tenants, "allow_tenants", u32), deleted or None, ext or None,
        _dev_ptr(calib[0], "mu", f32) if calib is not None else None,
        _dev_ptr(calib[1], "a", f32) if calib is not None else None, k,
        _dev_ptr(out_ids, "out_ids", torch.int64),
        _dev_ptr(out_scores, "out_scores", f32), _dev_ptr(workspace, "workspace", contiguous=True),
        workspace.numel() * workspace.element_size(), _stream_handle(stream)))
    return out_ids, out_scores


def search_host_staging(nq: int, d: int, k: int) -> int:
    """Bytes of device staging tq_search_host needs (queries and results)."""
    out = C.c_size_t()
    check(load().tq_search_host_staging(nq, d, k, C.byref(out)))
    return out.value


def search_from_host(Q_host, R, centroids, bits: int, codes, scale, k: int, ids_host, scores_host,
                     filter: Filter | None = None, allow_off=None, allow_tenants=None, workspace=None,
                     staging=None, stream=None, idmap: IdMap | None = None, calib=None):
    """tq_search_host: queries in host memory (a CPU float32 tensor, page-locked
    for asynchronous copies), results into the host tensors ids_host (int64
    [nq, k]) and scores_host (float32 [nq, k]).  The library queues the query
    copy, the search and the result copies on `stream`; synchronise it before
    reading the results."""
    torch = _torch()
    nq, d = Q_host.shape
    n = codes.shape[0]
    for t, name, dt in ((Q_host, "Q_host", torch.float32), (ids_host, "ids_host", torch.int64),
                        (scores_host, "scores_host", torch.float32)):
        if t.is_cuda or t.dtype != dt or not t.is_contiguous():
            raise TypeError(f"{name} must be a contiguous host {dt} tensor")
    if ids_host.shape != (nq, k) or scores_host.shape != (nq, k):
        raise ValueError("ids_host and scores_host must be [nq, k]")
    deleted = ext = 0
    if idmap is not None:
        deleted, ext = idmap.device()
    dev = codes.device
    with _on_stream(stream):
        if workspace is None:
            workspace = torch.empty(max(search_workspace(nq, n, d, bits, k, filter), 1), dtype=torch.uint8,
                                    device=dev)
        if staging is None:
            staging = torch.empty(search_host_staging(nq, d, k), dtype=torch.uint8, device=dev)
    f32 = torch.float32
    u32 = (torch.int32, getattr(torch, "uint32", torch.int32))
    check(load().tq_search_host(
        int(Q_host.data_ptr()), nq, d, _dev_ptr(R, "R", f32), _dev_ptr(centroids, "centroids", f32), bits,
        _dev_ptr(codes, "codes", torch.uint8), _dev_ptr(scale, "scale", f32), n,
        filter.handle if filter else None, _dev_ptr(allow_off, "allow_off", torch.int64),
        _dev_ptr(allow_tenants, "allow_tenants", u32), deleted or None, ext or None,
        _dev_ptr(calib[0], "mu", f32) if calib is not None else None,
        _dev_ptr(calib[1], "a", f32) if calib is not None else None, k,
        int(ids_host.data_ptr()), int(scores_host.data_ptr()), _dev_ptr(staging, "staging"),
        staging.numel() * staging.element_size(), _dev_ptr(workspace, "workspace"),
        workspace.numel() * workspace.element_size(), _stream_handle(stream)))
    return ids_host, scores_host


def merge_topk(cand_ids, cand_scores, k: int, out_ids=None, out_scores=None, stream=None):
    """tq_merge_topk on CUDA tensors laid out [n_src, nq, m] (or [nq, m] for a
    single source): returns (ids int64 [nq, k], scores f32 [nq, k])."""
    torch = _torch()
    if cand_ids.dim() == 2:
        cand_ids, cand_scores = cand_ids.unsqueeze(0), cand_scores.unsqueeze(0)
    if cand_ids.shape != cand_scores.shape or cand_ids.dim() != 3:
        raise ValueError("cand_ids and cand_scores must both be [n_src, nq, m]")
    n_src, nq, m = cand_ids.shape
    dev = cand_ids.device
    with _on_stream(stream):
        if out_ids is None:
            out_ids = torch.empty((nq, k), dtype=torch.int64, device=dev)
        if out_scores is None:
            out_scores = torch.empty((nq, k), dtype=torch.float32, device=dev)
    check(load().tq_merge_topk(
        _dev_ptr(cand_ids, "cand_ids", torch.int64), _dev_ptr(cand_scores, "cand_scores", torch.float32),
        n_src, nq, m, k, _dev_ptr(out_ids, "out_ids", torch.int64),
        _dev_ptr(out_scores, "out_scores", torch.float32), _stream_handle(stream)))
    return out_ids, out_scores


def search_check(workspace, stream=None) -> None:
    """tq_search_check: waits for the stream; raises TQError (TQ_ETIMEOUT) if
    the last search that used `workspace` gave up on a bounded wait."""
    check(load().tq_search_check(_dev_ptr(workspace, "workspace"), _stream_handle(stream)))


def set_search_path(path: str) -> None:
    """'auto' (default), 'lut' or 'mma' for later searches on this thread."""
    check(load().tq_set_search_path(PATHS[path]))


def profile_events(start=None, stop=None) -> None:
    """Record two torch.cuda.Events around the scan kernel of later searches.
    torch creates an event's CUDA handle on its first record(), so events that
    have never been recorded are recorded once here first."""
    handles = []
    for ev in (start, stop):
        if ev is None:
            handles.append(None)
            continue
        if not int(ev.cuda_event):
            ev.record()
        handles.append(int(ev.cuda_event))
    check(load().tq_profile_events(*handles))


from .index import Index  # noqa: E402  (index.py builds on the calls above)
