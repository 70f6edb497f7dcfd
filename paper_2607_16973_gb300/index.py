"""A TurboQuant index on one GPU: online ingest, deletion, filtered search and
persistence (Sec. III-A).

The paper names two index types, a flat scan addressed by position and an
id-mapped one (external uint64 ids, O(1) deletion); both ingest vectors
without a training step and persist to disk.  `Index` is both: with
`id_map=True` it keeps a `tq_idmap` and reports external ids, otherwise rows.
With `tenants=True` every row carries a tenant id and searches can take
allowlists (Sec. III-B), the per-block tenant bitmaps growing with the index.

Everything here is bookkeeping around the C ABI: rows are encoded by
tq_encode straight into the index's device arrays, the filter grows by
tq_filter_append, and search is tq_search_ex.  With `tq_plus=True` the first
batch added fixes a TQ+ calibration (tq_calibrate) that every later encode and
search uses.  Files use the flat format of `flatfile`.
"""
from __future__ import annotations

import numpy as np

from . import Filter, IdMap, calibrate, codebook, encode, encode_plan, encode_plan_bytes, rotation, row_bytes, search
from . import _used_on, flatfile

FORMAT_VERSION = 1


def _torch():
    import torch
    return torch


class Index:
    """Flat index of up to `capacity` vectors of dimension d at `bits` bits.

    d: multiple of 32; bits: 2, 3, 4 or 8; seed: the rotation's seed
    (tq_rotation); marginal / scale_mode: as for tq_codebook / tq_encode.
    tables: optional (R [d, d], centroids, boundaries) host arrays to use
    instead of tq_rotation(d, seed) and tq_codebook(d, bits, marginal).
    """

    def __init__(self, d: int, bits: int = 4, capacity: int = 1 << 20, *, seed: int = 1536,
                 marginal: str = "beta", scale_mode: str = "norm", id_map: bool = False,
                 tenants: bool = False, block: int = 64, device=None, tables=None, tq_plus: bool = False):
        torch = _torch()
        self.device = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        self.d, self.bits, self.capacity = int(d), int(bits), int(capacity)
        self.seed, self.marginal, self.scale_mode, self.block = int(seed), marginal, scale_mode, int(block)
        self.n = 0
        if tables is None:
            c, t, _ = codebook(self.d, self.bits, marginal)
            tables = (rotation(self.d, self.seed), c, t)
        R, c, t = (np.asarray(a, np.float32) for a in tables)
        if R.shape != (self.d, self.d) or c.shape != (1 << self.bits,) or t.shape != ((1 << self.bits) - 1,):
            raise ValueError("tables must be R [d, d], centroids [2^bits] and boundaries [2^bits - 1]")
        self._set_tables(R, c, t)
        self.codes = torch.empty((self.capacity, row_bytes(self.d, self.bits)), dtype=torch.uint8,
                                 device=self.device)
        self.scale = torch.empty(self.capacity, dtype=torch.float32, device=self.device)
        self.id_map = IdMap(self.capacity) if id_map else None
        self.tenant_ids = torch.empty(self.capacity, dtype=torch.int32, device=self.device) if tenants else None
        self.filter: Filter | None = None
        # TQ+ (Sec. II-B): per-coordinate shift and scale fitted on the first
        # add() batch, then used for every encode and search
        self.tq_plus = bool(tq_plus)
        self.calib = None

    def _set_tables(self, R, centroids, boundaries) -> None:
        torch = _torch()
        self.R = torch.from_numpy(np.ascontiguousarray(R, np.float32)).to(self.device)
        self.centroids = torch.from_numpy(np.ascontiguousarray(centroids, np.float32)).to(self.device)
        self.boundaries = torch.from_numpy(np.ascontiguousarray(boundaries, np.float32)).to(self.device)
        # the tensor-core encoder's split of R, where it applies (else the FFMA encoder runs)
        with torch.cuda.device(self.device):
            self.plan = encode_plan(self.R) if encode_plan_bytes(self.d) is not None else None

    def __len__(self) -> int:
        return self.n

    @property
    def live(self) -> int:
        """Rows that a search can return (all rows without an id map)."""
        return self.id_map.info()["live"] if self.id_map is not None else self.n

    def add(self, X, ids=None, tenant_ids=None, stream=None) -> int:
        """Appends the rows of X ([m, d] float32; a CUDA tensor or host array),
        encoded on the GPU into rows n .. n+m-1; returns n.  `ids` (host
        uint64 [m]) is required with an id map, `tenant_ids` ([m] int32/uint32,
        host or device) with tenants.

        The rows are encoded first and committed by the id map and the filter
        after: rejected ids (live, repeated or -1) leave the index unchanged.
        A filter that cannot grow (device memory) raises after the id map
        took the rows; the index should then be rebuilt or reloaded."""
        torch = _torch()
        X = torch.as_tensor(X, dtype=torch.float32, device=self.device).contiguous()
        if X.dim() != 2 or X.shape[1] != self.d:
            raise ValueError(f"X must be [m, {self.d}]")
        m = X.shape[0]
        if self.n + m > self.capacity:
            raise ValueError(f"{self.n} rows + {m} new exceed the capacity {self.capacity}")
        if (self.id_map is not None) != (ids is not None):
            raise ValueError("ids are required with an id map, and only then")
        if (self.tenant_ids is not None) != (tenant_ids is not None):
            raise ValueError("tenant_ids are required with tenants, and only then")
        if m == 0:
            return self.n
        if ids is not None and len(np.asarray(ids).reshape(-1)) != m:
            raise ValueError("one id per row")
        ten = None
        if tenant_ids is not None:
            if not isinstance(tenant_ids, torch.Tensor):  # host ids: uint32 values
                tenant_ids = torch.from_numpy(np.asarray(tenant_ids).astype(np.uint32).view(np.int32))
            ten = tenant_ids.to(self.device).reshape(-1)
            if ten.numel() != m or ten.dtype not in (torch.int32, getattr(torch, "uint32", torch.int32)):
                raise ValueError("one int32/uint32 tenant id per row")
        if stream is not None:
            # X and ten were made on the current stream: the work queued on
            # `stream` waits for them, and their memory stays theirs until it ends
            stream.wait_stream(torch.cuda.current_stream(self.device))
            _used_on(X, stream)
            _used_on(ten, stream)
        first = self.n
        rows = slice(first, first + m)
        codes, scale = self.codes[rows], self.scale[rows]
        if self.tq_plus and self.calib is None:  # the first batch fixes the calibration
            self.calib = calibrate(X, self.R, stream=stream)
        if codes.data_ptr() % 16 == 0:
            encode(X, self.R, self.centroids, self.boundaries, self.bits, self.scale_mode, codes, scale,
                   stream=stream, calib=self.calib, plan=self.plan)
        else:  # a row offset off the 16-byte grid tq_encode needs: encode aside, then copy
            c, s = encode(X, self.R, self.centroids, self.boundaries, self.bits, self.scale_mode, stream=stream,
                          calib=self.calib, plan=self.plan)
            with torch.cuda.stream(stream) if stream is not None else _null():
                codes.copy_(c)
                scale.copy_(s)
        if self.id_map is not None:  # validates the ids; a rejection leaves n as it was
            self.id_map.add(ids, stream=stream)
        if ten is not None:
            with torch.cuda.stream(stream) if stream is not None else _null():
                self.tenant_ids[rows].copy_(ten.view(torch.int32))
            if self.filter is None:
                self.filter = Filter(self.tenant_ids[: first + m], block=self.block, stream=stream)
            else:
                self.filter.append(self.tenant_ids[rows], stream=stream)
        self.n = first + m
        return first

    def remove(self, ids, stream=None) -> int:
        """Deletes the rows of these external ids (id map only); returns how
        many were live."""
        if self.id_map is None:
            raise ValueError("deletion needs an id map (Index(..., id_map=True))")
        return self.id_map.remove(ids, stream=stream)

    def search(self, Q, k: int, allow=None, stream=None, workspace=None):
        """Top-k of each query row of Q ([nq, d] float32): (ids int64 [nq, k],
        scores float32 [nq, k]); ids are external ids with an id map, rows
        otherwise; empty slots are (-1, -inf).  `allow` (tenants only): one
        list of allowed tenant ids per query, or a (allow_off, allow_tenants)
        pair of CUDA tensors in tq_search's CSR layout."""
        torch = _torch()
        Q = torch.as_tensor(Q, dtype=torch.float32, device=self.device).contiguous()
        nq = Q.shape[0]
        if self.n == 0:
            return (torch.full((nq, k), -1, dtype=torch.int64, device=self.device),
                    torch.full((nq, k), float("-inf"), dtype=torch.float32, device=self.device))
        off = ten = None
        if allow is not None:
            if self.filter is None:
                raise ValueError("allowlists need an index built with tenants=True")
            if isinstance(allow, tuple):
                off, ten = allow
            else:
                if len(allow) != nq:
                    raise ValueError("one allowlist per query")
                lens = np.array([len(a) for a in allow], np.int64)
                off_h = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
                ten_h = (np.concatenate([np.asarray(a, np.uint32).reshape(-1) for a in allow])
                         if off_h[-1] else np.zeros(1, np.uint32))
                off = torch.from_numpy(off_h).to(self.device)
                ten = torch.from_numpy(ten_h.view(np.int32)).to(self.device)
        if stream is not None:  # inputs made on the current stream, used on `stream`
            stream.wait_stream(torch.cuda.current_stream(self.device))
            for t in (Q, off, ten):
                _used_on(t, stream)
        return search(Q, self.R, self.centroids, self.bits, self.codes[: self.n], self.scale[: self.n], k,
                      filter=self.filter if allow is not None else None, allow_off=off, allow_tenants=ten,
                      workspace=workspace, stream=stream, idmap=self.id_map, calib=self.calib)

    # ----------------------------------------------------------- persistence
    def save(self, path: str) -> None:
        """Writes the index (tables, codes, scales, tenants, id map) to one
        flat file; waits for the device work queued so far."""
        torch = _torch()
        torch.cuda.synchronize(self.device)
        n = self.n
        fields = {"format": "turboquant-index", "version": FORMAT_VERSION, "d": self.d, "bits": self.bits,
                  "n": n, "seed": self.seed, "marginal": self.marginal, "scale_mode": self.scale_mode,
                  "block": self.block, "id_map": self.id_map is not None, "tenants": self.tenant_ids is not None,
                  "tq_plus": self.tq_plus}
        arrays = {"R": self.R.cpu().numpy(), "centroids": self.centroids.cpu().numpy(),
                  "boundaries": self.boundaries.cpu().numpy(), "codes": self.codes[:n].cpu().numpy(),
                  "scale": self.scale[:n].cpu().numpy()}
        if self.tenant_ids is not None:
            arrays["tenant_ids"] = self.tenant_ids[:n].cpu().numpy().view(np.uint32)
        if self.id_map is not None:
            arrays["ext_ids"], arrays["deleted"] = self.id_map.export()
        if self.calib is not None:
            arrays["calib_mu"], arrays["calib_a"] = (t.cpu().numpy() for t in self.calib)
        flatfile.write(path, fields, arrays)

    @classmethod
    def load(cls, path: str, capacity: int | None = None, device=None) -> "Index":
        """Reads a file written by save() into a new index (capacity defaults
        to the file's row count)."""
        fields, a = flatfile.read(path)
        if fields.get("format") != "turboquant-index" or fields.get("version") != FORMAT_VERSION:
            raise ValueError(f"{path}: unsupported index file ({fields.get('format')} v{fields.get('version')})")
        n = int(fields["n"])
        cap = max(n, 1) if capacity is None else int(capacity)
        if cap < n:
            raise ValueError(f"capacity {cap} < the file's {n} rows")
        idx = cls.__new__(cls)
        torch = _torch()
        idx.device = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
        idx.d, idx.bits, idx.capacity = int(fields["d"]), int(fields["bits"]), cap
        idx.seed, idx.marginal, idx.scale_mode = int(fields["seed"]), fields["marginal"], fields["scale_mode"]
        idx.block, idx.n = int(fields["block"]), n
        rb = row_bytes(idx.d, idx.bits)
        if a["codes"].shape != (n, rb) or a["scale"].shape != (n,) or a["R"].shape != (idx.d, idx.d):
            raise ValueError(f"{path}: array shapes do not match d={idx.d}, bits={idx.bits}, n={n}")
        idx._set_tables(a["R"], a["centroids"], a["boundaries"])
        idx.codes = torch.empty((cap, rb), dtype=torch.uint8, device=idx.device)
        idx.scale = torch.empty(cap, dtype=torch.float32, device=idx.device)
        idx.codes[:n].copy_(torch.from_numpy(a["codes"]))
        idx.scale[:n].copy_(torch.from_numpy(a["scale"]))
        idx.tq_plus = bool(fields.get("tq_plus", False))
        idx.calib = None
        if "calib_mu" in a:
            idx.calib = tuple(torch.from_numpy(np.ascontiguousarray(a[k], np.float32)).to(idx.device)
                              for k in ("calib_mu", "calib_a"))
        idx.id_map = None
        if fields["id_map"]:
            idx.id_map = IdMap(cap)
            idx.id_map.import_(a["ext_ids"], a["deleted"])
        idx.tenant_ids, idx.filter = None, None
        if fields["tenants"]:
            idx.tenant_ids = torch.empty(cap, dtype=torch.int32, device=idx.device)
            if n:
                idx.tenant_ids[:n].copy_(torch.from_numpy(a["tenant_ids"].view(np.int32)))
                idx.filter = Filter(idx.tenant_ids[:n], block=idx.block)
        torch.cuda.synchronize(idx.device)
        return idx

    def close(self) -> None:
        if self.filter is not None:
            self.filter.close()
            self.filter = None
        if self.id_map is not None:
            self.id_map.close()


class _null:
    def __enter__(self):
        return self

    def __exit__(self, *exc):
        return False


__all__ = ["Index", "FORMAT_VERSION"]
