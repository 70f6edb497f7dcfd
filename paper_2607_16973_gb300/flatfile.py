"""Flat file format of a persisted index (Sec. III-A: indexes persist to disk).

Layout, all integers little-endian:

    bytes 0-7     magic b"TQINDEX1"
    bytes 8-15    uint64 length L of the header
    bytes 16-     the header: UTF-8 JSON, an object with the index's scalar
                  fields and "arrays": {name: {"dtype", "shape", "offset",
                  "nbytes"}}
    then          each array's raw bytes (C order) at its "offset", a multiple
                  of 64 from the start of the file

Host-only (numpy): writing and reading move no data to or from a device.
"""
from __future__ import annotations

import json
import os
import struct

import numpy as np

MAGIC = b"TQINDEX1"
ALIGN = 64
DTYPES = {"uint8", "uint32", "uint64", "int32", "int64", "float32"}


def _pad(n: int) -> int:
    return (n + ALIGN - 1) // ALIGN * ALIGN


def write(path: str, fields: dict, arrays: dict[str, np.ndarray]) -> None:
    """Writes `fields` (JSON-serialisable scalars) and `arrays` to `path`
    (through a temporary file renamed into place, so a reader never sees a
    partial file)."""
    specs, blobs = {}, []
    # the header's size depends on the offsets it lists: lay the arrays out
    # after a generous header estimate, then check it fits
    est = len(json.dumps({**fields, "arrays": {k: {"dtype": "float32", "shape": list(v.shape),
                                                    "offset": 1 << 62, "nbytes": 1 << 62}
                                                for k, v in arrays.items()}}).encode()) + 64
    off = _pad(16 + est)
    for name, a in arrays.items():
        a = np.ascontiguousarray(a)
        if a.dtype.name not in DTYPES:
            raise TypeError(f"array {name}: dtype {a.dtype} is not one of {sorted(DTYPES)}")
        specs[name] = {"dtype": a.dtype.name, "shape": list(a.shape), "offset": off, "nbytes": int(a.nbytes)}
        blobs.append((off, a))
        off = _pad(off + a.nbytes)
    header = json.dumps({**fields, "arrays": specs}).encode()
    if blobs and 16 + len(header) > blobs[0][0]:
        raise AssertionError("header estimate too small")
    tmp = path + ".tmp"
    with open(tmp, "wb") as f:
        f.write(MAGIC)
        f.write(struct.pack("<Q", len(header)))
        f.write(header)
        for o, a in blobs:
            f.seek(o)
            f.write(a.tobytes())
        f.truncate(off if blobs else 16 + len(header))
    os.replace(tmp, path)


def read(path: str, mmap: bool = False) -> tuple[dict, dict[str, np.ndarray]]:
    """Returns (fields, arrays) of a file written by write().  Raises
    ValueError on a wrong magic, a malformed header or a truncated file.
    mmap=True maps the arrays read-only instead of reading them."""
    size = os.path.getsize(path)
    with open(path, "rb") as f:
        if f.read(8) != MAGIC:
            raise ValueError(f"{path}: not a TurboQuant index file (bad magic)")
        raw = f.read(8)
        if len(raw) != 8:
            raise ValueError(f"{path}: truncated header")
        (hlen,) = struct.unpack("<Q", raw)
        if 16 + hlen > size:
            raise ValueError(f"{path}: truncated header")
        try:
            fields = json.loads(f.read(hlen).decode())
            specs = fields.pop("arrays")
        except (UnicodeDecodeError, json.JSONDecodeError, KeyError) as e:
            raise ValueError(f"{path}: malformed header ({e})") from None
        arrays = {}
        for name, sp in specs.items():
            if sp["dtype"] not in DTYPES:
                raise ValueError(f"{path}: array {name} has unknown dtype {sp['dtype']}")
            dt = np.dtype(sp["dtype"])
            shape = tuple(int(x) for x in sp["shape"])
            nbytes = int(np.prod(shape, dtype=np.int64)) * dt.itemsize
            off = int(sp["offset"])
            if nbytes != sp["nbytes"] or off % ALIGN or off + nbytes > size:
                raise ValueError(f"{path}: array {name} is truncated or inconsistent")
            if nbytes == 0:
                arrays[name] = np.zeros(shape, dt)
            elif mmap:
                arrays[name] = np.memmap(path, dtype=dt, mode="r", offset=off, shape=shape)
            else:
                f.seek(off)
                arrays[name] = np.frombuffer(f.read(nbytes), dtype=dt).reshape(shape).copy()
    return fields, arrays
