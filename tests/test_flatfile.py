"""The flat index file format (persistence, Sec. III-A) on the host: round
trips, 64-byte alignment, and rejection of damaged files."""
import json
import struct

import numpy as np
import pytest

from paper_2607_16973_gb300 import flatfile


def _arrays():
    rng = np.random.default_rng(0)
    return {"R": rng.standard_normal((32, 32)).astype(np.float32),
            "codes": rng.integers(0, 256, (77, 16), dtype=np.uint8),
            "scale": rng.random(77).astype(np.float32),
            "ext_ids": rng.integers(0, 2**63, 77, dtype=np.int64).view(np.uint64) | np.uint64(1 << 63),
            "deleted": np.array([5, 0, 1 << 31], np.uint32),
            "empty": np.zeros((0, 16), np.uint8)}


@pytest.mark.parametrize("mmap", [False, True])
def test_round_trip(tmp_path, mmap):
    p = str(tmp_path / "a.tqi")
    arrays = _arrays()
    fields = {"format": "turboquant-index", "version": 1, "d": 32, "n": 77, "marginal": "beta"}
    flatfile.write(p, fields, arrays)
    f2, a2 = flatfile.read(p, mmap=mmap)
    assert f2 == fields
    assert set(a2) == set(arrays)
    for k, v in arrays.items():
        assert a2[k].dtype == v.dtype and a2[k].shape == v.shape and np.array_equal(a2[k], v), k


def test_layout_is_aligned_and_documented(tmp_path):
    p = str(tmp_path / "b.tqi")
    flatfile.write(p, {"x": 1}, _arrays())
    raw = open(p, "rb").read()
    assert raw[:8] == b"TQINDEX1"
    (hlen,) = struct.unpack("<Q", raw[8:16])
    hdr = json.loads(raw[16:16 + hlen])
    for name, sp in hdr["arrays"].items():
        assert sp["offset"] % 64 == 0 and sp["offset"] >= 16 + hlen
        blob = raw[sp["offset"]:sp["offset"] + sp["nbytes"]]
        assert blob == np.ascontiguousarray(_arrays()[name]).tobytes()


def test_damaged_files_rejected(tmp_path):
    p = str(tmp_path / "c.tqi")
    flatfile.write(p, {"x": 1}, _arrays())
    raw = open(p, "rb").read()
    bad = tmp_path / "bad.tqi"
    bad.write_bytes(b"NOTANIDX" + raw[8:])
    with pytest.raises(ValueError, match="bad magic"):
        flatfile.read(str(bad))
    bad.write_bytes(raw[: len(raw) - 200])
    with pytest.raises(ValueError, match="truncated"):
        flatfile.read(str(bad))
    bad.write_bytes(raw[:20])
    with pytest.raises(ValueError, match="truncated header"):
        flatfile.read(str(bad))
    (hlen,) = struct.unpack("<Q", raw[8:16])
    bad.write_bytes(raw[:16] + b"{" * hlen + raw[16 + hlen:])
    with pytest.raises(ValueError, match="malformed header"):
        flatfile.read(str(bad))


def test_unsupported_dtype_refused(tmp_path):
    with pytest.raises(TypeError, match="dtype"):
        flatfile.write(str(tmp_path / "d.tqi"), {}, {"x": np.zeros(3, np.float16)})
