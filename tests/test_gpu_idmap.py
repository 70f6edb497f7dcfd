"""Id-mapped index on the GPU (Sec. III-A: external uint64 ids, O(1)
deletion): tq_search_ex through an IdMap against the oracle, on every scan
kernel, and the id map's host semantics."""
import json
import os

import numpy as np
import pytest

import oracle as O
from conftest import GOLDEN
from paper_2607_16973_gb300 import synth
from parity import TOL_LUT, TOL_MMA, check_topk

pytestmark = pytest.mark.gpu


def _t(torch, dev, a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


@pytest.fixture(scope="module")
def torch_dev(cuda_lib):
    import torch
    return torch, torch.device("cuda:0")


def _cb(d, bits):
    """Oracle codebook: the committed oracle output at d = 1536 (the 8-bit
    Lloyd iteration takes minutes), else computed (2-bit only here)."""
    if d == 1536:
        with open(os.path.join(GOLDEN, "codebooks.json")) as f:
            e = [e for e in json.load(f)["entries"] if e["bits"] == bits and e["marginal"] == "beta"][0]
        return np.asarray(e["centroids"], np.float32), np.asarray(e["boundaries"], np.float32)
    cb = O.codebook(d, bits)
    return cb.centroids32, cb.boundaries32


def _ext_ids(n, seed):
    rng = np.random.default_rng(seed)
    ext = rng.choice(1 << 50, size=n, replace=False).astype(np.uint64)
    ext[::3] |= np.uint64(1 << 63)  # ids with the high bit set (negative as int64)
    return ext


def _rows_of(ids, ext):
    """External ids (int64 bit patterns) back to rows; -1 stays -1."""
    to_row = {int(e): r for r, e in enumerate(ext.view(np.int64))}
    return np.vectorize(lambda v: -1 if v == -1 else to_row[int(v)])(ids)


@pytest.mark.parametrize("bits,path,d,n,nq,k", [
    (4, "lut", 1536, 3000, 3, 10),     # byte-pair lookup scan
    (4, "lut_fold", 1536, 3000, 3, 10),  # query-folded lookup scan
    (2, "lut", 256, 1500, 2, 7),       # per-code lookup scan
    (3, "lut", 1536, 700, 2, 5),
    (8, "lut", 1536, 900, 4, 12),
    (4, "mma", 1536, 3000, 130, 10),   # tensor-core scan, two query tiles
    (8, "mma", 1536, 1000, 40, 8),     # one query tile
])
def test_idmap_search_parity(cuda_lib, torch_dev, bits, path, d, n, nq, k):
    torch, dev = torch_dev
    tq = cuda_lib
    X = synth.mixture_corpus(n, d, 16, seed=bits + n)
    R = O.rotation(d, 11).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits)
    src = synth.query_sources(n, nq)
    Q = synth.perturb(X[src])
    rng = np.random.default_rng(n)
    deleted = rng.random(n) < 0.25
    deleted[src[: nq // 2 + 1]] = True  # some queries' own sources are gone
    ext = _ext_ids(n, seed=n)
    m = tq.IdMap(n + 100)
    assert m.add(ext) == 0
    assert m.remove(ext[deleted]) == int(deleted.sum())
    assert m.info() == {"rows": n, "capacity": n + 100, "live": n - int(deleted.sum())}
    tq.set_search_path(path)
    try:
        ids, sc = tq.search(_t(torch, dev, Q), _t(torch, dev, R), _t(torch, dev, c32), bits,
                            _t(torch, dev, enc.packed), _t(torch, dev, enc.scale), k, idmap=m)
        torch.cuda.synchronize()
    finally:
        tq.set_search_path("auto")
    ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
    ref = O.search(Q, R, c32, bits, enc.packed, enc.scale, k, d, deleted=deleted, ext_ids=ext)
    allowed = np.broadcast_to(~deleted, (nq, n))
    check_topk(_rows_of(ids, ext), sc, _rows_of(ref.ids, ext), ref.scores64, allowed, k,
               TOL_LUT if path.startswith("lut") else TOL_MMA)
    m.close()


def test_idmap_filtered_and_incremental_delete(cuda_lib, torch_dev):
    """A tenant filter and tombstones together; a removal queued on the
    search stream is seen by the next search; deleting every row pads."""
    torch, dev = torch_dev
    tq = cuda_lib
    d, n, bits, k, T = 1536, 4000, 4, 10, 10
    X = synth.mixture_corpus(n, d, 32, seed=3)
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits)
    src = synth.query_sources(n, 8)
    Q = synth.perturb(X[src])
    tid, values = synth.zipf_tenants(n, T)
    off, allow = synth.allowlists(src, tid, values)
    ext = _ext_ids(n, seed=5)
    m = tq.IdMap(n)
    m.add(ext)
    filt = tq.Filter(_t(torch, dev, tid.view(np.int32)), block=64)
    args = (_t(torch, dev, Q), _t(torch, dev, R), _t(torch, dev, c32), bits, _t(torch, dev, enc.packed),
            _t(torch, dev, enc.scale), k)
    fkw = dict(filter=filt, allow_off=_t(torch, dev, off), allow_tenants=_t(torch, dev, allow.view(np.int32)),
               idmap=m)
    deleted = np.zeros(n, bool)
    for step in range(3):
        ids, sc = tq.search(*args, **fkw)
        ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
        ref = O.search(Q, R, c32, bits, enc.packed, enc.scale, k, d, tid, off, allow, deleted=deleted,
                       ext_ids=ext)
        allowed = O.allowed_mask(tid, off, allow, len(Q), n) & ~deleted[None, :]
        check_topk(_rows_of(ids, ext), sc, _rows_of(ref.ids, ext), ref.scores64, allowed, k, TOL_LUT)
        # delete this search's results before the next one
        gone = np.unique(ids[ids != -1])
        assert m.remove(gone) == len(gone)
        deleted[_rows_of(gone, ext)] = True
    m.remove(ext)  # everything
    ids, sc = tq.search(*args, **fkw)
    assert np.all(ids.cpu().numpy() == -1) and np.all(np.isneginf(sc.cpu().numpy()))
    filt.close()
    m.close()


def test_idmap_host_semantics(cuda_lib):
    tq = cuda_lib
    m = tq.IdMap(8)
    assert m.add(np.array([10, 20, 30], np.uint64)) == 0
    assert [m.lookup(v) for v in (10, 20, 30, 40)] == [0, 1, 2, -1]
    with pytest.raises(tq.TQError, match="already live"):
        m.add(np.array([40, 20], np.uint64))            # 20 is live: nothing added
    assert m.lookup(40) == -1 and m.info()["rows"] == 3
    with pytest.raises(tq.TQError, match="already live"):
        m.add(np.array([50, 50], np.uint64))            # twice in one batch
    with pytest.raises(tq.TQError, match="empty result slots"):
        m.add(np.array([-1], np.int64))
    assert m.remove(np.array([20, 99], np.uint64)) == 1  # 99 is not live
    assert m.lookup(20) == -1
    assert m.add(np.array([20], np.uint64)) == 3         # re-added as a new row
    assert m.lookup(20) == 3
    assert m.info() == {"rows": 4, "capacity": 8, "live": 3}   # 10, 30 and the new 20
    with pytest.raises(tq.TQError, match="capacity"):
        m.add(np.arange(100, 105, dtype=np.uint64))
    assert m.add(np.arange(100, 104, dtype=np.uint64)) == 4
    big = np.uint64((1 << 64) - 2)
    m2 = tq.IdMap(1)
    m2.add(np.array([big], np.uint64))
    assert m2.lookup(int(big)) == 0
    m2.close()
    m.close()


def test_idmap_shorter_than_corpus_rejected(cuda_lib, torch_dev):
    torch, dev = torch_dev
    tq = cuda_lib
    d = 64
    m = tq.IdMap(10)
    m.add(np.arange(5, dtype=np.uint64))
    with pytest.raises(ValueError, match="id map holds 5 rows"):
        tq.search(torch.zeros((1, d), device=dev), torch.eye(d, device=dev), torch.zeros(16, device=dev), 4,
                  torch.zeros((10, 32), dtype=torch.uint8, device=dev), None, 3, idmap=m)
    m.close()
