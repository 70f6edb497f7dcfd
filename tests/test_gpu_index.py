"""Online ingest and persistence on the GPU (Sec. III-A): an Index built in
pieces equals one built at once (codes, scales, tenant filter, results), its
searches match the oracle, and a saved index loads back to the same results."""
import json
import os

import numpy as np
import pytest

import oracle as O
from conftest import GOLDEN
from paper_2607_16973_gb300 import synth
from parity import TOL_LUT, TOL_MMA, check_encode, check_topk

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch_dev(cuda_lib):
    import torch
    return torch, torch.device("cuda:0")


def _golden_cb(bits):
    with open(os.path.join(GOLDEN, "codebooks.json")) as f:
        e = [e for e in json.load(f)["entries"] if e["bits"] == bits and e["marginal"] == "beta"][0]
    return np.asarray(e["centroids"], np.float32), np.asarray(e["boundaries"], np.float32)


def _rows_of(ids, ext):
    to_row = {int(e): r for r, e in enumerate(ext.view(np.int64))}
    return np.vectorize(lambda v: -1 if v == -1 else to_row[int(v)])(ids)


def test_filter_append_equals_build(cuda_lib, torch_dev):
    """In place, grown and rebuilt (a new tenant) appends give the filter a
    build over all rows gives: same tenant count and identical searches."""
    torch, dev = torch_dev
    tq = cuda_lib
    d, n, bits, k = 64, 3000, 4, 10
    packed = synth.random_codes(n, d * bits // 8, seed=4)
    scale = synth.random_scales(n, seed=4)
    R = O.rotation(d, 3).astype(np.float32)
    cb = O.codebook(d, bits)
    tid = np.random.default_rng(1).choice(np.array([7, 11, 13, 99], np.uint32), n)
    tid[2500:] = np.where(tid[2500:] == 7, 12345, tid[2500:])  # a tenant first seen at row 2500
    cuts = [0, 700, 1100, 1300, 2500, 3000]                    # grow, in place, grow, rebuild
    t = torch.from_numpy(tid.view(np.int32)).to(dev)
    f = tq.Filter(t[:cuts[1]], block=32)
    for a, b in zip(cuts[1:-1], cuts[2:]):
        f.append(t[a:b])
    assert f.info() == {"n": n, "block": 32, "n_tenants": 5}
    g = tq.Filter(t, block=32)
    Q = torch.from_numpy(synth.gaussian_rows(6, d, seed=2)).to(dev)
    off = torch.tensor([0, 1, 2, 4, 5, 6, 8], dtype=torch.int64, device=dev)
    allow = torch.from_numpy(np.array([7, 12345, 11, 13, 99, 5, 7, 12345], np.uint32).view(np.int32)).to(dev)
    args = (Q, torch.from_numpy(R).to(dev), torch.from_numpy(cb.centroids32).to(dev), bits,
            torch.from_numpy(packed).to(dev), torch.from_numpy(scale).to(dev), k)
    a_ids, a_sc = tq.search(*args, filter=f, allow_off=off, allow_tenants=allow)
    b_ids, b_sc = tq.search(*args, filter=g, allow_off=off, allow_tenants=allow)
    assert torch.equal(a_ids, b_ids) and torch.equal(a_sc, b_sc)
    ref = O.search(Q.cpu().numpy(), R, cb.centroids32, bits, packed, scale, k, d, tid, off.cpu().numpy(),
                   allow.cpu().numpy().view(np.uint32))
    allowed = O.allowed_mask(tid, off.cpu().numpy(), allow.cpu().numpy().view(np.uint32), 6, n)
    check_topk(a_ids.cpu().numpy(), a_sc.cpu().numpy(), ref.ids, ref.scores64, allowed, k, TOL_LUT)
    f.close()
    g.close()


@pytest.mark.parametrize("d,bits,chunks", [(1536, 4, [1000, 1, 2999]), (32, 2, [3, 5, 700])])
def test_index_ingest_in_pieces(cuda_lib, torch_dev, d, bits, chunks):
    """Rows added in pieces (including offsets off the 16-byte grid at d=32,
    2 bits) encode exactly as one encode of all rows (with the index's
    tensor-core plan where d allows one: a row's codes do not depend on the
    batch it came in)."""
    torch, dev = torch_dev
    tq = cuda_lib
    n = sum(chunks)
    X = synth.mixture_corpus(n, d, 8, seed=d)
    idx = tq.Index(d, bits, capacity=n + 10)
    r0 = 0
    for m in chunks:
        assert idx.add(X[r0:r0 + m]) == r0
        r0 += m
    assert (idx.plan is not None) == (d == 1536)
    codes, scale = tq.encode(torch.from_numpy(X).to(dev), idx.R, idx.centroids, idx.boundaries, bits,
                             plan=idx.plan)
    torch.cuda.synchronize()
    assert torch.equal(idx.codes[:n], codes) and torch.equal(idx.scale[:n], scale)
    with pytest.raises(ValueError, match="capacity"):
        idx.add(X[:11])
    idx.close()


def test_index_search_delete_filter_and_persist(cuda_lib, torch_dev, tmp_path):
    """An id-mapped, tenant-filtered index grown in three pieces: its searches
    match the oracle (deleted rows never returned, ids external), and after
    save/load the results are identical and ingest continues."""
    torch, dev = torch_dev
    tq = cuda_lib
    d, bits, k = 1536, 4, 10
    n = 5000
    X = synth.mixture_corpus(n, d, 64, seed=9)
    tid, values = synth.zipf_tenants(n, 20)
    ext = np.random.default_rng(3).choice(1 << 60, n, replace=False).astype(np.uint64)
    # the rotation and codebook are inputs to both sides: the oracle's
    c32, t32 = _golden_cb(bits)
    R = O.rotation(d, synth.SEED_ROTATION).astype(np.float32)
    idx = tq.Index(d, bits, capacity=8000, id_map=True, tenants=True, block=64, tables=(R, c32, t32))
    for a, b in [(0, 1200), (1200, 1201), (1201, n)]:
        idx.add(X[a:b], ids=ext[a:b], tenant_ids=tid[a:b])
    # the index's codes are the oracle's up to boundary-window flips; rows with
    # a flip score differently on the two sides, so they are deleted along
    # with a random 600 and no search below can return them
    enc = O.encode(X, R, c32, t32, bits)
    gpu_codes = idx.codes[:n].cpu().numpy()
    check_encode(gpu_codes, idx.scale[:n].cpu().numpy(), X, enc, c32, t32, d, bits, "norm")
    flipped = np.nonzero(np.any(gpu_codes != enc.packed, axis=1))[0]
    gone = np.union1d(np.random.default_rng(4).choice(n, 600, replace=False), flipped)
    assert idx.remove(ext[gone]) == len(gone)
    assert len(idx) == n and idx.live == n - len(gone)
    src = synth.query_sources(n, 12)
    Q = synth.perturb(X[src])
    off, allow = synth.allowlists(src, tid, values)
    allow_lists = [allow[off[q]:off[q + 1]] for q in range(len(Q))]
    ids, sc = idx.search(Q, k, allow=allow_lists)
    ids_u, sc_u = idx.search(Q, k)  # no allowlist: every tenant
    # oracle: its own encoding of the same rows, the same deletions and ids
    deleted = np.zeros(n, bool)
    deleted[gone] = True
    ref = O.search(Q, R, c32, bits, enc.packed, enc.scale, k, d, tid, off, allow, deleted=deleted, ext_ids=ext)
    allowed = O.allowed_mask(tid, off, allow, len(Q), n) & ~deleted[None, :]
    check_topk(_rows_of(ids.cpu().numpy(), ext), sc.cpu().numpy(), _rows_of(ref.ids, ext), ref.scores64,
               allowed, k, TOL_LUT)
    ref_u = O.search(Q, R, c32, bits, enc.packed, enc.scale, k, d, deleted=deleted, ext_ids=ext)
    check_topk(_rows_of(ids_u.cpu().numpy(), ext), sc_u.cpu().numpy(), _rows_of(ref_u.ids, ext),
               ref_u.scores64, np.broadcast_to(~deleted, (len(Q), n)), k, TOL_LUT)
    # tensor-core path through the index (batch >= 16, no allowlist)
    Qb = synth.perturb(X[synth.query_sources(n, 40)])
    tq.set_search_path("mma")
    try:
        ids_b, sc_b = idx.search(Qb, k)
    finally:
        tq.set_search_path("auto")
    ref_b = O.search(Qb, R, c32, bits, enc.packed, enc.scale, k, d, deleted=deleted, ext_ids=ext)
    check_topk(_rows_of(ids_b.cpu().numpy(), ext), sc_b.cpu().numpy(), _rows_of(ref_b.ids, ext),
               ref_b.scores64, np.broadcast_to(~deleted, (len(Qb), n)), k, TOL_MMA)
    # persistence
    path = str(tmp_path / "index.tqi")
    idx.save(path)
    back = tq.Index.load(path, capacity=8000)
    assert len(back) == n and back.live == n - len(gone)
    ids2, sc2 = back.search(Q, k, allow=allow_lists)
    assert torch.equal(ids, ids2) and torch.equal(sc, sc2)
    live_row = int(np.setdiff1d(np.arange(n), gone)[0])
    assert back.id_map.lookup(int(ext[gone[0]])) == -1 and back.id_map.lookup(int(ext[live_row])) == live_row
    # ingest continues after a load: a new tenant and new ids
    extra = synth.mixture_corpus(100, d, 4, seed=77)
    back.add(extra, ids=np.arange(100, dtype=np.uint64) + np.uint64(1 << 62),
             tenant_ids=np.full(100, 4242, np.uint32))
    ids3, _ = back.search(extra[:3], 1, allow=[[4242]] * 3)
    assert ids3.cpu().numpy()[:, 0].tolist() == [(1 << 62) + i for i in range(3)]
    for x in (idx, back):
        x.close()


def test_index_rejected_ids_leave_it_unchanged(cuda_lib, torch_dev):
    torch, dev = torch_dev
    tq = cuda_lib
    d = 64
    X = synth.mixture_corpus(20, d, 2, seed=6)
    idx = tq.Index(d, 4, capacity=100, id_map=True)
    idx.add(X[:10], ids=np.arange(10, dtype=np.uint64))
    with pytest.raises(tq.TQError, match="already live"):
        idx.add(X[10:15], ids=np.array([10, 11, 3, 12, 13], np.uint64))
    assert len(idx) == 10 and idx.live == 10 and idx.id_map.info()["rows"] == 10
    assert idx.add(X[10:15], ids=np.arange(10, 15, dtype=np.uint64)) == 10
    ids, _ = idx.search(X[[12]], 1)
    assert ids.cpu().numpy().tolist() == [[12]]
    idx.close()
