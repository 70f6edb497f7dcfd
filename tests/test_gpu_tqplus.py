"""TQ+ calibration (Sec. II-B) on the GPU against the oracle's reading of it.

The paper gives no formula, so the reading itself is unpinned (its pins are
in test_oracle_pins.py); these tests check that the CUDA path computes that
reading: the calibration from a first batch, the calibrated encode, and the
calibrated search on both scans, filtered or not.  Both sides get the
oracle's calibration, rounded to float32, for encode and search.
"""
import json
import os

import numpy as np
import pytest

import oracle as O
from conftest import GOLDEN
from paper_2607_16973_gb300 import synth
from parity import TOL_LUT, TOL_MMA, check_encode, check_topk, recall

pytestmark = pytest.mark.gpu


def _cb(bits):
    with open(os.path.join(GOLDEN, "codebooks.json")) as f:
        e = [e for e in json.load(f)["entries"] if e["bits"] == bits and e["marginal"] == "beta"][0]
    return np.asarray(e["centroids"], np.float32), np.asarray(e["boundaries"], np.float32)


def _skewed_corpus(n, d, seed):
    """Mixture rows with coordinate-dependent offsets and spreads, so that the
    rotated coordinates are off the canonical marginal and TQ+ matters."""
    rng = np.random.default_rng(seed)
    X = synth.mixture_corpus(n, d, 16, seed=seed).astype(np.float64)
    X = X * rng.uniform(0.3, 3.0, d)[None, :] + rng.normal(0, 0.05, d)[None, :]
    return X.astype(np.float32)


@pytest.fixture(scope="module")
def tdev(cuda_lib):
    import torch
    dev = torch.device("cuda:0")
    return torch, dev, (lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev))


@pytest.mark.parametrize("n,d", [(3000, 1536), (257, 96), (1, 64)])
def test_calibrate_parity(cuda_lib, tdev, n, d):
    """Shift and scale from the GPU (fixed summation order) equal the oracle's
    float64 moments: mu to 2e-7 absolute, a to 2e-5 relative.  Zero rows do
    not count; a single row gives a = 1."""
    torch, dev, T = tdev
    tq = cuda_lib
    X = _skewed_corpus(max(n, 2), d, seed=n)[:n]
    if n > 10:
        X[3] = 0.0
        X[n - 1] = 0.0
    R = O.rotation(d, 9).astype(np.float32)
    ref = O.calibrate(X, R)
    mu, a = tq.calibrate(T(X), T(R))
    torch.cuda.synchronize()
    assert np.max(np.abs(mu.cpu().numpy() - ref.mu)) <= 2e-7
    assert np.max(np.abs(a.cpu().numpy() / ref.a - 1)) <= 2e-5
    if n == 1:
        assert np.all(a.cpu().numpy() == 1.0)
    mu2, a2 = tq.calibrate(T(X), T(R))
    assert torch.equal(mu, mu2) and torch.equal(a, a2)  # deterministic


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
@pytest.mark.parametrize("mode", ["norm", "unbiased"])
def test_encode_tqplus_parity(cuda_lib, tdev, bits, mode):
    torch, dev, T = tdev
    tq = cuda_lib
    d, n = 1536, 1300
    X = _skewed_corpus(n, d, seed=3)
    X[7] = 0.0
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(bits)
    cal = O.calibration32(O.calibrate(X[:500], R))
    enc = O.encode(X, R, c32, t32, bits, mode, calib=cal)
    codes, scale = tq.encode(T(X), T(R), T(c32), T(t32), bits, mode,
                             calib=(T(cal.mu.astype(np.float32)), T(cal.a.astype(np.float32))))
    torch.cuda.synchronize()
    check_encode(codes.cpu().numpy(), scale.cpu().numpy(), X, enc, c32, t32, d, bits, mode, calib=cal)


@pytest.fixture(scope="module")
def tqp_corpus(tdev):
    d, n, bits = 1536, 8000, 4
    X = _skewed_corpus(n, d, seed=5)
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(bits)
    cal = O.calibration32(O.calibrate(X[:2000], R))
    enc = O.encode(X, R, c32, t32, bits, calib=cal)
    src = synth.query_sources(n, 60)
    Q = synth.perturb(X[src] / np.linalg.norm(X[src], axis=1, keepdims=True))
    return dict(X=X, R=R, c32=c32, cal=cal, enc=enc, src=src, Q=Q, d=d, n=n, bits=bits)


@pytest.mark.parametrize("path,nq", [("lut", 5), ("lut_fold", 5), ("mma", 60)])
def test_search_tqplus_parity(cuda_lib, tdev, tqp_corpus, path, nq):
    """Calibrated search: the lookup scan and the tensor-core scan add the
    query's term sum_j q'_j mu_j to every raw score before the per-vector
    scale, on queries pre-scaled by a."""
    torch, dev, T = tdev
    tq = cuda_lib
    c = tqp_corpus
    cal = c["cal"]
    calib = (T(cal.mu.astype(np.float32)), T(cal.a.astype(np.float32)))
    k = 10
    tq.set_search_path(path)
    try:
        ids, sc = tq.search(T(c["Q"][:nq]), T(c["R"]), T(c["c32"]), c["bits"], T(c["enc"].packed),
                            T(c["enc"].scale), k, calib=calib)
        torch.cuda.synchronize()
    finally:
        tq.set_search_path("auto")
    ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
    ref = O.search(c["Q"][:nq], c["R"], c["c32"], c["bits"], c["enc"].packed, c["enc"].scale, k, c["d"], calib=cal)
    check_topk(ids, sc, ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k,
               TOL_LUT if path.startswith("lut") else TOL_MMA)
    exact, _ = O.exact_knn(c["X"], c["Q"][:nq], k)
    assert abs(recall(ids, exact) - recall(ref.ids, exact)) <= 0.002


def test_search_tqplus_filtered(cuda_lib, tdev, tqp_corpus):
    torch, dev, T = tdev
    tq = cuda_lib
    c = tqp_corpus
    cal = c["cal"]
    nq, k = 6, 8
    tid, values = synth.zipf_tenants(c["n"], 50)
    off, allow = synth.allowlists(c["src"][:nq], tid, values)
    filt = tq.Filter(T(tid.view(np.int32)))
    try:
        ids, sc = tq.search(T(c["Q"][:nq]), T(c["R"]), T(c["c32"]), c["bits"], T(c["enc"].packed),
                            T(c["enc"].scale), k, filter=filt, allow_off=T(off), allow_tenants=T(allow.view(np.int32)),
                            calib=(T(cal.mu.astype(np.float32)), T(cal.a.astype(np.float32))))
        torch.cuda.synchronize()
    finally:
        filt.close()
    ref = O.search(c["Q"][:nq], c["R"], c["c32"], c["bits"], c["enc"].packed, c["enc"].scale, k, c["d"], tid, off,
                   allow, calib=cal)
    check_topk(ids.cpu().numpy(), sc.cpu().numpy(), ref.ids, ref.scores64,
               O.allowed_mask(tid, off, allow, nq, c["n"]), k, TOL_LUT)


def test_index_tqplus_ingest_and_persist(cuda_lib, tdev, tmp_path):
    """An Index with tq_plus=True fits its calibration on the first batch (equal
    to the oracle's within the calibration tolerances), encodes every later
    batch with it exactly as one calibrated tq_encode of all rows does, and
    saves and reloads to identical searches."""
    torch, dev, T = tdev
    tq = cuda_lib
    d, bits, k = 256, 4, 10
    X = _skewed_corpus(3000, d, seed=8)
    idx = tq.Index(d, bits, capacity=4000, tq_plus=True)
    idx.add(X[:1200])
    idx.add(X[1200:])
    ref = O.calibrate(X[:1200], idx.R.cpu().numpy())
    mu, a = (t.cpu().numpy() for t in idx.calib)
    assert np.max(np.abs(mu - ref.mu)) <= 2e-7 and np.max(np.abs(a / ref.a - 1)) <= 2e-5
    codes, scale = tq.encode(T(X), idx.R, idx.centroids, idx.boundaries, bits, calib=idx.calib,
                             plan=idx.plan)
    torch.cuda.synchronize()
    assert torch.equal(codes, idx.codes[:3000]) and torch.equal(scale, idx.scale[:3000])
    Q = T(synth.perturb(X[:7] / np.linalg.norm(X[:7], axis=1, keepdims=True)))
    ids, sc = idx.search(Q, k)
    path = str(tmp_path / "tqp.idx")
    idx.save(path)
    back = tq.Index.load(path)
    ids2, sc2 = back.search(Q, k)
    torch.cuda.synchronize()
    assert back.tq_plus and torch.equal(ids, ids2) and torch.equal(sc, sc2)
    idx.close()
    back.close()
