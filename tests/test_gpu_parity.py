"""Parity of the CUDA path with the oracle, element by element, on seeded
inputs the oracle finishes in seconds (several tiles plus ragged tails), and
the edge cases of the method.  Every call goes through the C ABI."""
import json
import os

import numpy as np
import pytest

import oracle as O
from paper_2607_16973_gb300 import synth
from conftest import GOLDEN
from parity import TOL_LUT, TOL_MMA, check_encode, check_topk, recall

pytestmark = pytest.mark.gpu


def _cb(d, bits, marginal="beta"):
    if d == 1536:
        with open(os.path.join(GOLDEN, "codebooks.json")) as f:
            e = [e for e in json.load(f)["entries"] if e["bits"] == bits and e["marginal"] == marginal][0]
        return np.asarray(e["centroids"], np.float32), np.asarray(e["boundaries"], np.float32)
    cb = O.codebook(d, bits, marginal)
    return cb.centroids32, cb.boundaries32


@pytest.fixture(scope="module")
def torch_dev(cuda_lib):
    import torch
    return torch, torch.device("cuda:0")


def _t(torch, dev, a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


# ------------------------------------------------------------------- encode --
@pytest.mark.parametrize("bits", [2, 3, 4, 8])
@pytest.mark.parametrize("mode", ["norm", "none", "unbiased"])
def test_encode_parity(cuda_lib, torch_dev, bits, mode):
    torch, dev = torch_dev
    tq = cuda_lib
    d, n = 1536, 2077                       # 16 panels of 128 rows + a ragged 29
    X = synth.mixture_corpus(n, d, 64, seed=42)
    X[5] = 0.0                              # zero row: codes L/2-1, scale 0
    X[6] *= 3.0
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits, mode)
    codes, scale = tq.encode(_t(torch, dev, X), _t(torch, dev, R), _t(torch, dev, c32), _t(torch, dev, t32),
                             bits, mode)
    torch.cuda.synchronize()
    check_encode(codes.cpu().numpy(), scale.cpu().numpy(), X, enc, c32, t32, d, bits, mode)
    assert np.all(codes.cpu().numpy()[5] == enc.packed[5]) and scale.cpu().numpy()[5] == 0.0


@pytest.mark.parametrize("d", [32, 96, 160, 2048])
def test_encode_parity_dims(cuda_lib, torch_dev, d):
    torch, dev = torch_dev
    tq = cuda_lib
    n, bits = 300, 4
    X = synth.mixture_corpus(n, d, 8, seed=7)
    R = O.rotation(d, 11).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits)
    codes, scale = tq.encode(_t(torch, dev, X), _t(torch, dev, R), _t(torch, dev, c32), _t(torch, dev, t32), bits)
    torch.cuda.synchronize()
    check_encode(codes.cpu().numpy(), scale.cpu().numpy(), X, enc, c32, t32, d, bits, "norm")


def test_encode_empty_and_single(cuda_lib, torch_dev):
    torch, dev = torch_dev
    tq = cuda_lib
    d, bits = 64, 4
    R = O.rotation(d, 3).astype(np.float32)
    c32, t32 = _cb(d, bits)
    X = synth.mixture_corpus(1, d, 2, seed=1)
    enc = O.encode(X, R, c32, t32, bits)
    codes, scale = tq.encode(_t(torch, dev, X), _t(torch, dev, R), _t(torch, dev, c32), _t(torch, dev, t32), bits)
    check_encode(codes.cpu().numpy(), scale.cpu().numpy(), X, enc, c32, t32, d, bits, "norm")
    empty = torch.empty((0, d), dtype=torch.float32, device=dev)
    codes, scale = tq.encode(empty, _t(torch, dev, R), _t(torch, dev, c32), _t(torch, dev, t32), bits)
    assert codes.shape == (0, d * bits // 8)


# ------------------------------------------------------------------- search --
@pytest.fixture(scope="module")
def tiny_config():
    """The tiny exact-check workload: N=10,000, d=1536, 64-component mixture,
    100 perturbed-corpus queries, 4-bit codes, top-10, no filtering."""
    d, n, nq, bits = 1536, 10_000, 100, 4
    X = synth.mixture_corpus(n, d, 64)
    R = O.rotation(d, synth.SEED_ROTATION).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits)
    src = synth.query_sources(n, nq)
    Q = synth.perturb(X[src])
    return dict(X=X, R=R, c32=c32, t32=t32, enc=enc, Q=Q, d=d, n=n, bits=bits)


def _gpu_search(tq, torch, dev, Q, R, c32, bits, packed, scale, k, **kw):
    ids, sc = tq.search(_t(torch, dev, Q), _t(torch, dev, R), _t(torch, dev, c32), bits,
                        _t(torch, dev, packed), None if scale is None else _t(torch, dev, scale), k, **kw)
    torch.cuda.synchronize()
    return ids.cpu().numpy(), sc.cpu().numpy()


@pytest.mark.parametrize("path", ["lut", "lut_fixed", "lut_fold", "mma"])
def test_search_tiny_config(cuda_lib, torch_dev, tiny_config, path):
    torch, dev = torch_dev
    tq = cuda_lib
    c = tiny_config
    k = 10
    tq.set_search_path(path)
    try:
        ids, sc = _gpu_search(tq, torch, dev, c["Q"], c["R"], c["c32"], c["bits"], c["enc"].packed,
                              c["enc"].scale, k)
    finally:
        tq.set_search_path("auto")
    ref = O.search(c["Q"], c["R"], c["c32"], c["bits"], c["enc"].packed, c["enc"].scale, k, c["d"])
    allowed = np.ones_like(ref.scores64, dtype=bool)
    check_topk(ids, sc, ref.ids, ref.scores64, allowed, k, TOL_MMA if path == "mma" else TOL_LUT)
    exact, _ = O.exact_knn(c["X"], c["Q"], k)
    assert abs(recall(ids, exact) - recall(ref.ids, exact)) <= 0.002


@pytest.mark.parametrize("path", ["lut", "mma"])
def test_rag_metrics_tiny_config(cuda_lib, torch_dev, tiny_config, path):
    """Hit@1/3/5/10 and MRR@20 against the exact top-1 (Sec. IV-E, Table III)
    from the CUDA path's top-20 equal the oracle's, up to one query of the
    100 (a near-tie at the exact top-1 may rank differently)."""
    torch, dev = torch_dev
    tq = cuda_lib
    c = tiny_config
    tq.set_search_path(path)
    try:
        ids, _ = _gpu_search(tq, torch, dev, c["Q"], c["R"], c["c32"], c["bits"], c["enc"].packed,
                             c["enc"].scale, 20)
    finally:
        tq.set_search_path("auto")
    ref = O.search(c["Q"], c["R"], c["c32"], c["bits"], c["enc"].packed, c["enc"].scale, 20, c["d"])
    exact, _ = O.exact_knn(c["X"], c["Q"], 1)
    one = 1.0 / len(c["Q"]) + 1e-9
    for kk in (1, 3, 5, 10):
        assert abs(O.hit_at_k(ids, exact, kk) - O.hit_at_k(ref.ids, exact, kk)) <= one
    assert abs(O.mrr_at(ids, exact, 20) - O.mrr_at(ref.ids, exact, 20)) <= one
    assert O.hit_at_k(ref.ids, exact, 10) > 0.9  # the workload is retrievable at 4 bits


@pytest.mark.parametrize("bits,path", [(2, "lut"), (3, "lut"), (8, "lut"), (2, "mma"), (3, "mma"), (8, "mma")])
def test_search_bit_widths(cuda_lib, torch_dev, bits, path):
    torch, dev = torch_dev
    tq = cuda_lib
    d, n, nq, k = 1536, 4000, 20, 10
    X = synth.mixture_corpus(n, d, 64, seed=42)
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits)
    Q = synth.perturb(X[synth.query_sources(n, nq)])
    tq.set_search_path(path)
    try:
        ids, sc = _gpu_search(tq, torch, dev, Q, R, c32, bits, enc.packed, enc.scale, k)
    finally:
        tq.set_search_path("auto")
    ref = O.search(Q, R, c32, bits, enc.packed, enc.scale, k, d)
    check_topk(ids, sc, ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k,
               TOL_LUT if path == "lut" else TOL_MMA)


@pytest.mark.parametrize("d,n,nq,k", [(32, 5, 3, 10), (64, 64 * 3 + 17, 9, 7), (96, 1000, 8, 1),
                                      (160, 777, 2, 256), (512, 2000, 3, 10), (2048, 1500, 1, 5)])
@pytest.mark.parametrize("path", ["auto", "lut_fixed"])
def test_search_shapes_and_edges(cuda_lib, torch_dev, d, n, nq, k, path):
    """n below one block, ragged blocks, small d (lanes idle), k = 1 and 256,
    the GEMV (nq <= 8) and GEMM (nq > 8) query rotations, d = 2048, both
    4-bit tables (the fixed-point one from d = 512 on).  The exact table
    takes raw Gaussian queries (norms up to 45); the fixed-point one takes
    unit queries, as in the workloads (its error scales with the query norm)."""
    torch, dev = torch_dev
    tq = cuda_lib
    bits = 4
    packed = synth.random_codes(n, d * bits // 8, seed=d)
    scale = synth.random_scales(n, seed=n)
    scale[0] = 0.0
    R = O.rotation(d, 5).astype(np.float32)
    c32, _ = _cb(d, bits)
    Q = synth.gaussian_rows(nq, d, seed=nq)
    if path == "lut_fixed":
        Q /= np.linalg.norm(Q, axis=1, keepdims=True)
    tq.set_search_path(path)
    try:
        ids, sc = _gpu_search(tq, torch, dev, Q, R, c32, bits, packed, scale, k)
    finally:
        tq.set_search_path("auto")
    ref = O.search(Q, R, c32, bits, packed, scale, k, d)
    check_topk(ids, sc, ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k, TOL_LUT)


@pytest.mark.parametrize("d,marginal,bound", [(512, "beta", 1e-5), (1536, "beta", 3e-6), (1536, "gauss", 3e-6)])
def test_fixed_point_table_error(cuda_lib, torch_dev, d, marginal, bound):
    """The fixed-point 4-bit table against the float64 oracle on unit queries:
    256 results per query, each within `bound` of the oracle's score, and the
    exact fp32 table within 1e-6.  The fixed-point error is the centroids'
    rounding to the table's step (about 2^-16 of the largest centroid, which
    grows as 1/sqrt(d)) weighted by the rotated query: about 1.2e-6 rms at
    d = 512 and 2.5e-7 at d = 1536 for random codes."""
    torch, dev = torch_dev
    tq = cuda_lib
    bits, n, nq, k = 4, 6000, 24, 256
    packed = synth.random_codes(n, d * bits // 8, seed=d + 1)
    scale = synth.random_scales(n, seed=d + 1)
    R = O.rotation(d, 6).astype(np.float32)
    c32 = _cb(d, bits, marginal)[0]
    Q = synth.gaussian_rows(nq, d, seed=d + 2)
    Q /= np.linalg.norm(Q, axis=1, keepdims=True)
    ref = O.search(Q, R, c32, bits, packed, scale, k, d)
    for path, tol in (("lut_fixed", bound), ("lut", 1e-6)):
        tq.set_search_path(path)
        try:
            ids, sc = _gpu_search(tq, torch, dev, Q, R, c32, bits, packed, scale, k)
        finally:
            tq.set_search_path("auto")
        check_topk(ids, sc, ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k, tol)


def test_search_unit_scale_and_ties(cuda_lib, torch_dev):
    """scale=NULL means 1; duplicated rows tie exactly and come back by id."""
    torch, dev = torch_dev
    tq = cuda_lib
    d, bits, k = 64, 4, 6
    packed = synth.random_codes(300, d * bits // 8, seed=3)
    packed = np.concatenate([packed, packed[[17, 17, 250]]])
    R = O.rotation(d, 2).astype(np.float32)
    c32, _ = _cb(d, bits)
    C = c32.astype(np.float64)[O.unpack(packed, d, bits)]
    Q = (C[17] @ R.astype(np.float64))[None].astype(np.float32)   # R q = c[row 17]
    ids, sc = _gpu_search(tq, torch, dev, Q, R, c32, bits, packed, None, k)
    ref = O.search(Q, R, c32, bits, packed, None, k, d)
    check_topk(ids, sc, ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k, TOL_LUT)
    assert ids[0][:3].tolist() == [17, 300, 301]


# ---------------------------------------------------------------- filtering --
@pytest.fixture(scope="module")
def filtered_corpus():
    d, n, bits = 1536, 20_000, 4
    X = synth.mixture_corpus(n, d, 256, seed=42)
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits)
    src = synth.query_sources(n, 200)
    Q = synth.perturb(X[src])
    return dict(X=X, R=R, c32=c32, enc=enc, src=src, Q=Q, d=d, n=n, bits=bits)


@pytest.mark.parametrize("T", [10, 100, 1000])
@pytest.mark.parametrize("block", [64, 32])
@pytest.mark.parametrize("path", ["lut", "lut_fold"])
def test_filtered_search(cuda_lib, torch_dev, filtered_corpus, T, block, path):
    """Zipf(1.1) tenants in interleaved order; 1 allowed tenant per query, 10%
    of queries with 5 (Sec. III-B, the filtered workload).  The query-folded
    scan runs one CTA per query here: four passes of 6,656 rows each."""
    torch, dev = torch_dev
    tq = cuda_lib
    c = filtered_corpus
    k = 10
    tid, values = synth.zipf_tenants(c["n"], T)
    off, allow = synth.allowlists(c["src"], tid, values)
    filt = tq.Filter(_t(torch, dev, tid.view(np.int32)), block=block)
    assert filt.info() == {"n": c["n"], "block": block, "n_tenants": T}
    tq.set_search_path(path)  # a lookup scan (a batch of 200 would take the tensor-core scan)
    try:
        ids, sc = _gpu_search(tq, torch, dev, c["Q"], c["R"], c["c32"], c["bits"], c["enc"].packed,
                              c["enc"].scale, k, filter=filt, allow_off=_t(torch, dev, off),
                              allow_tenants=_t(torch, dev, allow.view(np.int32)))
    finally:
        tq.set_search_path("auto")
    ref = O.search(c["Q"], c["R"], c["c32"], c["bits"], c["enc"].packed, c["enc"].scale, k, c["d"],
                   tid, off, allow)
    allowed = O.allowed_mask(tid, off, allow, len(c["Q"]), c["n"])
    check_topk(ids, sc, ref.ids, ref.scores64, allowed, k, TOL_LUT)
    exact, _ = O.exact_knn(c["X"], c["Q"], k, tid, off, allow)
    assert abs(recall(ids, exact) - recall(ref.ids, exact)) <= 0.002
    filt.close()


@pytest.mark.parametrize("path", ["lut", "lut_fixed", "lut_fold"])
def test_filter_every_tenant_equals_unfiltered(cuda_lib, torch_dev, filtered_corpus, path):
    """At d = 1536, with each 4-bit lookup scan: allowing every tenant gives
    the unfiltered search bit for bit (the same operations on every score)."""
    torch, dev = torch_dev
    tq = cuda_lib
    c = filtered_corpus
    k, nq = 10, 40
    tid, values = synth.zipf_tenants(c["n"], 100)
    off = np.arange(nq + 1, dtype=np.int64) * len(values)
    allow = np.tile(values, nq)
    filt = tq.Filter(_t(torch, dev, tid.view(np.int32)), block=64)
    tq.set_search_path(path)
    try:
        ids_f, sc_f = _gpu_search(tq, torch, dev, c["Q"][:nq], c["R"], c["c32"], c["bits"], c["enc"].packed,
                                  c["enc"].scale, k, filter=filt, allow_off=_t(torch, dev, off),
                                  allow_tenants=_t(torch, dev, allow.view(np.int32)))
        ids_u, sc_u = _gpu_search(tq, torch, dev, c["Q"][:nq], c["R"], c["c32"], c["bits"], c["enc"].packed,
                                  c["enc"].scale, k)
    finally:
        tq.set_search_path("auto")
        filt.close()
    assert np.array_equal(ids_f, ids_u) and np.array_equal(sc_f, sc_u)


def test_filter_edge_cases(cuda_lib, torch_dev):
    """Empty allowlists, ids absent from the corpus, a tenant smaller than k,
    and a filter allowing every tenant equal to no filter."""
    torch, dev = torch_dev
    tq = cuda_lib
    d, n, bits, k = 64, 500, 4, 12
    packed = synth.random_codes(n, d * bits // 8, seed=9)
    scale = synth.random_scales(n, seed=9)
    R = O.rotation(d, 9).astype(np.float32)
    c32, _ = _cb(d, bits)
    tid = np.full(n, 7, np.uint32)
    tid[::50] = 99                           # a tenant of 10 vectors (< k)
    tid[3] = 12345
    Q = synth.gaussian_rows(4, d, seed=4)
    off = np.array([0, 0, 1, 3, 5], np.int64)
    allow = np.array([99, 555, 12345, 7, 99], np.uint32)
    filt = tq.Filter(_t(torch, dev, tid.view(np.int32)), block=32)
    ids, sc = _gpu_search(tq, torch, dev, Q, R, c32, bits, packed, scale, k, filter=filt,
                          allow_off=_t(torch, dev, off), allow_tenants=_t(torch, dev, allow.view(np.int32)))
    ref = O.search(Q, R, c32, bits, packed, scale, k, d, tid, off, allow)
    allowed = O.allowed_mask(tid, off, allow, 4, n)
    check_topk(ids, sc, ref.ids, ref.scores64, allowed, k, TOL_LUT)
    assert np.all(ids[0] == -1)              # empty allowlist
    assert np.sum(ids[1] >= 0) == 10         # tenant of 10 vectors, k = 12
    # every tenant allowed == unfiltered
    off2 = np.array([0, 3, 6, 9, 12], np.int64)
    allow2 = np.tile(np.array([7, 99, 12345], np.uint32), 4)
    ids_f, sc_f = _gpu_search(tq, torch, dev, Q, R, c32, bits, packed, scale, k, filter=filt,
                              allow_off=_t(torch, dev, off2), allow_tenants=_t(torch, dev, allow2.view(np.int32)))
    ids_u, sc_u = _gpu_search(tq, torch, dev, Q, R, c32, bits, packed, scale, k)
    assert np.array_equal(ids_f, ids_u) and np.array_equal(sc_f, sc_u)
    filt.close()


def test_invalid_calls_on_gpu(cuda_lib, torch_dev):
    torch, dev = torch_dev
    tq = cuda_lib
    d, bits = 64, 4
    Q = torch.zeros((2, d), device=dev)
    R = torch.eye(d, device=dev)
    c = torch.zeros(16, device=dev)
    codes = torch.zeros((10, 32), dtype=torch.uint8, device=dev)
    with pytest.raises(tq.TQError, match="workspace"):
        tq.search(Q, R, c, bits, codes, None, 5, workspace=torch.zeros(16, dtype=torch.uint8, device=dev))
    tid = torch.zeros(11, dtype=torch.int32, device=dev)
    f = tq.Filter(tid)
    with pytest.raises(tq.TQError, match="filter built for n=11"):
        tq.search(Q, R, c, bits, codes, None, 5, filter=f, allow_off=torch.zeros(3, dtype=torch.int64, device=dev),
                  allow_tenants=torch.zeros(1, dtype=torch.int32, device=dev))
    f.close()


# ------------------------------------------------------- tensor-core scan --
@pytest.mark.parametrize("bits,d,n,nq,k", [(4, 1536, 3000, 130, 10), (2, 1536, 1000, 17, 5),
                                           (8, 1536, 777, 64, 8), (4, 64, 513, 200, 1),
                                           (4, 2048, 2049, 129, 64), (4, 128, 255, 1, 3),
                                           (8, 1536, 777, 300, 8), (4, 1536, 1500, 257, 5),
                                           (3, 1536, 1000, 17, 5), (3, 1536, 777, 300, 8), (3, 256, 600, 40, 10)])
def test_search_mma_parity(cuda_lib, torch_dev, bits, d, n, nq, k):
    """Query tiles of 128 with a ragged last tile, vector tiles of 256 with a
    ragged tail (rows past n are filled with zeros by the tensor map), one
    query, k = 1 and 64, 2/3/4/8-bit codes (fp16 products, float32 sums)."""
    torch, dev = torch_dev
    tq = cuda_lib
    packed = synth.random_codes(n, d * bits // 8, seed=bits * n)
    scale = synth.random_scales(n, seed=n + 1)
    R = O.rotation(d, 7).astype(np.float32)
    c32, _ = _cb(d, bits)
    Q = synth.gaussian_rows(nq, d, seed=nq + d)
    Q /= np.linalg.norm(Q, axis=1, keepdims=True)   # unit queries, as in the workloads (fp16 error ~ |q|)
    tq.set_search_path("mma")
    try:
        ids, sc = _gpu_search(tq, torch, dev, Q, R, c32, bits, packed, scale, k)
    finally:
        tq.set_search_path("auto")
    ref = O.search(Q, R, c32, bits, packed, scale, k, d)
    check_topk(ids, sc, ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k, TOL_MMA)


@pytest.mark.parametrize("path,nq", [("lut", 40), ("mma", 3500)])
def test_search_rotation_splits(cuda_lib, torch_dev, path, nq):
    """The tensor-core query rotation (batches of 16 or more) with its
    contraction split over several CTAs (40 queries: one query tile, many
    splits, and the lookup scan's float32 tolerance) and with one split
    writing the rotated queries directly (3,500 queries: 28 query tiles)."""
    torch, dev = torch_dev
    tq = cuda_lib
    d, n, bits, k = 1536, 1200, 4, 10
    packed = synth.random_codes(n, d * bits // 8, seed=nq)
    scale = synth.random_scales(n, seed=nq + 1)
    R = O.rotation(d, 13).astype(np.float32)
    c32, _ = _cb(d, bits)
    Q = synth.gaussian_rows(nq, d, seed=nq + 2)
    Q /= np.linalg.norm(Q, axis=1, keepdims=True)
    tq.set_search_path(path)
    try:
        ids, sc = _gpu_search(tq, torch, dev, Q, R, c32, bits, packed, scale, k)
    finally:
        tq.set_search_path("auto")
    ref = O.search(Q, R, c32, bits, packed, scale, k, d)
    check_topk(ids, sc, ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k,
               TOL_LUT if path == "lut" else TOL_MMA)


def test_search_mma_unsupported(cuda_lib, torch_dev):
    """Forcing the tensor-core scan where it does not apply is an error, not a
    silent switch: k > 64, d not a multiple of 64 (of 128 for 3-bit codes)."""
    torch, dev = torch_dev
    tq = cuda_lib
    tq.set_search_path("mma")
    try:
        for bits, d, k in ((3, 160, 5), (4, 1536, 65), (4, 96, 5)):
            Q = torch.zeros((4, d), device=dev)
            R = torch.eye(d, device=dev)
            c = torch.zeros(1 << bits, device=dev)
            codes = torch.zeros((100, d * bits // 8), dtype=torch.uint8, device=dev)
            with pytest.raises(tq.TQError, match="TQ_EUNSUPPORTED"):
                tq.search(Q, R, c, bits, codes, None, k)
    finally:
        tq.set_search_path("auto")


def test_search_on_side_stream_keeps_its_temporaries(cuda_lib, torch_dev):
    """search() on a side stream with library-made workspace and outputs: the
    caller then allocates and fills blocks of the same sizes on its current
    stream while the scan is still running.  The temporaries belong to the
    side stream's pool, so the results equal a search run alone."""
    torch, dev = torch_dev
    tq = cuda_lib
    d, n, bits, k, nq = 1536, 300_000, 4, 10, 48
    packed = synth.random_codes(n, d * bits // 8, seed=31)
    scale = synth.random_scales(n, seed=31)
    R = O.rotation(d, 5).astype(np.float32)
    c32, _ = _cb(d, bits)
    Q = synth.gaussian_rows(nq, d, seed=31)
    Qd, Rd, cd, pd, sd = (_t(torch, dev, a) for a in (Q, R, c32, packed, scale))
    tq.set_search_path("lut")  # one full corpus pass per query: milliseconds of work
    try:
        want_i, want_s = tq.search(Qd, Rd, cd, bits, pd, sd, k)
        torch.cuda.synchronize()
        want_i, want_s = want_i.cpu(), want_s.cpu()
        ws_bytes = tq.search_workspace(nq, n, d, bits, k)
        side = torch.cuda.Stream(device=dev)
        side.wait_stream(torch.cuda.current_stream())
        for _ in range(3):
            got_i, got_s = tq.search(Qd, Rd, cd, bits, pd, sd, k, stream=side)
            junk = [torch.full((ws_bytes,), 255, dtype=torch.uint8, device=dev),
                    torch.full((nq, k), -5, dtype=torch.int64, device=dev),
                    torch.full((nq, k), 9.0, dtype=torch.float32, device=dev)]
            side.synchronize()
            assert torch.equal(got_i.cpu(), want_i) and torch.equal(got_s.cpu(), want_s)
            del junk
    finally:
        tq.set_search_path("auto")


@pytest.mark.parametrize("bits,filtered,nq", [(4, False, 1), (4, False, 5), (3, False, 2), (2, False, 1),
                                              (4, True, 3), (8, True, 1)])
def test_search_on_created_stream_matches_default_stream(cuda_lib, torch_dev, filtered_corpus, bits, filtered, nq):
    """On a created stream the lookup scan is launched as a programmatic
    dependent of the kernel before it (its prologue overlaps that kernel's
    tail) and merges in its last CTA; the results equal the default-stream
    search (no overlap) bit for bit, in back-to-back searches and with the
    scan bracketed by profiling events."""
    torch, dev = torch_dev
    tq = cuda_lib
    c = filtered_corpus
    d, n, k = c["d"], 12_000, 10
    packed = synth.random_codes(n, d * bits // 8, seed=bits + nq)
    scale = synth.random_scales(n, seed=bits)
    c32, _ = _cb(d, bits)
    Qd, Rd, cd = _t(torch, dev, c["Q"][:nq]), _t(torch, dev, c["R"]), _t(torch, dev, c32)
    pd, sd = _t(torch, dev, packed), _t(torch, dev, scale)
    kw = {}
    if filtered:
        tid, values = synth.zipf_tenants(n, 100)
        off, allow = synth.allowlists(np.arange(nq), tid, values)
        kw = dict(filter=tq.Filter(_t(torch, dev, tid.view(np.int32))), allow_off=_t(torch, dev, off),
                  allow_tenants=_t(torch, dev, allow.view(np.int32)))
    tq.set_search_path("lut")
    try:
        want_i, want_s = tq.search(Qd, Rd, cd, bits, pd, sd, k, **kw)
        torch.cuda.synchronize()
        side = torch.cuda.Stream(device=dev)
        side.wait_stream(torch.cuda.current_stream())
        ws = torch.empty(tq.search_workspace(nq, n, d, bits, k, kw.get("filter")), dtype=torch.uint8, device=dev)
        outs = []
        for rep in range(4):
            if rep == 3:
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                tq.profile_events(e0, e1)
            try:
                outs.append(tq.search(Qd, Rd, cd, bits, pd, sd, k, workspace=ws, stream=side, **kw))
            finally:
                tq.profile_events(None, None)
            tq.search_check(ws, stream=side)
        side.synchronize()
        for i, s_ in outs:
            assert torch.equal(i, want_i) and torch.equal(s_, want_s)
    finally:
        tq.set_search_path("auto")
        if filtered:
            kw["filter"].close()
    ref = O.search(c["Q"][:nq], c["R"], c32, bits, packed, scale, k, d, *(
        (tid, off, allow) if filtered else ()))
    allowed = O.allowed_mask(tid, off, allow, nq, n) if filtered else np.ones((nq, n), bool)
    check_topk(want_i.cpu().numpy(), want_s.cpu().numpy(), ref.ids, ref.scores64, allowed, k, TOL_LUT)


@pytest.mark.parametrize("filtered,nq,pinned", [(False, 7, True), (True, 7, True), (False, 7, False),
                                                (False, 40, True), (True, 40, False)])
def test_search_host_buffers(cuda_lib, torch_dev, filtered_corpus, filtered, nq, pinned):
    """tq_search_host (queries from host memory, results back to host memory,
    all queued by the library on one stream) returns what tq_search on device
    buffers returns, bit for bit: page-locked buffers used in place (the
    queries only below 16 per batch), pageable ones through the staging
    copies."""
    torch, dev = torch_dev
    tq = cuda_lib
    c = filtered_corpus
    k = 10
    args = (_t(torch, dev, c["R"]), _t(torch, dev, c["c32"]), c["bits"], _t(torch, dev, c["enc"].packed),
            _t(torch, dev, c["enc"].scale), k)
    kw = {}
    if filtered:
        tid, values = synth.zipf_tenants(c["n"], 100)
        off, allow = synth.allowlists(c["src"][:nq], tid, values)
        kw = dict(filter=tq.Filter(_t(torch, dev, tid.view(np.int32))), allow_off=_t(torch, dev, off),
                  allow_tenants=_t(torch, dev, allow.view(np.int32)))
    pin = (lambda t: t.pin_memory()) if pinned else (lambda t: t)
    Qh = pin(torch.from_numpy(c["Q"][:nq].copy()))
    ih = pin(torch.full((nq, k), 3, dtype=torch.int64))
    sh = pin(torch.full((nq, k), 3.0, dtype=torch.float32))
    side = torch.cuda.Stream(device=dev)
    try:
        tq.search_from_host(Qh, *args, ih, sh, stream=side, **kw)
        side.synchronize()
        want_i, want_s = tq.search(Qh.to(dev), *args, **kw)
        torch.cuda.synchronize()
    finally:
        if filtered:
            kw["filter"].close()
    assert torch.equal(ih, want_i.cpu()) and torch.equal(sh, want_s.cpu())


@pytest.mark.parametrize("T,nq,k", [(10, 200, 10), (100, 200, 10), (1000, 200, 10), (100, 40, 64)])
def test_filtered_search_mma(cuda_lib, torch_dev, filtered_corpus, T, nq, k):
    """Filtered batches on the tensor-core scan: the epilogue drops a vector
    whose tenant the query does not allow before it can enter the query's
    list (Sec. III-B).  Two query tiles (nq = 200) and one (nq = 40, k = 64)."""
    torch, dev = torch_dev
    tq = cuda_lib
    c = filtered_corpus
    tid, values = synth.zipf_tenants(c["n"], T)
    off, allow = synth.allowlists(c["src"][:nq], tid, values)
    filt = tq.Filter(_t(torch, dev, tid.view(np.int32)), block=64)
    tq.set_search_path("mma")
    try:
        ids, sc = _gpu_search(tq, torch, dev, c["Q"][:nq], c["R"], c["c32"], c["bits"], c["enc"].packed,
                              c["enc"].scale, k, filter=filt, allow_off=_t(torch, dev, off),
                              allow_tenants=_t(torch, dev, allow.view(np.int32)))
    finally:
        tq.set_search_path("auto")
        filt.close()
    ref = O.search(c["Q"][:nq], c["R"], c["c32"], c["bits"], c["enc"].packed, c["enc"].scale, k, c["d"],
                   tid, off, allow)
    allowed = O.allowed_mask(tid, off, allow, nq, c["n"])
    check_topk(ids, sc, ref.ids, ref.scores64, allowed, k, TOL_MMA)
    exact, _ = O.exact_knn(c["X"], c["Q"][:nq], k, tid, off, allow)
    assert abs(recall(ids, exact) - recall(ref.ids, exact)) <= 0.002


def test_filter_every_tenant_equals_unfiltered_mma(cuda_lib, torch_dev, filtered_corpus):
    """On the tensor-core scan, allowing every tenant gives the unfiltered
    result bit for bit (AUTO picks the tensor-core scan for 40 queries)."""
    torch, dev = torch_dev
    tq = cuda_lib
    c = filtered_corpus
    k, nq = 10, 40
    tid, values = synth.zipf_tenants(c["n"], 100)
    off = np.arange(nq + 1, dtype=np.int64) * len(values)
    allow = np.tile(values, nq)
    filt = tq.Filter(_t(torch, dev, tid.view(np.int32)), block=64)
    try:
        ids_f, sc_f = _gpu_search(tq, torch, dev, c["Q"][:nq], c["R"], c["c32"], c["bits"], c["enc"].packed,
                                  c["enc"].scale, k, filter=filt, allow_off=_t(torch, dev, off),
                                  allow_tenants=_t(torch, dev, allow.view(np.int32)))
        ids_u, sc_u = _gpu_search(tq, torch, dev, c["Q"][:nq], c["R"], c["c32"], c["bits"], c["enc"].packed,
                                  c["enc"].scale, k)
    finally:
        filt.close()
    assert np.array_equal(ids_f, ids_u) and np.array_equal(sc_f, sc_u)
