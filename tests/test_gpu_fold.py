"""The query-folded 4-bit lookup scan (k_scan_fold, TQ_PATH_LUT_FOLD) against
the oracle's float64 search (Sec. II-B step 5, Sec. III-B), element by
element within the lookup scans' 1e-5.  The cases reach: one and several
slices of 256 coordinates, a last slice cut short (d = 288, 1824: the TMA
box reads past the row's end, which fills zeros, and those positions' tables
are zero), the largest d, rows not filling a 32-row tile, CTAs that run
several 6,656-row passes (the accumulators reused), one row, k = 1 and the
largest k, and the cases the scan refuses."""
import json
import os

import numpy as np
import pytest

import oracle as O
from conftest import GOLDEN
from paper_2607_16973_gb300 import synth
from parity import TOL_LUT, check_topk

pytestmark = pytest.mark.gpu


def _cb(d, bits=4):
    if d == 1536:
        with open(os.path.join(GOLDEN, "codebooks.json")) as f:
            e = [e for e in json.load(f)["entries"] if e["bits"] == bits and e["marginal"] == "beta"][0]
        return np.asarray(e["centroids"], np.float32), np.asarray(e["boundaries"], np.float32)
    cb = O.codebook(d, bits, "beta")
    return cb.centroids32, cb.boundaries32


@pytest.fixture(scope="module")
def tdev(cuda_lib):
    import torch
    dev = torch.device("cuda:0")
    return torch, (lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev))


def _fold_search(tq, torch, T, Q, R, c32, packed, scale, k):
    tq.set_search_path("lut_fold")
    try:
        ids, sc = tq.search(T(Q), T(R), T(c32), 4, T(packed), None if scale is None else T(scale), k)
        torch.cuda.synchronize()
    finally:
        tq.set_search_path("auto")
    return ids.cpu().numpy(), sc.cpu().numpy()


# (d, n, nq, k): with nq queries each query gets 152 // nq CTAs (at least
# one), so nq = 15 over 70,001 rows gives CTAs of 7,008 rows: two passes
@pytest.mark.parametrize("d,n,nq,k", [
    (256, 70_001, 15, 10),    # one slice, two passes per CTA
    (288, 5_000, 1, 1),       # two slices, the second 16 bytes wide
    (1536, 20_000, 1, 32),    # six slices, largest k
    (1536, 3_001, 4, 10),     # ragged last tile
    (1824, 2_000, 2, 5),      # eight slices, the last 16 bytes wide
    (2048, 600, 1, 10),       # the largest d a search takes: eight full slices
    (512, 1, 1, 10),          # one row: k - 1 empty slots
    (512, 31, 3, 7),          # less than one tile
])
def test_fold_parity(cuda_lib, tdev, d, n, nq, k):
    torch, T = tdev
    tq = cuda_lib
    packed = synth.random_codes(n, d // 2, seed=d + n)
    scale = synth.random_scales(n, seed=n)
    scale[0] = 0.0
    R = O.rotation(d, 5).astype(np.float32)
    c32, _ = _cb(d)
    Q = synth.gaussian_rows(nq, d, seed=nq)
    Q /= np.linalg.norm(Q, axis=1, keepdims=True)
    ids, sc = _fold_search(tq, torch, T, Q, R, c32, packed, scale, k)
    ref = O.search(Q, R, c32, 4, packed, scale, k, d)
    check_topk(ids, sc, ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k, TOL_LUT)
    if n < k:
        assert np.all(ids[:, n:] == -1) and np.all(np.isneginf(sc[:, n:]))


def test_fold_encoded_corpus_agrees_with_byte_pair_scan(cuda_lib, tdev):
    """On an encoded corpus (the scale workload's distribution, 40,000 rows)
    both 4-bit lookup scans return the oracle's top-10 within 1e-5, and their
    scores agree with each other to the same bound."""
    torch, T = tdev
    tq = cuda_lib
    d, n, nq, k = 1536, 40_000, 6, 10
    X = synth.mixture_corpus(n, d, 64, seed=17)
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(d)
    enc = O.encode(X, R, c32, t32, 4)
    Q = synth.perturb(X[synth.query_sources(n, nq)])
    ids_f, sc_f = _fold_search(tq, torch, T, Q, R, c32, enc.packed, enc.scale, k)
    tq.set_search_path("lut")
    try:
        ids_l, sc_l = tq.search(T(Q), T(R), T(c32), 4, T(enc.packed), T(enc.scale), k)
        torch.cuda.synchronize()
    finally:
        tq.set_search_path("auto")
    ids_l, sc_l = ids_l.cpu().numpy(), sc_l.cpu().numpy()
    ref = O.search(Q, R, c32, 4, enc.packed, enc.scale, k, d)
    ones = np.ones_like(ref.scores64, bool)
    check_topk(ids_f, sc_f, ref.ids, ref.scores64, ones, k, TOL_LUT)
    check_topk(ids_l, sc_l, ref.ids, ref.scores64, ones, k, TOL_LUT)
    assert np.max(np.abs(sc_f - sc_l)) <= 2 * TOL_LUT


def test_fold_unsupported(cuda_lib, tdev):
    """Forced onto shapes it does not take (2-bit codes, d < 256, k > 32),
    the query-folded path refuses with TQ_EUNSUPPORTED; AUTO still serves
    them with another scan."""
    torch, T = tdev
    tq = cuda_lib
    for bits, d, k in ((2, 512, 10), (4, 128, 10), (4, 512, 33)):
        n = 100
        packed = synth.random_codes(n, d * bits // 8, seed=1)
        scale = synth.random_scales(n, seed=1)
        R = O.rotation(d, 3).astype(np.float32)
        c32 = O.codebook(d, bits, "beta").centroids32
        Q = synth.gaussian_rows(1, d, seed=2)
        tq.set_search_path("lut_fold")
        try:
            with pytest.raises(tq.TQError) as ei:
                tq.search(T(Q), T(R), T(c32), bits, T(packed), T(scale), k)
            assert ei.value.status == tq.TQ_EUNSUPPORTED
        finally:
            tq.set_search_path("auto")
        ids, sc = tq.search(T(Q), T(R), T(c32), bits, T(packed), T(scale), k)
        torch.cuda.synchronize()
        ref = O.search(Q, R, c32, bits, packed, scale, k, d)
        check_topk(ids.cpu().numpy(), sc.cpu().numpy(), ref.ids, ref.scores64,
                   np.ones_like(ref.scores64, bool), k, TOL_LUT)
