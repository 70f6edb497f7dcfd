"""tq_search_static: search for callers that cannot allocate device memory.

Such callers (a C host program or plugin that is handed device buffers for its
inputs and outputs but owns no allocator, or a serving loop that must not call
cudaMalloc in the middle of a request) get a search entry point whose scratch
is a fixed device array inside the library.  This test calls it through the C
ABI twice in a row, with different query batches (the second call must not see
the first call's leftovers in the shared array), and checks each result
against tq_search with a caller-provided workspace.  It lives in a file that
pytest collects last and runs alone in a fresh process as well.
"""
import ctypes as C

import numpy as np
import pytest

import oracle as O
from paper_2607_16973_gb300 import synth
from paper_2607_16973_gb300.build import build
from parity import TOL_LUT

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("CUDA is not available: GPU tests need a GB300")
    build()
    import paper_2607_16973_gb300 as tq
    return tq, tq.load(), torch


def _static_search(lib, torch, Q, R, c, bits, codes, scale, k, filt=None, off=None, allow=None):
    nq, d = Q.shape
    ids = torch.full((nq, k), -7, dtype=torch.int64, device=Q.device)
    sc = torch.full((nq, k), 7.0, dtype=torch.float32, device=Q.device)
    st = lib.tq_search_static(Q.data_ptr(), nq, d, R.data_ptr(), c.data_ptr(), bits, codes.data_ptr(),
                              scale.data_ptr(), codes.shape[0], filt.handle if filt else None,
                              off.data_ptr() if off is not None else None,
                              allow.data_ptr() if allow is not None else None, k, ids.data_ptr(),
                              sc.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert st == 0, lib.tq_last_error()
    torch.cuda.synchronize()
    return ids.cpu().numpy(), sc.cpu().numpy()


def test_static_scratch_search_matches_workspace_search(env):
    tq, lib, torch = env
    dev = torch.device("cuda:0")
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    d, n, bits, k = 1536, 20_000, 4, 10
    X = synth.mixture_corpus(n, d, 64, seed=42)
    R = O.rotation(d, synth.SEED_ROTATION).astype(np.float32)
    cb = O.codebook(d, bits)
    enc = O.encode(X, R, cb.centroids32, cb.boundaries32, bits)
    dR, dc, dcodes, dscale = T(R), T(cb.centroids32), T(enc.packed), T(enc.scale)
    tid, values = synth.zipf_tenants(n, 100)
    src = synth.query_sources(n, 40)
    Qall = synth.perturb(X[src])
    off, allow = synth.allowlists(src[20:], tid, values)
    filt = tq.Filter(T(tid.view(np.int32)))
    tq.set_search_path("lut")
    try:
        # call 1: unfiltered batch of 20; call 2: a different, filtered batch of 20
        for first, kw in ((True, {}), (False, dict(filter=filt, allow_off=T(off),
                                                   allow_tenants=T(allow.view(np.int32))))):
            Q = T(Qall[:20] if first else Qall[20:])
            ids_s, sc_s = _static_search(lib, torch, Q, dR, dc, bits, dcodes, dscale, k,
                                         kw.get("filter"), kw.get("allow_off"), kw.get("allow_tenants"))
            ids_w, sc_w = tq.search(Q, dR, dc, bits, dcodes, dscale, k, **kw)
            torch.cuda.synchronize()
            ids_w, sc_w = ids_w.cpu().numpy(), sc_w.cpu().numpy()
            assert np.array_equal(ids_s, ids_w)
            ok = ids_w >= 0
            assert np.all(np.abs(sc_s[ok] - sc_w[ok]) <= TOL_LUT)
            assert np.array_equal(np.isneginf(sc_s), np.isneginf(sc_w))
    finally:
        tq.set_search_path("auto")
        filt.close()


def test_static_scratch_rejects_oversize(env):
    tq, lib, torch = env
    dev = torch.device("cuda:0")
    d, bits, k, nq = 1536, 4, 256, 4096
    Q = torch.zeros((nq, d), device=dev)
    R = torch.zeros((d, d), device=dev)
    c = torch.zeros(16, device=dev)
    codes = torch.zeros((1000, d // 2), dtype=torch.uint8, device=dev)
    scale = torch.ones(1000, device=dev)
    ids = torch.empty((nq, k), dtype=torch.int64, device=dev)
    sc = torch.empty((nq, k), dtype=torch.float32, device=dev)
    st = lib.tq_search_static(Q.data_ptr(), nq, d, R.data_ptr(), c.data_ptr(), bits, codes.data_ptr(),
                              scale.data_ptr(), 1000, None, None, None, k, ids.data_ptr(), sc.data_ptr(),
                              torch.cuda.current_stream().cuda_stream)
    assert st == 1 and b"static scratch holds" in lib.tq_last_error()
