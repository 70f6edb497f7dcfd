"""tq_search_static: search for callers that cannot allocate device memory.

Such callers (a C host program or plugin that is handed device buffers for its
inputs and outputs but owns no allocator, or a serving loop that must not call
cudaMalloc in the middle of a request) get a search entry point whose scratch
is a fixed device array inside the library.  This test calls it through the C
ABI twice in a row, with different query batches (the second call must not see
the first call's leftovers in the shared array), and checks each result
against tq_search with a caller-provided workspace and against the oracle.
It checks that a call after the first one on the device takes no device
memory, and runs the comparison once more alone in a fresh process.  It
lives in a file that pytest collects last.
"""
import ctypes as C
import os
import subprocess
import sys

import numpy as np
import pytest

import oracle as O
from paper_2607_16973_gb300 import synth
from paper_2607_16973_gb300.build import build
from parity import TOL_LUT, check_topk

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
            # and against the oracle's search of the same codes
            Qh = Qall[:20] if first else Qall[20:]
            if first:
                ref = O.search(Qh, R, cb.centroids32, bits, enc.packed, enc.scale, k, d)
                allowed = np.ones((20, n), bool)
            else:
                ref = O.search(Qh, R, cb.centroids32, bits, enc.packed, enc.scale, k, d, tid, off, allow)
                allowed = O.allowed_mask(tid, off, allow, 20, n)
            check_topk(ids_s, sc_s, ref.ids, ref.scores64, allowed, k, TOL_LUT)
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


def test_static_scratch_call_takes_no_device_memory(env):
    """After the first call on the device (which may reserve the array), a
    call leaves the device's free memory exactly as it was."""
    tq, lib, torch = env
    dev = torch.device("cuda:0")
    d, n, bits, k, nq = 256, 5000, 4, 8, 12
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    packed = T(synth.random_codes(n, d * bits // 8, seed=12))
    scale = T(synth.random_scales(n, seed=12))
    R = T(O.rotation(d, 3).astype(np.float32))
    c = T(O.codebook(d, bits).centroids32)
    Q = T(synth.gaussian_rows(nq, d, seed=12))
    first = _static_search(lib, torch, Q, R, c, bits, packed, scale, k)
    ids = torch.empty((nq, k), dtype=torch.int64, device=dev)
    sc = torch.empty((nq, k), dtype=torch.float32, device=dev)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    st = lib.tq_search_static(Q.data_ptr(), nq, d, R.data_ptr(), c.data_ptr(), bits, packed.data_ptr(),
                              scale.data_ptr(), n, None, None, None, k, ids.data_ptr(), sc.data_ptr(),
                              torch.cuda.current_stream().cuda_stream)
    assert st == 0, lib.tq_last_error()
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert np.array_equal(ids.cpu().numpy(), first[0])


def test_static_scratch_fresh_process(env):
    """The comparison above, alone in a new process: the first call there is
    also the first on the device."""
    if os.environ.get("TQ_NO_ALLOC_CHILD"):
        pytest.skip("already the child process")
    here = os.path.dirname(os.path.abspath(__file__))
    envv = dict(os.environ, TQ_NO_ALLOC_CHILD="1")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-p", "no:cacheprovider", "-m", "gpu",
                        os.path.join(here, "test_zz_no_alloc.py"), "-k", "matches_workspace_search"],
                       cwd=os.path.dirname(here), env=envv, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "1 passed" in r.stdout
