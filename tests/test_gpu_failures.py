"""Failure paths on the GPU, exercised without faulting it: an injected
device-allocation failure comes back as TQ_ENOMEM and leaks nothing, and a
bounded wait that can never be satisfied gives up, is reported by
tq_search_check as TQ_ETIMEOUT, and leaves the context usable."""
import numpy as np
import pytest

import oracle as O
from paper_2607_16973_gb300 import synth
from parity import TOL_LUT, check_topk

pytestmark = pytest.mark.gpu


def test_injected_allocation_failure_is_enomem(cuda_lib):
    import torch
    tq = cuda_lib
    dev = torch.device("cuda:0")
    tid = torch.from_numpy(np.arange(1000, dtype=np.uint32).view(np.int32) % 7).to(dev)
    free0 = torch.cuda.mem_get_info()[0]
    for count in (1, 2, 3):
        tq.load().tq_debug_fail_allocs(count)
        with pytest.raises(tq.TQError, match="TQ_ENOMEM"):
            tq.Filter(tid)
        tq.load().tq_debug_fail_allocs(0)
    f = tq.Filter(tid)  # allocations work again
    assert f.info()["n_tenants"] == 7
    f.close()
    torch.cuda.synchronize()
    assert abs(torch.cuda.mem_get_info()[0] - free0) < (8 << 20)


def test_allocation_failure_in_idmap_and_filter_growth(cuda_lib):
    """An id map that cannot allocate either of its device arrays is
    TQ_ENOMEM; a filter whose growth cannot allocate (in place of doubling, or
    of a rebuild for a new tenant) is TQ_ENOMEM and left exactly as it was."""
    import torch
    tq = cuda_lib
    dev = torch.device("cuda:0")
    tid = torch.from_numpy((np.arange(2000, dtype=np.uint32) % 7).view(np.int32)).to(dev)
    extra = torch.full((10,), 99, dtype=torch.int32, device=dev)
    # run every path once first: a first launch of a kernel or a copy can
    # reserve device memory for good, which is not a leak
    warm = tq.Filter(tid[:1000])
    warm.append(tid[1000:1500])
    warm.append(extra)
    warm.close()
    tq.IdMap(1000).close()
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for count in (1, 2):
        tq.load().tq_debug_fail_allocs(count)
        with pytest.raises(tq.TQError, match="TQ_ENOMEM"):
            tq.IdMap(1000)
        tq.load().tq_debug_fail_allocs(0)
    f = tq.Filter(tid[:1000])
    for new in (tid[1000:1500], extra):  # grow, rebuild
        for count in (1, 2):
            tq.load().tq_debug_fail_allocs(count)
            with pytest.raises(tq.TQError, match="TQ_ENOMEM"):
                f.append(new)
            tq.load().tq_debug_fail_allocs(0)
            assert f.info() == {"n": 1000, "block": 64, "n_tenants": 7}
    f.append(tid[1000:2000])
    assert f.info()["n"] == 2000
    f.close()
    torch.cuda.synchronize()
    assert abs(torch.cuda.mem_get_info()[0] - free0) < (8 << 20)


def test_bounded_wait_timeout_is_reported_and_context_survives(cuda_lib):
    import torch
    tq = cuda_lib
    dev = torch.device("cuda:0")
    n, d, bits, k, nq = 3000, 256, 4, 10, 3
    packed = synth.random_codes(n, d * bits // 8, seed=21)
    scale = synth.random_scales(n, seed=22)
    R = O.rotation(d, 9).astype(np.float32)
    cb = O.codebook(d, bits)
    Q = synth.gaussian_rows(nq, d, seed=23)
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    args = (T(Q), T(R), T(cb.centroids32), bits, T(packed), T(scale), k)
    ws = torch.empty(tq.search_workspace(nq, n, d, bits, k), dtype=torch.uint8, device=dev)
    ids0, sc0 = tq.search(*args, workspace=ws)
    tq.search_check(ws)                                  # a normal search: TQ_OK
    # a wait on an mbarrier nothing completes, budget ~1 ms of SM clock
    tq._lib.check(tq.load().tq_debug_bounded_wait(2_000_000, ws.data_ptr(), None))
    with pytest.raises(tq.TQError, match="TQ_ETIMEOUT.*site 99"):
        tq.search_check(ws)
    ids1, sc1 = tq.search(*args, workspace=ws)           # the next search clears the word
    tq.search_check(ws)
    assert torch.equal(ids0, ids1) and torch.equal(sc0, sc1)
    ref = O.search(Q, R, cb.centroids32, bits, packed, scale, k, d)
    check_topk(ids1.cpu().numpy(), sc1.cpu().numpy(), ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k,
               TOL_LUT)
