"""Full-size parity on sampled outputs: the 999,000 x 1536 4-bit workload in
the launch configurations the benchmark times (batch 1 and batch 1024, top-5).

The oracle cannot search every query at this size, so it checks sampled
queries (each a full float64 scan of the corpus) and sampled encoded rows.
"""
import numpy as np
import pytest

import oracle as O
from paper_2607_16973_gb300 import synth
from parity import TOL_LUT, TOL_MMA, check_encode, check_topk

pytestmark = pytest.mark.gpu

N, D, BITS, K = 999_000, 1536, 4, 5


@pytest.fixture(scope="module")
def corpus(cuda_lib):
    """Random codes and scales (every byte pattern is a valid 4-bit row)."""
    import torch
    dev = torch.device("cuda:0")
    packed = synth.random_codes(N, D * BITS // 8, seed=999)
    scale = synth.random_scales(N, seed=999)
    R = O.rotation(D, synth.SEED_ROTATION).astype(np.float32)
    cb = O.codebook(D, BITS)
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    return dict(packed=packed, scale=scale, R=R, c32=cb.centroids32, t32=cb.boundaries32,
                d_packed=T(packed), d_scale=T(scale), d_R=T(R), d_c=T(cb.centroids32), T=T)


@pytest.mark.parametrize("batch,sampled,tol", [(1, [0], TOL_LUT), (1024, [0, 517, 1023], TOL_MMA)])
def test_fullsize_search_sampled(cuda_lib, corpus, batch, sampled, tol):
    """Batch 1 runs the lookup scan, batch 1024 the tensor-core scan (AUTO)."""
    import torch
    tq = cuda_lib
    c = corpus
    Q = synth.gaussian_rows(batch, D, seed=batch)
    Q /= np.linalg.norm(Q, axis=1, keepdims=True)   # unit queries, as in the workload
    ids, sc = tq.search(c["T"](Q), c["d_R"], c["d_c"], BITS, c["d_packed"], c["d_scale"], K)
    torch.cuda.synchronize()
    ids, sc = ids.cpu().numpy(), sc.cpu().numpy()
    assert np.all(ids >= 0) and np.all(ids < N)
    for q in sampled:
        ref = O.search(Q[q:q + 1], c["R"], c["c32"], BITS, c["packed"], c["scale"], K, D)
        check_topk(ids[q:q + 1], sc[q:q + 1], ref.ids, ref.scores64, np.ones((1, N), bool), K, tol)


def test_fullsize_encode_sampled_rows(cuda_lib, corpus):
    """Encode all 999,000 rows of the mixture corpus on the GPU; the oracle
    re-encodes sampled rows (first, last, panel edges, random)."""
    import torch
    tq = cuda_lib
    c = corpus
    X = synth.mixture_corpus(N, D, 1024, workers=16)
    codes, scale = tq.encode(c["T"](X), c["d_R"], c["d_c"], c["T"](c["t32"]), BITS)
    torch.cuda.synchronize()
    rng = np.random.default_rng(5)
    rows = np.unique(np.concatenate([[0, 127, 128, N - 1, N - 24, N - 25],
                                     rng.integers(0, N, 120)]))
    enc = O.encode(X[rows], c["R"], c["c32"], c["t32"], BITS)
    check_encode(codes[torch.from_numpy(rows).cuda()].cpu().numpy(), scale.cpu().numpy()[rows], X[rows], enc,
                 c["c32"], c["t32"], D, BITS, "norm")
