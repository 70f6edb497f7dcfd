"""Sharded search on one GPU: tq_merge_topk against the ranking rule on
random candidate lists, and S row shards searched separately and merged
against the unsharded search and the oracle.  The multi-rank exchange itself
is covered on the CPU (gloo) in test_shard.py; here one NCCL rank drives
sharded_search end to end."""
import os
import socket

import numpy as np
import pytest

import oracle as O
from paper_2607_16973_gb300 import synth
from paper_2607_16973_gb300.shard import shard_rows, to_global
from parity import TOL_LUT, TOL_MMA, check_topk, merge_candidates

pytestmark = pytest.mark.gpu


def _t(torch, dev, a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


@pytest.mark.parametrize("S,nq,m,k", [(1, 3, 5, 10), (3, 4, 10, 10), (8, 2, 300, 256), (2, 5, 0, 4),
                                      (4, 1, 64, 1), (16, 3, 256, 256)])
def test_merge_topk_matches_ranking_rule(cuda_lib, S, nq, m, k):
    """Random lists with -1 padding and tied scores (ids break ties); more
    candidates than one merge pass holds (chunked) in the larger cases."""
    import torch
    tq = cuda_lib
    dev = torch.device("cuda:0")
    rng = np.random.default_rng(S * 1000 + m)
    ids = np.empty((S, nq, m), np.int64)
    for q in range(nq):
        ids[:, q, :] = rng.permutation(10 * S * m + 1)[:S * m].reshape(S, m)
    sc = rng.integers(-20, 20, size=(S, nq, m)).astype(np.float32) / 4  # many ties
    pad = rng.random((S, nq, m)) < 0.2
    ids[pad] = -1
    sc[pad] = -np.inf
    gi, gs = tq.merge_topk(_t(torch, dev, ids), _t(torch, dev, sc), k)
    torch.cuda.synchronize()
    ri, rs = merge_candidates(ids, sc, k)
    np.testing.assert_array_equal(gi.cpu().numpy(), ri)
    np.testing.assert_array_equal(gs.cpu().numpy(), rs)


def _corpus(n, d, bits, seed):
    packed = synth.random_codes(n, d * bits // 8, seed=seed)
    scale = synth.random_scales(n, seed=seed + 1)
    R = O.rotation(d, 9).astype(np.float32)
    cb = O.codebook(d, bits)
    return packed, scale, R, cb.centroids32


@pytest.mark.parametrize("S", [2, 3, 5])
@pytest.mark.parametrize("path,nq", [("lut", 2), ("mma", 32)])
def test_shards_merged_equal_unsharded(cuda_lib, S, path, nq):
    """Row shards searched one by one, ids shifted, merged: the same ids and
    scores as one search of the whole corpus (a row's score does not depend
    on which rows share its launch), and within tolerance of the oracle."""
    import torch
    tq = cuda_lib
    dev = torch.device("cuda:0")
    n, d, bits, k = 20_000, 512, 4, 10
    packed, scale, R, c32 = _corpus(n, d, bits, seed=S)
    Q = synth.gaussian_rows(nq, d, seed=nq)
    Q /= np.linalg.norm(Q, axis=1, keepdims=True)
    Qd, Rd, cd = _t(torch, dev, Q), _t(torch, dev, R), _t(torch, dev, c32)
    codes, scl = _t(torch, dev, packed), _t(torch, dev, scale)
    tq.set_search_path(path)
    try:
        full_i, full_s = tq.search(Qd, Rd, cd, bits, codes, scl, k)
        parts_i, parts_s = [], []
        for r in range(S):
            lo, hi = shard_rows(n, S, r, 64)
            i, s = tq.search(Qd, Rd, cd, bits, codes[lo:hi], scl[lo:hi], k)
            parts_i.append(to_global(i, lo))
            parts_s.append(s)
        mi, ms = tq.merge_topk(torch.stack(parts_i), torch.stack(parts_s), k)
        torch.cuda.synchronize()
    finally:
        tq.set_search_path("auto")
    np.testing.assert_array_equal(mi.cpu().numpy(), full_i.cpu().numpy())
    np.testing.assert_array_equal(ms.cpu().numpy(), full_s.cpu().numpy())
    ref = O.search(Q, R, c32, bits, packed, scale, k, d)
    check_topk(mi.cpu().numpy(), ms.cpu().numpy(), ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k,
               TOL_LUT if path == "lut" else TOL_MMA)


def test_filtered_shards_merged_equal_oracle(cuda_lib):
    """Tenant filter built per shard; a query whose tenants live in one shard
    gets padding from the others."""
    import torch
    tq = cuda_lib
    dev = torch.device("cuda:0")
    n, d, bits, k, S = 6_000, 256, 4, 10, 3
    packed, scale, R, c32 = _corpus(n, d, bits, seed=77)
    ten = np.full(n, 1, np.uint32)
    ten[::3] = 2
    ten[[4500, 4501, 5999]] = 9
    off = np.array([0, 1, 3, 4], np.int64)
    allow = np.array([9, 1, 9, 2], np.uint32)
    Q = synth.gaussian_rows(3, d, seed=3)
    Qd, Rd, cd = _t(torch, dev, Q), _t(torch, dev, R), _t(torch, dev, c32)
    parts_i, parts_s = [], []
    for r in range(S):
        lo, hi = shard_rows(n, S, r, 64)
        f = tq.Filter(_t(torch, dev, ten[lo:hi].view(np.int32)), block=64)
        i, s = tq.search(Qd, Rd, cd, bits, _t(torch, dev, packed[lo:hi]), _t(torch, dev, scale[lo:hi]), k,
                         filter=f, allow_off=_t(torch, dev, off), allow_tenants=_t(torch, dev, allow.view(np.int32)))
        parts_i.append(to_global(i, lo))
        parts_s.append(s)
    mi, ms = tq.merge_topk(torch.stack(parts_i), torch.stack(parts_s), k)
    torch.cuda.synchronize()
    ref = O.search(Q, R, c32, bits, packed, scale, k, d, ten, off, allow)
    allowed = O.allowed_mask(ten, off, allow, 3, n)
    check_topk(mi.cpu().numpy(), ms.cpu().numpy(), ref.ids, ref.scores64, allowed, k, TOL_LUT)
    assert sorted(mi[0, :3].tolist()) == [4500, 4501, 5999] and mi[0, 3:].eq(-1).all()


def test_sharded_search_one_nccl_rank(cuda_lib):
    """sharded_search through a real NCCL process group of one rank."""
    import torch
    import torch.distributed as dist
    from paper_2607_16973_gb300.shard import sharded_search
    tq = cuda_lib
    dev = torch.device("cuda:0")
    with socket.socket() as s_:
        s_.bind(("127.0.0.1", 0))
        port = s_.getsockname()[1]
    dist.init_process_group("nccl", init_method=f"tcp://127.0.0.1:{port}", rank=0, world_size=1)
    try:
        n, d, bits, k = 3_000, 256, 4, 7
        packed, scale, R, c32 = _corpus(n, d, bits, seed=5)
        Q = synth.gaussian_rows(2, d, seed=8)
        ids, sc = sharded_search(_t(torch, dev, Q), _t(torch, dev, R), _t(torch, dev, c32), bits,
                                 _t(torch, dev, packed), _t(torch, dev, scale), k, offset=0)
        torch.cuda.synchronize()
    finally:
        dist.destroy_process_group()
    ref = O.search(Q, R, c32, bits, packed, scale, k, d)
    check_topk(ids.cpu().numpy(), sc.cpu().numpy(), ref.ids, ref.scores64, np.ones_like(ref.scores64, bool), k,
               TOL_LUT)
