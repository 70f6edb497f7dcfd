"""Comparison helpers for the GPU parity tests (CUDA result vs the oracle).

Tolerances come from what is fixed about this path:
* codes: bit-exact except a coordinate whose rotated value lies within 1e-5 of
  the boundary between the two codes (the GPU forms y in float32 FFMA order);
* scores: 1e-5 absolute on the float32 lookup path, 2e-3 on the fp16
  tensor-core path;
* top-k ids: the same set except among candidates tied with the k-th score
  within the score tolerance; padding (-1, -inf) bit-exact;
* Recall@k: within 0.002 of the oracle's.
"""
import numpy as np

import oracle as O

CODE_WINDOW = 1e-5
TOL_LUT = 1e-5
TOL_MMA = 2e-3


def check_encode(gpu_packed, gpu_scale, X, enc, centroids32, boundaries32, d, bits, mode, calib=None,
                 max_rate=1e-4):
    """Returns the number of boundary-window code flips (all of them checked).
    With a TQ+ calibration (the oracle's, as given to both sides) enc.y holds
    the quantised z and the scalar is checked on the reconstruction a c + mu.
    `max_rate` bounds the fraction of flipped codes: about 2 E|y error| times
    the density of boundaries, so it grows with the bit width."""
    gpu_packed = np.asarray(gpu_packed)
    gpu_scale = np.asarray(gpu_scale)
    assert gpu_packed.shape == enc.packed.shape
    U = O.unpack(gpu_packed, d, bits).astype(np.int64)
    ref = enc.codes.astype(np.int64)
    mism = U != ref
    rows, cols = np.nonzero(mism)
    if len(rows):
        lo = np.minimum(U[rows, cols], ref[rows, cols])
        assert np.all(np.abs(U[rows, cols] - ref[rows, cols]) == 1), "code off by more than one cell"
        y = enc.y[rows, cols]
        assert np.all(np.abs(y - boundaries32[lo].astype(np.float64)) < CODE_WINDOW), \
            "code differs away from a boundary"
    assert mism.mean() < max_rate, f"flip rate {mism.mean():.2e}"
    clean = ~mism.any(axis=1)
    assert np.array_equal(gpu_packed[clean], enc.packed[clean])
    # scale: against the oracle on clean rows, against the definition on the rest
    n = np.linalg.norm(np.asarray(X, np.float64), axis=1)
    c = centroids32.astype(np.float64)[U]
    yy = enc.y
    if calib is not None:
        c = calib.a[None, :] * c + calib.mu[None, :]
        yy = enc.y * calib.a[None, :] + calib.mu[None, :]   # back from z to y
    if mode == "norm":
        cn = np.linalg.norm(c, axis=1)
        want = np.where(n > 0, n / np.where(cn > 0, cn, 1), 0.0)
        rtol = 2e-6
    elif mode == "none":
        want = n
        rtol = 2e-6
    else:
        yc = np.sum(yy * c, axis=1)
        want = np.where(n > 0, n / np.where(yc != 0, yc, 1), 0.0)
        rtol = 2e-5
    assert np.allclose(gpu_scale[clean], enc.scale[clean], rtol=rtol, atol=1e-30)
    assert np.allclose(gpu_scale, want, rtol=rtol, atol=1e-30)
    return int(mism.sum())


def check_topk(gpu_ids, gpu_scores, oracle_ids, scores64, allowed, k, tol):
    """gpu_ids/gpu_scores [nq, k] against the oracle's ids [nq, k]; scores64
    [nq, n] are the oracle's float64 scores of every vector; allowed [nq, n]."""
    gpu_ids = np.asarray(gpu_ids)
    gpu_scores = np.asarray(gpu_scores)
    nq = gpu_ids.shape[0]
    for q in range(nq):
        ref = np.asarray(oracle_ids[q])
        n_valid = int(np.sum(ref >= 0))
        assert n_valid == min(k, int(allowed[q].sum()))
        g = gpu_ids[q]
        gs = gpu_scores[q]
        assert np.all(g[:n_valid] >= 0), f"query {q}: missing results"
        assert np.all(g[n_valid:] == -1) and np.all(np.isneginf(gs[n_valid:])), f"query {q}: bad padding"
        g = g[:n_valid]
        gs = gs[:n_valid]
        assert len(set(g.tolist())) == n_valid, f"query {q}: duplicate ids"
        assert np.all(allowed[q, g]), f"query {q}: disallowed id returned"
        s = scores64[q]
        assert np.all(np.abs(gs.astype(np.float64) - s[g]) <= tol), f"query {q}: score off"
        assert np.all(np.diff(gs) <= 0), f"query {q}: not sorted"
        # ties on equal float32 scores are ordered by id
        eq = np.nonzero(np.diff(gs) == 0)[0]
        assert np.all(g[eq] < g[eq + 1]), f"query {q}: tie not ordered by id"
        if n_valid == 0:
            continue
        ref = ref[:n_valid]
        kth = s[ref[-1]]
        diff = set(g.tolist()) ^ set(ref.tolist())
        for i in diff:
            assert abs(s[i] - kth) <= 2 * tol, f"query {q}: id {i} differs and is not tied with the k-th"


def recall(ids, exact_ids):
    return O.recall_at_k(np.asarray(ids), np.asarray(exact_ids))


def merge_candidates(cand_ids, cand_scores, k):
    """Top-k of the union of candidate lists [S, nq, m] by (score desc, id asc),
    padding (id -1) dropped, result padded with (-1, -inf): the ranking rule of
    the search, applied to the gathered lists."""
    S, nq, m = cand_ids.shape
    ids = np.full((nq, k), -1, np.int64)
    sc = np.full((nq, k), -np.inf, np.float32)
    for q in range(nq):
        i = cand_ids[:, q, :].reshape(-1)
        s = cand_scores[:, q, :].reshape(-1)
        keep = i >= 0
        i, s = i[keep], s[keep]
        order = np.lexsort((i, -s.astype(np.float64)))[:k]
        ids[q, :len(order)] = i[order]
        sc[q, :len(order)] = s[order]
    return ids, sc
