"""Plain, slow CPU oracle of the TurboQuant search path (TEST INFRASTRUCTURE).

This module is a checker, not part of the product.  Only tests/,
__graft_entry__.smoke() and bench.py's CPU-baseline leg may import it.  It
shares no code with the CUDA library (paper_2607_16973_gb300/csrc): it is
numpy/scipy in float64, written step by step from the paper:

* Sec. II-B, steps 1-5 (the TurboQuant pipeline): normalise and keep the norm,
  rotate by a fixed random orthogonal R, quantise each coordinate with a
  Lloyd-Max quantiser derived from the Beta / N(0, 1/d) coordinate marginal
  (no corpus data), bit-pack, and score with a per-vector length
  renormalisation scalar;
* Sec. III-B: allowlist filtering (a vector whose tenant is not allowed never
  enters the top-k);
* Sec. III-A: the id-mapped index (a deleted row never enters the top-k; rows
  are reported by their external uint64 ids);
* Sec. IV-A: exact brute-force inner-product ground truth and Recall@k;
  Sec. IV-E: Hit@k and MRR@20 against the exact top-1;
* Sec. V-C: the over-fetch post-filter baseline that filtering is compared with;
* Sec. II-B, TQ+: per-coordinate shift and scale from the first batch (a
  reading; parity unpinned, see `calibrate`).

Readings where the paper is silent:
* marginal: the exact coordinate density of a uniformly random unit vector,
  f_d(x) proportional to (1-x^2)^((d-3)/2) on [-1, 1]; N(0, 1/d) is an option;
* Lloyd-Max: centroids start at the (i+1/2)/L quantiles of the marginal and the
  plain Lloyd iteration (midpoint boundaries, conditional-mean centroids) runs
  until the largest centroid move is below 1e-13 of the largest centroid (the
  Beta cell masses carry ~1e-14 relative rounding noise at d = 1536); the
  fixed point of a symmetric log-concave density is unique and symmetric, so
  the result is symmetrised exactly before the boundaries are taken;
* rotation: y = R x, R row-major, R = Q diag(sign(diag(Rqr))) from the QR
  factorisation of a d x d standard Gaussian matrix drawn by splitmix64 and
  Box-Muller (definitions in `gaussian_matrix`);
* a coordinate exactly on a boundary goes to the lower cell: code = #{i: t_i < y};
  the comparison is taken in float32 (the precision the GPU encoder works in);
* packing: each row is a little-endian bit stream, code j in bits [b*j, b*j+b);
* per-vector scalar: "norm" = ||x|| / ||c[code]|| (length renormalisation,
  default), "none" = ||x||, "unbiased" = ||x|| / <y, c[code]>;  a zero row has
  y = 0 and scale 0;
* ranking: score descending, ties by id ascending, taken on float32 scores;
  fewer than k allowed vectors pad with id -1 and score -inf;
* id map: deletion excludes a row as a disallowed tenant does; the tie-break
  stays on the row (insertion order), which is then reported as its external
  id; the all-ones id (-1) is reserved for empty slots.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np
from scipy import special as sp

SCALE_MODES = ("norm", "none", "unbiased")

# ---------------------------------------------------------------------------
# Random rotation (Sec. II-B step 2)
# ---------------------------------------------------------------------------
_SM_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_SM_M1 = np.uint64(0xBF58476D1CE4E5B9)
_SM_M2 = np.uint64(0x94D049BB133111EB)


def splitmix64(seed: int, counters: np.ndarray) -> np.ndarray:
    """Vigna's splitmix64, counter form: output number c (c = 0, 1, ...) of the
    generator started in state `seed` is mix(seed + (c + 1) * 0x9E3779B97F4A7C15)
    with mix(z) = z ^ z>>30, * 0xBF58476D1CE4E5B9, ^ >>27, * 0x94D049BB133111EB,
    ^ >>31 (all mod 2^64)."""
    c = np.asarray(counters, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(seed) + (c + np.uint64(1)) * _SM_GAMMA
        z = (z ^ (z >> np.uint64(30))) * _SM_M1
        z = (z ^ (z >> np.uint64(27))) * _SM_M2
        z = z ^ (z >> np.uint64(31))
    return z


def gaussian_matrix(d: int, seed: int) -> np.ndarray:
    """d x d standard normal matrix, float64, filled row-major.

    Element pair (2p, 2p+1) comes from Box-Muller on two splitmix64 outputs
    a = out(2p), b = out(2p+1):  u1 = ((a >> 11) + 1) 2^-53 in (0, 1],
    u2 = (b >> 11) 2^-53 in [0, 1),  r = sqrt(-2 ln u1),
    g[2p] = r cos(2 pi u2),  g[2p+1] = r sin(2 pi u2).
    """
    total = d * d
    pairs = (total + 1) // 2
    p = np.arange(pairs, dtype=np.uint64)
    a = splitmix64(seed, 2 * p)
    b = splitmix64(seed, 2 * p + np.uint64(1))
    u1 = ((a >> np.uint64(11)).astype(np.float64) + 1.0) * 2.0 ** -53
    u2 = (b >> np.uint64(11)).astype(np.float64) * 2.0 ** -53
    r = np.sqrt(-2.0 * np.log(u1))
    g = np.empty(2 * pairs, dtype=np.float64)
    g[0::2] = r * np.cos(2.0 * np.pi * u2)
    g[1::2] = r * np.sin(2.0 * np.pi * u2)
    return g[:total].reshape(d, d)


def rotation(d: int, seed: int) -> np.ndarray:
    """Haar-random orthogonal R (float64, row-major, y = R x).

    G = Q Rqr (QR factorisation);  R = Q diag(s) with s_i = sign(Rqr_ii), which
    makes the factorisation unique (positive diagonal) and Q Haar distributed.
    """
    G = gaussian_matrix(d, seed)
    Q, Rqr = np.linalg.qr(G)
    s = np.sign(np.diag(Rqr))
    s[s == 0] = 1.0
    return Q * s[None, :]


# ---------------------------------------------------------------------------
# Codebook (Sec. II-B step 3; Sec. II-A: derived from the marginal, no data)
# ---------------------------------------------------------------------------
@dataclass
class Codebook:
    centroids: np.ndarray   # float64 [L]
    boundaries: np.ndarray  # float64 [L-1]
    distortion: float       # per-coordinate MSE, sum_i int_cell (x - c_i)^2 f
    iterations: int

    @property
    def centroids32(self) -> np.ndarray:
        return self.centroids.astype(np.float32)

    @property
    def boundaries32(self) -> np.ndarray:
        return self.boundaries.astype(np.float32)


def _beta_params(d: int) -> tuple[float, float, float]:
    """f_d(x) = C_d (1 - x^2)^m on [-1, 1], m = (d-3)/2; (x+1)/2 ~ Beta(a, a),
    a = (d-1)/2;  log C_d = lgamma(d/2) - lgamma((d-1)/2) - log(sqrt(pi))."""
    m = (d - 3) / 2.0
    a = (d - 1) / 2.0
    log_c = sp.gammaln(d / 2.0) - sp.gammaln((d - 1) / 2.0) - 0.5 * np.log(np.pi)
    return m, a, log_c


def marginal_pdf(x: np.ndarray, d: int, marginal: str = "beta") -> np.ndarray:
    """Coordinate density after the random rotation (Sec. II-B step 2)."""
    x = np.asarray(x, dtype=np.float64)
    if marginal == "gauss":
        s = 1.0 / np.sqrt(d)
        return np.exp(-0.5 * (x / s) ** 2) / (s * np.sqrt(2.0 * np.pi))
    m, _, log_c = _beta_params(d)
    out = np.zeros_like(x)
    inside = np.abs(x) < 1.0
    out[inside] = np.exp(log_c + m * np.log1p(-x[inside] ** 2))
    return out


def _std_pdf(z: np.ndarray) -> np.ndarray:
    """Standard normal density, 0 at +-inf."""
    fin = np.isfinite(z)
    zz = np.where(fin, z, 0.0)
    return np.where(fin, np.exp(-0.5 * zz * zz) / np.sqrt(2.0 * np.pi), 0.0)


def _z_pdf(z: np.ndarray) -> np.ndarray:
    """z * phi(z), 0 at +-inf."""
    fin = np.isfinite(z)
    return np.where(fin, np.where(fin, z, 0.0) * _std_pdf(z), 0.0)


def cell_moments(edges: np.ndarray, d: int, marginal: str = "beta"):
    """Zeroth, first and second moments of the marginal over each cell
    [edges[i], edges[i+1]].

    Beta:  M0 = I_u(a, a) differences (u = (x+1)/2, upper-tail form for cells
    in x >= 0);  M1 from the antiderivative of x (1-x^2)^m,
    -(1-x^2)^(m+1) / (2(m+1));  M2 = M0 - 2a/(2a+1) * [I_u(a+1, a+1)] because
    x^2 = 1 - (1 - x^2) and C_d int (1-x^2)^(m+1) = 2a/(2a+1) dI(a+1, a+1).
    Gauss N(0, s^2), z = x/s:  M0 = dPhi(z), M1 = s [phi(z_lo) - phi(z_hi)],
    M2 = s^2 (dPhi - [z phi(z)]).
    """
    e = np.asarray(edges, dtype=np.float64)
    lo, hi = e[:-1], e[1:]
    if marginal == "gauss":
        s = 1.0 / np.sqrt(d)
        zl, zh = lo / s, hi / s
        upper = zl >= 0
        M0 = np.where(upper, sp.ndtr(-zl) - sp.ndtr(-zh), sp.ndtr(zh) - sp.ndtr(zl))
        M1 = s * (_std_pdf(zl) - _std_pdf(zh))
        M2 = s * s * (M0 - (_z_pdf(zh) - _z_pdf(zl)))
        return M0, M1, M2
    m, a, log_c = _beta_params(d)
    ul, uh = (lo + 1.0) / 2.0, (hi + 1.0) / 2.0
    upper = lo >= 0
    M0 = np.where(upper, sp.betaincc(a, a, ul) - sp.betaincc(a, a, uh),
                  sp.betainc(a, a, uh) - sp.betainc(a, a, ul))
    J = np.where(upper, sp.betaincc(a + 1, a + 1, ul) - sp.betaincc(a + 1, a + 1, uh),
                 sp.betainc(a + 1, a + 1, uh) - sp.betainc(a + 1, a + 1, ul))

    def prim(x):  # C_d * -(1-x^2)^(m+1) / (2(m+1))
        with np.errstate(divide="ignore"):
            p = np.where(np.abs(x) >= 1.0, 0.0,
                         np.exp(log_c + (m + 1.0) * np.log1p(-np.minimum(x * x, 1.0))))
        return -p / (2.0 * (m + 1.0))

    M1 = prim(hi) - prim(lo)
    M2 = M0 - (2.0 * a / (2.0 * a + 1.0)) * J
    return M0, M1, M2


def _quantile(p: np.ndarray, d: int, marginal: str) -> np.ndarray:
    if marginal == "gauss":
        return sp.ndtri(p) / np.sqrt(d)
    _, a, _ = _beta_params(d)
    return 2.0 * sp.betaincinv(a, a, p) - 1.0


def codebook(d: int, bits: int, marginal: str = "beta", tol: float = 1e-13,
             max_iter: int = 1_000_000) -> Codebook:
    """Lloyd-Max quantiser of the coordinate marginal (Sec. II-B step 3).

    Repeats: boundaries t_i = (c_i + c_{i+1}) / 2, then c_i = E[x | t_{i-1} < x <= t_i]
    (outer edges -1, +1 for the Beta marginal, -inf, +inf for the Gaussian).
    """
    if marginal not in ("beta", "gauss"):
        raise ValueError(marginal)
    if bits < 1 or d < (2 if marginal == "beta" else 1):
        raise ValueError("need bits >= 1 and d >= 2 (Beta) or d >= 1 (Gaussian)")
    L = 1 << bits
    end = 1.0 if marginal == "beta" else np.inf
    c = _quantile((np.arange(L) + 0.5) / L, d, marginal)
    it = 0
    for it in range(1, max_iter + 1):
        edges = np.concatenate([[-end], (c[:-1] + c[1:]) / 2.0, [end]])
        M0, M1, _ = cell_moments(edges, d, marginal)
        c_new = M1 / M0
        move = np.max(np.abs(c_new - c))
        c = c_new
        if move <= tol * np.max(np.abs(c)):
            break
    c = (c - c[::-1]) / 2.0                     # exact symmetry c_i = -c_{L-1-i}
    t = (c[:-1] + c[1:]) / 2.0
    edges = np.concatenate([[-end], t, [end]])
    M0, M1, M2 = cell_moments(edges, d, marginal)
    D = float(np.sum(M2 - 2.0 * c * M1 + c * c * M0))
    return Codebook(centroids=c, boundaries=t, distortion=D, iterations=it)


# ---------------------------------------------------------------------------
# Packing (Sec. II-B step 4)
# ---------------------------------------------------------------------------
def row_bytes(d: int, bits: int) -> int:
    """Bytes of one packed row: d*b/8 (1536-d at 4 bits -> 768 B, Sec. II-B)."""
    if (d * bits) % 8:
        raise ValueError("d * bits must be a multiple of 8")
    return d * bits // 8


def pack(codes: np.ndarray, bits: int) -> np.ndarray:
    """codes uint [n, d] (< 2^bits) -> uint8 [n, d*bits/8]: little-endian bit
    stream, code j in bits [bits*j, bits*j + bits) of its row.

    Written group by group: g = lcm(bits, 8) / 8 bytes hold 8g/bits whole
    codes, code r of a group adding code << bits*r to the group's
    little-endian integer value."""
    codes = np.asarray(codes)
    n, d = codes.shape
    g = int(np.lcm(bits, 8)) // 8
    per = 8 * g // bits
    nb = (d * bits + 7) // 8
    groups = -(-nb // g)
    c = np.zeros((n, groups * per), dtype=np.uint64)
    c[:, :d] = codes
    v = np.zeros((n, groups), dtype=np.uint64)
    for r in range(per):
        v |= c[:, r::per] << np.uint64(bits * r)
    out = np.empty((n, groups * g), dtype=np.uint8)
    for i in range(g):
        out[:, i::g] = ((v >> np.uint64(8 * i)) & np.uint64(255)).astype(np.uint8)
    return out[:, :nb]


def unpack(packed: np.ndarray, d: int, bits: int) -> np.ndarray:
    """Inverse of `pack`: uint8 [n, d*bits/8] -> codes uint16 [n, d].

    The row is read in groups of g = lcm(bits, 8) / 8 bytes, each holding
    8g/bits whole codes: the group's little-endian integer value v gives code
    r of the group as (v >> bits*r) & (2^bits - 1)."""
    packed = np.asarray(packed, dtype=np.uint8)
    n = packed.shape[0]
    g = int(np.lcm(bits, 8)) // 8
    per = 8 * g // bits
    nb = (d * bits + 7) // 8
    groups = -(-nb // g)
    rows = np.zeros((n, groups * g), dtype=np.uint8)
    rows[:, :nb] = packed[:, :nb]
    v = np.zeros((n, groups), dtype=np.uint64)
    for i in range(g):
        v |= rows[:, i::g].astype(np.uint64) << np.uint64(8 * i)
    shifts = (np.arange(per, dtype=np.uint64) * np.uint64(bits))
    codes = (v[:, :, None] >> shifts) & np.uint64((1 << bits) - 1)
    return codes.reshape(n, groups * per)[:, :d].astype(np.uint16)


# ---------------------------------------------------------------------------
# Encode (Sec. II-B steps 1-5)
# ---------------------------------------------------------------------------
@dataclass
class Encoded:
    packed: np.ndarray   # uint8 [n, d*b/8]
    scale: np.ndarray    # float32 [n]
    codes: np.ndarray    # uint16 [n, d]
    y: np.ndarray        # float64 [n, d]: R x / ||x||
    norm: np.ndarray     # float64 [n]


def rotate_normalize(X: np.ndarray, R: np.ndarray):
    """Steps 1-2 of the encoder: n = ||x|| and y = R x / n (y = 0 when n = 0),
    float64.  R is the float32 array the GPU path also gets, promoted.
    Returns (y [rows, d], n [rows])."""
    X64 = np.asarray(X, dtype=np.float64)
    R64 = np.asarray(R, dtype=np.float32).astype(np.float64)
    n = np.sqrt(np.sum(X64 * X64, axis=1))
    y = X64 @ R64.T
    nz = n > 0
    y[nz] /= n[nz, None]
    y[~nz] = 0.0
    return y, n


def encode(X: np.ndarray, R: np.ndarray, centroids: np.ndarray, boundaries: np.ndarray,
           bits: int, scale_mode: str = "norm", calib: "Calibration | None" = None) -> Encoded:
    """Encode rows of X.

    Step 1: n = ||x||.  Step 2: y = R x / n (y = 0 when n = 0).  Step 3:
    code_j = #{i : t_i < y_j} with y_j rounded to float32 and the float32
    boundaries t.  Step 4: pack.  Step 5: the per-vector scalar (module header).
    R, centroids and boundaries are the float32 arrays the GPU path also gets;
    they are promoted to float64 here.  With a TQ+ calibration the quantiser
    sees z_j = (y_j - mu_j) / a_j instead of y_j (see `calibrate`).
    """
    y, n = rotate_normalize(X, R)
    return quantize(y, n, centroids, boundaries, bits, scale_mode, calib)


def quantize(y: np.ndarray, n: np.ndarray, centroids: np.ndarray, boundaries: np.ndarray,
             bits: int, scale_mode: str = "norm", calib: "Calibration | None" = None) -> Encoded:
    """Steps 3-5 of the encoder on rotated, normalised rows y (float64) with
    norms n: nearest-centroid codes, packing and the per-vector scalar.  With a
    TQ+ calibration the codes are those of z = (y - mu) / a and the
    reconstruction the scalar is taken on is y^ = a c[code] + mu; Encoded.y
    then holds z, the value compared with the boundaries."""
    if scale_mode not in SCALE_MODES:
        raise ValueError(scale_mode)
    c64 = np.asarray(centroids, dtype=np.float32).astype(np.float64)
    t32 = np.asarray(boundaries, dtype=np.float32)
    assert len(c64) == 1 << bits and len(t32) == len(c64) - 1
    nz = n > 0
    if calib is not None:
        yq = (y - calib.mu[None, :]) / calib.a[None, :]
        code = np.searchsorted(t32, yq.astype(np.float32), side="left").astype(np.uint16)
        c = calib.a[None, :] * c64[code] + calib.mu[None, :]
    else:
        yq = y
        code = np.searchsorted(t32, y.astype(np.float32), side="left").astype(np.uint16)
        c = c64[code]
    if scale_mode == "norm":
        cn = np.sqrt(np.sum(c * c, axis=1))
        scale = np.where(nz & (cn > 0), n / np.where(cn > 0, cn, 1.0), 0.0)
    elif scale_mode == "none":
        scale = n
    else:
        yc = np.sum(y * c, axis=1)
        scale = np.where(nz & (yc != 0), n / np.where(yc != 0, yc, 1.0), 0.0)
    return Encoded(packed=pack(code, bits), scale=scale.astype(np.float32),
                   codes=code, y=yq, norm=n)


def decode(packed: np.ndarray, scale: np.ndarray, R: np.ndarray, centroids: np.ndarray,
           d: int, bits: int, calib: "Calibration | None" = None) -> np.ndarray:
    """Reconstruction x_hat = scale * R^T c[code] (float64 [n, d]); with a TQ+
    calibration x_hat = scale * R^T (a c[code] + mu)."""
    codes = unpack(packed, d, bits)
    c = np.asarray(centroids, dtype=np.float32).astype(np.float64)[codes]
    if calib is not None:
        c = calib.a[None, :] * c + calib.mu[None, :]
    R64 = np.asarray(R, dtype=np.float32).astype(np.float64)
    return (c @ R64) * np.asarray(scale, dtype=np.float64)[:, None]


# ---------------------------------------------------------------------------
# TQ+ calibration (Sec. II-B, "TQ+ calibration and data dependence")
# PARITY UNPINNED as a reading: the paper says only that per-coordinate shift
# and scale parameters are fitted from the first batch of indexed vectors to
# align the empirical coordinate quantiles with the canonical marginal, and
# that only per-coordinate first and second moments are kept.  The pins in the
# tests check what the mathematics fixes about this reading, not the reading.
# ---------------------------------------------------------------------------
@dataclass
class Calibration:
    mu: np.ndarray   # float64 [d]: per-coordinate shift (first moment)
    a: np.ndarray    # float64 [d]: per-coordinate scale (spread / canonical spread)


def calibrate(X: np.ndarray, R: np.ndarray) -> Calibration:
    """Per-coordinate shift and scale from a first batch X of rows.

    Reading: over the batch's non-zero rows, y = R x / ||x|| (steps 1-2 of the
    encoder); mu_j = mean of y_j and sigma_j = its population standard
    deviation (the first and second moments); a_j = sigma_j * sqrt(d), the
    ratio to the canonical marginal's spread (1/sqrt(d) for the coordinate of
    a uniform unit vector, the Beta marginal, and for N(0, 1/d)), and a_j = 1
    where sigma_j = 0.  z_j = (y_j - mu_j) / a_j then has the canonical first
    two moments over the batch, and the canonical codebook quantises z.  A
    batch without a non-zero row gives mu = 0, a = 1 (plain TurboQuant)."""
    y, n = rotate_normalize(X, R)
    d = y.shape[1]
    y = y[n > 0]
    if len(y) == 0:
        return Calibration(mu=np.zeros(d), a=np.ones(d))
    mu = y.mean(axis=0)
    sigma = np.sqrt(np.mean((y - mu[None, :]) ** 2, axis=0))
    a = np.where(sigma > 0, sigma * np.sqrt(d), 1.0)
    return Calibration(mu=mu, a=a)


def calibration32(calib: Calibration) -> Calibration:
    """The calibration as the float32 values the GPU path is given, promoted."""
    return Calibration(mu=calib.mu.astype(np.float32).astype(np.float64),
                       a=calib.a.astype(np.float32).astype(np.float64))


# ---------------------------------------------------------------------------
# Search (Sec. II-B step 5, Sec. III-B filtering, Sec. IV-A ground truth)
# ---------------------------------------------------------------------------
def allowed_mask(tenant_ids, allow_off, allow_ids, nq: int, n: int) -> np.ndarray:
    """bool [nq, n]: vector i may be returned for query q iff its tenant is in
    q's allowlist (Sec. III-B).  No filter -> all True."""
    if tenant_ids is None:
        return np.ones((nq, n), dtype=bool)
    tid = np.asarray(tenant_ids, dtype=np.uint32)
    out = np.zeros((nq, n), dtype=bool)
    for q in range(nq):
        allow = np.asarray(allow_ids[allow_off[q]:allow_off[q + 1]], dtype=np.uint32)
        out[q] = np.isin(tid, allow)
    return out


def rank_topk(scores32: np.ndarray, allowed: np.ndarray, k: int):
    """Top-k of one query: sort by (score desc, id asc) over allowed ids, pad
    with (-1, -inf)."""
    idx = np.nonzero(allowed)[0]
    s = scores32[idx]
    if len(idx) > k:
        # a vector scoring below the k-th largest score has k better ones and
        # cannot be in the top k; every vector tied with that score stays
        kth = np.partition(s, len(s) - k)[len(s) - k]
        keep = s >= kth
        idx, s = idx[keep], s[keep]
    order = np.lexsort((idx, -s.astype(np.float64)))
    top = idx[order[:k]]
    ids = np.full(k, -1, dtype=np.int64)
    sc = np.full(k, -np.inf, dtype=np.float32)
    ids[: len(top)] = top
    sc[: len(top)] = scores32[top]
    return ids, sc


@dataclass
class SearchResult:
    ids: np.ndarray        # int64 [nq, k]
    scores: np.ndarray     # float32 [nq, k]
    scores64: np.ndarray   # float64 [nq, n]: every vector's score (allowed or not)


def quantized_scores(Q, R, centroids, bits, packed, scale, d, row_chunk=16384,
                     calib: Calibration | None = None) -> np.ndarray:
    """s[q, i] = scale_i * sum_j q'_j c[code_ij] with q' = R q, float64 [nq, n];
    with a TQ+ calibration the reconstruction a_j c[code_ij] + mu_j takes the
    place of c[code_ij]."""
    Q64 = np.asarray(Q, dtype=np.float64)
    R64 = np.asarray(R, dtype=np.float32).astype(np.float64)
    c64 = np.asarray(centroids, dtype=np.float32).astype(np.float64)
    qr = Q64 @ R64.T
    n = packed.shape[0]
    S = np.empty((Q64.shape[0], n), dtype=np.float64)
    sc = np.asarray(scale, dtype=np.float32).astype(np.float64) if scale is not None else np.ones(n)
    for r0 in range(0, n, row_chunk):
        r1 = min(n, r0 + row_chunk)
        C = c64[unpack(packed[r0:r1], d, bits)]
        if calib is not None:
            C = calib.a[None, :] * C + calib.mu[None, :]
        S[:, r0:r1] = (qr @ C.T) * sc[None, r0:r1]
    return S


def search(Q, R, centroids, bits, packed, scale, k, d,
           tenant_ids=None, allow_off=None, allow_ids=None, deleted=None, ext_ids=None,
           calib: Calibration | None = None) -> SearchResult:
    """Top-k inner-product search over the quantised corpus.

    Id-mapped index (Sec. III-A: external uint64 ids, O(1) deletion): a row
    with deleted[i] True is never returned, exactly like a row whose tenant
    is not allowed; with ext_ids the k rows, ranked as usual (ties by row,
    i.e. insertion order), are reported as ext_ids[row] (their int64 bit
    pattern; empty slots stay -1).  With a TQ+ calibration the scores are
    those of the calibrated reconstruction (quantized_scores)."""
    S = quantized_scores(Q, R, centroids, bits, packed, scale, d, calib=calib)
    nq, n = S.shape
    allowed = allowed_mask(tenant_ids, allow_off, allow_ids, nq, n)
    if deleted is not None:
        allowed = allowed & ~np.asarray(deleted, dtype=bool)[None, :]
    ids = np.empty((nq, k), dtype=np.int64)
    sc = np.empty((nq, k), dtype=np.float32)
    S32 = S.astype(np.float32)
    for q in range(nq):
        ids[q], sc[q] = rank_topk(S32[q], allowed[q], k)
    if ext_ids is not None:
        ext = np.asarray(ext_ids, dtype=np.uint64).view(np.int64)
        ids = np.where(ids >= 0, ext[np.maximum(ids, 0)], -1)
    return SearchResult(ids=ids, scores=sc, scores64=S)


def exact_knn(X, Q, k, tenant_ids=None, allow_off=None, allow_ids=None, row_chunk=65536):
    """Ground truth: brute-force float64 inner product on the unquantised rows
    (Sec. IV-A), same tie rule and allowlist.  Returns (ids, scores64).  The
    corpus is converted to float64 `row_chunk` rows at a time."""
    Q64 = np.asarray(Q, dtype=np.float64)
    n = X.shape[0]
    S = np.empty((Q64.shape[0], n), dtype=np.float64)
    for r0 in range(0, n, row_chunk):
        S[:, r0:r0 + row_chunk] = Q64 @ np.asarray(X[r0:r0 + row_chunk], dtype=np.float64).T
    nq = S.shape[0]
    allowed = allowed_mask(tenant_ids, allow_off, allow_ids, nq, n)
    ids = np.empty((nq, k), dtype=np.int64)
    sc = np.empty((nq, k), dtype=np.float64)
    for q in range(nq):
        idx = np.nonzero(allowed[q])[0]
        s = S[q, idx]
        if len(idx) > k:  # only scores >= the k-th largest can be in the top k
            kth = np.partition(s, len(s) - k)[len(s) - k]
            keep = s >= kth
            idx, s = idx[keep], s[keep]
        order = np.lexsort((idx, -s))
        top = idx[order[:k]]
        ids[q] = -1
        sc[q] = -np.inf
        ids[q, : len(top)] = top
        sc[q, : len(top)] = S[q, top]
    return ids, sc


def hit_at_k(approx_ids: np.ndarray, exact_ids: np.ndarray, k: int) -> float:
    """Hit@k (Sec. IV-E, Table III): the share of queries whose exact top-1
    result is among the first k approximate results.  Queries without an
    exact result are skipped."""
    vals = [int(e[0]) in set(int(v) for v in a[:k]) for a, e in zip(approx_ids, exact_ids) if e[0] >= 0]
    return float(np.mean(vals)) if vals else 1.0


def mrr_at(approx_ids: np.ndarray, exact_ids: np.ndarray, depth: int = 20) -> float:
    """MRR@depth (Sec. IV-E, Table III): the mean over queries of 1 / rank of
    the exact top-1 result in the approximate list (rank 1 = first), counted
    as 0 when it is not among the first `depth`."""
    vals = []
    for a, e in zip(approx_ids, exact_ids):
        if e[0] < 0:
            continue
        ranks = [r for r, v in enumerate(a[:depth], start=1) if v == e[0]]
        vals.append(1.0 / ranks[0] if ranks else 0.0)
    return float(np.mean(vals)) if vals else 1.0


def postfilter_topk(cand_ids: np.ndarray, allowed: np.ndarray, k: int) -> np.ndarray:
    """The over-fetch post-filter baseline (Sec. V-C, Table V): from each
    query's unfiltered candidate list (best first, -1 = empty), keep the
    candidates whose vector is allowed, in order, and return the first k,
    padded with -1.  allowed: bool [nq, n]."""
    out = np.full((len(cand_ids), k), -1, dtype=np.int64)
    for q, row in enumerate(cand_ids):
        keep = [int(v) for v in row if v >= 0 and allowed[q, v]][:k]
        out[q, :len(keep)] = keep
    return out


def recall_at_k(approx_ids: np.ndarray, exact_ids: np.ndarray) -> float:
    """Recall@k = mean over queries of |approx ∩ exact| / |exact| (Sec. IV-A);
    padding ids (-1) are not results."""
    vals = []
    for a, e in zip(approx_ids, exact_ids):
        e = set(int(v) for v in e if v >= 0)
        if not e:
            continue
        a = set(int(v) for v in a if v >= 0)
        vals.append(len(a & e) / len(e))
    return float(np.mean(vals)) if vals else 1.0
