"""Seeded synthetic inputs shaped like the paper's workloads.

The paper evaluates on DBpedia entity descriptions embedded with OpenAI
text-embedding-3-large (d=1536, L2-normalised, 100K-999K vectors, 1,000
held-out queries, seed 42; Sec. IV-A), with tenant partitions for the filtered
experiment (Sec. V-C).  That dataset is not available here, so these generators
stand in for it with the same shapes:

* corpus: a Gaussian mixture (centres ~ N(0, I_d), per-cluster spread 0.5),
  each row L2-normalised;
* queries: corpus rows drawn without replacement plus per-coordinate Gaussian
  noise, renormalised;
* tenants: Zipf(s)-sized tenants with distinct random uint32 ids, stored in a
  shuffled (tenant-interleaved) order; allowlists of one tenant, a fraction
  carrying extra tenants.

This module is shared by the oracle, the tests and the benchmark.  It holds no
arithmetic of the method itself (no rotation, quantisation, packing or scoring):
it only draws numbers.  Every generator is chunked with a per-chunk seed so any
row range can be regenerated on its own (the CPU baseline uses that to draw a
bounded sample of a large corpus).
"""
from __future__ import annotations

import numpy as np

CHUNK_ROWS = 8192

# Default seeds of the synthetic workloads: data 42 (the paper's seed, Sec. IV-A),
# rotation 1536, queries 43, tenants 44.
SEED_DATA = 42
SEED_ROTATION = 1536
SEED_QUERIES = 43
SEED_TENANTS = 44


def mixture_centers(d: int, n_clusters: int, seed: int = SEED_DATA) -> np.ndarray:
    """Cluster centres ~ N(0, I_d), float64 [n_clusters, d]."""
    rng = np.random.default_rng([seed, 0xC0FFEE, n_clusters, d])
    return rng.standard_normal((n_clusters, d))


def mixture_rows(start: int, stop: int, d: int, n_clusters: int,
                 seed: int = SEED_DATA, spread: float = 0.5,
                 centers: np.ndarray | None = None, workers: int = 1) -> np.ndarray:
    """Rows [start, stop) of the seeded mixture corpus, float32, unit L2 norm.

    Row r belongs to chunk r // CHUNK_ROWS; chunk c draws from the stream
    seeded by (seed, c), so any range is reproducible on its own (and the
    result does not depend on `workers`).
    """
    if centers is None:
        centers = mixture_centers(d, n_clusters, seed)
    out = np.empty((max(stop - start, 0), d), dtype=np.float32)
    c0 = start // CHUNK_ROWS
    c1 = (stop + CHUNK_ROWS - 1) // CHUNK_ROWS

    def one(c: int) -> None:
        # every chunk draws all CHUNK_ROWS rows so a row never depends on
        # which range asked for it
        rng = np.random.default_rng([seed, c, n_clusters, d])
        z = rng.integers(0, n_clusters, size=CHUNK_ROWS)
        noise = rng.standard_normal((CHUNK_ROWS, d), dtype=np.float32)
        lo = max(start, c * CHUNK_ROWS)
        hi = min(stop, (c + 1) * CHUNK_ROWS)
        a, b = lo - c * CHUNK_ROWS, hi - c * CHUNK_ROWS
        block = centers[z[a:b]] + spread * noise[a:b].astype(np.float64)
        block /= np.linalg.norm(block, axis=1, keepdims=True)
        out[lo - start: hi - start] = block.astype(np.float32)

    if workers > 1 and c1 - c0 > 1:
        from concurrent.futures import ThreadPoolExecutor
        with ThreadPoolExecutor(max_workers=workers) as ex:
            list(ex.map(one, range(c0, c1)))
    else:
        for c in range(c0, c1):
            one(c)
    return out


def mixture_corpus(n: int, d: int, n_clusters: int, seed: int = SEED_DATA,
                   spread: float = 0.5, workers: int = 1) -> np.ndarray:
    """The whole seeded mixture corpus, float32 [n, d], unit rows."""
    centers = mixture_centers(d, n_clusters, seed)
    return mixture_rows(0, n, d, n_clusters, seed, spread, centers, workers)


def query_sources(n: int, nq: int, seed: int = SEED_QUERIES) -> np.ndarray:
    """Indices of the corpus rows the queries are drawn from (no replacement)."""
    rng = np.random.default_rng([seed, 1])
    return rng.choice(n, size=nq, replace=False).astype(np.int64)


def perturb(rows: np.ndarray, seed: int = SEED_QUERIES, sigma: float = 0.1,
            per_coordinate: bool = True) -> np.ndarray:
    """Add N(0, s^2) noise to each coordinate and renormalise, float32.

    per_coordinate=True reads "N(0, 0.1^2) noise" literally (s = sigma per
    coordinate); False spreads sigma over the vector (s = sigma / sqrt(d)).
    """
    rows = np.asarray(rows, dtype=np.float64)
    d = rows.shape[1]
    s = sigma if per_coordinate else sigma / np.sqrt(d)
    rng = np.random.default_rng([seed, 2])
    q = rows + s * rng.standard_normal(rows.shape)
    q /= np.linalg.norm(q, axis=1, keepdims=True)
    return q.astype(np.float32)


def zipf_sizes(n: int, n_tenants: int, s: float = 1.1) -> np.ndarray:
    """Tenant sizes proportional to r^-s (r = 1..T), summing to n.

    Rounded by largest remainder with a minimum of one vector per tenant.
    """
    if n_tenants > n:
        raise ValueError("more tenants than vectors")
    w = np.arange(1, n_tenants + 1, dtype=np.float64) ** (-s)
    share = (n - n_tenants) * w / w.sum()
    base = np.floor(share).astype(np.int64)
    rem = (n - n_tenants) - int(base.sum())
    order = np.argsort(-(share - base), kind="stable")
    base[order[:rem]] += 1
    return base + 1


def zipf_tenants(n: int, n_tenants: int, s: float = 1.1,
                 seed: int = SEED_TENANTS) -> tuple[np.ndarray, np.ndarray]:
    """Per-vector uint32 tenant ids, Zipf-sized, in shuffled (interleaved) order.

    Returns (tenant_ids [n] uint32, tenant_values [T] uint32) where
    tenant_values[r] is the id of the r-th largest tenant.
    """
    rng = np.random.default_rng([seed, 3, n_tenants])
    values = np.unique(rng.integers(0, 2**32, size=4 * n_tenants + 16, dtype=np.uint64))
    values = rng.permutation(values)[:n_tenants].astype(np.uint32)
    if len(values) < n_tenants:
        raise RuntimeError("could not draw distinct tenant ids")
    sizes = zipf_sizes(n, n_tenants, s)
    ids = np.repeat(values, sizes)
    rng.shuffle(ids)
    return ids.astype(np.uint32), values


def equal_tenants(n: int, n_tenants: int, seed: int = SEED_TENANTS) -> np.ndarray:
    """Equal-size tenant partitions (the paper's Sec. V-C setup), interleaved."""
    rng = np.random.default_rng([seed, 4, n_tenants])
    values = rng.permutation(np.arange(n_tenants, dtype=np.uint32) * 7919 + 13)
    ids = np.resize(values, n)
    rng.shuffle(ids)
    return ids.astype(np.uint32)


def allowlists(query_src: np.ndarray, tenant_ids: np.ndarray, tenant_values: np.ndarray,
               frac_multi: float = 0.1, extra: int = 4,
               seed: int = SEED_TENANTS) -> tuple[np.ndarray, np.ndarray]:
    """CSR allowlists: each query allows the tenant of its source row; a
    fraction frac_multi of the queries also allow `extra` other tenants drawn
    uniformly without replacement.  Returns (offsets int64 [nq+1], ids uint32).
    """
    rng = np.random.default_rng([seed, 5])
    nq = len(query_src)
    multi = rng.random(nq) < frac_multi
    off = [0]
    out: list[int] = []
    values = np.asarray(tenant_values, dtype=np.uint32)
    for i in range(nq):
        own = int(tenant_ids[query_src[i]])
        lst = [own]
        if multi[i] and len(values) > 1:
            others = values[values != own]
            k = min(extra, len(others))
            lst += [int(v) for v in rng.choice(others, size=k, replace=False)]
        out += lst
        off.append(len(out))
    return np.asarray(off, dtype=np.int64), np.asarray(out, dtype=np.uint32)


def random_codes(n: int, row_bytes: int, seed: int) -> np.ndarray:
    """Uniform random code bytes [n, row_bytes] (every bit pattern is a valid
    packed row for b in {2, 3, 4, 8})."""
    rng = np.random.default_rng([seed, 6])
    return rng.integers(0, 256, size=(n, row_bytes), dtype=np.uint8)


def random_scales(n: int, seed: int, lo: float = 0.9, hi: float = 1.1) -> np.ndarray:
    """Per-vector positive scales, float32."""
    rng = np.random.default_rng([seed, 7])
    return rng.uniform(lo, hi, size=n).astype(np.float32)


def gaussian_rows(n: int, d: int, seed: int) -> np.ndarray:
    """Plain N(0, 1) rows, float32 (not normalised: used for norm edge cases)."""
    rng = np.random.default_rng([seed, 8])
    return rng.standard_normal((n, d), dtype=np.float32)
