"""The tensor-core encoder (tq_encode_planned: the rotation of Sec. II-B step 2
in TF32 with a three-product split) against the oracle's float64 encode, with
the same checks as the FFMA encoder: codes equal except one-cell flips within
the boundary window, scalars to the tolerance of each scale mode.  The sizes
reach several panels per CTA (more panels than SMs), partial last chunks of
256 coordinates, panels with a ragged tail and rows of zeros.

Its y carries about 1e-7 of error at d = 1536 (at most ~1e-6), mostly from
the float32 accumulation inside the tensor cores, against ~5e-9 for the FFMA
encoder.  The expected flip rate is about 2 E|error| times the density of
boundaries: ~3e-5 at 4 bits, but ~5e-4 at 8 bits, whose 255 boundaries sit
about 1e-4 apart near the centre.  So the rate bound is 1e-3 at 8 bits and
1e-4 below; the window (codes differ only within 1e-5 of a boundary) and
everything else is as for the FFMA encoder."""
import json
import os

import numpy as np
import pytest

import oracle as O
from conftest import GOLDEN
from paper_2607_16973_gb300 import synth
from parity import check_encode

pytestmark = pytest.mark.gpu


def _cb(d, bits):
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
    return torch, dev, (lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev))


def _rate(bits):
    return 1e-3 if bits == 8 else 1e-4


def _planned(tq, T, X, R, c32, t32, bits, mode="norm", calib=None):
    import torch
    plan = tq.encode_plan(T(R))
    codes, scale = tq.encode(T(X), None, T(c32), T(t32), bits, mode, plan=plan, calib=calib)
    tq.encode_check(plan)
    torch.cuda.synchronize()
    return codes.cpu().numpy(), scale.cpu().numpy()


def test_plan_is_a_tf32_split(cuda_lib, tdev):
    """The plan holds R_hi = tf32(R) and R_lo = tf32(R - R_hi): both have the
    13 low mantissa bits clear, |R_lo| <= 2^-11 |R|, and R_hi + R_lo is R to
    2^-22 relative; the status word is clear."""
    torch, dev, T = tdev
    tq = cuda_lib
    d = 384
    R = O.rotation(d, 5).astype(np.float32)
    plan = tq.encode_plan(T(R)).cpu().numpy()
    assert plan.size == 256 + 2 * d * d * 4
    assert np.all(plan[:256] == 0)
    parts = plan[256:].view(np.float32).reshape(2, d, d)
    hi, lo = parts[0], parts[1]
    for p in (hi, lo):
        assert np.all((p.view(np.uint32) & 0x1FFF) == 0)
    r = R.astype(np.float64)
    assert np.all(np.abs(hi - r) <= 2.0 ** -11 * np.abs(r))
    assert np.all(np.abs(hi.astype(np.float64) + lo - r) <= 2.0 ** -22 * np.abs(r))


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
@pytest.mark.parametrize("mode", ["norm", "none", "unbiased"])
def test_encode_planned_parity(cuda_lib, tdev, bits, mode):
    torch, dev, T = tdev
    tq = cuda_lib
    d, n = 1536, 2077                       # 16 panels of 128 rows + a ragged 29
    X = synth.mixture_corpus(n, d, 64, seed=42)
    X[5] = 0.0                              # zero row: codes L/2-1, scale 0
    X[6] *= 3.0
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits, mode)
    codes, scale = _planned(tq, T, X, R, c32, t32, bits, mode)
    check_encode(codes, scale, X, enc, c32, t32, d, bits, mode, max_rate=_rate(bits))
    assert np.all(codes[5] == enc.packed[5]) and scale[5] == 0.0


@pytest.mark.parametrize("bits,mode", [(4, "norm"), (3, "unbiased")])
def test_encode_planned_many_panels(cuda_lib, tdev, bits, mode):
    """More panels than SMs: each CTA runs 2-3 panels, so the per-panel norm
    and sum buffers and both accumulator sets are reused."""
    torch, dev, T = tdev
    tq = cuda_lib
    d, n = 1536, 40_000 + 77
    X = synth.mixture_corpus(n, d, 64, seed=8)
    X[n - 1] = 0.0
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits, mode)
    codes, scale = _planned(tq, T, X, R, c32, t32, bits, mode)
    check_encode(codes, scale, X, enc, c32, t32, d, bits, mode)


@pytest.mark.parametrize("d", [128, 160, 384, 2048, 4096])
def test_encode_planned_dims(cuda_lib, tdev, d):
    """One partial chunk (128, 160), a partial last chunk (384), several full
    chunks (2048, 4096)."""
    torch, dev, T = tdev
    tq = cuda_lib
    n, bits = 300, 4
    X = synth.mixture_corpus(n, d, 8, seed=7)
    R = O.rotation(d, 11).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits)
    codes, scale = _planned(tq, T, X, R, c32, t32, bits)
    check_encode(codes, scale, X, enc, c32, t32, d, bits, "norm")


@pytest.mark.parametrize("n", [1, 5, 127, 128, 129])
def test_encode_planned_small_batches(cuda_lib, tdev, n):
    """Fewer rows than one panel (the X tile is zero-filled past row n) and
    the panel edge."""
    torch, dev, T = tdev
    tq = cuda_lib
    d, bits = 1536, 4
    X = synth.mixture_corpus(n, d, 4, seed=n)
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(d, bits)
    enc = O.encode(X, R, c32, t32, bits)
    codes, scale = _planned(tq, T, X, R, c32, t32, bits)
    check_encode(codes, scale, X, enc, c32, t32, d, bits, "norm")


def test_encode_planned_empty_and_offsets(cuda_lib, tdev):
    """n = 0 is a no-op; codes and scale written into a larger array at a row
    offset land only in their rows."""
    torch, dev, T = tdev
    tq = cuda_lib
    d, bits, n = 256, 4, 200
    R = O.rotation(d, 2).astype(np.float32)
    c32, t32 = _cb(d, bits)
    plan = tq.encode_plan(T(R))
    empty = torch.empty((0, d), dtype=torch.float32, device=dev)
    codes, scale = tq.encode(empty, None, T(c32), T(t32), bits, plan=plan)
    assert codes.shape == (0, d * bits // 8)
    X = synth.mixture_corpus(n, d, 4, seed=3)
    big_c = torch.full((n + 64, d * bits // 8), 0xAB, dtype=torch.uint8, device=dev)
    big_s = torch.full((n + 64,), -7.0, dtype=torch.float32, device=dev)
    tq.encode(T(X), None, T(c32), T(t32), bits, "norm", big_c[32:32 + n], big_s[32:32 + n], plan=plan)
    torch.cuda.synchronize()
    bc, bs = big_c.cpu().numpy(), big_s.cpu().numpy()
    assert np.all(bc[:32] == 0xAB) and np.all(bc[32 + n:] == 0xAB)
    assert np.all(bs[:32] == -7.0) and np.all(bs[32 + n:] == -7.0)
    enc = O.encode(X, R, c32, t32, bits)
    check_encode(bc[32:32 + n], bs[32:32 + n], X, enc, c32, t32, d, bits, "norm")


@pytest.mark.parametrize("bits", [3, 4])
def test_encode_planned_tqplus(cuda_lib, tdev, bits):
    """A TQ+ calibration (the oracle's, rounded to float32, on both sides)."""
    torch, dev, T = tdev
    tq = cuda_lib
    d, n = 1536, 1300
    rng = np.random.default_rng(3)
    X = synth.mixture_corpus(n, d, 16, seed=3).astype(np.float64)
    X = (X * rng.uniform(0.3, 3.0, d)[None, :] + rng.normal(0, 0.05, d)[None, :]).astype(np.float32)
    X[7] = 0.0
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(d, bits)
    cal = O.calibration32(O.calibrate(X[:500], R))
    enc = O.encode(X, R, c32, t32, bits, "unbiased", calib=cal)
    codes, scale = _planned(tq, T, X, R, c32, t32, bits, "unbiased",
                            calib=(T(cal.mu.astype(np.float32)), T(cal.a.astype(np.float32))))
    check_encode(codes, scale, X, enc, c32, t32, d, bits, "unbiased", calib=cal)


def test_encode_planned_matches_ffma_encoder(cuda_lib, tdev):
    """The two encoders differ only in the rounding of y: their codes agree
    except for one-cell flips, at most a few in 10^5."""
    torch, dev, T = tdev
    tq = cuda_lib
    d, n, bits = 1536, 3000, 4
    X = synth.mixture_corpus(n, d, 64, seed=21)
    R = O.rotation(d, 1536).astype(np.float32)
    c32, t32 = _cb(d, bits)
    a, sa = tq.encode(T(X), T(R), T(c32), T(t32), bits)
    b, sb = _planned(tq, T, X, R, c32, t32, bits)
    ua = O.unpack(a.cpu().numpy(), d, bits).astype(np.int64)
    ub = O.unpack(b, d, bits).astype(np.int64)
    diff = ua != ub
    assert np.all(np.abs(ua - ub)[diff] == 1)
    assert diff.mean() < 1e-4
    same = ~diff.any(axis=1)
    assert np.allclose(sa.cpu().numpy()[same], sb[same], rtol=2e-6)
