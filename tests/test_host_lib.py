"""libtq.so on the CPU: it loads, exports every symbol include/tq.h declares,
its host-only math (tq_codebook, tq_rotation) matches the oracle, and every
device call rejects invalid arguments before touching CUDA."""
import ctypes as C
import json
import os
import re

import numpy as np
import pytest

import oracle as O
import paper_2607_16973_gb300 as tq
from paper_2607_16973_gb300 import _lib
from paper_2607_16973_gb300.build import build
from conftest import GOLDEN, ROOT


@pytest.fixture(scope="module")
def lib():
    build()
    return tq.load()


def _header_functions():
    with open(os.path.join(ROOT, "include", "tq.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(tq_[a-z0-9_]+)\s*\(", text)))


def test_exports_every_declared_symbol(lib):
    names = _header_functions()
    assert "tq_search" in names and "tq_encode" in names and "tq_codebook" in names
    for name in names:
        assert hasattr(lib, name), name
    assert set(names) == set(_lib.SIGNATURES), "binding and header disagree"
    assert lib.tq_version() == 100


@pytest.mark.parametrize("marginal", ["beta", "gauss"])
@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_codebook_matches_oracle_golden(lib, marginal, bits):
    with open(os.path.join(GOLDEN, "codebooks.json")) as f:
        e = [e for e in json.load(f)["entries"] if e["bits"] == bits and e["marginal"] == marginal][0]
    c, t, D = tq.codebook(1536, bits, marginal)
    want_c = np.asarray(e["centroids"])
    want_t = np.asarray(e["boundaries"])
    # float32 outputs: within one float32 ulp of the float64 oracle (the oracle's
    # own fixed-point error is < 1e-9 relative at 8 bits)
    ulp_c = np.spacing(np.abs(want_c).astype(np.float32)).astype(np.float64)
    ulp_t = np.spacing(np.abs(want_t).astype(np.float32)).astype(np.float64)
    assert np.all(np.abs(c - want_c) <= ulp_c + 2e-9 * np.abs(want_c))
    assert np.all(np.abs(t - want_t) <= ulp_t + 2e-9 * np.abs(want_t) + 1e-30)
    assert D == pytest.approx(e["distortion"], rel=1e-8)
    assert t[len(t) // 2] == 0.0 and np.array_equal(c, -c[::-1])


@pytest.mark.parametrize("d", [32, 96, 512])
@pytest.mark.parametrize("bits", [2, 4])
def test_codebook_matches_oracle_small_d(lib, d, bits):
    c, t, D = tq.codebook(d, bits)
    ref = O.codebook(d, bits)
    assert np.allclose(c, ref.centroids, rtol=1.5e-7, atol=0)
    assert np.allclose(t, ref.boundaries, rtol=1.5e-7, atol=1e-30)
    assert D == pytest.approx(ref.distortion, rel=1e-9)


def test_codebook_is_data_free_and_deterministic(lib):
    a = tq.codebook(1536, 4)
    b = tq.codebook(1536, 4)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1]) and a[2] == b[2]


@pytest.mark.parametrize("d", [32, 160, 1536])
def test_rotation_matches_oracle(lib, d):
    R = tq.rotation(d, 1536)
    ref = O.rotation(d, 1536).astype(np.float32)
    diff = np.abs(R.astype(np.float64) - ref.astype(np.float64))
    assert np.all(diff <= np.spacing(np.abs(ref)).astype(np.float64))
    assert np.mean(R == ref) > 0.999


def _status(fn, *args):
    return fn(*args)


def test_invalid_arguments_rejected_without_gpu(lib):
    null = None
    # codebook / rotation
    assert lib.tq_codebook(4, 4, 0, null, null, null) == _lib.TQ_EINVAL
    assert lib.tq_codebook(64, 9, 0, null, null, null) == _lib.TQ_EINVAL
    assert lib.tq_codebook(64, 4, 7, null, null, null) == _lib.TQ_EINVAL
    assert lib.tq_rotation(1, 0, null) == _lib.TQ_EINVAL
    assert b"d=1" in lib.tq_last_error()
    # encode: d not a multiple of 32, bad bits, bad scale mode, NULL pointers, misalignment
    p = 4096
    assert lib.tq_encode(p, 10, 48, p, p, p, 4, 0, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_encode(p, 10, 64, p, p, p, 5, 0, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_encode(p, 10, 64, p, p, p, 4, 9, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_encode(null, 10, 64, p, p, p, 4, 0, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_encode(p + 4, 10, 64, p, p, p, 4, 0, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_encode(null, 0, 64, null, null, null, 4, 0, null, null, null) == _lib.TQ_OK
    # search
    args = [p, 1, 64, p, p, 4, p, p, 100, null, null, null, 10, p, p, p, 1 << 20, null]

    def search(**kw):
        a = list(args)
        names = ["Q", "nq", "d", "R", "cen", "bits", "codes", "scale", "n", "filter", "off",
                 "ten", "k", "ids", "scores", "ws", "wsb", "stream"]
        for k_, v in kw.items():
            a[names.index(k_)] = v
        return lib.tq_search(*a)

    assert search(k=0) == _lib.TQ_EINVAL
    assert search(k=257) == _lib.TQ_EINVAL
    assert search(bits=1) == _lib.TQ_EINVAL
    assert search(d=40) == _lib.TQ_EINVAL
    assert search(n=0) == _lib.TQ_EINVAL
    assert search(Q=null) == _lib.TQ_EINVAL
    assert search(codes=p + 8) == _lib.TQ_EINVAL
    assert search(ws=null) == _lib.TQ_EINVAL
    assert search(nq=0) == _lib.TQ_OK
    # search over an id map: misaligned tombstone bitmap / external ids
    ex = list(args[:12]) + [p + 2, null, null, null] + list(args[12:])
    assert lib.tq_search_ex(*ex) == _lib.TQ_EINVAL
    ex[12], ex[13] = null, p + 4
    assert lib.tq_search_ex(*ex) == _lib.TQ_EINVAL
    ex[13], ex[16] = null, 0
    assert lib.tq_search_ex(*ex) == _lib.TQ_EINVAL
    # a TQ+ calibration needs both arrays, 4-byte aligned
    ex[16] = 5
    ex[14] = p
    assert lib.tq_search_ex(*ex) == _lib.TQ_EINVAL and b"both mu and a" in lib.tq_last_error()
    ex[14], ex[15] = p + 1, p
    assert lib.tq_search_ex(*ex) == _lib.TQ_EINVAL
    # TQ+ calibration and calibrated encode: argument checks (no device memory is touched)
    sz = C.c_size_t()
    assert lib.tq_calibrate_workspace(0, 64, C.byref(sz)) == _lib.TQ_EINVAL
    assert lib.tq_calibrate_workspace(10, 48, C.byref(sz)) == _lib.TQ_EINVAL
    assert lib.tq_calibrate_workspace(300, 64, C.byref(sz)) == _lib.TQ_OK
    assert sz.value == 3 * 64 * 16 + 3 * 4   # 3 panels of 128 rows: sums, squares (double), counts
    assert lib.tq_calibrate(p, 300, 64, p, p, p, p, sz.value - 1, null) == _lib.TQ_EINVAL
    assert lib.tq_calibrate(null, 300, 64, p, p, p, p, sz.value, null) == _lib.TQ_EINVAL
    assert lib.tq_encode_ex(p, 10, 64, p, p, p, 4, 0, p, null, p, p, null) == _lib.TQ_EINVAL
    # tensor-core encode plan: sizes and argument checks (no device memory is touched)
    assert lib.tq_encode_plan_bytes(1536, C.byref(sz)) == _lib.TQ_OK
    assert sz.value == 256 + 2 * 1536 * 1536 * 4    # status header, R_hi, R_lo
    for d in (64, 96, 130, 8224):
        assert lib.tq_encode_plan_bytes(d, C.byref(sz)) == _lib.TQ_EUNSUPPORTED
    assert lib.tq_encode_plan_bytes(128, null) == _lib.TQ_EINVAL
    assert lib.tq_encode_plan(p, 96, p, 1 << 20, null) == _lib.TQ_EUNSUPPORTED
    assert lib.tq_encode_plan(p, 128, p + 8, 1 << 20, null) == _lib.TQ_EINVAL
    assert lib.tq_encode_plan(p, 128, p, 1000, null) == _lib.TQ_EINVAL
    planned = lambda **kw: lib.tq_encode_planned(*[kw.get(k, v) for k, v in (
        ("X", p), ("n", 10), ("d", 128), ("plan", p), ("c", p), ("b", p), ("bits", 4), ("mode", 0),
        ("mu", null), ("a", null), ("codes", p), ("scale", p), ("s", null))])
    assert planned(d=96) == _lib.TQ_EUNSUPPORTED
    assert planned(d=100) == _lib.TQ_EINVAL
    assert planned(bits=5) == _lib.TQ_EINVAL
    assert planned(plan=null) == _lib.TQ_EINVAL
    assert planned(plan=p + 4) == _lib.TQ_EINVAL
    assert planned(mu=p) == _lib.TQ_EINVAL
    assert planned(n=-1) == _lib.TQ_EINVAL
    assert planned(n=0) == _lib.TQ_OK
    assert lib.tq_encode_check(null, null) == _lib.TQ_EINVAL
    # id map: capacity, NULL handle / ids (no device memory is touched)
    m = C.c_void_p()
    assert lib.tq_idmap_create(0, C.byref(m)) == _lib.TQ_EINVAL
    assert lib.tq_idmap_create(1 << 31, C.byref(m)) == _lib.TQ_EINVAL
    assert lib.tq_idmap_create(10, null) == _lib.TQ_EINVAL
    r = C.c_int64()
    assert lib.tq_idmap_add(null, p, 1, C.byref(r), null) == _lib.TQ_EINVAL
    assert lib.tq_idmap_remove(null, p, 1, C.byref(r), null) == _lib.TQ_EINVAL
    assert lib.tq_idmap_lookup(null, 5, C.byref(r)) == _lib.TQ_EINVAL
    assert lib.tq_idmap_info(null, null, null, null) == _lib.TQ_EINVAL
    assert lib.tq_idmap_device(null, null, null) == _lib.TQ_EINVAL
    assert lib.tq_idmap_destroy(null) == _lib.TQ_OK
    assert lib.tq_idmap_export(null, p, p) == _lib.TQ_EINVAL
    assert lib.tq_idmap_import(null, p, p, 1, null) == _lib.TQ_EINVAL
    assert lib.tq_filter_append(null, p, 1, null) == _lib.TQ_EINVAL
    # filter
    h = C.c_void_p()
    assert lib.tq_filter_build(p, 10, 48, C.byref(h), null) == _lib.TQ_EINVAL
    assert lib.tq_filter_build(p, 0, 64, C.byref(h), null) == _lib.TQ_EINVAL
    assert lib.tq_filter_destroy(null) == _lib.TQ_OK
    # merge: sources, candidates per source, k, NULL and misaligned pointers
    assert lib.tq_merge_topk(p, p, 0, 4, 10, 5, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_merge_topk(p, p, 2, 4, -1, 5, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_merge_topk(p, p, 2, 4, 10, 0, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_merge_topk(p, p, 2, 4, 10, 257, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_merge_topk(null, p, 2, 4, 10, 5, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_merge_topk(p + 4, p, 2, 4, 10, 5, p, p, null) == _lib.TQ_EINVAL
    assert lib.tq_merge_topk(null, null, 2, 0, 10, 5, null, null, null) == _lib.TQ_OK
    # status check and testing hooks
    assert lib.tq_search_check(null, null) == _lib.TQ_EINVAL
    assert lib.tq_search_check(p + 4, null) == _lib.TQ_EINVAL
    assert lib.tq_debug_fail_allocs(-1) == _lib.TQ_EINVAL
    assert lib.tq_debug_fail_allocs(0) == _lib.TQ_OK
    assert lib.tq_debug_bounded_wait(0, p, null) == _lib.TQ_EINVAL
    assert lib.tq_debug_bounded_wait(5_000_000_000, p, null) == _lib.TQ_EINVAL
    assert lib.tq_debug_bounded_wait(1000, null, null) == _lib.TQ_EINVAL
    assert lib.tq_set_search_path(7) == _lib.TQ_EINVAL
    assert lib.tq_set_search_path(-1) == _lib.TQ_EINVAL
    for name, path in _lib.PATHS.items():  # every named path is accepted (auto last)
        assert lib.tq_set_search_path(path) == _lib.TQ_OK, name
    assert lib.tq_set_search_path(_lib.PATHS["auto"]) == _lib.TQ_OK
    assert lib.tq_profile_events(p, null) == _lib.TQ_EINVAL


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(_lib, "_lib", None)
    monkeypatch.setattr(_lib, "LIB_PATH", str(tmp_path / "libtq.so"))
    with pytest.raises(RuntimeError, match="missing"):
        _lib.load()
