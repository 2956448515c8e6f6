"""The C ABI library: it loads, exports every entry point the header declares,
and rejects invalid shapes, budgets and workspaces on the host before any
launch (CPU only; no compute call reaches a GPU)."""
import ctypes
import os
import re

import pytest

from paper_2608_21541_gb300 import build as B
from paper_2608_21541_gb300 import certkv as ck

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "certkv.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return ck.load_library()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(certkv_[a-z_]+)\s*\(", text)))


def test_header_declares_the_entry_points():
    names = declared_functions()
    assert set(names) == set(ck.EXPORTED), names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def shape(**kw):
    s = dict(batch=1, layers=2, hq=32, hkv=8, n=4096, d=128, w=32)
    s.update(kw)
    return ck.certkv_shape(**s)


def test_defaults_and_budget(lib):
    p = ck.certkv_default_params()
    assert (p.pool_kernel, p.protect_window, p.alpha_num, p.alpha_den, p.bisect_steps,
            p.statistic, p.tail_slot) == (5, 1, 1, 5, 40, 0, 1)
    assert ck.certkv_live_budget(4096, 8, 1, 10) == 8 * 409
    assert ck.certkv_live_budget(65536, 8, 1, 10) == 8 * 6553
    assert ck.certkv_live_budget(131072, 8, 1, 20) == 8 * 6553
    assert ck.certkv_live_budget(4000, 1, 1, 10) == 400  # exact rational, no float floor
    assert ck.certkv_live_budget(10, 1, 3, 2) == -1


@pytest.mark.parametrize("bad", [dict(d=64), dict(hkv=33, hq=33), dict(hq=24, hkv=8),
                                 dict(hq=12, hkv=4), dict(w=0), dict(w=4096), dict(n=(1 << 24) + 1),
                                 dict(batch=0)])
def test_invalid_shapes_have_no_workspace(lib, bad):
    assert ck.certkv_workspace_bytes(shape(**bad)) == 0


def test_workspace_size_grows_with_the_problem(lib):
    a = ck.certkv_workspace_bytes(shape(n=4096))
    b = ck.certkv_workspace_bytes(shape(n=8192))
    assert 0 < a < b
    assert ck.certkv_decode_workspace_bytes(shape()) > 0


def _call_compress(lib, shp, budget, params=None, ws_bytes=None, ws_ptr=256, cap=None,
                   k_ptr=1 << 20):
    params = params or ck.certkv_default_params()
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: validation fails first
    need = lib.certkv_workspace_bytes(ctypes.byref(shp), ctypes.byref(params))
    packed = ck.certkv_packed(fake, fake, fake, fake, fake,
                              cap if cap is not None else 1 << 40, None, None)
    return lib.certkv_compress(ctypes.byref(shp), ctypes.c_void_p(k_ptr), fake, fake, budget,
                               ctypes.byref(params),
                               ctypes.byref(packed),
                               ctypes.c_void_p(ws_ptr) if ws_ptr else None,
                               need if ws_bytes is None else ws_bytes, None)


def test_host_validation_errors(lib):
    s = shape()
    H, n = s.hkv, s.n
    assert _call_compress(lib, shape(d=64), 2 * H) == ck.EINVAL
    assert _call_compress(lib, s, 2 * H - 1) == ck.EBUDGET          # n_keep < 2
    assert _call_compress(lib, s, H * n + 1) == ck.EBUDGET          # beyond H * n
    assert _call_compress(lib, s, -5) == ck.EBUDGET
    assert _call_compress(lib, s, 2 * H, ws_ptr=0) == ck.EWORKSPACE
    assert _call_compress(lib, s, 2 * H, ws_ptr=257) == ck.EWORKSPACE  # misaligned
    assert _call_compress(lib, s, 2 * H, ws_bytes=1024) == ck.EWORKSPACE
    assert _call_compress(lib, s, 2 * H, k_ptr=(1 << 20) + 8) == ck.EINVAL  # K not 16-B aligned
    assert _call_compress(lib, s, 40 * H, cap=10) == ck.ECAPACITY
    bad = ck.certkv_default_params(pool_kernel=4)
    assert _call_compress(lib, s, 2 * H, params=bad) == ck.EINVAL
    bad = ck.certkv_default_params(alpha_num=6, alpha_den=5)
    assert _call_compress(lib, s, 2 * H, params=bad) == ck.EINVAL
    bad = ck.certkv_default_params(statistic=3)
    assert _call_compress(lib, s, 2 * H, params=bad) == ck.EINVAL
    bad = ck.certkv_default_params(allocator=3)
    assert _call_compress(lib, s, 2 * H, params=bad) == ck.EINVAL
    # without a tail slot the smallest budget is H
    ns = ck.certkv_default_params(tail_slot=0)
    assert _call_compress(lib, s, H - 1, params=ns) == ck.EBUDGET
    assert ck.certkv_strerror(ck.EBUDGET).startswith("infeasible")


def test_binding_refuses_a_missing_library(tmp_path):
    saved = ck._lib
    try:
        ck._lib = None
        with pytest.raises(RuntimeError, match="not found"):
            ck.load_library(str(tmp_path / "missing.so"))
    finally:
        ck._lib = saved


def test_host_entry_point_validation(lib):
    s = shape()
    params = ck.certkv_default_params()
    need_dev = lib.certkv_workspace_bytes(ctypes.byref(s), ctypes.byref(params))
    need = lib.certkv_host_workspace_bytes(ctypes.byref(s), ctypes.byref(params), 0)
    assert need > need_dev  # device workspace of a chunk plus two staging halves
    assert lib.certkv_host_workspace_bytes(ctypes.byref(s), ctypes.byref(params), -1) == 0
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: validation fails first
    packed = ck.certkv_packed(fake, fake, fake, fake, fake, 1 << 40, None, None)

    def call(chunk=0, ws=256, ws_bytes=None, budget=2 * s.hkv, k=fake):
        return lib.certkv_compress_host(ctypes.byref(s), k, fake, fake, budget,
                                        ctypes.byref(params), chunk, ctypes.byref(packed),
                                        ctypes.c_void_p(ws) if ws else None,
                                        need if ws_bytes is None else ws_bytes, None)

    assert call(chunk=-1) == ck.EINVAL
    assert call(k=None) == ck.EINVAL
    assert call(budget=-3) == ck.EBUDGET
    assert call(ws=0) == ck.EWORKSPACE
    assert call(ws=257) == ck.EWORKSPACE
    assert call(ws_bytes=need - 1) == ck.EWORKSPACE


def test_host_copyback_validation(lib):
    s = shape()
    params = ck.certkv_default_params()
    need = lib.certkv_host_workspace_bytes(ctypes.byref(s), ctypes.byref(params), 0)
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: validation fails first
    budget = 2 * s.hkv
    slots = budget * s.batch * s.layers
    packed = ck.certkv_packed(fake, fake, fake, fake, fake, 1 << 40, None, None)

    def host(k=fake, cap=slots, pos=fake):
        return ck.certkv_packed(k, fake, fake, fake, pos, cap, None, None)

    def call(h, ws=256):
        return lib.certkv_compress_host_copyback(
            ctypes.byref(s), fake, fake, fake, budget, ctypes.byref(params), 0,
            ctypes.byref(packed), ctypes.byref(h) if h is not None else None,
            ctypes.c_void_p(ws) if ws else None, need, None)

    assert call(None) == ck.EINVAL               # no host output
    assert call(host(k=None)) == ck.EINVAL       # a missing host buffer
    assert call(host(pos=None)) == ck.EINVAL
    assert call(host(cap=slots - 1)) == ck.EINVAL  # too few host slots
    assert call(host(), ws=0) == ck.EWORKSPACE   # the rest as certkv_compress_host


def test_coverage_profile_validation(lib):
    s = shape()
    need = lib.certkv_coverage_workspace_bytes(ctypes.byref(s))
    assert need > 16 * s.n * s.batch * s.layers * s.hq
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: validation fails first

    def arr(*x):
        return (ctypes.c_double * max(len(x), 1))(*x)

    def call(eta=(0.1,), rel=(0.1,), ab=(0.01,), out=fake, ws=256, ws_bytes=None, scale=0.0,
             n_eta=None):
        return lib.certkv_coverage_profile(
            ctypes.byref(s), fake, fake, scale, arr(*eta), len(eta) if n_eta is None else n_eta,
            arr(*rel), len(rel), arr(*ab), len(ab), out, out, out, fake, None, None,
            ctypes.c_void_p(ws) if ws else None, need if ws_bytes is None else ws_bytes, None)

    assert call(eta=(1.0,)) == ck.EINVAL          # eta must lie in (0, 1)
    assert call(eta=(0.0,)) == ck.EINVAL
    assert call(rel=(0.0,)) == ck.EINVAL          # thresholds positive
    assert call(ab=(float("inf"),)) == ck.EINVAL
    assert call(out=None) == ck.EINVAL            # an output missing for a nonzero count
    assert call(n_eta=17) == ck.EINVAL            # at most 16 thresholds per kind
    assert call(scale=-1.0) == ck.EINVAL
    assert call(ws=0) == ck.EWORKSPACE
    assert call(ws_bytes=need - 1) == ck.EWORKSPACE
    # counts of zero need no arrays
    assert lib.certkv_coverage_profile(
        ctypes.byref(s), fake, fake, 0.0, None, 0, None, 0, None, 0, None, None, None, fake,
        None, None, None, need, None) == ck.EWORKSPACE


def test_sampled_compensation_validation(lib):
    s = shape()
    need = lib.certkv_sampled_workspace_bytes(ctypes.byref(s))
    assert need > lib.certkv_fixed_row_workspace_bytes(ctypes.byref(s))
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: validation fails first
    packed = ck.certkv_packed(fake, fake, fake, fake, fake, 1 << 40, None, None)

    def call(m=4, unif=fake, ws=256, ws_bytes=None, scale=0.0):
        return lib.certkv_sampled_compensation(ctypes.byref(s), fake, fake, fake,
                                               ctypes.byref(packed), scale, m, unif, None, fake,
                                               ctypes.c_void_p(ws) if ws else None,
                                               need if ws_bytes is None else ws_bytes, None)

    assert call(m=0) == ck.EINVAL
    assert call(m=65) == ck.EINVAL  # at most CERTKV_MAX_SAMPLES
    assert call(unif=None) == ck.EINVAL
    assert call(scale=float("nan")) == ck.EINVAL
    assert call(ws=0) == ck.EWORKSPACE
    assert call(ws_bytes=need - 1) == ck.EWORKSPACE


def test_workspace_guards_refuse_bad_arguments_on_the_host(lib):
    """Guard words: an invalid shape or a missing, misaligned or short
    workspace returns -1 before anything is enqueued."""
    s, p = shape(), ck.certkv_default_params()
    need = ck.certkv_workspace_bytes(s, p)
    assert need > 0
    for fn in (lib.certkv_workspace_guard_arm, lib.certkv_workspace_guard_check):
        assert fn(ctypes.byref(s), ctypes.byref(p), None, need, None) == -1
        assert fn(ctypes.byref(s), ctypes.byref(p), ctypes.c_void_p(256), need - 1, None) == -1
        assert fn(ctypes.byref(s), ctypes.byref(p), ctypes.c_void_p(16), need, None) == -1
        assert fn(ctypes.byref(shape(d=64)), ctypes.byref(p), ctypes.c_void_p(256), need, None) == -1


def test_bounds_checking_build_compiles_and_exports_the_same_symbols():
    """The -DCERTKV_DEBUG build (bounds checks on every ragged index) links
    with the same entry points (compiled here; its GPU test is
    tests/test_gpu_debug.py)."""
    path = B.build(debug=True)
    dbg = ctypes.CDLL(path)
    for name in declared_functions():
        assert hasattr(dbg, name), name
