"""The C-ABI library builds, loads and exports every entry point that
include/hc.h declares; host-side argument checks reject bad calls before
anything reaches a GPU. No compute call is made here (no GPU needed)."""
import ctypes
import os
import re

import pytest

from paper_2608_09388_gb300 import build, hc

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "hc.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(hc_[a-z_0-9]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return hc.load_library()


def test_header_declares_the_boundary():
    d = _declared()
    for name in ("hc_mask_compact", "hc_sparse_spiral_conv_fwd", "hc_sparse_linear_fwd",
                 "hc_scatter_dense", "hc_spiral_conv_fwd", "hc_get_device_status",
                 "hc_last_error_string"):
        assert name in d
    assert set(hc.EXPORTS) <= set(d)


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), f"libhc.so does not export {name}"


def test_version(lib):
    assert re.match(r"^\d+\.\d+\.\d+$", hc.hc_version())


# Host-side validation returns before any CUDA call, so it runs without a GPU.
def test_invalid_arguments_rejected_on_host(lib):
    P = ctypes.c_void_p
    fake = P(0x1000)
    assert lib.hc_mask_compact(fake, -1, 5, fake, None, None, fake, None) == hc.HC_ERR_INVALID_ARG
    assert lib.hc_mask_compact(fake, 2, 5, fake, None, None, None, None) == hc.HC_ERR_INVALID_ARG
    assert "count" in hc.hc_last_error_string()
    # unknown dtype
    assert lib.hc_sparse_spiral_conv_fwd(fake, 0, 7, fake, fake, fake, fake, 1, 4, 3, 8, 8, fake,
                                         None, 1, fake, None) == hc.HC_ERR_INVALID_ARG
    # spiral longer than supported
    assert lib.hc_sparse_spiral_conv_fwd(fake, 0, 1, fake, fake, fake, fake, 1, 40, 33, 8, 8, fake,
                                         None, 1, fake, None) == hc.HC_ERR_UNSUPPORTED
    # unknown activation
    assert lib.hc_spiral_conv_fwd(fake, 1, fake, 1, 4, 3, 8, 8, fake, None, 9, fake,
                                  None) == hc.HC_ERR_INVALID_ARG
    # a negative row estimate
    lib.hc_sparse_conv_rulebook_fwd_hint.argtypes = [P, ctypes.c_int, ctypes.c_int, P, P,
                                                     ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                                     ctypes.c_int, P, P, ctypes.c_int, P, P,
                                                     ctypes.c_int, ctypes.c_int, P,
                                                     ctypes.c_longlong, P]
    assert lib.hc_sparse_conv_rulebook_fwd_hint(fake, 1, 10, fake, fake, 10, 9, 16, 128, fake,
                                                None, 1, fake, None, 0, 0, None, -1,
                                                None) == hc.HC_ERR_INVALID_ARG
    assert "rows_hint" in hc.hc_last_error_string()
    # misaligned pointer for the element size
    assert lib.hc_spiral_conv_fwd(P(0x1001), 1, fake, 1, 4, 3, 8, 8, fake, None, 1, fake,
                                  None) == hc.HC_ERR_INVALID_ARG
    # neither coords nor (with zero_fill) row_of
    assert lib.hc_scatter_dense(fake, 1, None, None, fake, 2, 3, 8, 1, fake,
                                None) == hc.HC_ERR_INVALID_ARG
    assert lib.hc_scatter_dense(fake, 1, None, fake, fake, 2, 3, 8, 0, fake,
                                None) == hc.HC_ERR_INVALID_ARG
    # test hooks: unknown option, group-norm path out of range (no CUDA call)
    assert lib.hc_test_set_option(99, 0) == hc.HC_ERR_INVALID_ARG
    assert lib.hc_test_set_option(hc.HC_TEST_GROUP_NORM_PATH, 3) == hc.HC_ERR_INVALID_ARG
    assert lib.hc_test_set_option(hc.HC_TEST_WAIT_LIMIT_NS, -5) == hc.HC_ERR_INVALID_ARG
    # negative capacity
    assert lib.hc_sparse_linear_fwd(fake, 1, fake, -1, 8, 8, fake, None, 0, fake,
                                    None) == hc.HC_ERR_INVALID_ARG
    # C_in < 1
    assert lib.hc_sparse_linear_fwd(fake, 1, fake, 4, 0, 8, fake, None, 0, fake,
                                    None) == hc.HC_ERR_INVALID_ARG


def test_missing_library_fails_loudly(tmp_path, monkeypatch):
    monkeypatch.setattr(hc, "_lib", None)
    with pytest.raises(RuntimeError, match="not built"):
        hc.load_library(str(tmp_path / "nope.so"))


def test_group_norm_arguments_rejected_on_host(lib):
    fake = ctypes.c_void_p(0x1000)
    f = ctypes.c_float
    gn = lib.hc_sparse_group_norm_fwd
    bad = [
        (fake, 0, fake, 2, 10, 10, 3, f(1e-5), None, None, 0, fake, None),  # C % G != 0
        (fake, 0, fake, 2, 10, 8, 0, f(1e-5), None, None, 0, fake, None),   # G = 0
        (fake, 0, fake, 2, 10, 8, 2, f(-1.0), None, None, 0, fake, None),   # eps < 0
        (fake, 7, fake, 2, 10, 8, 2, f(1e-5), None, None, 0, fake, None),   # dtype
        (fake, 0, fake, 2, 10, 8, 2, f(1e-5), None, None, 9, fake, None),   # activation
        (fake, 0, None, 2, 10, 8, 2, f(1e-5), None, None, 0, fake, None),   # no offsets
    ]
    for args in bad:
        assert gn(*args) == hc.HC_ERR_INVALID_ARG
    # nothing to do: returns before any device call
    assert gn(fake, 0, fake, 0, 10, 8, 2, f(1e-5), None, None, 0, fake, None) == hc.HC_OK


def test_conv_gn_arguments_rejected_on_host(lib):
    fake = ctypes.c_void_p(0x1000)
    f = ctypes.c_float
    cg = lib.hc_sparse_conv_gn_fwd

    def call(dt=1, x_rows=100, count=fake, capacity=100, L=9, C_in=16, C_out=64, coords=fake,
             offs=fake, B=2, G=8, eps=1e-5, act=1):
        return cg(fake, dt, x_rows, fake, count, capacity, L, C_in, C_out, fake, None, coords,
                  offs, B, G, f(eps), None, None, act, fake, None)

    for kw in (dict(G=7), dict(G=0), dict(B=0), dict(eps=-1.0), dict(dt=5), dict(act=9),
               dict(coords=None), dict(offs=None), dict(count=None), dict(x_rows=0),
               dict(capacity=-1), dict(C_out=0)):
        assert call(**kw) == hc.HC_ERR_INVALID_ARG, kw
    assert call(L=10 ** 4) == hc.HC_ERR_UNSUPPORTED
    # nothing to do: returns before any device call
    assert call(capacity=0) == hc.HC_OK


def test_compact_rulebook_arguments_rejected_on_host(lib):
    fake = ctypes.c_void_p(0x1000)
    f = lib.hc_mask_compact_rulebook

    def call(mask=fake, B=2, V=100, spiral=fake, L=9, layout=0, coords=fake, row_of=fake,
             count=fake, rb=fake):
        return f(mask, B, V, spiral, L, layout, coords, row_of, None, count, rb, None)

    for kw in (dict(B=-1), dict(V=-3), dict(L=0), dict(layout=5), dict(count=None),
               dict(mask=None), dict(spiral=None), dict(coords=None), dict(row_of=None),
               dict(rb=None), dict(B=1 << 16, V=1 << 15)):
        assert call(**kw) == hc.HC_ERR_INVALID_ARG, kw
    assert call(L=33) == hc.HC_ERR_UNSUPPORTED


def test_gather_rows_arguments_rejected_on_host(lib):
    fake = ctypes.c_void_p(0x1000)
    g = lib.hc_gather_rows

    def call(x=fake, dt=1, B_in=2, V=100, C=64, coords=fake, count=fake, cap=200, fps=1, y=fake):
        return g(x, dt, B_in, V, C, coords, count, cap, fps, y, None)

    for kw in (dict(dt=9), dict(B_in=-1), dict(C=0), dict(fps=0), dict(cap=-1), dict(count=None),
               dict(x=None), dict(y=None), dict(x=ctypes.c_void_p(0x1001))):
        assert call(**kw) == hc.HC_ERR_INVALID_ARG, kw
    assert call(cap=0) == hc.HC_OK  # nothing to gather: no device call
    assert call(cap=0, coords=None) == hc.HC_OK  # rows in order: coords are optional


def test_binding_refuses_pageable_host_tensors(lib):
    """Host memory is accepted only pinned, and only by hc_gather_rows (its
    input and output); a pageable tensor is refused before any library call."""
    torch = pytest.importorskip("torch")
    x = torch.zeros((2, 10, 8), dtype=torch.float32)
    coords = torch.zeros((20, 2), dtype=torch.int32)
    count = torch.zeros((1,), dtype=torch.int32)
    y = torch.zeros((20, 8), dtype=torch.float32)
    with pytest.raises(ValueError):
        hc.hc_gather_rows(x, coords, count, 1, y)
    with pytest.raises(ValueError):
        hc.hc_sparse_linear_fwd(y, count, torch.zeros((8, 8)), None, hc.HC_ACT_NONE, y)
