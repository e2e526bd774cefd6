"""The row-count-dispatched tensor-core kernel (conv_tc_auto_kernel): a
128-channel rulebook call without a row estimate, whose capacity could give
every SM a two-half item, reads N' on the device and runs two-half
transposed items when N' >= 256 x CTAs (one CTA per SM), one-half items
below. Around that threshold, and at no rows, one row, a ragged last item
and the full capacity: every row against the oracle (Eqs. 4-5 with the bias
and ELU), bit-identical to the calls that force each item shape through a
row estimate, rows past N' untouched; bad rulebook entries reported in both
branches and contributing nothing."""
import os

import numpy as np
import pytest

import oracle
from paper_2608_09388_gb300 import hc, inputs

from _util import check_close, sample_rows, to_numpy, to_torch

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
NCPU = len(os.sched_getaffinity(0))
B, V, L, C_IN = 4, 10475, 9, 64


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_09388_gb300 import build
    build.build()
    hc.load_library()
    assert hc.hc_get_device_status() == hc.HC_OK


@pytest.fixture(scope="module")
def case():
    """Random spiral (slot 0 the vertex itself, ~10% absent entries),
    features, weights and bias of a 64 -> 128 ELU layer on 4 x 10475
    vertices: a capacity of 41,900 rows, above 256 rows per SM."""
    rng = np.random.default_rng(2024)
    sp = rng.integers(0, V, size=(V, L)).astype(np.int32)
    sp[rng.random((V, L)) < 0.1] = -1
    sp[:, 0] = np.arange(V)
    x = inputs.features(rng, (B, V, C_IN), "bf16")
    W = inputs.weights(rng, L * C_IN, 128, "bf16")
    b = rng.standard_normal(128).astype(np.float32)
    order = rng.permutation(B * V)  # vertices made active, in this order
    return sp, x, W, b, order


def threshold():
    return 256 * torch.cuda.get_device_properties(0).multi_processor_count


def mask_with(order, n):
    m = np.zeros(B * V, np.uint8)
    m[order[:n]] = 1
    return m.reshape(B, V)


def rulebook(m, sp):
    coords = torch.empty((B * V, 2), dtype=torch.int32, device="cuda")
    row_of = torch.empty((B, V), dtype=torch.int32, device="cuda")
    offs = torch.empty((B + 1,), dtype=torch.int32, device="cuda")
    count = torch.empty((1,), dtype=torch.int32, device="cuda")
    rb = torch.empty((sp.shape[1], B * V), dtype=torch.int32, device="cuda")
    hc.hc_mask_compact_rulebook(to_torch(m), to_torch(sp), hc.HC_LAYOUT_DENSE, coords, row_of,
                                offs, count, rb)
    return rb, count


def run(x, rb, count, W, b, hint=None):
    y = torch.full((B * V, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    if hint is None:
        hc.hc_sparse_conv_rulebook_fwd(x, rb, count, W, b, hc.HC_ACT_ELU, y)
    else:
        hc.hc_sparse_conv_rulebook_fwd_hint(x, rb, count, W, b, hc.HC_ACT_ELU, y, hint)
    return y


@pytest.mark.parametrize("offset", [-1, 0, 1, 255, 256, 300])
def test_both_branches_at_the_threshold(case, offset):
    """N' = 256 x SMs + offset: one-half items just below, two-half
    transposed items from the threshold up (exact, one row into a new item,
    a full last item, a ragged one)."""
    sp, x, W, b, order = case
    n = threshold() + offset
    assert n <= B * V
    m = mask_with(order, n)
    rb, count = rulebook(m, sp)
    assert int(count.item()) == n
    xt, Wt, bt = to_torch(x), to_torch(W), to_torch(b)
    y = run(xt, rb, count, Wt, bt)
    assert hc.hc_get_device_status() == hc.HC_OK
    assert torch.isnan(y[n:].float()).all()
    for hint in (1, B * V):  # forced one-half, forced two-half transposed
        assert torch.equal(run(xt, rb, count, Wt, bt, hint)[:n], y[:n]), f"hint {hint}"
    c, r, _, _ = oracle.mask_compact(m)
    y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c, r, sp, W, b, oracle.ACT_ELU,
                                         n_threads=NCPU)
    check_close(to_numpy(y)[:n], y_pre, f"auto N'={n}")


@pytest.mark.parametrize("n", [0, 1, 5000, B * V])
def test_small_and_full_counts(case, n):
    """No rows, one row, a count far below the threshold (one-half items on
    a few CTAs), every vertex active."""
    sp, x, W, b, order = case
    m = mask_with(order, n)
    rb, count = rulebook(m, sp)
    xt, Wt, bt = to_torch(x), to_torch(W), to_torch(b)
    y = run(xt, rb, count, Wt, bt)
    assert hc.hc_get_device_status() == hc.HC_OK
    assert torch.isnan(y[n:].float()).all()
    assert torch.equal(run(xt, rb, count, Wt, bt, 1)[:n], y[:n])
    if n:
        c, r, _, _ = oracle.mask_compact(m)
        y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c, r, sp, W, b,
                                             oracle.ACT_ELU, n_threads=NCPU)
        check_close(to_numpy(y)[:n], y_pre, f"auto N'={n}")


@pytest.mark.parametrize("offset", [-1, 0])
def test_bad_entries_reported_in_both_branches(case, offset):
    """Out-of-range rulebook entries of active rows, in the first item of a
    CTA (the one-half roles' prefetched table) and in a later one: the call
    reports HC_ERR_INVALID_INDEX and its rows are those of the same rulebook
    with the entries absent."""
    sp, x, W, b, order = case
    n = threshold() + offset
    rb, count = rulebook(mask_with(order, n), sp)
    xt, Wt, bt = to_torch(x), to_torch(W), to_torch(b)
    bad = [(2, 5, B * V), (1, 7, -3), (4, n - 3, B * V + 11), (0, 200 * 128 + 9, -2)]
    for l, col, v in bad:
        rb[l, col] = v
    y = run(xt, rb, count, Wt, bt)
    assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
    for l, col, _ in bad:
        rb[l, col] = -1
    y_abs = run(xt, rb, count, Wt, bt)
    assert hc.hc_get_device_status() == hc.HC_OK
    assert torch.equal(y[:n], y_abs[:n])


@pytest.mark.parametrize("L,C_in,act", [(1, 64, hc.HC_ACT_ELU), (12, 64, hc.HC_ACT_RELU),
                                        (32, 64, hc.HC_ACT_NONE), (9, 45, hc.HC_ACT_ELU),
                                        (5, 200, hc.HC_ACT_ELU)])
@pytest.mark.parametrize("branch", ["one-half", "two-half"])
def test_spiral_lengths_and_channels(L, C_in, act, branch):
    """Other spiral lengths (one k-block per slot up to 32 slots: the rings'
    stage counts change with the tables' size), 45 input channels (padded to
    48 by the channel-padding pass, then this kernel), 200 (a ragged last
    k-block), each activation, in both branches: sampled rows (all of the
    first and last item) against the oracle, every row bit-identical to the
    call forcing that item shape, rows past N' untouched."""
    rng = np.random.default_rng(L * 1000 + C_in)
    sp = rng.integers(0, V, size=(V, L)).astype(np.int32)
    sp[rng.random((V, L)) < 0.1] = -1
    sp[:, 0] = np.arange(V)
    x = inputs.features(rng, (B, V, C_in), "bf16")
    W = inputs.weights(rng, L * C_in, 128, "bf16")
    b = rng.standard_normal(128).astype(np.float32)
    n = threshold() + 123 if branch == "two-half" else 20000
    m = mask_with(rng.permutation(B * V), n)
    rb, count = rulebook(m, sp)
    xt, Wt, bt = to_torch(x), to_torch(W), to_torch(b)
    y = torch.full((B * V, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    hc.hc_sparse_conv_rulebook_fwd(xt, rb, count, Wt, bt, act, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    assert torch.isnan(y[n:].float()).all()
    forced = torch.full_like(y, float("nan"))
    hc.hc_sparse_conv_rulebook_fwd_hint(xt, rb, count, Wt, bt, act, forced,
                                        B * V if branch == "two-half" else 1)
    assert torch.equal(forced[:n], y[:n])
    c, r, _, _ = oracle.mask_compact(m)
    rows = np.unique(np.concatenate([np.arange(256), np.arange(n - 256, n),
                                     sample_rows(n, 3000, seed=L)]))
    y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c, r, sp, W, b, act, rows=rows,
                                         n_threads=NCPU)
    check_close(to_numpy(y)[rows], y_pre, f"auto L={L} C_in={C_in} {branch}")


@pytest.mark.parametrize("layout", [hc.HC_LAYOUT_DENSE, hc.HC_LAYOUT_COMPACT])
@pytest.mark.parametrize("offset", [-1, 7, None])
def test_resolved_taps_both_layouts(case, layout, offset):
    """hc_sparse_spiral_conv_fwd (taps resolved from coords, spiral and
    row_of inside the kernel) goes through the same dispatch: one-half items
    below 256 rows per SM, two-half transposed items from there up to every
    vertex active (offset None), dense and compact inputs; bit-identical to
    the rulebook call on the same layout, sampled rows (all of the first and
    last item) against the oracle, rows past N' untouched."""
    sp, x, W, b, order = case
    n = B * V if offset is None else threshold() + offset
    m = mask_with(order, n)
    coords = torch.empty((B * V, 2), dtype=torch.int32, device="cuda")
    row_of = torch.empty((B, V), dtype=torch.int32, device="cuda")
    offs = torch.empty((B + 1,), dtype=torch.int32, device="cuda")
    count = torch.empty((1,), dtype=torch.int32, device="cuda")
    rb = torch.empty((L, B * V), dtype=torch.int32, device="cuda")
    hc.hc_mask_compact_rulebook(to_torch(m), to_torch(sp), layout, coords, row_of, offs, count, rb)
    c, r, _, n_ref = oracle.mask_compact(m)
    assert int(count.item()) == n == n_ref
    if layout == hc.HC_LAYOUT_DENSE:
        xin, x_np = to_torch(x), x
    else:
        x_np = np.zeros((B * V, C_IN), x.dtype)
        x_np[:n] = x[c[:, 0], c[:, 1]]
        xin = to_torch(x_np)
    Wt, bt = to_torch(W), to_torch(b)
    y = torch.full((B * V, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    hc.hc_sparse_spiral_conv_fwd(xin, layout, coords, row_of, count, to_torch(sp), B, V, Wt, bt,
                                 hc.HC_ACT_ELU, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    assert torch.isnan(y[n:].float()).all()
    ref = run(xin.view(-1, C_IN), rb, count, Wt, bt)
    assert torch.equal(y[:n], ref[:n])
    rows = np.unique(np.concatenate([np.arange(256), np.arange(n - 256, n),
                                     sample_rows(n, 3000, seed=n)]))
    lay = oracle.LAYOUT_DENSE if layout == hc.HC_LAYOUT_DENSE else oracle.LAYOUT_COMPACT
    y_pre, _ = oracle.sparse_spiral_conv(x_np if layout == hc.HC_LAYOUT_COMPACT else x, lay, c, r,
                                         sp, W, b, oracle.ACT_ELU, rows=rows, n_threads=NCPU)
    check_close(to_numpy(y)[rows], y_pre, f"resolved taps layout={layout} N'={n}")
