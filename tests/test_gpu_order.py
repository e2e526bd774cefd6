"""The row order of the rulebook conv (hc_conv_rulebook_order) and the conv
run in that order (hc_sparse_conv_rulebook_ordered_fwd).

The order is a schedule, not part of the paper's method: several orders are
correct (rows of equal tap pattern in any order), so the tests check what is
unique (the sorted keys, each tile's tap union, the set of rows) and that the
rest is valid (a permutation). The ordered conv must give every row exactly
the result of the unordered one (it only leaves out k-blocks whose taps are
absent from every row of a tile, i.e. exact zeros) and match the oracle."""
import os

import numpy as np
import pytest

import oracle
from paper_2608_09388_gb300 import hc, inputs

from _util import check_close, sample_rows, to_numpy, to_torch

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
NCPU = len(os.sched_getaffinity(0))


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_09388_gb300 import build
    build.build()
    hc.load_library()
    assert hc.hc_get_device_status() == hc.HC_OK


def _mapping(mask, spiral, layout=hc.HC_LAYOUT_DENSE):
    B, V = mask.shape
    L = spiral.shape[1]
    coords = torch.empty((max(B * V, 1), 2), dtype=torch.int32, device="cuda")
    row_of = torch.empty((B, V), dtype=torch.int32, device="cuda")
    offs = torch.empty((B + 1,), dtype=torch.int32, device="cuda")
    count = torch.empty((1,), dtype=torch.int32, device="cuda")
    rb = torch.empty((L, max(B * V, 1)), dtype=torch.int32, device="cuda")
    hc.hc_mask_compact_rulebook(to_torch(mask), to_torch(spiral), layout, coords, row_of, offs,
                                count, rb)
    return coords, row_of, count, rb


def _order(rb, count):
    L, cap = rb.shape
    order = torch.full((cap,), -7, dtype=torch.int32, device="cuda")
    taps = torch.full(((cap + 127) // 128,), -7, dtype=torch.int32, device="cuda")
    srb = torch.full((L, cap), -7, dtype=torch.int32, device="cuda")
    hc.hc_conv_rulebook_order(rb, count, order, taps, srb)
    assert hc.hc_get_device_status() == hc.HC_OK
    return order, taps, srb


def _keys(mask, spiral, layout=0):
    """Tap-presence pattern of every active row, from the oracle's mapping."""
    c, r, _, n = oracle.mask_compact(mask)
    rb = oracle.conv_rulebook(c, r, spiral, layout)[:, :n]
    L = rb.shape[0]
    return ((rb >= 0).astype(np.uint64) << np.arange(L, dtype=np.uint64)[:, None]).sum(0), n


def _check_order(mask, spiral):
    coords, row_of, count, rb = _mapping(mask, spiral)
    order, taps, srb = _order(rb, count)
    keys, n = _keys(mask, spiral)
    assert int(count.item()) == n
    o = to_numpy(order)[:n].astype(np.int64)
    np.testing.assert_array_equal(np.sort(o), np.arange(n))  # a permutation
    L = spiral.shape[1]
    low = keys & np.uint64((1 << min(L, 12)) - 1)
    np.testing.assert_array_equal(low[o], np.sort(low, kind="stable"))  # sorted keys
    t = to_numpy(taps).view(np.uint32)
    for i in range((n + 127) // 128):
        assert int(t[i]) == int(np.bitwise_or.reduce(keys[o[128 * i:128 * (i + 1)]]))
    # the sorted rulebook: column p is row order[p]'s column (bit for bit)
    np.testing.assert_array_equal(to_numpy(srb)[:, :n], to_numpy(rb)[:, o])
    return order, taps, n


@pytest.mark.parametrize("density", [0.0, 0.01, 0.1, 0.5, 1.0])
def test_order_sweep_masks(density):
    w = inputs.make_workload("sweep10475_bf16", B=8)
    m = inputs.uniform_mask(np.random.default_rng(int(density * 100)), 8, w.V, density)
    _check_order(m, w.spiral)


@pytest.mark.parametrize("L", [1, 3, 12, 13, 32])
def test_order_spiral_lengths(L):
    """L > 12: the sort uses the low 12 bits of the key, the unions all of it;
    -1 spiral entries give rows without some taps."""
    sp, m, *_ = inputs.random_case(300 + L, 5, 700, L, 16, 16, "bf16", 0.3, neg_frac=0.2)
    _check_order(m, sp)


def _run(x, rb, count, W, b, act, C_out, ordering=None, coords=None, out=None):
    n_cap = rb.shape[1]
    y = torch.full((n_cap, C_out), float("nan"), dtype=torch.bfloat16, device="cuda")
    if ordering is None:
        hc.hc_sparse_conv_rulebook_fwd(x, rb, count, W, b, act, y, coords=coords, out=out)
    else:
        order, taps, srb = ordering
        hc.hc_sparse_conv_rulebook_ordered_fwd(x, rb, count, W, b, act, y, order, taps, srb,
                                               coords=coords, out=out)
    assert hc.hc_get_device_status() == hc.HC_OK
    return y


@pytest.mark.parametrize("C_in,C_out,L,density,act,bias", [
    (16, 64, 9, 0.1, oracle.ACT_ELU, True),     # four taps per 64-deep k-block
    (32, 128, 9, 0.3, oracle.ACT_RELU, False),  # two taps per k-block, no bias
    (64, 128, 12, 0.05, oracle.ACT_ELU, True),  # the bench layer's shape
    (128, 128, 9, 0.1, oracle.ACT_NONE, True),  # the sweep's shape, two k-blocks per tap
    (128, 64, 32, 0.2, oracle.ACT_ELU, True),   # 64 k-blocks: the most a tile skips over
    (24, 40, 5, 0.5, oracle.ACT_ELU, True),     # k-blocks across tap boundaries
])
def test_ordered_conv_same_as_unordered_and_oracle(C_in, C_out, L, density, act, bias):
    sp, m, x, W, b = inputs.random_case(C_in * 7 + L, 6, 1500, L, C_in, C_out, "bf16", density,
                                        neg_frac=0.1)
    if not bias:
        b = None
    coords, row_of, count, rb = _mapping(m, sp)
    ordering = _order(rb, count)
    xt, Wt, bt = to_torch(x), to_torch(W), None if b is None else to_torch(b)
    y0 = _run(xt, rb, count, Wt, bt, act, C_out)
    y1 = _run(xt, rb, count, Wt, bt, act, C_out, ordering)
    n = int(count.item())
    assert torch.equal(y0[:n], y1[:n])
    assert torch.isnan(y1[n:].float()).all()  # rows past N' untouched
    c, r, _, _ = oracle.mask_compact(m)
    y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c, r, sp, W, b, act,
                                         n_threads=NCPU)
    check_close(to_numpy(y1)[:n], y_pre, f"ordered conv C_in={C_in} L={L}")


def test_ordered_conv_fused_scatter():
    """The dense scatter of the ordered conv writes each row at its own
    coordinate and leaves the inactive rows alone."""
    sp, m, x, W, b = inputs.random_case(77, 4, 2000, 9, 64, 128, "bf16", 0.1)
    B, V = m.shape
    coords, row_of, count, rb = _mapping(m, sp)
    ordering = _order(rb, count)
    prev = inputs.features(np.random.default_rng(5), (B, V, 128), "bf16")
    out = to_torch(prev)
    y = _run(to_torch(x), rb, count, to_torch(W), to_torch(b), oracle.ACT_ELU, 128, ordering,
             coords=coords, out=out)
    c, r, _, n = oracle.mask_compact(m)
    y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c, r, sp, W, b, oracle.ACT_ELU,
                                         n_threads=NCPU)
    o = to_numpy(out)
    check_close(o[c[:, 0], c[:, 1]], y_pre, "ordered conv, dense scatter")
    inactive = np.ones((B, V), bool)
    inactive[c[:, 0], c[:, 1]] = False
    np.testing.assert_array_equal(o[inactive], prev[inactive])
    np.testing.assert_array_equal(to_numpy(y)[:n], o[c[:, 0], c[:, 1]])


@pytest.mark.parametrize("density", [0.01, 0.05, 0.1, 0.25, 0.5, 1.0])
def test_ordered_sweep_full_size(density):
    """The density sweep's layer (V = 10475, L = 9, B = 64, 128 -> 128) in
    the order: bit-identical to the unordered call on every row, and the
    oracle on all rows at 1% and 5%, 10k rows above."""
    w = inputs.make_workload("sweep10475_bf16")
    ly = w.layers[0]
    m = w.masks[list(w.densities).index(density)]
    coords, row_of, count, rb = _mapping(m, w.spiral)
    ordering = _order(rb, count)
    xt, Wt, bt = to_torch(w.x), to_torch(ly.W), to_torch(ly.b)
    y0 = _run(xt, rb, count, Wt, bt, ly.act, ly.C_out)
    y1 = _run(xt, rb, count, Wt, bt, ly.act, ly.C_out, ordering)
    n = int(count.item())
    assert torch.equal(y0[:n], y1[:n])
    c, r, _, _ = oracle.mask_compact(m)
    rows = np.arange(n) if density <= 0.05 else sample_rows(n, 10000, seed=8)
    y_pre, _ = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, c, r, w.spiral, ly.W, ly.b,
                                         ly.act, rows=rows, n_threads=NCPU)
    check_close(to_numpy(y1)[rows], y_pre, f"ordered sweep {density}")


def test_order_empty_and_host_checks():
    rb = torch.zeros((9, 10), dtype=torch.int32, device="cuda")
    count = torch.zeros((1,), dtype=torch.int32, device="cuda")
    order, taps, srb = _order(rb, count)  # N' = 0: nothing written, no error
    assert (to_numpy(order) == -7).all()
    assert (to_numpy(srb) == -7).all()
