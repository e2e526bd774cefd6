"""The exact call chains the benchmark times, at their full sizes, against
the oracle on every output row (or, for the densest sweep masks, on at least
10k sampled rows): compaction fused with the Eq. 4 mapping
(hc_mask_compact_rulebook), then the tensor-core conv through the rulebook
(hc_sparse_conv_rulebook_fwd) with the scatter into the dense tensor fused
into its epilogue, as the bench step runs them; the density sweep's call;
the dense layer the speed-ups divide by."""
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


def _chain(mask, x, spiral, W, bias, act, out_fill=None):
    """The bench step: compaction + mapping, then the conv writing compact
    rows and, when out_fill is given, the dense tensor (prefilled with it)."""
    B, V = mask.shape
    L = spiral.shape[1]
    C_out = W.shape[1]
    coords = torch.full((B * V, 2), -7, dtype=torch.int32, device="cuda")
    row_of = torch.full((B, V), -7, dtype=torch.int32, device="cuda")
    offs = torch.full((B + 1,), -7, dtype=torch.int32, device="cuda")
    count = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    rb = torch.full((L, B * V), -7, dtype=torch.int32, device="cuda")
    hc.hc_mask_compact_rulebook(to_torch(mask), spiral, hc.HC_LAYOUT_DENSE, coords, row_of, offs,
                                count, rb)
    y = torch.full((B * V, C_out), float("nan"), dtype=torch.bfloat16, device="cuda")
    out = None if out_fill is None else to_torch(out_fill)
    hc.hc_sparse_conv_rulebook_fwd(x, rb, count, W, bias, act, y,
                                   coords=None if out is None else coords, out=out)
    assert hc.hc_get_device_status() == hc.HC_OK
    n = int(count.item())
    return n, to_numpy(coords)[:n], to_numpy(y), None if out is None else to_numpy(out)


def _rulebook(mask, spiral):
    """Compaction + Eq. 4 mapping (dense layout): rulebook, coords, row_of, count."""
    B, V = mask.shape
    L = spiral.shape[1]
    coords = torch.empty((B * V, 2), dtype=torch.int32, device="cuda")
    row_of = torch.empty((B, V), dtype=torch.int32, device="cuda")
    offs = torch.empty((B + 1,), dtype=torch.int32, device="cuda")
    count = torch.empty((1,), dtype=torch.int32, device="cuda")
    rb = torch.empty((L, B * V), dtype=torch.int32, device="cuda")
    hc.hc_mask_compact_rulebook(to_torch(mask), to_torch(spiral), hc.HC_LAYOUT_DENSE, coords,
                                row_of, offs, count, rb)
    return rb, coords, row_of, count


def test_bench_step_every_row():
    """The 10475-vertex layer (32 clustered frames, L = 12, 64 -> 128, ELU):
    every active row of the compact output and of the dense scatter against
    the oracle, every inactive dense row untouched."""
    w = inputs.make_workload("layer10475_bf16")
    ly = w.layers[0]
    B, V = w.B, w.V
    prev = inputs.features(np.random.default_rng(11), (B, V, ly.C_out), "bf16")
    n, coords, y, out = _chain(w.masks[0], to_torch(w.x), to_torch(w.spiral), to_torch(ly.W),
                               to_torch(ly.b), ly.act, out_fill=prev)
    c, r, _, n_ref = oracle.mask_compact(w.masks[0])
    assert n == n_ref and n > 16000
    np.testing.assert_array_equal(coords, c)
    y_pre, _ = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, c, r, w.spiral, ly.W, ly.b,
                                         ly.act, n_threads=NCPU)
    check_close(y[:n], y_pre, "bench step, compact rows")
    check_close(out[c[:, 0], c[:, 1]], y_pre, "bench step, dense scatter")
    inactive = np.ones((B, V), bool)
    inactive[c[:, 0], c[:, 1]] = False
    np.testing.assert_array_equal(out[inactive], prev[inactive])


@pytest.mark.parametrize("density", [0.01, 0.05, 0.1, 0.25, 0.5, 1.0])
def test_sweep_call_full_size(density):
    """The density sweep's call (V = 10475, L = 9, B = 64, 128 -> 128): all
    rows at 1% and 5%, at least 10k rows (first, last, tile boundaries and a
    seeded sample) above."""
    w = inputs.make_workload("sweep10475_bf16")
    ly = w.layers[0]
    m = w.masks[list(w.densities).index(density)]
    n, coords, y, _ = _chain(m, to_torch(w.x), to_torch(w.spiral), to_torch(ly.W),
                             to_torch(ly.b), ly.act)
    c, r, _, n_ref = oracle.mask_compact(m)
    assert n == n_ref
    np.testing.assert_array_equal(coords, c)
    rows = np.arange(n) if density <= 0.05 else sample_rows(n, 10000, seed=5)
    y_pre, _ = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, c, r, w.spiral, ly.W, ly.b,
                                         ly.act, rows=rows, n_threads=NCPU)
    check_close(y[rows], y_pre, f"sweep density {density}")


@pytest.mark.parametrize("act,bias", [(oracle.ACT_ELU, True), (oracle.ACT_RELU, False),
                                      (oracle.ACT_NONE, True)])
def test_dense_layer_transposed_mma(act, bias):
    """The dense layer with 128 output channels and enough rows for two-half
    items (at least two per SM) takes the transposed MMA (W^T times the
    gathered rows: lanes = channels, columns = rows); 79,999 rows leave the
    last item ragged. Every row against the oracle, for each activation,
    with and without bias, and rows past B*V untouched."""
    B, V, L, C_in = 1, 79999, 9, 32
    rng = np.random.default_rng(11 + act)
    sp = rng.integers(0, V, size=(V, L)).astype(np.int32)
    sp[:, 0] = np.arange(V)
    sp[rng.random((V, L)) < 0.1] = -1
    sp[:, 0] = np.arange(V)
    x = inputs.features(rng, (B, V, C_in), "bf16")
    W = inputs.weights(rng, L * C_in, 128, "bf16")
    b = rng.standard_normal(128).astype(np.float32) if bias else None
    yd = torch.full((B * V + 7, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    hc.hc_spiral_conv_fwd(to_torch(x), to_torch(sp), to_torch(W), None if b is None else to_torch(b),
                          act, yd[:B * V].view(B, V, 128))
    assert hc.hc_get_device_status() == hc.HC_OK
    y_pre, _ = oracle.dense_spiral_conv(x, sp, W, b, act, n_threads=NCPU)
    check_close(to_numpy(yd)[:B * V], y_pre, f"dense transposed act={act} bias={bias}")
    assert torch.isnan(yd[B * V:].float()).all()


@pytest.mark.parametrize("density", [0.01, 0.1, 0.5, 1.0])
def test_row_hint_same_bits(density):
    """hc_sparse_conv_rulebook_fwd_hint on the density sweep's layer: with the
    exact count as the estimate (two-half transposed items from 10% up, the
    one-half kernel at 1%), with a wrong one in each direction, and with
    none, every row is bit-identical to hc_sparse_conv_rulebook_fwd; the
    oracle on 3000 sampled rows; rows past N' untouched."""
    w = inputs.make_workload("sweep10475_bf16")
    ly = w.layers[0]
    m = w.masks[list(w.densities).index(density)]
    B, V = m.shape
    rb, coords, row_of, count = _rulebook(m, w.spiral)
    n = int(count.item())
    xt, Wt, bt = to_torch(w.x), to_torch(ly.W), to_torch(ly.b)
    ref = torch.full((B * V, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    hc.hc_sparse_conv_rulebook_fwd(xt, rb, count, Wt, bt, ly.act, ref)
    for hint in (n, 0, B * V, 1000):
        y = torch.full((B * V, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
        hc.hc_sparse_conv_rulebook_fwd_hint(xt, rb, count, Wt, bt, ly.act, y, hint)
        assert hc.hc_get_device_status() == hc.HC_OK
        assert torch.equal(y[:n], ref[:n]), f"hint {hint}"
        assert torch.isnan(y[n:].float()).all()
    c, r, _, _ = oracle.mask_compact(m)
    rows = sample_rows(n, 3000, seed=12)
    y_pre, _ = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, c, r, w.spiral, ly.W, ly.b,
                                         ly.act, rows=rows, n_threads=NCPU)
    check_close(to_numpy(ref)[rows], y_pre, f"hinted sweep {density}")


@pytest.mark.parametrize("L,C_in,act,bias,density", [
    (9, 64, oracle.ACT_ELU, True, 0.4),
    (9, 45, oracle.ACT_RELU, False, 0.4),   # channel-padded input, then the two-half items
    (12, 128, oracle.ACT_NONE, True, 0.3),
    (1, 16, oracle.ACT_ELU, True, 0.5),     # one slot: a single k-block
    (5, 200, oracle.ACT_ELU, True, 0.2),    # K = 1000: a ragged last k-block
    (9, 64, oracle.ACT_ELU, True, 0.0),     # no active rows
])
def test_row_hint_forces_two_half_items_on_small_calls(L, C_in, act, bias, density):
    """A row estimate far above the real count makes small calls run the
    two-half transposed items (few items, the last ragged): every row
    against the oracle and bit-identical to the default call; rows past N'
    untouched."""
    sp, m, x, W, b = inputs.random_case(L * 100 + C_in + int(density * 10), 3, 1001, L, C_in,
                                        128, "bf16", density, neg_frac=0.1)
    if not bias:
        b = None
    B, V = m.shape
    rb, coords, row_of, count = _rulebook(m, sp)
    n = int(count.item())
    xt, Wt, bt = to_torch(x), to_torch(W), None if b is None else to_torch(b)
    ref = torch.full((B * V, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    hc.hc_sparse_conv_rulebook_fwd(xt, rb, count, Wt, bt, act, ref)
    y = torch.full((B * V, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    hc.hc_sparse_conv_rulebook_fwd_hint(xt, rb, count, Wt, bt, act, y, 10 ** 7)
    assert hc.hc_get_device_status() == hc.HC_OK
    assert torch.equal(y[:n], ref[:n])
    assert torch.isnan(y[n:].float()).all()
    if n:
        c, r, _, _ = oracle.mask_compact(m)
        y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c, r, sp, W, b, act,
                                             n_threads=NCPU)
        check_close(to_numpy(y)[:n], y_pre, f"hinted L={L} C_in={C_in}")


@pytest.mark.parametrize("name", ["sweep10475_bf16", "layer10475_bf16"])
def test_dense_layer_full_size(name):
    """The dense layer of the speed-up denominators on 10k sampled rows."""
    w = inputs.make_workload(name)
    ly = w.layers[0]
    B, V = w.B, w.V
    yd = torch.full((B, V, ly.C_out), float("nan"), dtype=torch.bfloat16, device="cuda")
    hc.hc_spiral_conv_fwd(to_torch(w.x), to_torch(w.spiral), to_torch(ly.W), to_torch(ly.b),
                          ly.act, yd)
    assert hc.hc_get_device_status() == hc.HC_OK
    rows = sample_rows(B * V, 10000, seed=6)
    y_pre, _ = oracle.dense_spiral_conv(w.x, w.spiral, ly.W, ly.b, ly.act, rows=rows,
                                        n_threads=NCPU)
    check_close(to_numpy(yd).reshape(B * V, -1)[rows], y_pre, f"dense {name}")
