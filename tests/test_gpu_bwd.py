"""GPU parity of the sparse conv backward through the C-ABI: the transposed
Eq. 4 mapping (bit-exact) and the input, weight and bias gradients against
the CPU oracle.

Tolerance. A gradient entry is a sum over many rows; rounding one operand
of each term (bf16 dz, bf16 per-tap products) or accumulating in fp32 moves
the sum by a fraction of the L2 norm of its terms, not of the sum itself
(an entry can cancel to near zero). So an entry passes when
    |gpu - oracle| <= tol * max(1, |oracle|, ||terms||_2)
with tol = 1e-4 for fp32 and 2e-2 for bf16 (the forward's bars), where
||terms||_2 is computed by the oracle itself: the same backward on squared
inputs with no activation sums the squared terms exactly."""
import os

import numpy as np
import pytest

import oracle
from paper_2608_09388_gb300 import hc, inputs

from _util import to_numpy, to_torch, widen

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_09388_gb300 import build
    build.build()
    hc.load_library()
    assert hc.hc_get_device_status() == hc.HC_OK


def _case(seed, B, V, L, C_in, C_out, dtype, layout, act, density=0.3):
    sp, m, x_dense, W, b = inputs.random_case(seed, B, V, L, C_in, C_out, dtype, density)
    coords, row_of, _, n = oracle.mask_compact(m)
    x = x_dense.reshape(B * V, C_in) if layout == oracle.LAYOUT_DENSE else \
        oracle.gather_rows(x_dense, coords)
    rb = oracle.conv_rulebook(coords, row_of, sp, layout, stride=B * V)
    _, y = oracle.sparse_spiral_conv(x_dense if layout == oracle.LAYOUT_DENSE else x, layout,
                                     coords, row_of, sp, W, b, act)
    rng = np.random.default_rng(seed + 99)
    dy = inputs.features(rng, (n, C_out), dtype)
    return dict(x=x, W=W, y=y, dy=dy, rb=rb, n=n, cap=B * V, act=act, dtype=dtype)


def _terms_norms(c):
    """L2 norms of the summands of every dx / dW / dbias entry (oracle,
    squared inputs, identity activation)."""
    def sq(a):
        return (widen(a) ** 2).astype(np.float32)
    ad = widen(c["dy"]) * np.where(
        c["act"] == oracle.ACT_NONE, 1.0,
        np.where(widen(c["y"]) > 0, 1.0,
                 (widen(c["y"]) + 1.0) if c["act"] == oracle.ACT_ELU else 0.0))
    dz2 = (ad ** 2).astype(np.float32)
    zeros = np.zeros_like(dz2)
    dx2, dW2, db2 = oracle.sparse_conv_bwd(sq(c["x"]), c["rb"][:, :c["n"]], sq(c["W"]), zeros, dz2,
                                           oracle.ACT_NONE)
    return np.sqrt(dx2), np.sqrt(dW2), np.sqrt(db2)


def _check(name, got, ref, norm, tol):
    scale = np.maximum(np.maximum(np.abs(ref), norm), 1.0)
    err = np.abs(got - ref) / scale
    worst = np.unravel_index(np.argmax(err), err.shape) if err.size else None
    assert err.size == 0 or err.max() <= tol, (
        f"{name}: err {err.max():.3e} at {worst}: gpu {got[worst]} oracle {ref[worst]} "
        f"norm {norm[worst]}")


def run_bwd(c, want=("dx", "dW", "db")):
    x = to_torch(c["x"])
    L, cap = c["rb"].shape
    rb = to_torch(c["rb"])
    count = torch.tensor([c["n"]], dtype=torch.int32, device="cuda")
    x_rows = x.shape[0]
    row_ptr = torch.full((x_rows + 1,), -7, dtype=torch.int32, device="cuda")
    taps = torch.full((L * cap,), -7, dtype=torch.int32, device="cuda")
    hc.hc_conv_rulebook_transpose(rb, count, x_rows, row_ptr, taps)
    C_out = c["W"].shape[1]
    y = torch.zeros((cap, C_out), dtype=x.dtype, device="cuda")
    dy = torch.zeros_like(y)
    y[:c["n"]] = to_torch(c["y"])
    dy[:c["n"]] = to_torch(c["dy"])
    dx = torch.full_like(x, float("nan")) if "dx" in want else None
    dW = torch.full(c["W"].shape, float("nan"), device="cuda") if "dW" in want else None
    db = torch.full((C_out,), float("nan"), device="cuda") if "db" in want else None
    hc.hc_sparse_conv_rulebook_bwd(x, rb, count, to_torch(c["W"]), y, dy, c["act"], row_ptr,
                                   taps, dx, dW, db)
    assert hc.hc_get_device_status() == hc.HC_OK
    return (None if dx is None else widen(to_numpy(dx)),
            None if dW is None else dW.cpu().numpy().astype(np.float64),
            None if db is None else db.cpu().numpy().astype(np.float64),
            to_numpy(row_ptr), to_numpy(taps))


def check_against_oracle(c, got, want=("dx", "dW", "db")):
    dx, dW, db, _, _ = got
    rdx, rdW, rdb = oracle.sparse_conv_bwd(c["x"], c["rb"][:, :c["n"]], c["W"], c["y"], c["dy"],
                                           c["act"])
    ndx, ndW, ndb = _terms_norms(c)
    tol = 1e-4 if c["dtype"] == "f32" else 2e-2
    if "dx" in want:
        _check("dx", dx, rdx, ndx, tol)
    if "dW" in want:
        _check("dW", dW, rdW, ndW, tol)
    if "db" in want:
        _check("dbias", db, rdb, ndb, tol)


def test_rulebook_transpose_bit_exact():
    c = _case(1, 4, 300, 9, 16, 32, "bf16", oracle.LAYOUT_COMPACT, oracle.ACT_ELU)
    _, _, _, ptr, taps = run_bwd(c, want=())
    L, cap = c["rb"].shape
    n = c["n"]
    lists = [[] for _ in range(c["x"].shape[0])]
    for l in range(L):
        for r in range(n):
            j = c["rb"][l, r]
            if j >= 0:
                lists[j].append(r * L + l)
    ref_ptr = np.concatenate([[0], np.cumsum([len(v) for v in lists])])
    np.testing.assert_array_equal(ptr, ref_ptr)
    np.testing.assert_array_equal(taps[:ref_ptr[-1]],
                                  np.concatenate([sorted(v) for v in lists]).astype(np.int32))


def test_rulebook_transpose_long_rows():
    """A synthetic mapping whose entries land on 10 input rows (hundreds of
    taps per row, past the 32 a warp sorts at once), with absent taps."""
    rng = np.random.default_rng(3)
    L, cap, n, x_rows = 6, 500, 431, 10
    rb_np = rng.integers(-1, x_rows, size=(L, cap)).astype(np.int32)
    rb = to_torch(rb_np)
    count = torch.tensor([n], dtype=torch.int32, device="cuda")
    row_ptr = torch.empty(x_rows + 1, dtype=torch.int32, device="cuda")
    taps = torch.full((L * cap,), -7, dtype=torch.int32, device="cuda")
    hc.hc_conv_rulebook_transpose(rb, count, x_rows, row_ptr, taps)
    assert hc.hc_get_device_status() == hc.HC_OK
    lists = [[] for _ in range(x_rows)]
    for l in range(L):
        for r in range(n):
            if rb_np[l, r] >= 0:
                lists[rb_np[l, r]].append(r * L + l)
    ref_ptr = np.concatenate([[0], np.cumsum([len(v) for v in lists])])
    np.testing.assert_array_equal(to_numpy(row_ptr), ref_ptr)
    np.testing.assert_array_equal(to_numpy(taps)[:ref_ptr[-1]],
                                  np.concatenate([sorted(v) for v in lists]).astype(np.int32))


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("layout", [oracle.LAYOUT_DENSE, oracle.LAYOUT_COMPACT])
@pytest.mark.parametrize("shape", [(3, 200, 9, 16, 64), (2, 333, 12, 64, 128),
                                   (5, 100, 5, 8, 24), (2, 150, 7, 12, 20), (1, 64, 3, 3, 5)])
@pytest.mark.parametrize("act", [oracle.ACT_ELU, oracle.ACT_RELU, oracle.ACT_NONE])
def test_backward(shape, layout, dtype, act):
    """Tensor-core weight gradient (bf16, channels multiples of 8) and the
    CUDA-core one (fp32, or odd channel counts), several tiles of
    L*C_in and C_out, ragged row counts, both input layouts."""
    B, V, L, C_in, C_out = shape
    c = _case(sum(shape) + layout * 7 + act, B, V, L, C_in, C_out, dtype, layout, act)
    check_against_oracle(c, run_bwd(c))


def test_backward_partial_outputs_and_no_rows():
    c = _case(5, 2, 120, 9, 16, 32, "bf16", oracle.LAYOUT_DENSE, oracle.ACT_ELU)
    for want in (("dx",), ("dW",), ("db",), ("dW", "db")):
        check_against_oracle(c, run_bwd(c, want), want)
    c0 = _case(6, 2, 50, 5, 8, 8, "f32", oracle.LAYOUT_DENSE, oracle.ACT_ELU, density=0.0)
    assert c0["n"] == 0
    dx, dW, db, _, _ = run_bwd(c0)
    assert not dx.any() and not dW.any() and not db.any()


def test_backward_full_size_layer():
    """The 10475-vertex bf16 layer (32 frames, clustered ~5% masks, L = 12,
    64 -> 128 channels, dense input) that the bench times."""
    w = inputs.make_workload("layer10475_bf16")
    ly = w.layers[0]
    B, V = w.B, w.V
    coords, row_of, _, n = oracle.mask_compact(w.masks[0])
    rb = oracle.conv_rulebook(coords, row_of, w.spiral, oracle.LAYOUT_DENSE, stride=B * V)
    _, y = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, coords, row_of, w.spiral, ly.W,
                                     ly.b, ly.act, n_threads=len(os.sched_getaffinity(0)))
    dy = inputs.features(np.random.default_rng(5), (n, ly.C_out), "bf16")
    c = dict(x=w.x.reshape(B * V, ly.C_in), W=ly.W, y=y, dy=dy, rb=rb, n=n, cap=B * V,
             act=ly.act, dtype="bf16")
    check_against_oracle(c, run_bwd(c))


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_backward_many_taps_per_range(dtype):
    """A synthetic mapping with ~48 taps per input row: the first 256-row
    range holds more keys than the input gradient stages in shared memory
    (8192), so it reads them from global memory; the tail range stages them."""
    rng = np.random.default_rng(11)
    L, n, x_rows, C_in, C_out = 24, 600, 300, 16, 32
    rb = rng.integers(-1, x_rows, size=(L, n)).astype(np.int32)
    x = inputs.features(rng, (x_rows, C_in), dtype)
    W = inputs.weights(rng, L * C_in, C_out, dtype)
    y = np.zeros((n, C_out), dtype=x.dtype)
    dy = inputs.features(rng, (n, C_out), dtype)
    c = dict(x=x, W=W, y=y, dy=dy, rb=rb, n=n, cap=n, act=oracle.ACT_NONE, dtype=dtype)
    check_against_oracle(c, run_bwd(c, want=("dx",)), want=("dx",))


def test_backward_bad_taps_reported():
    """A malformed transposed mapping is reported and its entries skipped."""
    c = _case(8, 2, 80, 5, 8, 16, "f32", oracle.LAYOUT_DENSE, oracle.ACT_NONE)
    x = to_torch(c["x"])
    L, cap = c["rb"].shape
    rb = to_torch(c["rb"])
    count = torch.tensor([c["n"]], dtype=torch.int32, device="cuda")
    row_ptr = torch.zeros(x.shape[0] + 1, dtype=torch.int32, device="cuda")
    taps = torch.zeros(L * cap, dtype=torch.int32, device="cuda")
    hc.hc_conv_rulebook_transpose(rb, count, x.shape[0], row_ptr, taps)
    taps[0] = L * cap + 5  # a key past the last P row
    y = torch.zeros((cap, 16), device="cuda")
    dx = torch.empty_like(x)
    hc.hc_sparse_conv_rulebook_bwd(x, rb, count, to_torch(c["W"]), y, y, 0, row_ptr, taps,
                                   dx, None, None)
    assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
