"""GPU parity of the mask-score update (Eq. 3) and of inference with the
kappa kept masks (Sec. 3.1): top-kappa selection, kappa masks per sample,
the S' row gather of Eq. 2, and the whole chain into a sparse conv, each
against the CPU oracle through the C-ABI.

Tolerances: indices, masks and gathered rows are bit-exact. Scores: the
Gram sums are fp32 (tensor-core accumulation for bf16 inputs, FFMA for
fp32) and S, sim and alpha are formed from them in fp32, so |alpha -
alpha_oracle| and |sim - sim_oracle| <= 1e-4 (the fp32 bar)."""
import os

import numpy as np
import pytest

import oracle
from paper_2608_09388_gb300 import hc, inputs

from _util import check_close, to_numpy, to_torch

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
NCPU = len(os.sched_getaffinity(0))
SCORE_TOL = 1e-4


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_09388_gb300 import build
    build.build()
    hc.load_library()
    assert hc.hc_get_device_status() == hc.HC_OK


def _outputs(rng, K, N, D, dtype, shift=0.2):
    O = (rng.standard_normal((K, N, D)) + shift).astype(np.float32)
    return O if dtype == "f32" else inputs.to_bf16_bits(O)


def run_score(O_np, alpha_np, in_place=False):
    O = to_torch(O_np)
    K = O_np.shape[0]
    a_in = torch.tensor(alpha_np, dtype=torch.float32, device="cuda")
    a_out = a_in if in_place else torch.full((K,), float("nan"), device="cuda")
    sim = torch.full((K, K), float("nan"), device="cuda")
    hc.hc_mask_score_update(O, a_in, a_out, sim)
    assert hc.hc_get_device_status() == hc.HC_OK
    return a_out.cpu().numpy().astype(np.float64), sim.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("K,N,D", [(2, 100, 8), (3, 1000, 64), (4, 777, 5), (5, 300, 1),
                                   (1, 50, 16), (6, 333, 130), (10, 4000, 42), (3, 64, 8),
                                   (2, 1, 3), (40, 500, 16), (10, 3000, 128), (9, 700, 130),
                                   (11, 500, 101), (10, 2000, 96), (8, 900, 121)])
def test_mask_score(K, N, D, dtype):
    """Multi-tile Gram matrices (K*D > 128; K*D >= 512 whose padding to 256
    keeps >= 80% of the Gram useful takes the 256-wide tensor-core tiles:
    1280, 1170, 960, 968 here; 1111, 780 and 640 stay on 128-wide tiles),
    ragged row counts, D a multiple of 8 (16-byte pieces), even (4-byte
    pieces) and odd (the packed copy), D = 1, K = 1, one row."""
    rng = np.random.default_rng(K * 1000 + N + D)
    O = _outputs(rng, K, N, D, dtype)
    alpha = rng.standard_normal(K)
    a_ref, sim_ref, _ = oracle.mask_score(O, alpha.astype(np.float32), n_threads=NCPU)
    a, sim = run_score(O, alpha)
    np.testing.assert_allclose(a, a_ref, rtol=0, atol=SCORE_TOL)
    np.testing.assert_allclose(sim, sim_ref, rtol=0, atol=SCORE_TOL)


def test_mask_score_in_place_and_edge_cases():
    rng = np.random.default_rng(7)
    O = _outputs(rng, 4, 500, 24, "bf16")
    O[2] = 0  # a mask with an all-zero output: similarity 0 to every mask
    alpha = rng.standard_normal(4)
    a_ref, sim_ref, _ = oracle.mask_score(O, alpha.astype(np.float32))
    a, sim = run_score(O, alpha, in_place=True)
    np.testing.assert_allclose(a, a_ref, atol=SCORE_TOL)
    np.testing.assert_allclose(sim, sim_ref, atol=SCORE_TOL)
    # identical outputs: fully similar, alpha unchanged
    same = np.repeat(O[:1], 3, axis=0)
    a, sim = run_score(same, alpha[:3])
    np.testing.assert_allclose(a, alpha[:3].astype(np.float32), atol=SCORE_TOL)
    np.testing.assert_allclose(sim, np.ones((3, 3)), atol=SCORE_TOL)
    # N = 0: every Gram norm is 0, so every term is 1
    empty = np.zeros((3, 0, 8), np.float32)
    a, _ = run_score(empty, alpha[:3])
    np.testing.assert_allclose(a, alpha[:3].astype(np.float32) + 1, atol=1e-6)


def test_mask_score_encoder_outputs_full_size():
    """K = 10 masks of the 4-layer encoder's output rows (64 frames of the
    655-vertex sphere, 64 features, bf16): the size the bench measures."""
    rng = np.random.default_rng(11)
    O = _outputs(rng, 10, 64 * 655, 64, "bf16")
    alpha = np.zeros(10)
    a_ref, sim_ref, _ = oracle.mask_score(O, alpha.astype(np.float32), n_threads=NCPU)
    a, sim = run_score(O, alpha)
    np.testing.assert_allclose(a, a_ref, atol=SCORE_TOL)
    np.testing.assert_allclose(sim, sim_ref, atol=SCORE_TOL)


def test_mask_score_rejects_oversize():
    O = torch.zeros((2, 4, 8192), dtype=torch.bfloat16, device="cuda")
    a = torch.zeros(2, device="cuda")
    with pytest.raises(hc.HcError) as e:
        hc.hc_mask_score_update(O, a, a)
    assert e.value.status == hc.HC_ERR_UNSUPPORTED


@pytest.mark.parametrize("K,kappa", [(10, 3), (50, 10), (7, 7), (1, 1), (3000, 50)])
def test_select_topk(K, kappa):
    rng = np.random.default_rng(K + kappa)
    alpha = (rng.integers(-4, 5, size=K) * 0.25).astype(np.float32)  # many ties
    if K > 5:
        alpha[[1, K // 2]] = np.nan
        alpha[K - 1] = np.inf
    sel = torch.full((kappa,), -7, dtype=torch.int32, device="cuda")
    hc.hc_mask_select_topk(to_torch(alpha), kappa, sel)
    assert hc.hc_get_device_status() == hc.HC_OK
    np.testing.assert_array_equal(to_numpy(sel), oracle.select_topk(alpha, kappa))


@pytest.mark.parametrize("V", [655, 10475, 17])
def test_kappa_masks(V):
    rng = np.random.default_rng(V)
    K, B = 10, 9
    masks = inputs.uniform_mask(rng, K, V, 0.1)
    sel = np.array([7, 2, 9], np.int32)
    out = torch.full((B * 3, V), 7, dtype=torch.uint8, device="cuda")
    hc.hc_kappa_masks(to_torch(masks), to_torch(sel), B, out)
    assert hc.hc_get_device_status() == hc.HC_OK
    np.testing.assert_array_equal(to_numpy(out), oracle.kappa_masks(masks, sel, B))
    bad = to_torch(np.array([7, 10, 0], np.int32))
    hc.hc_kappa_masks(to_torch(masks), bad, B, out)
    assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
    assert not to_numpy(out).reshape(B, 3, V)[:, 1].any()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("C,fps", [(64, 1), (16, 3), (45, 3), (3, 1)])
def test_gather_rows(C, fps, dtype):
    rng = np.random.default_rng(C * 10 + fps)
    B, V = 6, 300
    masks = inputs.uniform_mask(rng, B * fps, V, 0.2)
    x = inputs.features(rng, (B, V, C), dtype)
    c_ref, _, _, n = oracle.mask_compact(masks)
    coords = torch.full((B * fps * V, 2), -1, dtype=torch.int32, device="cuda")
    coords[:n] = to_torch(c_ref)
    count = torch.tensor([n], dtype=torch.int32, device="cuda")
    xt = to_torch(x)
    y = torch.zeros((B * fps * V, C), dtype=xt.dtype, device="cuda")
    hc.hc_gather_rows(xt, coords, count, fps, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    np.testing.assert_array_equal(to_numpy(y)[:n], oracle.gather_rows(x, c_ref, fps))
    # a coordinate outside the input is reported and its row left alone
    coords[0, 0] = B * fps
    y.zero_()
    hc.hc_gather_rows(xt, coords, count, fps, y)
    assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
    assert not to_numpy(y)[0].any()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_gather_rows_from_pinned_host_memory(dtype):
    """x in pinned host memory (read over the host link): the same rows, bit
    for bit, as from device memory."""
    rng = np.random.default_rng(17)
    B, V, C = 4, 2000, 64
    masks = inputs.uniform_mask(rng, B, V, 0.05)
    x = inputs.features(rng, (B, V, C), dtype)
    c_ref, _, _, n = oracle.mask_compact(masks)
    coords = torch.full((B * V, 2), -1, dtype=torch.int32, device="cuda")
    coords[:n] = to_torch(c_ref)
    count = torch.tensor([n], dtype=torch.int32, device="cuda")
    xt = to_torch(x)
    xh = xt.cpu().pin_memory()
    y = torch.zeros((B * V, C), dtype=xt.dtype, device="cuda")
    hc.hc_gather_rows(xh, coords, count, 1, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    np.testing.assert_array_equal(to_numpy(y)[:n], oracle.gather_rows(x, c_ref, 1))
    with pytest.raises(ValueError):  # pageable host memory is refused by the binding
        hc.hc_gather_rows(xt.cpu(), coords, count, 1, y)


@pytest.mark.parametrize("dtype,C", [("bf16", 128), ("f32", 2), ("bf16", 3)])
def test_gather_rows_in_order_into_pinned_host_memory(dtype, C):
    """coords NULL: the first N' rows of a device tensor copied in order into
    pinned host memory, the count read on the device (16-, 4- and 2-byte
    chunks); rows past N' untouched; N' above the capacity clamped
    (HC_ERR_CAPACITY), N' above the input's rows reported
    (HC_ERR_INVALID_INDEX) with those rows untouched."""
    rng = np.random.default_rng(C)
    cap = 5000
    x = inputs.features(rng, (1, cap, C), dtype)
    xt = to_torch(x)
    for n in (0, 1, 3777, cap):
        count = torch.tensor([n], dtype=torch.int32, device="cuda")
        yh = torch.full((cap, C), 7, dtype=xt.dtype).pin_memory()
        hc.hc_gather_rows(xt, None, count, 1, yh)
        torch.cuda.synchronize()
        assert hc.hc_get_device_status() == hc.HC_OK
        assert torch.equal(yh[:n], xt[0, :n].cpu())
        assert (yh[n:] == 7).all()
    # capacity below N': clamped
    count = torch.tensor([cap], dtype=torch.int32, device="cuda")
    yh = torch.full((100, C), 7, dtype=xt.dtype).pin_memory()
    hc.hc_gather_rows(xt, None, count, 1, yh)
    torch.cuda.synchronize()
    assert hc.hc_get_device_status() == hc.HC_ERR_CAPACITY
    assert torch.equal(yh, xt[0, :100].cpu())
    # input rows below N': the rows past the input reported and untouched
    xs = xt[:, :1000].contiguous()
    count = torch.tensor([1200], dtype=torch.int32, device="cuda")
    yh = torch.full((cap, C), 7, dtype=xt.dtype).pin_memory()
    hc.hc_gather_rows(xs, None, count, 1, yh)
    torch.cuda.synchronize()
    assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
    assert torch.equal(yh[:1000], xs[0].cpu())
    assert (yh[1000:] == 7).all()


def test_kappa_inference_chain():
    """alpha -> top-3 -> kappa masks for every sample -> compaction -> S'
    -> sparse spiral conv on the compact rows, against the same chain on
    the oracle."""
    w = inputs.make_workload("encoder655_bf16", B=8)
    rng = np.random.default_rng(12)
    K, kappa, V = 10, 3, w.V
    masks = inputs.uniform_mask(rng, K, V, 0.1)
    alpha = rng.standard_normal(K).astype(np.float32)
    sel_ref = oracle.select_topk(alpha, kappa)
    fm_ref = oracle.kappa_masks(masks, sel_ref, w.B)
    c_ref, r_ref, _, n = oracle.mask_compact(fm_ref)
    s_ref = oracle.gather_rows(w.x, c_ref, kappa)
    ly = w.layers[0]
    y_pre, _ = oracle.sparse_spiral_conv(s_ref, oracle.LAYOUT_COMPACT, c_ref, r_ref, w.spiral,
                                         ly.W, ly.b, ly.act)

    sel = torch.empty(kappa, dtype=torch.int32, device="cuda")
    hc.hc_mask_select_topk(to_torch(alpha), kappa, sel)
    fm = torch.empty((w.B * kappa, V), dtype=torch.uint8, device="cuda")
    hc.hc_kappa_masks(to_torch(masks), sel, w.B, fm)
    F = w.B * kappa
    coords = torch.empty((F * V, 2), dtype=torch.int32, device="cuda")
    row_of = torch.empty((F, V), dtype=torch.int32, device="cuda")
    offs = torch.empty(F + 1, dtype=torch.int32, device="cuda")
    count = torch.empty(1, dtype=torch.int32, device="cuda")
    hc.hc_mask_compact(fm, coords, row_of, offs, count)
    xs = torch.empty((F * V, ly.C_in), dtype=torch.bfloat16, device="cuda")
    hc.hc_gather_rows(to_torch(w.x), coords, count, kappa, xs)
    y = torch.empty((F * V, ly.C_out), dtype=torch.bfloat16, device="cuda")
    hc.hc_sparse_spiral_conv_fwd(xs, hc.HC_LAYOUT_COMPACT, coords, row_of, count,
                                 to_torch(w.spiral), F, V, to_torch(ly.W), to_torch(ly.b),
                                 ly.act, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    np.testing.assert_array_equal(to_numpy(sel), sel_ref)
    np.testing.assert_array_equal(to_numpy(fm), fm_ref)
    assert int(count.item()) == n
    np.testing.assert_array_equal(to_numpy(xs)[:n], s_ref)
    check_close(to_numpy(y)[:n], y_pre, "kappa chain conv")
