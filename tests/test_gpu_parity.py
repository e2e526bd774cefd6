"""Parity of the CUDA path (through the C-ABI) with the CPU oracle.

Indices (coords, row_of, offsets, count) must match bit for bit; fp32 outputs
within 1e-4 absolute of the oracle's fp64 value; bf16 outputs within
2e-2 * max(|r|, 1) of the oracle's fp64 value r before rounding. Small cases
are compared element by element; full-size workloads on sampled rows that
the oracle computes one by one."""
import os

import numpy as np
import pytest

import oracle
from paper_2608_09388_gb300 import hc, inputs

from _util import check_close, sample_rows, to_numpy, to_torch

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
NCPU = len(os.sched_getaffinity(0))


@pytest.fixture
def gn_force():
    """Force the group-norm kernel choice ("auto", "slice" = one CTA per
    frame and group, "rows" = the row-range kernels) through the library's
    test hook; the automatic choice is restored afterwards."""
    paths = {"auto": 0, "slice": 1, "rows": 2}

    def force(path):
        hc.hc_test_set_option(hc.HC_TEST_GROUP_NORM_PATH, paths[path])

    yield force
    hc.hc_test_set_option(hc.HC_TEST_GROUP_NORM_PATH, 0)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_09388_gb300 import build
    build.build()
    hc.load_library()
    assert hc.hc_get_device_status() == hc.HC_OK


def gpu_compact(mask_np, offset=0):
    """Run hc_mask_compact; returns torch (coords, row_of, offsets, count).
    `offset` > 0 places the mask at a misaligned address."""
    B, V = mask_np.shape
    if offset:
        buf = torch.zeros(B * V + offset, dtype=torch.uint8, device="cuda")
        buf[offset:] = torch.from_numpy(mask_np.ravel()).cuda()
        mask = buf[offset:].view(B, V)
    else:
        mask = to_torch(mask_np)
    coords = torch.full((max(B * V, 1), 2), -7, dtype=torch.int32, device="cuda")
    row_of = torch.full((B, V), -7, dtype=torch.int32, device="cuda")
    offs = torch.full((B + 1,), -7, dtype=torch.int32, device="cuda")
    count = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    hc.hc_mask_compact(mask, coords, row_of, offs, count)
    return coords, row_of, offs, count


def assert_compact_equal(mask_np, got):
    coords, row_of, offs, count = got
    c_ref, r_ref, o_ref, n = oracle.mask_compact(mask_np)
    assert int(count.item()) == n
    np.testing.assert_array_equal(to_numpy(coords)[:n], c_ref)
    np.testing.assert_array_equal(to_numpy(row_of), r_ref)
    np.testing.assert_array_equal(to_numpy(offs), o_ref)


def run_sparse_conv(x_np, x_layout, mask_np, sp_np, W_np, b_np, act, coords=None, row_of=None,
                    count=None, y_fill=None):
    B, V = mask_np.shape
    if coords is None:
        coords, row_of, _, count = gpu_compact(mask_np)
    C_out = W_np.shape[1]
    x = to_torch(x_np)
    dt = torch.float32 if x_np.dtype == np.float32 else torch.bfloat16
    y = torch.full((B * V, C_out), float("nan") if y_fill is None else y_fill, dtype=dt,
                   device="cuda")
    hc.hc_sparse_spiral_conv_fwd(x, x_layout, coords, row_of, count, to_torch(sp_np), B, V,
                                 to_torch(W_np), None if b_np is None else to_torch(b_np), act, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    return to_numpy(y), int(count.item())


# ------------------------------------------------------------------ compaction

@pytest.mark.parametrize("B,V", [(1, 1), (1, 31), (7, 32), (7, 33), (64, 655), (256, 655),
                                 (3, 10475), (32, 10475)])
@pytest.mark.parametrize("density", [0.0, 0.01, 0.1, 0.5, 1.0])
def test_compact_bit_exact(B, V, density):
    m = inputs.uniform_mask(np.random.default_rng(B * 7919 + V), B, V, density)
    assert_compact_equal(m, gpu_compact(m))


@pytest.mark.parametrize("offset", [1, 3, 8])
def test_compact_misaligned_mask(offset):
    m = inputs.uniform_mask(np.random.default_rng(offset), 9, 777, 0.3)
    assert_compact_equal(m, gpu_compact(m, offset))


def test_compact_nonbinary_and_many_tiles():
    rng = np.random.default_rng(4)
    m = (rng.integers(0, 4, size=(520, 10475)) * (rng.random((520, 10475)) < 0.1)).astype(np.uint8)
    assert_compact_equal(m, gpu_compact(m))  # > 1024 tiles: pre-scanned offsets


def test_compact_empty_sizes():
    for B, V in [(0, 5), (3, 0), (0, 0)]:
        m = np.zeros((B, V), np.uint8)
        coords = torch.zeros((1, 2), dtype=torch.int32, device="cuda")
        offs = torch.full((B + 1,), -7, dtype=torch.int32, device="cuda")
        count = torch.full((1,), -7, dtype=torch.int32, device="cuda")
        hc.hc_mask_compact(torch.zeros((B, V), dtype=torch.uint8, device="cuda"), coords, None,
                           offs, count)
        assert int(count.item()) == 0 and (to_numpy(offs) == 0).all()


def test_compact_repeated_sizes_and_streams():
    """Calls of changing sizes back to back (more tiles, then fewer, then
    more; the per-stream workspace grows and is reused) on the default
    stream and on a second stream stay bit-exact."""
    side = torch.cuda.Stream()
    shapes = [(64, 10475), (3, 100), (1, 5000), (130, 10475), (2, 7), (64, 10475)]
    for i, (B, V) in enumerate(shapes):
        m = inputs.uniform_mask(np.random.default_rng(100 + i), B, V, 0.2)
        assert_compact_equal(m, gpu_compact(m))
        got = (torch.full((B * V, 2), -7, dtype=torch.int32, device="cuda"),
               torch.full((B, V), -7, dtype=torch.int32, device="cuda"),
               torch.full((B + 1,), -7, dtype=torch.int32, device="cuda"),
               torch.full((1,), -7, dtype=torch.int32, device="cuda"))
        mt = to_torch(m)
        torch.cuda.synchronize()
        with torch.cuda.stream(side):
            hc.hc_mask_compact(mt, *got, side)
        torch.cuda.synchronize()
        assert_compact_equal(m, got)
    assert hc.hc_get_device_status() == hc.HC_OK


def test_compact_graph_replays():
    """One compaction captured in a CUDA graph and replayed with new mask
    contents each time (empty, dense and sparse masks): every replay
    bit-exact."""
    B, V = 32, 10475
    stream = torch.cuda.Stream()
    mask = torch.zeros((B, V), dtype=torch.uint8, device="cuda")
    coords = torch.empty((B * V, 2), dtype=torch.int32, device="cuda")
    row_of = torch.empty((B, V), dtype=torch.int32, device="cuda")
    offs = torch.empty((B + 1,), dtype=torch.int32, device="cuda")
    count = torch.empty((1,), dtype=torch.int32, device="cuda")
    with torch.cuda.stream(stream):
        hc.hc_mask_compact(mask, coords, row_of, offs, count, stream)  # sets up the state
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            hc.hc_mask_compact(mask, coords, row_of, offs, count, stream)
    for i, d in enumerate((0.05, 0.0, 0.5, 1.0, 0.01)):
        m = inputs.uniform_mask(np.random.default_rng(200 + i), B, V, d)
        mask.copy_(torch.from_numpy(m))
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            g.replay()
        torch.cuda.synchronize()
        assert_compact_equal(m, (coords, row_of, offs, count))
    assert hc.hc_get_device_status() == hc.HC_OK


def test_compact_workload_masks():
    for name in ("layer655_f32", "encoder655_bf16", "motion655_bf16", "layer10475_bf16"):
        w = inputs.make_workload(name)
        for m in w.masks:
            assert_compact_equal(m, gpu_compact(m))


# ------------------------------------------------------------------ sparse conv

def test_golden_octahedron_on_gpu():
    """The hand-worked octahedron cases (fp32 path)."""
    import json
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "octahedron.json")))
    acts = {"none": hc.HC_ACT_NONE, "elu": hc.HC_ACT_ELU}
    for case in g["cases"]:
        sp = np.array(g["spiral_L3"], dtype=np.int32)[:, : case.get("spiral_cols", 3)].copy()
        for k, row in case.get("spiral_override", {}).items():
            sp[int(k)] = row
        x = np.array(case["x"], dtype=np.float32)
        m = np.array(case["mask"], dtype=np.uint8)
        W = np.array(case["W"], dtype=np.float32)
        b = np.array(case["bias"], dtype=np.float32)
        y, n = run_sparse_conv(x, hc.HC_LAYOUT_DENSE, m, sp, W, b, acts[case["act"]])
        c_ref, r_ref, _, n_ref = oracle.mask_compact(m)
        y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c_ref, r_ref, sp, W, b,
                                             acts[case["act"]])
        check_close(y[:n], y_pre, case["name"])


def test_layer655_f32_full():
    w = inputs.make_workload("layer655_f32")
    ly = w.layers[0]
    y, n = run_sparse_conv(w.x, hc.HC_LAYOUT_DENSE, w.masks[0], w.spiral, ly.W, ly.b, ly.act)
    c, r, _, n_ref = oracle.mask_compact(w.masks[0])
    assert n == n_ref
    y_pre, _ = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, c, r, w.spiral, ly.W, ly.b,
                                         ly.act)
    check_close(y[:n], y_pre, "layer655_f32")


# (B, V, L, C_in, C_out, density, neg_frac): ragged N', several tiles, -1 entries
SHAPES = [
    (1, 40, 1, 8, 8, 0.5, 0.0),
    (3, 200, 9, 16, 64, 0.3, 0.1),
    (5, 300, 12, 64, 128, 0.4, 0.05),
    (2, 500, 9, 128, 128, 0.6, 0.0),
    (4, 333, 7, 24, 40, 0.5, 0.2),
    (2, 257, 5, 8, 136, 0.9, 0.0),
    (2, 400, 9, 64, 256, 0.5, 0.0),
    (1, 700, 12, 32, 72, 0.35, 0.1),
]


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("layout", [hc.HC_LAYOUT_DENSE, hc.HC_LAYOUT_COMPACT])
@pytest.mark.parametrize("shape", SHAPES)
def test_sparse_conv_shapes(shape, layout, dtype):
    B, V, L, C_in, C_out, dens, neg = shape
    sp, m, x, W, b = inputs.random_case(B * 1000 + V + L + C_in + C_out, B, V, L, C_in, C_out,
                                        dtype, dens, neg)
    c, r, _, n = oracle.mask_compact(m)
    xin = x if layout == hc.HC_LAYOUT_DENSE else np.ascontiguousarray(x[c[:, 0], c[:, 1]])
    y, n_gpu = run_sparse_conv(xin, layout, m, sp, W, b, hc.HC_ACT_ELU)
    assert n_gpu == n
    y_pre, _ = oracle.sparse_spiral_conv(xin, layout, c, r, sp, W, b, oracle.ACT_ELU)
    check_close(y[:n], y_pre, f"{shape} layout={layout} {dtype}")


@pytest.mark.parametrize("C_in,C_out", [(45, 64), (16, 42), (10, 3), (64, 1)])
def test_sparse_conv_odd_channels_bf16(C_in, C_out):
    sp, m, x, W, b = inputs.random_case(C_in * 100 + C_out, 3, 300, 9, C_in, C_out, "bf16", 0.3)
    c, r, _, n = oracle.mask_compact(m)
    y, _ = run_sparse_conv(x, hc.HC_LAYOUT_DENSE, m, sp, W, b, hc.HC_ACT_ELU)
    y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c, r, sp, W, b, oracle.ACT_ELU)
    check_close(y[:n], y_pre, f"odd channels {C_in}->{C_out}")


@pytest.mark.parametrize("entry", ["spiral_dense", "spiral_compact", "rulebook_scatter", "dense"])
@pytest.mark.parametrize("L,C_in,C_out", [
    (9, 45, 64),    # the motion encoder's first layer: chunks cross slots
    (12, 13, 128),  # several slots per k-block
    (32, 9, 64),    # K = 288: a ragged last k-block
    (5, 100, 136),  # two output tiles, the second ragged
    (9, 3, 64),     # C_in below 8: one 8-channel slot per tap
])
def test_tc_channels_not_multiple_of_8(entry, L, C_in, C_out):
    """bf16 with C_in % 8 != 0 runs on the tensor cores with element-wise
    gathers; several row tiles and a ragged tail, every entry point."""
    B, V = 4, 1500
    dens = 1.0 if entry == "dense" else 0.45
    sp, m, x, W, b = inputs.random_case(L * 1000 + C_in * 10 + C_out, B, V, L, C_in, C_out,
                                        "bf16", dens, neg_frac=0.1)
    c, r, _, n = oracle.mask_compact(m)
    assert n > 3 * 128
    if entry == "dense":
        yd = torch.full((B, V, C_out), float("nan"), dtype=torch.bfloat16, device="cuda")
        hc.hc_spiral_conv_fwd(to_torch(x), to_torch(sp), to_torch(W), to_torch(b),
                              hc.HC_ACT_ELU, yd)
        assert hc.hc_get_device_status() == hc.HC_OK
        y = to_numpy(yd).reshape(B * V, C_out)[c[:, 0] * V + c[:, 1]]
        layout, xin = oracle.LAYOUT_DENSE, x
    elif entry == "rulebook_scatter":
        layout, xin = oracle.LAYOUT_DENSE, x
        rb, coords, row_of, count = gpu_rulebook(m, sp, hc.HC_LAYOUT_DENSE)
        prev = inputs.features(np.random.default_rng(9), (B, V, C_out), "bf16")
        out = to_torch(prev)
        yt = torch.full((B * V, C_out), float("nan"), dtype=torch.bfloat16, device="cuda")
        hc.hc_sparse_conv_rulebook_fwd(to_torch(x), rb, count, to_torch(W), to_torch(b),
                                       hc.HC_ACT_ELU, yt, coords=coords, out=out)
        assert hc.hc_get_device_status() == hc.HC_OK
        y = to_numpy(yt)[:n]
        o = to_numpy(out)
        np.testing.assert_array_equal(o[c[:, 0], c[:, 1]], y)
        inactive = np.ones((B, V), bool)
        inactive[c[:, 0], c[:, 1]] = False
        np.testing.assert_array_equal(o[inactive], prev[inactive])
    else:
        layout = hc.HC_LAYOUT_DENSE if entry == "spiral_dense" else hc.HC_LAYOUT_COMPACT
        xin = x if layout == hc.HC_LAYOUT_DENSE else np.ascontiguousarray(x[c[:, 0], c[:, 1]])
        y, n_gpu = run_sparse_conv(xin, layout, m, sp, W, b, hc.HC_ACT_ELU)
        assert n_gpu == n
        y = y[:n]
    y_pre, _ = oracle.sparse_spiral_conv(xin, layout, c, r, sp, W, b, oracle.ACT_ELU,
                                         n_threads=NCPU)
    check_close(y, y_pre, f"{entry} L={L} {C_in}->{C_out}")


@pytest.mark.parametrize("act", [hc.HC_ACT_NONE, hc.HC_ACT_RELU])
def test_sparse_conv_activations(act):
    sp, m, x, W, b = inputs.random_case(31, 2, 300, 9, 64, 64, "bf16", 0.4)
    c, r, _, n = oracle.mask_compact(m)
    y, _ = run_sparse_conv(x, hc.HC_LAYOUT_DENSE, m, sp, W, None, act)
    y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c, r, sp, W, None, act)
    check_close(y[:n], y_pre, f"act {act}")


def test_empty_mask_leaves_output_untouched():
    sp, m, x, W, b = inputs.random_case(32, 2, 300, 9, 64, 128, "bf16", 0.0)
    y, n = run_sparse_conv(x, hc.HC_LAYOUT_DENSE, m, sp, W, b, hc.HC_ACT_ELU, y_fill=3.0)
    assert n == 0
    assert (y == to_numpy(torch.tensor([3.0], dtype=torch.bfloat16))[0]).all()


def test_all_ones_mask_equals_dense_operator():
    sp, m, x, W, b = inputs.random_case(33, 3, 300, 9, 64, 128, "bf16", 1.0)
    y, n = run_sparse_conv(x, hc.HC_LAYOUT_DENSE, m, sp, W, b, hc.HC_ACT_ELU)
    yd = torch.empty((3, 300, 128), dtype=torch.bfloat16, device="cuda")
    hc.hc_spiral_conv_fwd(to_torch(x), to_torch(sp), to_torch(W), to_torch(b), hc.HC_ACT_ELU, yd)
    np.testing.assert_array_equal(y[:n], to_numpy(yd).reshape(-1, 128))


def test_deterministic_and_stream_ordered():
    sp, m, x, W, b = inputs.random_case(34, 4, 500, 12, 64, 128, "bf16", 0.3)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        y1, _ = run_sparse_conv(x, hc.HC_LAYOUT_DENSE, m, sp, W, b, hc.HC_ACT_ELU)
        y2, _ = run_sparse_conv(x, hc.HC_LAYOUT_DENSE, m, sp, W, b, hc.HC_ACT_ELU)
    np.testing.assert_array_equal(y1, y2)


# ------------------------------------------------------------------ rulebook (Eq. 4 mapping)

def gpu_rulebook(m, sp, layout):
    B, V = m.shape
    coords, row_of, offs, count = gpu_compact(m)
    rb = torch.full((sp.shape[1], B * V), -7, dtype=torch.int32, device="cuda")
    hc.hc_conv_rulebook(coords, row_of, count, to_torch(sp), B, V, layout, rb)
    assert hc.hc_get_device_status() == hc.HC_OK
    return rb, coords, row_of, count


@pytest.mark.parametrize("layout", [hc.HC_LAYOUT_DENSE, hc.HC_LAYOUT_COMPACT])
@pytest.mark.parametrize("shape", [(1, 40, 1), (3, 200, 9), (5, 300, 12), (2, 1000, 32), (1, 5, 5)])
def test_rulebook_bit_exact(shape, layout):
    B, V, L = shape
    sp, m, x, W, b = inputs.random_case(B * 31 + V + L, B, V, L, 8, 8, "f32", 0.35, neg_frac=0.1)
    rb, *_ = gpu_rulebook(m, sp, layout)
    c, r, _, n = oracle.mask_compact(m)
    ref = oracle.conv_rulebook(c, r, sp, layout)
    np.testing.assert_array_equal(to_numpy(rb)[:, :n], ref[:, :n])


RB_SHAPES = [
    (3, 200, 9, 64, 64, 0.3, "bf16"),     # tensor cores, TMA gather
    (2, 300, 12, 128, 128, 0.5, "bf16"),  # tensor cores, TMA gather, 2 k-blocks per slot
    (4, 333, 7, 24, 40, 0.5, "bf16"),     # tensor cores, cp.async gather
    (2, 300, 9, 45, 64, 0.3, "bf16"),     # CUDA cores (C_in not a multiple of 8)
    (1, 655, 9, 16, 64, 0.1, "f32"),      # CUDA cores, fp32
    (2, 257, 5, 64, 136, 0.9, "bf16"),    # two N tiles
]


@pytest.mark.parametrize("layout", [hc.HC_LAYOUT_DENSE, hc.HC_LAYOUT_COMPACT])
@pytest.mark.parametrize("shape", RB_SHAPES)
def test_conv_through_rulebook(shape, layout):
    B, V, L, C_in, C_out, dens, dtype = shape
    sp, m, x, W, b = inputs.random_case(B + V + L + C_in + C_out, B, V, L, C_in, C_out, dtype,
                                        dens, neg_frac=0.1)
    rb, coords, row_of, count = gpu_rulebook(m, sp, layout)
    c, r, _, n = oracle.mask_compact(m)
    xin = x if layout == hc.HC_LAYOUT_DENSE else np.ascontiguousarray(x[c[:, 0], c[:, 1]])
    xt = to_torch(xin)
    y = torch.full((B * V, C_out), float("nan"), dtype=xt.dtype, device="cuda")
    hc.hc_sparse_conv_rulebook_fwd(xt, rb, count, to_torch(W), to_torch(b), hc.HC_ACT_ELU, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    y_pre, _ = oracle.sparse_spiral_conv(xin, layout, c, r, sp, W, b, oracle.ACT_ELU)
    check_close(to_numpy(y)[:n], y_pre, f"rulebook conv {shape} layout={layout}")


@pytest.mark.parametrize("shape", [(3, 200, 9, 64, 128, "bf16"), (2, 300, 9, 24, 40, "bf16"),
                                   (2, 300, 9, 45, 64, "bf16"), (1, 655, 9, 16, 64, "f32")])
@pytest.mark.parametrize("with_compact", [True, False])
def test_conv_through_rulebook_fused_scatter(shape, with_compact):
    """The rulebook conv writing the dense [B, V, C_out] tensor directly (the
    scatter fused into its epilogue): active rows hold the conv result, all
    other rows keep their previous contents."""
    B, V, L, C_in, C_out, dtype = shape
    sp, m, x, W, b = inputs.random_case(B * 7 + V + C_in, B, V, L, C_in, C_out, dtype, 0.3, 0.1)
    rb, coords, row_of, count = gpu_rulebook(m, sp, hc.HC_LAYOUT_DENSE)
    c, r, _, n = oracle.mask_compact(m)
    xt = to_torch(x)
    prev = inputs.features(np.random.default_rng(3), (B, V, C_out), dtype)
    out = to_torch(prev)
    y = torch.full((B * V, C_out), float("nan"), dtype=xt.dtype, device="cuda") if with_compact \
        else None
    hc.hc_sparse_conv_rulebook_fwd(xt, rb, count, to_torch(W), to_torch(b), hc.HC_ACT_ELU, y,
                                   coords=coords, out=out)
    assert hc.hc_get_device_status() == hc.HC_OK
    got = to_numpy(out)
    y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c, r, sp, W, b, oracle.ACT_ELU)
    check_close(got[c[:, 0], c[:, 1]], y_pre, f"fused scatter {shape}")
    inactive = np.ones((B, V), bool)
    inactive[c[:, 0], c[:, 1]] = False
    np.testing.assert_array_equal(got[inactive], prev[inactive])
    if with_compact:
        np.testing.assert_array_equal(to_numpy(y)[:n], got[c[:, 0], c[:, 1]])


def test_encoder_through_rulebooks():
    """Stacked layers sharing one mask: one rulebook for the dense-input first
    layer and one for the compact layers after it, reused by every layer."""
    w = inputs.make_workload("encoder655_bf16")
    m = w.masks[0]
    B, V = m.shape
    rb_d, coords, row_of, count = gpu_rulebook(m, w.spiral, hc.HC_LAYOUT_DENSE)
    rb_c = torch.empty_like(rb_d)
    hc.hc_conv_rulebook(coords, row_of, count, to_torch(w.spiral), B, V, hc.HC_LAYOUT_COMPACT, rb_c)
    h = to_torch(w.x)
    first = True
    for ly in w.layers:
        y = torch.empty((B * V, ly.C_out), dtype=torch.bfloat16, device="cuda")
        if ly.kind == "conv":
            hc.hc_sparse_conv_rulebook_fwd(h, rb_d if first else rb_c, count, to_torch(ly.W),
                                           to_torch(ly.b), ly.act, y)
        else:
            hc.hc_sparse_linear_fwd(h, count, to_torch(ly.W), to_torch(ly.b), ly.act, y)
        h, first = y, False
    assert hc.hc_get_device_status() == hc.HC_OK
    c, r, o, n, outs = oracle.encoder(w.x, m, w.spiral, w.layers, n_threads=NCPU)
    check_close(to_numpy(h)[:n], outs[-1][0], "encoder through rulebooks")


def test_rulebook_full_size_sampled():
    w = inputs.make_workload("layer10475_bf16")
    ly = w.layers[0]
    B, V = w.B, w.V
    rb, coords, row_of, count = gpu_rulebook(w.masks[0], w.spiral, hc.HC_LAYOUT_DENSE)
    c, r, _, n = oracle.mask_compact(w.masks[0])
    np.testing.assert_array_equal(to_numpy(rb)[:, :n], oracle.conv_rulebook(c, r, w.spiral, 0)[:, :n])
    y = torch.empty((B * V, ly.C_out), dtype=torch.bfloat16, device="cuda")
    hc.hc_sparse_conv_rulebook_fwd(to_torch(w.x), rb, count, to_torch(ly.W), to_torch(ly.b),
                                   ly.act, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    rows = sample_rows(n, 3000, seed=5)
    y_pre, _ = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, c, r, w.spiral, ly.W, ly.b,
                                         ly.act, rows=rows, n_threads=NCPU)
    check_close(to_numpy(y)[rows], y_pre, "rulebook conv, 10475-vertex layer")


def test_rulebook_entry_out_of_range_is_reported():
    sp, m, x, W, b = inputs.random_case(77, 2, 100, 5, 64, 64, "bf16", 1.0)
    rb, coords, row_of, count = gpu_rulebook(m, sp, hc.HC_LAYOUT_DENSE)
    rb[2, 5] = 200  # == x_rows: out of range
    rb[1, 7] = -3
    y = torch.empty((200, 64), dtype=torch.bfloat16, device="cuda")
    hc.hc_sparse_conv_rulebook_fwd(to_torch(x), rb, count, to_torch(W), to_torch(b), 1, y)
    assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
    # the bad entries contribute nothing: the same as absent taps
    rb[2, 5] = -1
    rb[1, 7] = -1
    y_abs = torch.empty_like(y)
    hc.hc_sparse_conv_rulebook_fwd(to_torch(x), rb, count, to_torch(W), to_torch(b), 1, y_abs)
    assert hc.hc_get_device_status() == hc.HC_OK
    n = int(count.item())
    assert torch.equal(y[:n], y_abs[:n])


# ------------------------------------------------------------------ dense conv

@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("shape", [(2, 300, 9, 64, 128), (3, 257, 12, 16, 64), (1, 100, 5, 40, 24)])
def test_dense_conv(shape, dtype):
    B, V, L, C_in, C_out = shape
    sp, m, x, W, b = inputs.random_case(sum(shape), B, V, L, C_in, C_out, dtype, 1.0, 0.1)
    xt = to_torch(x)
    y = torch.empty((B, V, C_out), dtype=xt.dtype, device="cuda")
    hc.hc_spiral_conv_fwd(xt, to_torch(sp), to_torch(W), to_torch(b), hc.HC_ACT_ELU, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    y_pre, _ = oracle.dense_spiral_conv(x, sp, W, b, oracle.ACT_ELU)
    check_close(to_numpy(y).reshape(B * V, C_out), y_pre, f"dense {shape} {dtype}")


# ------------------------------------------------------------------ linear

@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("C_in,C_out", [(64, 42), (64, 1), (64, 128), (128, 64), (45, 7)])
def test_sparse_linear(C_in, C_out, dtype):
    rng = np.random.default_rng(C_in * 1000 + C_out)
    cap, n = 1000, 777
    x = inputs.features(rng, (cap, C_in), dtype)
    W = inputs.weights(rng, C_in, C_out, dtype)
    b = inputs.bias(C_out)
    count = torch.tensor([n], dtype=torch.int32, device="cuda")
    xt = to_torch(x)
    y = torch.full((cap, C_out), float("nan"), dtype=xt.dtype, device="cuda")
    hc.hc_sparse_linear_fwd(xt, count, to_torch(W), to_torch(b), hc.HC_ACT_NONE, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    y_pre, _ = oracle.sparse_linear(x[:n], W, b, oracle.ACT_NONE)
    got = to_numpy(y)
    check_close(got[:n], y_pre, f"linear {C_in}->{C_out} {dtype}")
    assert np.isnan(got[n:].astype(np.float64) if dtype == "f32" else
                    (got[n:].astype(np.uint32) << 16).view(np.float32)).all()


# ------------------------------------------------------------------ scatter

@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("C", [1, 3, 8, 42, 128])
@pytest.mark.parametrize("zero_fill,inverse", [(0, "row_of"), (1, "row_of"), (1, "none")])
def test_scatter_dense(C, zero_fill, inverse, dtype):
    """Copy of the active rows, bit for bit; with zero_fill every other row
    becomes 0, through the inverse map (one pass) or, without it, a zero pass
    then the scatter (the call as the problem statement gives it)."""
    rng = np.random.default_rng(C * 10 + zero_fill)
    B, V = 5, 333
    m = inputs.uniform_mask(rng, B, V, 0.25)
    coords, row_of, offs, count = gpu_compact(m)
    c, r, _, n = oracle.mask_compact(m)
    y = inputs.features(rng, (n, C), dtype)
    prev = inputs.features(rng, (B, V, C), dtype)
    out = to_torch(prev)
    hc.hc_scatter_dense(to_torch(y), coords, row_of if inverse == "row_of" else None, count, B,
                        V, zero_fill, out)
    assert hc.hc_get_device_status() == hc.HC_OK
    ref = oracle.scatter_dense(y, c, B, V, zero_fill, out=prev)
    np.testing.assert_array_equal(to_numpy(out), ref)


# ------------------------------------------------------------------ group norm

def _gn_case(rng, sizes, C, dtype, shift=3.0, slack=5):
    """Compact rows for frames of the given row counts (plus `slack` rows
    that belong to no frame), features N(shift, 1)."""
    offs = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int32)
    cap = int(offs[-1]) + slack
    x = rng.standard_normal((cap, C)).astype(np.float32) + np.float32(shift)
    if dtype == "bf16":
        x = inputs.to_bf16_bits(x)
    return x, offs


def run_group_norm(x, offs, G, gamma, beta, act, eps=1e-5, in_place=False):
    xt = to_torch(x)
    y = xt if in_place else torch.full_like(xt, float("nan"))
    hc.hc_sparse_group_norm_fwd(xt, to_torch(offs), G, eps,
                                None if gamma is None else to_torch(gamma),
                                None if beta is None else to_torch(beta), act, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    return to_numpy(y)


def _as_f32(a):
    return (a.astype(np.uint32) << 16).view(np.float32) if a.dtype == np.uint16 else a


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("C,G", [(8, 1), (64, 4), (64, 8), (128, 32), (128, 64), (128, 128),
                                 (256, 16), (1024, 512), (42, 6), (48, 3)])
@pytest.mark.parametrize("affine,act", [(False, 0), (True, 1), (True, 2)])
@pytest.mark.parametrize("path", ["auto", "rows"])
def test_group_norm(C, G, affine, act, dtype, path, gn_force):
    """Frames of 0, 1, a few, a tile-ish and a large number of rows; rows
    after the last frame stay untouched. 'rows' forces the row-range kernels
    wherever the layout allows them."""
    gn_force(path)
    rng = np.random.default_rng(C * 100 + G * 7 + act)
    sizes = [0, 1, 3, 0, 130, 517, 2900, 64]
    x, offs = _gn_case(rng, sizes, C, dtype)
    gamma = (1.0 + 0.5 * rng.standard_normal(C)).astype(np.float32) if affine else None
    beta = (0.3 * rng.standard_normal(C)).astype(np.float32) if affine else None
    got = run_group_norm(x, offs, G, gamma, beta, act)
    y_pre, _ = oracle.sparse_group_norm(x, offs, G, 1e-5, gamma, beta, act)
    n = int(offs[-1])
    check_close(got[:n], y_pre[:n], f"group norm C={C} G={G} {dtype}")
    assert np.isnan(_as_f32(got[n:])).all()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("C,G", [(64, 8), (128, 32), (2048, 8)])
@pytest.mark.parametrize("path", ["rows", "slice"])
def test_group_norm_paths_and_frame_shapes(C, G, path, dtype, gn_force):
    """Both kernels (contiguous row ranges, and one CTA per frame and group)
    on many tiny frames (a row range holds dozens of frame segments) and on
    one frame spread over hundreds of row ranges (its partials are merged by
    a warp)."""
    gn_force(path)
    rng = np.random.default_rng(C + G)
    tiny = [int(v) for v in rng.integers(0, 6, size=300)]
    big = [40000 if C <= 128 else 3000]
    for sizes in (tiny, big, tiny[:40] + big + tiny[40:80]):
        x, offs = _gn_case(rng, sizes, C, dtype, shift=-1.5)
        gamma = (1.0 + 0.5 * rng.standard_normal(C)).astype(np.float32)
        got = run_group_norm(x, offs, G, gamma, None, 2)
        y_pre, _ = oracle.sparse_group_norm(x, offs, G, 1e-5, gamma, None, 2)
        n = int(offs[-1])
        check_close(got[:n], y_pre[:n], f"group norm {path} C={C} G={G} {dtype} B={len(sizes)}")


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_group_norm_in_place_and_misaligned(dtype):
    rng = np.random.default_rng(5)
    C, G = 64, 8
    x, offs = _gn_case(rng, [300, 0, 1100, 7], C, dtype)
    y_pre, _ = oracle.sparse_group_norm(x, offs, G, 1e-5, None, None, 1)
    n = int(offs[-1])
    check_close(run_group_norm(x, offs, G, None, None, 1, in_place=True)[:n], y_pre[:n],
                "in place")
    # a view starting one element in: the 16-byte paths are not taken
    xt = to_torch(x)
    buf = torch.empty(x.size + 1, dtype=xt.dtype, device="cuda")
    xs = buf[1:].view(x.shape)
    xs.copy_(xt)
    ys = torch.full_like(xs, float("nan"))
    hc.hc_sparse_group_norm_fwd(xs, to_torch(offs), G, 1e-5, None, None, 1, ys)
    assert hc.hc_get_device_status() == hc.HC_OK
    check_close(to_numpy(ys)[:n], y_pre[:n], "misaligned")


@pytest.mark.parametrize("path", ["rows", "slice"])
def test_group_norm_constant_group_and_eps(path, gn_force):
    """A group of equal values normalises to exactly 0 (then + beta); eps
    from 0 to large enters as 1/sqrt(var + eps)."""
    gn_force(path)
    C, G = 32, 4
    offs = np.array([0, 200, 201], dtype=np.int32)
    x = np.full((201, C), 100.25, dtype=np.float32)
    beta = np.linspace(-1, 1, C).astype(np.float32)
    got = run_group_norm(x, offs, G, None, beta, 0)
    np.testing.assert_array_equal(got, np.broadcast_to(beta, got.shape))
    rng = np.random.default_rng(9)
    x, offs = _gn_case(rng, [50, 400], C, "f32", shift=-2.0, slack=0)
    for eps in (0.0, 1e-5, 4.0):
        y_pre, _ = oracle.sparse_group_norm(x, offs, G, eps, None, None, 0)
        check_close(run_group_norm(x, offs, G, None, None, 0, eps=eps), y_pre, f"eps={eps}")


def test_group_norm_on_compacted_layer_output(gn_force):
    """The normalisation an encoder applies after a conv: a full-size
    compacted bf16 activation (32 clustered frames of the 10475-vertex
    sphere, 128 channels, G = 8), frame ranges from hc_mask_compact."""
    w = inputs.make_workload("layer10475_bf16")
    coords, row_of, offs, count = gpu_compact(w.masks[0])
    n = int(count.item())
    rng = np.random.default_rng(77)
    x = inputs.features(rng, (n, 128), "bf16")
    gamma = (1.0 + 0.2 * rng.standard_normal(128)).astype(np.float32)
    beta = (0.1 * rng.standard_normal(128)).astype(np.float32)
    xt = to_torch(x)
    y = torch.empty_like(xt)
    y_pre, _ = oracle.sparse_group_norm(x, to_numpy(offs), 8, 1e-5, gamma, beta, oracle.ACT_ELU)
    for path in ("auto", "rows"):
        gn_force(path)
        y.fill_(float("nan"))
        hc.hc_sparse_group_norm_fwd(xt, offs, 8, 1e-5, to_torch(gamma), to_torch(beta),
                                    hc.HC_ACT_ELU, y)
        assert hc.hc_get_device_status() == hc.HC_OK
        check_close(to_numpy(y), y_pre, f"group norm full size ({path})")


@pytest.mark.parametrize("path", ["rows", "slice"])
def test_group_norm_bad_offsets_reported(path, gn_force):
    gn_force(path)
    x = torch.zeros((10, 16), dtype=torch.float32, device="cuda")
    offs = torch.tensor([0, 4, 12], dtype=torch.int32, device="cuda")  # 12 > capacity
    hc.hc_sparse_group_norm_fwd(x, offs, 4, 1e-5, None, None, 0, x)
    assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
    offs = torch.tensor([0, 5, 3], dtype=torch.int32, device="cuda")  # decreasing
    hc.hc_sparse_group_norm_fwd(x, offs, 4, 1e-5, None, None, 0, x)
    assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
    assert hc.hc_get_device_status() == hc.HC_OK


# ------------------------------------------------------------------ encoders

def run_encoder_gpu(w):
    """The stacked sparse layers of a workload through the C-ABI: compact
    once, first conv on the dense input, later layers on compact rows, then
    the linear head."""
    m = w.masks[0]
    B, V = m.shape
    coords, row_of, offs, count = gpu_compact(m)
    h = to_torch(w.x)
    layout = hc.HC_LAYOUT_DENSE
    sp = to_torch(w.spiral)
    for ly in w.layers:
        y = torch.empty((B * V, ly.C_out), dtype=h.dtype, device="cuda")
        if ly.kind == "conv":
            hc.hc_sparse_spiral_conv_fwd(h, layout, coords, row_of, count, sp, B, V,
                                         to_torch(ly.W), to_torch(ly.b), ly.act, y)
        else:
            hc.hc_sparse_linear_fwd(h, count, to_torch(ly.W), to_torch(ly.b), ly.act, y)
        h, layout = y, hc.HC_LAYOUT_COMPACT
    assert hc.hc_get_device_status() == hc.HC_OK
    return to_numpy(h), int(count.item())


@pytest.mark.parametrize("name", ["encoder655_bf16", "motion655_bf16"])
def test_encoder_end_to_end(name):
    """Whole stack against the oracle's own stack (each layer stored in bf16
    on both sides). The final layer is compared under the bf16 tolerance."""
    w = inputs.make_workload(name)
    got, n = run_encoder_gpu(w)
    c, r, o, n_ref, outs = oracle.encoder(w.x, w.masks[0], w.spiral, w.layers, n_threads=NCPU)
    assert n == n_ref
    check_close(got[:n], outs[-1][0], name)


@pytest.mark.parametrize("name", ["layer655_f32", "encoder655_bf16", "motion655_bf16"])
def test_dense_layout_chain_against_oracle(name):
    """The configs' dense-layout chain: one dense-layout mapping, every conv
    reading the previous layer's dense rows and writing only its active rows
    into a dense tensor (fused scatter, no compact output), the per-vertex
    head as the rulebook conv on the centre slot; the head's compact rows
    against the oracle's stack, and the same bits as the compact chain."""
    w = inputs.make_workload(name)
    B, V = w.B, w.V
    dt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    rb, coords, row_of, count = gpu_rulebook(w.masks[0], w.spiral, hc.HC_LAYOUT_DENSE)
    h = to_torch(w.x)
    for i, ly in enumerate(w.layers):
        taps = rb if ly.kind == "conv" else rb[0:1]
        if i + 1 == len(w.layers):
            y = torch.full((B * V, ly.C_out), float("nan"), dtype=dt, device="cuda")
            hc.hc_sparse_conv_rulebook_fwd(h, taps, count, to_torch(ly.W), to_torch(ly.b),
                                           ly.act, y)
            h = y
        else:
            d = torch.full((B, V, ly.C_out), float("nan"), dtype=dt, device="cuda")
            hc.hc_sparse_conv_rulebook_fwd(h, taps, count, to_torch(ly.W), to_torch(ly.b),
                                           ly.act, None, coords=coords, out=d)
            h = d
    assert hc.hc_get_device_status() == hc.HC_OK
    n = int(count.item())
    c, r, o, n_ref, outs = oracle.encoder(w.x, w.masks[0], w.spiral, w.layers, n_threads=NCPU)
    assert n == n_ref
    check_close(to_numpy(h)[:n], outs[-1][0], f"{name} dense-layout chain")
    if len(w.layers) > 1:
        got, n2 = run_encoder_gpu(w)
        assert n2 == n
        np.testing.assert_array_equal(to_numpy(h)[:n], got[:n])


# ------------------------------------------------------------------ full size, sampled

def test_layer10475_full_size_sampled():
    w = inputs.make_workload("layer10475_bf16")
    ly = w.layers[0]
    y, n = run_sparse_conv(w.x, hc.HC_LAYOUT_DENSE, w.masks[0], w.spiral, ly.W, ly.b, ly.act)
    c, r, _, n_ref = oracle.mask_compact(w.masks[0])
    assert n == n_ref
    rows = sample_rows(n, 3000, seed=1)
    y_pre, _ = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, c, r, w.spiral, ly.W, ly.b,
                                         ly.act, rows=rows, n_threads=NCPU)
    check_close(y[rows], y_pre, "layer10475 sampled")


def test_sweep10475_full_size_sampled():
    w = inputs.make_workload("sweep10475_bf16")
    ly = w.layers[0]
    B, V = w.B, w.V
    xt = to_torch(w.x)
    for d, m in zip(w.densities, w.masks):
        y, n = run_sparse_conv(w.x, hc.HC_LAYOUT_DENSE, m, w.spiral, ly.W, ly.b, ly.act)
        c, r, _, n_ref = oracle.mask_compact(m)
        assert n == n_ref
        rows = sample_rows(n, 600, seed=2)
        y_pre, _ = oracle.sparse_spiral_conv(w.x, oracle.LAYOUT_DENSE, c, r, w.spiral, ly.W, ly.b,
                                             ly.act, rows=rows, n_threads=NCPU)
        check_close(y[rows], y_pre, f"sweep density {d}")
    yd = torch.empty((B, V, ly.C_out), dtype=torch.bfloat16, device="cuda")
    hc.hc_spiral_conv_fwd(xt, to_torch(w.spiral), to_torch(ly.W), to_torch(ly.b), ly.act, yd)
    assert hc.hc_get_device_status() == hc.HC_OK
    rows = sample_rows(B * V, 1500, seed=3)
    y_pre, _ = oracle.dense_spiral_conv(w.x, w.spiral, ly.W, ly.b, ly.act, rows=rows,
                                        n_threads=NCPU)
    check_close(to_numpy(yd).reshape(B * V, -1)[rows], y_pre, "dense full size")


# ------------------------------------------------------------------ device status

def test_out_of_range_spiral_entry_is_reported():
    """A spiral entry outside [-1, V) is caught by the kernel's own bounds
    check: the tap contributes nothing and HC_ERR_INVALID_INDEX is raised."""
    for C_out in (64, 42):  # tensor-core path and CUDA-core path
        sp, m, x, W, b = inputs.random_case(40 + C_out, 2, 100, 5, 16, C_out, "bf16", 1.0)
        sp[3, 2] = 100  # == V: out of range
        sp[7, 1] = -5
        coords, row_of, _, count = gpu_compact(m)
        out = torch.empty((200, C_out), dtype=torch.bfloat16, device="cuda")
        hc.hc_sparse_spiral_conv_fwd(to_torch(x), hc.HC_LAYOUT_DENSE, coords, row_of, count,
                                     to_torch(sp), 2, 100, to_torch(W), to_torch(b),
                                     hc.HC_ACT_ELU, out)
        assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
        assert hc.hc_get_device_status() == hc.HC_OK  # reading clears it


def test_count_above_capacity_is_reported():
    x = torch.zeros((10, 16), dtype=torch.bfloat16, device="cuda")
    W = torch.zeros((16, 16), dtype=torch.bfloat16, device="cuda")
    y = torch.zeros((10, 16), dtype=torch.bfloat16, device="cuda")
    count = torch.tensor([11], dtype=torch.int32, device="cuda")
    hc.hc_sparse_linear_fwd(x, count, W, None, hc.HC_ACT_NONE, y)
    assert hc.hc_get_device_status() == hc.HC_ERR_CAPACITY


def test_host_rejects_bad_arguments():
    x = torch.zeros((4, 16), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(hc.HcError) as e:
        hc.hc_sparse_linear_fwd(x, None, x, None, hc.HC_ACT_NONE, x)
    assert e.value.status == hc.HC_ERR_INVALID_ARG
