"""GPU parity of hc_mask_compact_rulebook (compaction fused with the Eq. 4
mapping) through the C-ABI: bit-exact against the oracle's mask_compact
followed by conv_rulebook. Shapes cover frames around the 16-byte chunks and
4096-byte tiles the kernels read, several 1024-vertex blocks per frame, the
frame-size limit of the fused pass (V = 65535 fused, larger frames through
the separate kernels), L up to 32, more than 1024 tiles (pre-scanned
tile counts), empty and full masks, absent neighbours, non-binary and
misaligned masks, and out-of-range spiral entries."""
import numpy as np
import pytest

import oracle
from paper_2608_09388_gb300 import hc, inputs

from _util import to_numpy, to_torch

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


def case(seed, B, V, L, density):
    """Mask and spiral: the geometric spiral table for small frames, a random
    table (slot 0 the vertex itself, ~10% absent entries) for large ones,
    whose nearest-neighbour construction would take minutes."""
    if V <= 5000:
        sp, m, *_ = inputs.random_case(seed, B, V, L, 8, 8, "f32", density, neg_frac=0.1)
        return sp, m
    rng = np.random.default_rng(seed)
    sp = rng.integers(0, V, size=(V, L)).astype(np.int32)
    sp[rng.random((V, L)) < 0.1] = -1
    sp[:, 0] = np.arange(V)
    return sp, inputs.uniform_mask(rng, B, V, density)


def run_fused(m, sp, layout, offset=0):
    B, V = m.shape
    L = sp.shape[1]
    if offset:
        buf = torch.zeros(B * V + offset, dtype=torch.uint8, device="cuda")
        buf[offset:] = torch.from_numpy(m.ravel()).cuda()
        mask = buf[offset:].view(B, V)
    else:
        mask = to_torch(m)
    cap = max(B * V, 1)
    coords = torch.full((cap, 2), -7, dtype=torch.int32, device="cuda")
    row_of = torch.full((B, V), -7, dtype=torch.int32, device="cuda")
    offs = torch.full((B + 1,), -7, dtype=torch.int32, device="cuda")
    count = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    rb = torch.full((L, cap), -7, dtype=torch.int32, device="cuda")
    hc.hc_mask_compact_rulebook(mask, to_torch(sp), layout, coords, row_of, offs, count, rb)
    return [to_numpy(t) for t in (coords, row_of, offs, count, rb)]


def check(m, sp, layout, got, sp_ref=None):
    coords, row_of, offs, count, rb = got
    c_ref, r_ref, o_ref, n = oracle.mask_compact(m)
    assert int(count[0]) == n
    np.testing.assert_array_equal(coords[:n], c_ref)
    assert (coords[n:] == -7).all()  # rows past the count untouched
    np.testing.assert_array_equal(row_of, r_ref)
    np.testing.assert_array_equal(offs, o_ref)
    ref = oracle.conv_rulebook(c_ref, r_ref, sp if sp_ref is None else sp_ref, layout)
    np.testing.assert_array_equal(rb[:, :n], ref[:, :n])
    assert (rb[:, n:] == -7).all()  # columns past the count untouched


@pytest.mark.parametrize("layout", [hc.HC_LAYOUT_DENSE, hc.HC_LAYOUT_COMPACT])
@pytest.mark.parametrize("B,V,L,density", [
    (1, 1, 1, 1.0), (1, 15, 3, 0.5), (3, 17, 5, 0.6), (7, 33, 9, 0.3), (2, 200, 9, 0.35),
    (5, 1023, 12, 0.2), (3, 1025, 12, 0.4), (4, 2049, 7, 0.1), (2, 4097, 12, 0.05),
    (32, 655, 9, 0.1), (64, 655, 16, 0.5), (1, 32767, 12, 0.05), (2, 5000, 1, 0.3),
    (2, 32768, 12, 0.2), (3, 300, 17, 0.2), (2, 100, 32, 0.2), (1, 65535, 9, 0.1)])
def test_fused_bit_exact(B, V, L, density, layout):
    sp, m = case(B * 131 + V * 7 + L, B, V, L, density)
    check(m, sp, layout, run_fused(m, sp, layout))
    assert hc.hc_get_device_status() == hc.HC_OK


@pytest.mark.parametrize("B,V,L", [(2, 65536, 12), (1, 70001, 5)])
def test_separate_kernels_past_the_fused_limits(B, V, L):
    """V > 65535: the compaction and mapping kernels of the two separate
    entry points, same results."""
    sp, m = case(B + V + L, B, V, L, 0.2)
    for layout in (hc.HC_LAYOUT_DENSE, hc.HC_LAYOUT_COMPACT):
        check(m, sp, layout, run_fused(m, sp, layout))


@pytest.mark.parametrize("density", [0.0, 1.0])
def test_empty_and_full_masks(density):
    sp, m, *_ = inputs.random_case(9, 6, 1500, 12, 8, 8, "f32", density)
    check(m, sp, hc.HC_LAYOUT_DENSE, run_fused(m, sp, hc.HC_LAYOUT_DENSE))


def test_workload_mask_and_many_tiles():
    """The bench layer's clustered mask (32 x 10475), and 420 frames of it
    (more than 1024 tiles of 4096 bytes: pre-scanned tile counts), with a
    non-binary mask value."""
    w = inputs.make_workload("layer10475_bf16")
    check(w.masks[0], w.spiral, hc.HC_LAYOUT_DENSE, run_fused(w.masks[0], w.spiral, 0))
    big = np.concatenate([w.masks[0]] * 13 + [w.masks[0][:4]], axis=0).copy()
    big[5, 17] = 3
    check(big, w.spiral, hc.HC_LAYOUT_COMPACT, run_fused(big, w.spiral, hc.HC_LAYOUT_COMPACT))


def test_many_frames_twice():
    """Many frames (6000 frames of 1200 vertices: 12000 CTAs of the write
    pass, more than the GPU holds at once; 16400 frames of 40 vertices),
    each twice in a row on the same buffers."""
    for B, V in ((6000, 1200), (16400, 40)):
        rng = np.random.default_rng(B)
        sp = rng.integers(0, V, size=(V, 5)).astype(np.int32)
        sp[:, 0] = np.arange(V)
        m = inputs.uniform_mask(rng, B, V, 0.07)
        for _ in range(2):
            check(m, sp, hc.HC_LAYOUT_COMPACT, run_fused(m, sp, hc.HC_LAYOUT_COMPACT))
            assert hc.hc_get_device_status() == hc.HC_OK


def test_streams_and_sizes_back_to_back():
    """Calls of changing frame counts back to back on two streams (each
    stream has its own workspace): every one bit-exact."""
    side = torch.cuda.Stream()
    for i, (B, V) in enumerate([(64, 655), (3, 10475), (200, 300), (1, 12), (64, 655)]):
        sp, m = case(300 + i, B, V, 9, 0.3)
        check(m, sp, hc.HC_LAYOUT_DENSE, run_fused(m, sp, hc.HC_LAYOUT_DENSE))
        torch.cuda.synchronize()
        with torch.cuda.stream(side):
            got = run_fused(m, sp, hc.HC_LAYOUT_COMPACT)
        check(m, sp, hc.HC_LAYOUT_COMPACT, got)
    assert hc.hc_get_device_status() == hc.HC_OK


@pytest.mark.parametrize("offset", [1, 5, 8])
def test_misaligned_mask(offset):
    sp, m, *_ = inputs.random_case(offset, 9, 777, 9, 8, 8, "f32", 0.3, neg_frac=0.2)
    check(m, sp, hc.HC_LAYOUT_DENSE, run_fused(m, sp, hc.HC_LAYOUT_DENSE, offset))


def test_out_of_range_spiral_entries_reported():
    sp, m, *_ = inputs.random_case(21, 3, 300, 9, 8, 8, "f32", 1.0)
    bad = sp.copy()
    bad[4, 2] = 300  # == V
    bad[10, 5] = -2
    got = run_fused(m, bad, hc.HC_LAYOUT_DENSE)
    assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
    fixed = bad.copy()
    fixed[4, 2] = -1
    fixed[10, 5] = -1
    check(m, bad, hc.HC_LAYOUT_DENSE, got, sp_ref=fixed)


def test_same_as_the_two_calls_then_conv():
    """The fused call feeds the rulebook conv exactly like hc_mask_compact +
    hc_conv_rulebook (same bits of the layer output)."""
    w = inputs.make_workload("layer10475_bf16")
    ly = w.layers[0]
    B, V, L = w.B, w.V, w.L
    coords, row_of, offs, count, rb = (to_torch(t) for t in run_fused(w.masks[0], w.spiral, 0))
    c2 = torch.empty_like(coords)
    r2 = torch.empty_like(row_of)
    o2 = torch.empty_like(offs)
    n2 = torch.empty_like(count)
    rb2 = torch.empty_like(rb)
    hc.hc_mask_compact(to_torch(w.masks[0]), c2, r2, o2, n2)
    hc.hc_conv_rulebook(c2, r2, n2, to_torch(w.spiral), B, V, 0, rb2)
    ys = []
    for r, n in ((rb, count), (rb2, n2)):
        y = torch.empty((B * V, ly.C_out), dtype=torch.bfloat16, device="cuda")
        hc.hc_sparse_conv_rulebook_fwd(to_torch(w.x), r, n, to_torch(ly.W), to_torch(ly.b),
                                       ly.act, y)
        ys.append(to_numpy(y)[:int(n.item())])
    assert hc.hc_get_device_status() == hc.HC_OK
    np.testing.assert_array_equal(ys[0], ys[1])
