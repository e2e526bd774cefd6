"""GPU parity of the convolution layer followed by group normalisation and
the activation (Eqs. 5-6, 7-9, 10) through hc_sparse_conv_gn_fwd.

The oracle computes the whole chain from the mask: compaction, the Eq. 4
mapping, the convolution without activation rounded to the stored dtype,
then the group norm with its activation over each frame's rows. The GPU
side runs hc_mask_compact, hc_conv_rulebook and the fused entry point. The
bar is that of the dtype (fp32 1e-4 absolute, bf16 2e-2 * max(|r|, 1)).
Shapes cover the fused path (statistics from the tensor-core epilogue:
C_out/G = 8 .. 128) and the two-call path it falls back to."""
import os

import numpy as np
import pytest

import oracle
from paper_2608_09388_gb300 import hc, inputs

from _util import check_close, to_numpy, to_torch, widen

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


def _mask(seed, B, V, density):
    """Bernoulli mask with an empty frame, a one-row frame and a full frame
    among the others (when B allows)."""
    m = inputs.uniform_mask(np.random.default_rng(seed), B, V, density)
    if B >= 3:
        m[1] = 0
        m[2] = 0
        m[2, V // 2] = 1
    if B >= 4:
        m[3] = 1
    return m


def _case(seed, B, V, L, C_in, C_out, G, dtype, affine, act, density=0.3, mask=None):
    sp, m, x, W, b = inputs.random_case(seed, B, V, L, C_in, C_out, dtype, density)
    if mask is not None:
        m = mask
    rng = np.random.default_rng(seed + 1)
    gamma = (1.0 + 0.4 * rng.standard_normal(C_out)).astype(np.float32) if affine else None
    beta = (0.2 * rng.standard_normal(C_out)).astype(np.float32) if affine else None
    return dict(sp=sp, m=m, x=x, W=W, b=b, G=G, gamma=gamma, beta=beta, act=act, dtype=dtype)


def oracle_conv_gn(c, eps=1e-5, n_threads=1):
    coords, row_of, offs, n = oracle.mask_compact(c["m"])
    _, z = oracle.sparse_spiral_conv(c["x"], oracle.LAYOUT_DENSE, coords, row_of, c["sp"], c["W"],
                                     c["b"], oracle.ACT_NONE, n_threads=n_threads)
    y_pre, _ = oracle.sparse_group_norm(z, offs, c["G"], eps, c["gamma"], c["beta"], c["act"])
    return y_pre, n


def gpu_conv_gn(c, eps=1e-5, fused=True):
    """The layer on the GPU: compaction, mapping, then either the fused entry
    point or the convolution and the group norm as two calls."""
    B, V = c["m"].shape
    L = c["sp"].shape[1]
    cap = B * V
    C_in = c["x"].shape[-1]
    C_out = c["W"].shape[1]
    mask = to_torch(c["m"])
    coords = torch.full((cap, 2), -7, dtype=torch.int32, device="cuda")
    row_of = torch.full((B, V), -7, dtype=torch.int32, device="cuda")
    offs = torch.full((B + 1,), -7, dtype=torch.int32, device="cuda")
    count = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    hc.hc_mask_compact(mask, coords, row_of, offs, count)
    rb = torch.full((L, cap), -7, dtype=torch.int32, device="cuda")
    hc.hc_conv_rulebook(coords, row_of, count, to_torch(c["sp"]), B, V, oracle.LAYOUT_DENSE, rb)
    x = to_torch(c["x"]).reshape(cap, C_in)
    W = to_torch(c["W"])
    bias = to_torch(c["b"])
    gamma = None if c["gamma"] is None else to_torch(c["gamma"])
    beta = None if c["beta"] is None else to_torch(c["beta"])
    y = torch.full((cap, C_out), float("nan"), dtype=x.dtype, device="cuda")
    if fused:
        hc.hc_sparse_conv_gn_fwd(x, rb, count, W, bias, coords, offs, c["G"], eps, gamma, beta,
                                 c["act"], y)
    else:
        hc.hc_sparse_conv_rulebook_fwd(x, rb, count, W, bias, oracle.ACT_NONE, y)
        hc.hc_sparse_group_norm_fwd(y, offs, c["G"], eps, gamma, beta, c["act"], y)
    assert hc.hc_get_device_status() == hc.HC_OK
    return to_numpy(y), int(count.item())


def check_case(c, what, eps=1e-5):
    y_pre, n = oracle_conv_gn(c, eps)
    got, n_gpu = gpu_conv_gn(c, eps)
    assert n_gpu == n
    check_close(got[:n], y_pre[:n], what)
    return got, n


# Fused: bf16, C_out/G a multiple of 8 dividing the tile (64 or 128 channels).
FUSED = [(3, 200, 9, 16, 64, 8),     # 8 channels per group, 4 groups per 32-column chunk
         (2, 333, 12, 64, 128, 8),   # 16 per group (the bench layer's shape)
         (4, 150, 9, 32, 128, 4),    # 32 per group
         (3, 300, 9, 16, 128, 2),    # 64 per group: merged over two chunks
         (3, 300, 9, 16, 128, 1),    # layer norm over 128 channels
         (4, 250, 9, 16, 64, 1),     # layer norm over the 64-channel tile
         (5, 200, 5, 8, 32, 4),      # C_out below the 64-channel tile
         (3, 180, 7, 16, 256, 8),    # two column tiles
         (3, 200, 9, 45, 64, 8),     # C_in not a multiple of 8: channel-padded x and W
         (2, 300, 9, 3, 128, 4)]     # C_in below 8
# Two calls: fp32, or a group layout the epilogue does not take.
UNFUSED = [(3, 200, 9, 16, 64, 16),  # 4 channels per group
           (3, 200, 9, 16, 48, 2),   # 24 per group
           (2, 200, 9, 16, 256, 1),  # 256 per group, wider than a tile
           (3, 200, 9, 16, 24, 3),   # C_out/8 not a power of two
           (3, 200, 9, 45, 48, 2)]   # padded channels, then the group norm's own workspace


@pytest.mark.parametrize("shape", FUSED + UNFUSED)
@pytest.mark.parametrize("affine,act", [(False, oracle.ACT_NONE), (True, oracle.ACT_ELU),
                                        (True, oracle.ACT_RELU)])
def test_conv_gn_bf16(shape, affine, act):
    B, V, L, C_in, C_out, G = shape
    c = _case(sum(shape) + act, B, V, L, C_in, C_out, G, "bf16", affine, act,
              mask=_mask(sum(shape), B, V, 0.3))
    check_case(c, f"conv+gn bf16 {shape} act={act}")


@pytest.mark.parametrize("shape", [(3, 200, 9, 16, 64, 8), (2, 150, 5, 12, 20, 5)])
def test_conv_gn_f32(shape):
    B, V, L, C_in, C_out, G = shape
    c = _case(sum(shape), B, V, L, C_in, C_out, G, "f32", True, oracle.ACT_ELU,
              mask=_mask(sum(shape), B, V, 0.4))
    check_case(c, f"conv+gn f32 {shape}")


@pytest.mark.parametrize("G", [8, 1])
def test_conv_gn_many_tiny_frames(G):
    """Frames of a few rows each: a 32-row block holds several frames, so
    one warp writes a partial for each of them."""
    B, V = 300, 24
    m = inputs.uniform_mask(np.random.default_rng(4), B, V, 0.15)
    c = _case(41, B, V, 9, 16, 128, G, "bf16", True, oracle.ACT_ELU, mask=m)
    check_case(c, f"tiny frames G={G}")


@pytest.mark.parametrize("G", [8, 2])
def test_conv_gn_frames_at_block_edges(G):
    """Frames of exactly 32 or 64 rows (every 32-row block inside one frame),
    one row more or less (blocks shared by two frames), empty and single-row
    frames: the block partials and the per-row partials of shared blocks."""
    sizes = [64, 32, 33, 31, 0, 96, 1, 63, 65, 32]
    B, V = len(sizes), 150
    rng = np.random.default_rng(12)
    m = np.zeros((B, V), np.uint8)
    for b, k in enumerate(sizes):
        m[b, rng.choice(V, size=k, replace=False)] = 1
    c = _case(46, B, V, 9, 16, 128, G, "bf16", True, oracle.ACT_ELU, mask=m)
    check_case(c, f"block edges G={G}")


def test_conv_gn_large_frame_and_eps():
    """One frame spread over hundreds of 32-row blocks, eps from 0 to large."""
    B, V = 2, 12000
    m = inputs.uniform_mask(np.random.default_rng(6), B, V, 0.7)
    c = _case(42, B, V, 9, 16, 64, 4, "bf16", False, oracle.ACT_NONE, mask=m)
    for eps in (0.0, 1e-5, 3.0):
        check_case(c, f"large frame eps={eps}", eps=eps)


def test_conv_gn_empty_mask():
    c = _case(43, 3, 100, 9, 16, 64, 8, "bf16", True, oracle.ACT_ELU,
              mask=np.zeros((3, 100), np.uint8))
    got, n = gpu_conv_gn(c)
    assert n == 0
    assert np.isnan(widen(got)).all()


def test_conv_gn_matches_two_calls():
    """The fused statistics against the two-call path on the same GPU
    convolution output: both normalise the same stored values, so they
    agree to a few bf16 rounding steps of the output."""
    c = _case(44, 6, 700, 12, 64, 128, 8, "bf16", True, oracle.ACT_ELU,
              mask=_mask(44, 6, 700, 0.25))
    a, n = gpu_conv_gn(c, fused=True)
    b, _ = gpu_conv_gn(c, fused=False)
    wa, wb = widen(a[:n]), widen(b[:n])
    assert np.abs(wa - wb).max() <= 2 ** -6 * max(1.0, np.abs(wb).max())


def test_conv_gn_full_size_layer():
    """The 10475-vertex bf16 layer (32 clustered frames, L = 12, 64 -> 128
    channels), G = 8, with affine terms and ELU."""
    w = inputs.make_workload("layer10475_bf16")
    ly = w.layers[0]
    rng = np.random.default_rng(8)
    c = dict(sp=w.spiral, m=w.masks[0], x=w.x, W=ly.W, b=ly.b, G=8,
             gamma=(1.0 + 0.3 * rng.standard_normal(ly.C_out)).astype(np.float32),
             beta=(0.1 * rng.standard_normal(ly.C_out)).astype(np.float32), act=oracle.ACT_ELU,
             dtype="bf16")
    y_pre, n = oracle_conv_gn(c, n_threads=NCPU)
    got, n_gpu = gpu_conv_gn(c)
    assert n_gpu == n
    check_close(got[:n], y_pre[:n], "conv+gn full size")


def test_conv_gn_frame_table_mismatch_reported():
    """A frame table that does not end at the row count is reported
    (HC_ERR_INVALID_INDEX) on the fused path."""
    c = _case(45, 3, 200, 9, 16, 64, 8, "bf16", False, oracle.ACT_NONE)
    B, V = c["m"].shape
    cap = B * V
    L = c["sp"].shape[1]
    coords = torch.zeros((cap, 2), dtype=torch.int32, device="cuda")
    row_of = torch.zeros((B, V), dtype=torch.int32, device="cuda")
    offs = torch.zeros((B + 1,), dtype=torch.int32, device="cuda")
    count = torch.zeros((1,), dtype=torch.int32, device="cuda")
    hc.hc_mask_compact(to_torch(c["m"]), coords, row_of, offs, count)
    rb = torch.empty((L, cap), dtype=torch.int32, device="cuda")
    hc.hc_conv_rulebook(coords, row_of, count, to_torch(c["sp"]), B, V, oracle.LAYOUT_DENSE, rb)
    assert int(count.item()) > 2
    offs[B] -= 1
    y = torch.empty((cap, 64), dtype=torch.bfloat16, device="cuda")
    hc.hc_sparse_conv_gn_fwd(to_torch(c["x"]).reshape(cap, 16), rb, count, to_torch(c["W"]),
                             to_torch(c["b"]), coords, offs, 8, 1e-5, None, None, 0, y)
    assert hc.hc_get_device_status() == hc.HC_ERR_INVALID_INDEX
    assert hc.hc_get_device_status() == hc.HC_OK
