"""hc_mask_compact_static: the mask compaction for callers that cannot
allocate device memory while they compact, such as a process that gives all
of its device memory to its own pool up front and must not allocate behind
that pool's back. It uses a fixed scratch array inside the library instead
of the workspace hc_mask_compact allocates per (device, stream), and must
give exactly what hc_mask_compact gives.

This file is collected last on purpose, so that a run stopping at the first
failure has already run every other test. It passes on its own in a fresh
process as well as after the other tests."""
import ctypes

import numpy as np
import pytest

from paper_2608_09388_gb300 import hc, inputs

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_09388_gb300 import build
    build.build()
    hc.load_library()


def _buffers(B, V):
    return (torch.full((max(B * V, 1), 2), -7, dtype=torch.int32, device="cuda"),
            torch.full((B, V), -7, dtype=torch.int32, device="cuda"),
            torch.full((B + 1,), -7, dtype=torch.int32, device="cuda"),
            torch.full((1,), -7, dtype=torch.int32, device="cuda"))


def _same(a, b):
    n = int(a[3].item())
    assert n == int(b[3].item())
    assert torch.equal(a[0][:n], b[0][:n])
    assert torch.equal(a[1], b[1])
    assert torch.equal(a[2], b[2])


# (7, 655): two tiles; (520, 10475): past 1024 tiles (the pre-scanned path);
# (4096, 4096): exactly HC_STATIC_MAX_MASK_BYTES, every int32 of the scratch
# array in use; (0, 655) and (3, 0): nothing to compact.
@pytest.mark.parametrize("B,V,density", [(7, 655, 0.1), (520, 10475, 0.05), (4096, 4096, 0.01),
                                         (0, 655, 0.1), (3, 0, 0.1)])
def test_static_compaction_matches_hc_mask_compact(B, V, density):
    """Two calls in a row through the C-ABI, each compared with the
    allocating entry point on the same mask (bit-exact, the tolerance of
    every compaction test). The second mask differs from the first, so stale
    scratch from the first call would show up."""
    assert B * V <= hc.HC_STATIC_MAX_MASK_BYTES
    rng = np.random.default_rng(B + V)
    for call in range(2):
        m = torch.from_numpy(inputs.uniform_mask(rng, B, V, density * (1 + call))).cuda()
        ref = _buffers(B, V)
        hc.hc_mask_compact(m, *ref)
        got = _buffers(B, V)
        hc.hc_mask_compact_static(m, *got)
        assert hc.hc_get_device_status() == hc.HC_OK
        _same(got, ref)


def test_static_compaction_allocates_nothing():
    """After a first call on the device (which looks up the scratch array's
    address), calls on a stream the library has never seen leave the
    device's free memory unchanged, and still succeed once device memory is
    exhausted: a workspace allocation (hc_mask_compact's first call on a new
    stream) would have to take memory in both cases."""
    B, V = 64, 10475
    rng = np.random.default_rng(3)
    masks = [torch.from_numpy(inputs.uniform_mask(rng, B, V, d)).cuda() for d in (0.1, 0.3)]
    refs = []
    for m in masks:
        ref = _buffers(B, V)
        hc.hc_mask_compact(m, *ref)
        refs.append(ref)
    got = [_buffers(B, V) for _ in masks]
    hc.hc_mask_compact_static(masks[0], *got[0])  # set-up call (default stream)
    torch.cuda.synchronize()
    fresh = torch.cuda.Stream()
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    hc.hc_mask_compact_static(masks[1], *got[1], stream=fresh)
    fresh.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    _same(got[1], refs[1])

    # device memory exhausted: hold blocks until the allocator refuses more
    # (nothing below allocates until they are released; the comparisons,
    # which do, come after)
    other = torch.cuda.Stream()
    for out in got:
        for t in out:
            t.fill_(-7)
    torch.cuda.synchronize()
    held = []
    block = max(torch.cuda.mem_get_info()[0] - (256 << 20), 2 << 20)
    while block >= (2 << 20):
        try:
            held.append(torch.empty(block, dtype=torch.uint8, device="cuda"))
        except torch.cuda.OutOfMemoryError:
            block //= 2
    try:
        for m, out in zip(masks, got):
            hc.hc_mask_compact_static(m, *out, stream=other)
        other.synchronize()
    finally:
        del held
        torch.cuda.empty_cache()
    for out, ref in zip(got, refs):
        _same(out, ref)
    assert hc.hc_get_device_status() == hc.HC_OK


def test_static_compaction_rejects_masks_above_the_limit():
    lib = hc.load_library()
    fake = ctypes.c_void_p(0x1000)
    V = 4096
    B = hc.HC_STATIC_MAX_MASK_BYTES // V + 1
    st = lib.hc_mask_compact_static(fake, B, V, fake, None, None, fake, None)
    assert st == hc.HC_ERR_UNSUPPORTED
    assert "limit" in hc.hc_last_error_string()
