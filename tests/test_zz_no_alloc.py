"""hc_mask_compact_static: compaction for callers that cannot allocate device
memory (for example code running while a stream is captured into a CUDA
graph, or a process whose device memory is all handed to its own pool). It
uses a fixed scratch array inside the library instead of a workspace that the
library allocates, and must give exactly what hc_mask_compact gives.

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


@pytest.mark.parametrize("B,V,density", [(7, 655, 0.1), (520, 10475, 0.05)])
def test_static_compaction_matches_hc_mask_compact(B, V, density):
    """Two calls in a row through the C-ABI, each compared with the
    allocating entry point on the same mask (bit-exact, the tolerance of
    every compaction test). The second mask differs from the first, so stale
    scratch from the first call would show up."""
    rng = np.random.default_rng(B + V)
    for call in range(2):
        m = torch.from_numpy(inputs.uniform_mask(rng, B, V, density * (1 + call))).cuda()
        ref = _buffers(B, V)
        hc.hc_mask_compact(m, *ref)
        got = _buffers(B, V)
        hc.hc_mask_compact_static(m, *got)
        assert hc.hc_get_device_status() == hc.HC_OK
        _same(got, ref)


def test_static_compaction_rejects_masks_above_the_limit():
    lib = hc.load_library()
    fake = ctypes.c_void_p(0x1000)
    V = 4096
    B = hc.HC_STATIC_MAX_MASK_BYTES // V + 1
    st = lib.hc_mask_compact_static(fake, B, V, fake, None, None, fake, None)
    assert st == hc.HC_ERR_UNSUPPORTED
    assert "limit" in hc.hc_last_error_string()
