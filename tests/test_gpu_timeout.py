"""The bounded-wait failure path of the pipelined kernels (tensor-core conv,
mask score, weight gradient): with the pipeline-wait limit lowered far below
the time their first pipeline stages take, a call gives up instead of
finishing, the device status reads HC_ERR_TIMEOUT, and once the limit is
back at its default the same call is correct again (the unwind freed the
CTA's tensor memory and let every copy and MMA it had issued finish).

No kernel is made to hang: every wait still ends, only sooner than the work
it waits for. The unwind's own waits keep the full limit."""
import os

import numpy as np
import pytest

import oracle
from paper_2608_09388_gb300 import hc, inputs

from _util import check_close, to_numpy, to_torch

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
NCPU = len(os.sched_getaffinity(0))

# Far below the few microseconds any of these kernels needs before its first
# accumulator is complete, so some role of every CTA gives up.
SHORT_LIMIT_NS = 500


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_09388_gb300 import build
    build.build()
    hc.load_library()
    assert hc.hc_get_device_status() == hc.HC_OK


@pytest.fixture
def short_waits():
    """Lower the wait limit for the body of a test; the default is restored
    (and any status the test left behind cleared) afterwards."""
    def lower():
        hc.hc_test_set_option(hc.HC_TEST_WAIT_LIMIT_NS, SHORT_LIMIT_NS)

    def restore():
        hc.hc_test_set_option(hc.HC_TEST_WAIT_LIMIT_NS, 0)

    yield lower, restore
    restore()
    hc.hc_get_device_status()


def _conv_case():
    sp, m, x, W, b = inputs.random_case(7001, 16, 4000, 9, 128, 128, "bf16", 1.0)
    c, r, _, n = oracle.mask_compact(m)
    B, V = m.shape
    L = sp.shape[1]
    t = {k: to_torch(v) for k, v in (("m", m), ("x", x), ("sp", sp), ("W", W), ("b", b))}
    coords = torch.empty((B * V, 2), dtype=torch.int32, device="cuda")
    row_of = torch.empty((B, V), dtype=torch.int32, device="cuda")
    offs = torch.empty((B + 1,), dtype=torch.int32, device="cuda")
    count = torch.empty((1,), dtype=torch.int32, device="cuda")
    rb = torch.empty((L, B * V), dtype=torch.int32, device="cuda")
    hc.hc_mask_compact_rulebook(t["m"], t["sp"], hc.HC_LAYOUT_DENSE, coords, row_of, offs, count,
                                rb)
    assert hc.hc_get_device_status() == hc.HC_OK
    return (sp, m, x, W, b, c, r, n), t, rb, count


def test_conv_wait_timeout_reported_then_correct(short_waits):
    lower, restore = short_waits
    (sp, m, x, W, b, c, r, n), t, rb, count = _conv_case()
    y = torch.full((n, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    lower()
    hc.hc_sparse_conv_rulebook_fwd(t["x"], rb, count, t["W"], t["b"], hc.HC_ACT_ELU, y)
    assert hc.hc_get_device_status() == hc.HC_ERR_TIMEOUT
    restore()
    assert hc.hc_get_device_status() == hc.HC_OK
    hc.hc_sparse_conv_rulebook_fwd(t["x"], rb, count, t["W"], t["b"], hc.HC_ACT_ELU, y)
    assert hc.hc_get_device_status() == hc.HC_OK
    rows = np.concatenate([np.arange(0, n, 97), [n - 1]])
    y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, c, r, sp, W, b, oracle.ACT_ELU,
                                         rows=rows, n_threads=NCPU)
    check_close(to_numpy(y)[rows], y_pre, "conv after a timed-out call")


def test_mask_score_wait_timeout_reported_then_correct(short_waits):
    lower, restore = short_waits
    rng = np.random.default_rng(7002)
    K, N, D = 10, 4096, 64
    O = inputs.features(rng, (K, N, D), "bf16")
    alpha = rng.standard_normal(K).astype(np.float32)
    Ot, at = to_torch(O), to_torch(alpha)
    out = torch.empty(K, dtype=torch.float32, device="cuda")
    sim = torch.empty((K, K), dtype=torch.float32, device="cuda")
    lower()
    hc.hc_mask_score_update(Ot, at, out, sim)
    assert hc.hc_get_device_status() == hc.HC_ERR_TIMEOUT
    restore()
    hc.hc_mask_score_update(Ot, at, out, sim)
    assert hc.hc_get_device_status() == hc.HC_OK
    a_ref, s_ref, _ = oracle.mask_score(O, alpha, n_threads=NCPU)
    np.testing.assert_allclose(to_numpy(out), a_ref, atol=1e-4, rtol=0)
    np.testing.assert_allclose(to_numpy(sim), s_ref, atol=1e-4, rtol=0)


def test_weight_gradient_wait_timeout_reported_then_correct(short_waits):
    lower, restore = short_waits
    (sp, m, x, W, b, c, r, n), t, rb, count = _conv_case()
    L, C_in, C_out = sp.shape[1], 128, 128
    y = torch.empty((n, C_out), dtype=torch.bfloat16, device="cuda")
    hc.hc_sparse_conv_rulebook_fwd(t["x"], rb, count, t["W"], t["b"], hc.HC_ACT_ELU, y)
    dy = torch.randn((n, C_out), generator=torch.Generator("cuda").manual_seed(3),
                     device="cuda").to(torch.bfloat16)
    dW = torch.empty((L * C_in, C_out), dtype=torch.float32, device="cuda")
    db = torch.empty((C_out,), dtype=torch.float32, device="cuda")
    assert hc.hc_get_device_status() == hc.HC_OK

    def bwd():
        hc.hc_sparse_conv_rulebook_bwd(t["x"], rb, count, t["W"], y, dy, hc.HC_ACT_ELU,
                                       None, None, None, dW, db)

    lower()
    bwd()
    assert hc.hc_get_device_status() == hc.HC_ERR_TIMEOUT
    restore()
    dW.fill_(float("nan"))
    bwd()
    assert hc.hc_get_device_status() == hc.HC_OK
    assert torch.isfinite(dW).all() and torch.isfinite(db).all()
    # against a second call under the default limit (the kernel's split
    # order is fixed, so the result repeats bit for bit)
    dW2 = dW.clone()
    bwd()
    assert torch.equal(dW, dW2)
