"""Helpers shared by the tests: moving seeded numpy inputs to torch, the
tolerance checks, and row sampling for full-size cases."""
import numpy as np

F32_ABS_TOL = 1e-4   # fp32 path: max |gpu - oracle_fp64| over all elements
BF16_REL_TOL = 2e-2  # bf16 path: |gpu - r| <= 2e-2 * max(|r|, 1), r = oracle fp64 before rounding


def to_torch(a, device="cuda"):
    """numpy -> torch; uint16 arrays are bf16 bit patterns."""
    import torch
    if a.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(device)
    return torch.from_numpy(np.ascontiguousarray(a)).to(device)


def to_numpy(t):
    """torch -> numpy; bf16 tensors come back as uint16 bit patterns."""
    import torch
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def widen(a):
    """float32 or bf16 bits -> float64 values."""
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def check_close(got, y_pre, what=""):
    """Compare a GPU result (float32 array or bf16 bits) with the oracle's fp64
    value before rounding, under the tolerance of its dtype."""
    g = widen(got)
    assert g.shape == y_pre.shape, (what, g.shape, y_pre.shape)
    if g.size == 0:
        return
    assert np.isfinite(g).all(), f"{what}: non-finite output"
    if got.dtype == np.uint16:
        err = np.abs(g - y_pre) / np.maximum(np.abs(y_pre), 1.0)
        worst = np.unravel_index(np.argmax(err), err.shape)
        assert err.max() <= BF16_REL_TOL, (
            f"{what}: bf16 rel err {err.max():.3e} at {worst}: gpu {g[worst]} oracle {y_pre[worst]}")
    else:
        err = np.abs(g - y_pre)
        worst = np.unravel_index(np.argmax(err), err.shape)
        assert err.max() <= F32_ABS_TOL, (
            f"{what}: f32 abs err {err.max():.3e} at {worst}: gpu {g[worst]} oracle {y_pre[worst]}")


def sample_rows(n, k, seed=0, tile=128):
    """Up to k row indices of [0, n): the first and last rows, rows around
    every few tile boundaries, and a seeded uniform sample."""
    if n <= k:
        return np.arange(n, dtype=np.int64)
    rng = np.random.default_rng(seed)
    s = set(range(min(n, 64))) | set(range(max(0, n - 64), n))
    for b in range(tile, n, tile * max(1, (n // tile) // 16)):
        s.update(range(b - 2, min(n, b + 2)))
    s.update(rng.choice(n, size=max(0, k - len(s)), replace=False).tolist())
    return np.array(sorted(s)[: max(k, len(s))], dtype=np.int64)
