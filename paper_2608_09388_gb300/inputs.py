"""Seeded synthetic inputs for the sparse spiral-conv operators.

This module is shared by the CPU oracle's tests and by the CUDA path's tests
and benchmark. It draws data only: mesh points, spiral neighbour tables,
contact masks, features, weights and biases. It performs none of the
operators' arithmetic (no compaction, gather, contraction, activation or
scatter), so that the oracle and the CUDA path stay independent of each other.

What the inputs stand in for. The paper measures on PROXD, GIMO and BEHAVE
with SMPL-X bodies (Sec. 4.1). None of those are available, so every input is
synthetic with the paper's workload statistics:

* a body mesh of 655 vertices (Table 4, "Original Input") and a large mesh of
  10475 vertices, both as points uniform on the unit sphere;
* a spiral of fixed length L per vertex: slot 0 is the vertex itself, then its
  L-1 nearest vertices by Euclidean distance (the spiral blocks the paper takes
  from POSA, Fig. 2 caption);
* contact masks drawn per vertex, the active fraction being the complement of
  the paper's "sparsity ratio" (Eq. 1 and Sec. 4.5: 90% sparsity, i.e. about
  66 of 655 vertices active per mask, Table 4);
* features N(0, 1), weights N(0, std = 1/sqrt(L*C_in)), bias 0.1.

Random numbers are drawn with numpy's PCG64 generator from a fixed seed per
workload, in a fixed order (mesh, masks, features, weights), so both sides of
every parity test see identical bytes.
"""
from __future__ import annotations

import functools
import math
from dataclasses import dataclass, field

import numpy as np

# ---------------------------------------------------------------------------
# dtype helpers (storage only)
# ---------------------------------------------------------------------------


def to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (round-to-nearest-even) and return the
    raw 16-bit patterns as uint16. Uses torch's conversion routine."""
    import torch

    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16).copy()


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widen raw bfloat16 bit patterns (uint16) to float32 exactly."""
    return (bits.astype(np.uint32) << 16).view(np.float32)


# ---------------------------------------------------------------------------
# mesh and spiral
# ---------------------------------------------------------------------------


def sphere_points(rng: np.random.Generator, V: int) -> np.ndarray:
    """V points uniform on the unit sphere (normalised 3-D Gaussians), fp64."""
    p = rng.standard_normal((V, 3))
    p /= np.linalg.norm(p, axis=1, keepdims=True)
    return p


def spiral_table(points: np.ndarray, L: int) -> np.ndarray:
    """Neighbour table [V, L] int32: slot 0 = the vertex itself, then its L-1
    nearest other vertices ordered by (squared distance, index).

    Squared distances are formed elementwise in fp64 (no BLAS), so the table
    is the same on every machine. Brute force over all pairs."""
    V = points.shape[0]
    if L > V:
        raise ValueError("spiral length exceeds vertex count")
    out = np.empty((V, L), dtype=np.int32)
    out[:, 0] = np.arange(V, dtype=np.int32)
    if L == 1:
        return out
    k = L - 1
    blk = 256
    for s in range(0, V, blk):
        e = min(V, s + blk)
        d = points[s:e, None, :] - points[None, :, :]
        d2 = d[..., 0] * d[..., 0] + d[..., 1] * d[..., 1] + d[..., 2] * d[..., 2]
        rows = np.arange(e - s)
        d2[rows, rows + s] = np.inf  # self is slot 0, never a neighbour
        if k < V - 1:
            cand = np.sort(np.argpartition(d2, k, axis=1)[:, : k + 1], axis=1)
        else:
            cand = np.tile(np.arange(V), (e - s, 1))
        dc = np.take_along_axis(d2, cand, axis=1)
        order = np.argsort(dc, axis=1, kind="stable")  # by distance, then index
        sel = np.take_along_axis(cand, order, axis=1)[:, :k]
        thr = np.take_along_axis(d2, sel[:, -1:], axis=1)
        # A tie at the cut could have been dropped by argpartition: redo such
        # a row with a full stable sort (a measure-zero event).
        bad = np.flatnonzero(np.count_nonzero(d2 <= thr, axis=1) != k)
        for i in bad:
            sel[i] = np.argsort(d2[i], kind="stable")[:k]
        out[s:e, 1:] = sel
    return out


# ---------------------------------------------------------------------------
# masks (the random draws of Eq. 1; the method receives them as inputs)
# ---------------------------------------------------------------------------


def uniform_mask(rng: np.random.Generator, B: int, V: int, density: float) -> np.ndarray:
    """Per-vertex Bernoulli mask, uint8 [B, V]: active iff a U(0,1) score falls
    below `density` (active fraction = 1 - sparsity ratio)."""
    u = rng.random((B, V))
    return (u < density).astype(np.uint8)


def score_mask(rng: np.random.Generator, B: int, V: int, threshold: float) -> np.ndarray:
    """Per-vertex mask, uint8 [B, V]: active iff a U(0,1) score exceeds
    `threshold` (0.9 gives the paper's 90% sparsity ratio)."""
    u = rng.random((B, V))
    return (u > threshold).astype(np.uint8)


def clustered_mask(rng: np.random.Generator, points: np.ndarray, B: int,
                   n_centres: int = 8, density: float = 0.05) -> np.ndarray:
    """Spatially clustered contact patches, uint8 [B, V].

    Per sample, `n_centres` centres are drawn uniform on the sphere; a vertex
    is active iff its geodesic distance to some centre is at most r, with r
    chosen so that each spherical cap covers density/n_centres of the sphere
    (cap area fraction (1 - cos r)/2). Overlapping caps make the realised
    density slightly lower than `density`."""
    V = points.shape[0]
    cos_r = 1.0 - 2.0 * density / n_centres
    out = np.zeros((B, V), dtype=np.uint8)
    for b in range(B):
        c = rng.standard_normal((n_centres, 3))
        c /= np.linalg.norm(c, axis=1, keepdims=True)
        dots = points @ c.T  # [V, P]; geodesic distance = arccos(dot)
        out[b] = (dots.max(axis=1) >= cos_r).astype(np.uint8)
    return out


def temporal_masks(rng: np.random.Generator, n_seq: int, T: int, V: int,
                   density0: float = 0.15, flip_frac: float = 0.02) -> np.ndarray:
    """Temporally correlated per-frame masks, uint8 [n_seq*T, V].

    Frame 0 of each sequence is Bernoulli(density0). Every later frame flips
    `flip_frac` of the previous frame's bits: half of them active->inactive and
    half inactive->active, chosen uniformly without replacement, so the density
    stays near density0 along the sequence."""
    out = np.zeros((n_seq * T, V), dtype=np.uint8)
    half = int(round(0.5 * flip_frac * V))
    for s in range(n_seq):
        m = (rng.random(V) < density0).astype(np.uint8)
        out[s * T] = m
        for t in range(1, T):
            m = m.copy()
            on = np.flatnonzero(m)
            off = np.flatnonzero(m == 0)
            a = min(half, on.size)
            d = min(half, off.size)
            if a:
                m[rng.choice(on, size=a, replace=False)] = 0
            if d:
                m[rng.choice(off, size=d, replace=False)] = 1
            out[s * T + t] = m
    return out


# ---------------------------------------------------------------------------
# tensors
# ---------------------------------------------------------------------------


def features(rng: np.random.Generator, shape, dtype: str) -> np.ndarray:
    """N(0,1) features; float32 array for 'f32', raw uint16 bits for 'bf16'."""
    x = rng.standard_normal(shape).astype(np.float32)
    return x if dtype == "f32" else to_bf16_bits(x)


def weights(rng: np.random.Generator, K: int, C_out: int, dtype: str) -> np.ndarray:
    """Weight [K, C_out] drawn N(0, std = 1/sqrt(K)), K = L*C_in."""
    w = (rng.standard_normal((K, C_out)) / math.sqrt(K)).astype(np.float32)
    return w if dtype == "f32" else to_bf16_bits(w)


def bias(C_out: int, value: float = 0.1) -> np.ndarray:
    return np.full(C_out, value, dtype=np.float32)


# ---------------------------------------------------------------------------
# the workloads
# ---------------------------------------------------------------------------

ACT_NONE, ACT_ELU, ACT_RELU = 0, 1, 2


@dataclass
class Layer:
    kind: str  # "conv" (spiral conv over the mesh) or "linear" (per-row)
    C_in: int
    C_out: int
    act: int
    W: np.ndarray  # [K, C_out], K = L*C_in for conv, C_in for linear
    b: np.ndarray  # [C_out] float32


@dataclass
class Workload:
    name: str
    dtype: str  # "f32" or "bf16"
    B: int
    V: int
    L: int
    points: np.ndarray
    spiral: np.ndarray  # [V, L] int32
    masks: list  # list of uint8 [B, V] (one entry, or one per density)
    x: np.ndarray  # dense input features [B, V, C_in] (f32 or bf16 bits)
    layers: list = field(default_factory=list)
    densities: list | None = None
    note: str = ""


SEEDS = {
    "layer655_f32": 20260,
    "encoder655_bf16": 20261,
    "layer10475_bf16": 20262,
    "sweep10475_bf16": 20263,
    "motion655_bf16": 20264,
}


@functools.lru_cache(maxsize=None)
def _mesh(seed: int, V: int, L: int):
    rng = np.random.default_rng(seed)
    pts = sphere_points(rng, V)
    return pts, spiral_table(pts, L), rng.bit_generator.state


def _rng_after_mesh(seed: int, V: int, L: int):
    pts, sp, state = _mesh(seed, V, L)
    rng = np.random.default_rng(seed)
    rng.bit_generator.state = state
    return rng, pts, sp


def _conv_stack(rng, L, chans, dtype, act=ACT_ELU):
    out = []
    for ci, co in zip(chans[:-1], chans[1:]):
        out.append(Layer("conv", ci, co, act, weights(rng, L * ci, co, dtype), bias(co)))
    return out


def make_workload(name: str, B: int | None = None) -> Workload:
    """Build one named workload. `B` overrides the batch (frames) for smaller
    test cases; the rest of the recipe is unchanged."""
    seed = SEEDS[name]
    if name == "layer655_f32":
        V, L = 655, 9
        B = 1 if B is None else B
        rng, pts, sp = _rng_after_mesh(seed, V, L)
        m = score_mask(rng, B, V, 0.9)
        x = features(rng, (B, V, 16), "f32")
        layers = _conv_stack(rng, L, [16, 64], "f32")
        return Workload(name, "f32", B, V, L, pts, sp, [m], x, layers,
                        note="single fp32 spiral-conv layer, 655-vertex sphere, ~10% active")
    if name == "encoder655_bf16":
        V, L = 655, 9
        B = 64 if B is None else B
        rng, pts, sp = _rng_after_mesh(seed, V, L)
        m = score_mask(rng, B, V, 0.9)
        x = features(rng, (B, V, 16), "bf16")
        layers = _conv_stack(rng, L, [16, 64, 64, 64, 64], "bf16")
        layers.append(Layer("linear", 64, 42, ACT_NONE, weights(rng, 64, 42, "bf16"), bias(42)))
        return Workload(name, "bf16", B, V, L, pts, sp, [m], x, layers,
                        note="4-layer bf16 sparse encoder + 64->42 linear, ~10% active")
    if name == "layer10475_bf16":
        V, L = 10475, 12
        B = 32 if B is None else B
        rng, pts, sp = _rng_after_mesh(seed, V, L)
        m = clustered_mask(rng, pts, B, 8, 0.05)
        x = features(rng, (B, V, 64), "bf16")
        layers = _conv_stack(rng, L, [64, 128], "bf16")
        return Workload(name, "bf16", B, V, L, pts, sp, [m], x, layers,
                        note="bf16 layer, 10475-vertex sphere, clustered ~5% active")
    if name == "sweep10475_bf16":
        V, L = 10475, 9
        B = 64 if B is None else B
        rng, pts, sp = _rng_after_mesh(seed, V, L)
        dens = [0.01, 0.05, 0.10, 0.25, 0.50, 1.00]
        ms = [uniform_mask(rng, B, V, d) for d in dens]
        x = features(rng, (B, V, 128), "bf16")
        layers = _conv_stack(rng, L, [128, 128], "bf16")
        return Workload(name, "bf16", B, V, L, pts, sp, ms, x, layers, densities=dens,
                        note="bf16 layer, 10475-vertex sphere, uniform masks at 1..100%")
    if name == "motion655_bf16":
        V, L = 655, 9
        n_seq, T = 4, 64
        if B is not None:
            n_seq, T = 1, B
        B = n_seq * T
        rng, pts, sp = _rng_after_mesh(seed, V, L)
        m = temporal_masks(rng, n_seq, T, V, 0.15, 0.02)
        x = features(rng, (B, V, 45), "bf16")
        layers = _conv_stack(rng, L, [45, 64, 128, 128, 64], "bf16")
        layers.append(Layer("linear", 64, 1, ACT_NONE, weights(rng, 64, 1, "bf16"), bias(1)))
        return Workload(name, "bf16", B, V, L, pts, sp, [m], x, layers,
                        note="256 frames (4 x 64) of the 655-vertex sphere, ~15% active, "
                             "2% of mask bits flipped per frame")
    raise KeyError(name)


WORKLOADS = tuple(SEEDS)


def random_case(seed: int, B: int, V: int, L: int, C_in: int, C_out: int,
                dtype: str, density: float, neg_frac: float = 0.0):
    """A small random case for shape fuzzing: random points and spiral, a
    Bernoulli mask, features, weights and bias. With `neg_frac` > 0 that
    fraction of spiral neighbour entries (slots >= 1) is replaced by -1
    ("no neighbour")."""
    rng = np.random.default_rng(seed)
    pts = sphere_points(rng, V)
    sp = spiral_table(pts, L)
    if neg_frac > 0 and L > 1:
        drop = rng.random((V, L - 1)) < neg_frac
        sp[:, 1:][drop] = -1
    m = uniform_mask(rng, B, V, density)
    x = features(rng, (B, V, C_in), dtype)
    W = weights(rng, L * C_in, C_out, dtype)
    b = (rng.standard_normal(C_out) * 0.1).astype(np.float32)
    return sp, m, x, W, b
