"""CPU oracle for the sparse contact operators (test infrastructure).

TEST INFRASTRUCTURE ONLY. Only the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may import this package; the product path never
does. It shares no code with the CUDA library: the arithmetic lives in plain C
(``hc_oracle.c``, fp64 accumulation) and this module only marshals numpy
arrays into it and chains layers.

Functions and the passages they follow:

* ``mask_compact``         decomposition into coordinates C' (Eq. 2) and the
                           inverse map idx() (Eq. 4)
* ``conv_rulebook``        the indexing matrix of Eq. 4 (tap -> input row)
* ``sparse_spiral_conv``   sparse convolution on the spiral neighbourhood
                           (Eqs. 4-5), bias (Eq. 6) and activation (Eq. 10)
* ``dense_spiral_conv``    the dense layer the sparse one replaces (Sec. 3.2)
* ``sparse_linear``        linear layer on compact rows (Eq. 6)
* ``sparse_group_norm``    group normalisation over each frame's active rows
                           (Eqs. 7-9)
* ``scatter_dense``        compact rows back to a dense tensor (inverse of Eq. 2)
* ``mask_score``           the mask-score update of Eq. 3
* ``select_topk``          the kappa highest-scoring masks kept at inference
                           (Sec. 3.1, Sparse Mask Selection)
* ``kappa_masks``          every kept mask applied to every sample (Eq. 1)
* ``gather_rows``          the feature matrix S' of Eq. 2
* ``sparse_conv_bwd``      gradients of the sparse convolution with respect
                           to input rows, weight and bias (chain rule on
                           Eqs. 4-5, 6, 10, through the Eq. 4 mapping)
* ``encoder``              a stack of sparse layers: coordinates fixed once by
                           the mask (Eqs. 5, 6, 10 keep C'), each layer's output
                           stored in the layer dtype before the next reads it
* ``bf16_round``           fp64 -> bf16 storage rounding

The shared library is compiled from ``hc_oracle.c`` with gcc on first use (or
by ``build()``) into ``oracle/_build``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hc_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libhc_oracle.so")
_lock = threading.Lock()
_lib = None

F32, BF16 = 0, 1
ACT_NONE, ACT_ELU, ACT_RELU = 0, 1, 2
LAYOUT_DENSE, LAYOUT_COMPACT = 0, 1


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP) unless an up-to-date build exists."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
           "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            I64 = ctypes.c_int64
            I = ctypes.c_int
            lib.hco_mask_compact.argtypes = [P, I64, I64, P, P, P]
            lib.hco_mask_compact.restype = I64
            lib.hco_sparse_spiral_conv.argtypes = [P, I, I, P, P, P, I64, P, I64, I64, I, I, I,
                                                   P, P, I, P, P, I]
            lib.hco_sparse_spiral_conv.restype = None
            lib.hco_dense_spiral_conv.argtypes = [P, I, P, I64, P, I64, I64, I, I, I, P, P, I,
                                                  P, P, I]
            lib.hco_dense_spiral_conv.restype = None
            lib.hco_sparse_linear.argtypes = [P, I, P, I64, I, I, P, P, I, P, P, I]
            lib.hco_sparse_linear.restype = None
            lib.hco_scatter_dense.argtypes = [P, I, P, I64, I64, I64, I, I, P]
            lib.hco_scatter_dense.restype = None
            lib.hco_sparse_group_norm.argtypes = [P, I, P, I64, I, I, ctypes.c_double, P, P, I,
                                                  P, P]
            lib.hco_sparse_group_norm.restype = None
            lib.hco_conv_rulebook.argtypes = [P, P, I64, P, I64, I, I, I64, P]
            lib.hco_conv_rulebook.restype = None
            lib.hco_mask_score.argtypes = [P, I, I64, I64, I64, P, P, P, P, I]
            lib.hco_mask_score.restype = None
            lib.hco_select_topk.argtypes = [P, I64, I64, P]
            lib.hco_select_topk.restype = None
            lib.hco_kappa_masks.argtypes = [P, I64, P, I64, I64, P]
            lib.hco_kappa_masks.restype = None
            lib.hco_gather_rows.argtypes = [P, I, I64, I, P, I64, I64, P]
            lib.hco_gather_rows.restype = None
            lib.hco_sparse_conv_bwd.argtypes = [P, I, I64, P, I64, I64, I, I, I, P, P, P, I, P,
                                                P, P]
            lib.hco_sparse_conv_bwd.restype = None
            lib.hco_bf16_round.argtypes = [ctypes.c_double]
            lib.hco_bf16_round.restype = ctypes.c_uint16
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _dtype_code(x: np.ndarray) -> int:
    if x.dtype == np.float32:
        return F32
    if x.dtype == np.uint16:
        return BF16
    raise TypeError(f"oracle takes float32 or bf16 bits (uint16), got {x.dtype}")


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def bf16_round(v: float) -> int:
    """fp64 -> bf16 (round to nearest even); returns the 16-bit pattern."""
    return int(_load().hco_bf16_round(float(v)))


def mask_compact(mask: np.ndarray):
    """Eq. 2 decomposition of a [B, V] mask.

    Returns (coords int32 [N', 2] of (b, v) ascending, row_of int32 [B, V]
    (position in coords or -1), offsets int32 [B+1], N')."""
    mask = _c(mask, np.uint8)
    B, V = mask.shape
    coords = np.empty((max(B * V, 1), 2), dtype=np.int32)
    row_of = np.empty((B, V), dtype=np.int32)
    offsets = np.empty(B + 1, dtype=np.int32)
    n = _load().hco_mask_compact(_ptr(mask), B, V, _ptr(coords), _ptr(row_of), _ptr(offsets))
    return coords[:n].copy(), row_of, offsets, int(n)


def conv_rulebook(coords, row_of, spiral, x_layout, stride=None):
    """Eq. 4 mapping: int32 [L, stride] with entry (l, n) = the input row read
    by slot l of output row n (dense row b*V+u, or compact row), -1 if absent.
    Columns n >= N' are -1."""
    coords = _c(coords, np.int32)
    row_of = _c(row_of, np.int32)
    spiral = _c(spiral, np.int32)
    B, V = row_of.shape
    L = spiral.shape[1]
    n = coords.shape[0]
    stride = B * V if stride is None else stride
    rb = np.full((L, stride), -1, dtype=np.int32)
    _load().hco_conv_rulebook(_ptr(coords), _ptr(row_of), n, _ptr(spiral), V, L, x_layout, stride,
                              _ptr(rb))
    return rb


def _rows_arg(rows, n_default):
    if rows is None:
        return None, n_default
    rows = _c(rows, np.int64)
    return rows, rows.shape[0]


def sparse_spiral_conv(x, x_layout, coords, row_of, spiral, W, bias, act, rows=None,
                       n_threads=1):
    """Sparse spiral conv (Eqs. 4-5, 6, 10) at the compact rows `rows`
    (default: all of coords). x: dense [B, V, C_in] (x_layout=LAYOUT_DENSE) or
    compact [N', C_in]; float32 or bf16 bits. Returns (y_pre fp64, y in the
    input dtype), both [n_rows, C_out]."""
    dt = _dtype_code(x)
    x = np.ascontiguousarray(x)
    W = _c(W, x.dtype)
    coords = _c(coords, np.int32)
    row_of = _c(row_of, np.int32)
    spiral = _c(spiral, np.int32)
    B, V = row_of.shape
    L = spiral.shape[1]
    C_in = x.shape[-1]
    C_out = W.shape[1]
    assert W.shape[0] == L * C_in
    rows, n = _rows_arg(rows, coords.shape[0])
    bias = None if bias is None else _c(bias, np.float32)
    y_pre = np.empty((n, C_out), dtype=np.float64)
    y = np.empty((n, C_out), dtype=x.dtype)
    _load().hco_sparse_spiral_conv(_ptr(x), x_layout, dt, _ptr(coords), _ptr(row_of), _ptr(rows),
                                   n, _ptr(spiral), B, V, L, C_in, C_out, _ptr(W), _ptr(bias), act,
                                   _ptr(y_pre), _ptr(y), int(n_threads))
    return y_pre, y


def dense_spiral_conv(x, spiral, W, bias, act, rows=None, n_threads=1):
    """Dense spiral conv over every (b, v) of x [B, V, C_in]. Row r of the
    output is (b, v) = divmod(r, V). Returns (y_pre fp64, y) [n_rows, C_out]."""
    dt = _dtype_code(x)
    x = np.ascontiguousarray(x)
    W = _c(W, x.dtype)
    spiral = _c(spiral, np.int32)
    B, V, C_in = x.shape
    L = spiral.shape[1]
    C_out = W.shape[1]
    assert W.shape[0] == L * C_in
    rows, n = _rows_arg(rows, B * V)
    bias = None if bias is None else _c(bias, np.float32)
    y_pre = np.empty((n, C_out), dtype=np.float64)
    y = np.empty((n, C_out), dtype=x.dtype)
    _load().hco_dense_spiral_conv(_ptr(x), dt, _ptr(rows), n, _ptr(spiral), B, V, L, C_in, C_out,
                                  _ptr(W), _ptr(bias), act, _ptr(y_pre), _ptr(y), int(n_threads))
    return y_pre, y


def sparse_linear(x, W, bias, act, rows=None, n_threads=1):
    """Eq. 6 on compact rows x [N', C_in]. Returns (y_pre fp64, y) [n_rows, C_out]."""
    dt = _dtype_code(x)
    x = np.ascontiguousarray(x)
    W = _c(W, x.dtype)
    C_in = x.shape[1]
    C_out = W.shape[1]
    assert W.shape[0] == C_in
    rows, n = _rows_arg(rows, x.shape[0])
    bias = None if bias is None else _c(bias, np.float32)
    y_pre = np.empty((n, C_out), dtype=np.float64)
    y = np.empty((n, C_out), dtype=x.dtype)
    _load().hco_sparse_linear(_ptr(x), dt, _ptr(rows), n, C_in, C_out, _ptr(W), _ptr(bias), act,
                              _ptr(y_pre), _ptr(y), int(n_threads))
    return y_pre, y


def sparse_group_norm(x, offsets, G, eps=1e-5, gamma=None, beta=None, act=ACT_NONE):
    """Eqs. 7-9 on compact rows x [N', C] with frame offsets [B+1]: returns
    (y_pre fp64, y in the input dtype), both [N', C]; rows outside every
    frame's range are left as NaN / zero."""
    dt = _dtype_code(x)
    x = np.ascontiguousarray(x)
    offsets = _c(offsets, np.int32)
    B = offsets.shape[0] - 1
    C = x.shape[1]
    assert C % G == 0
    gamma = None if gamma is None else _c(gamma, np.float32)
    beta = None if beta is None else _c(beta, np.float32)
    y_pre = np.full(x.shape, np.nan, dtype=np.float64)
    y = np.zeros_like(x)
    _load().hco_sparse_group_norm(_ptr(x), dt, _ptr(offsets), B, C, G, float(eps), _ptr(gamma),
                                  _ptr(beta), act, _ptr(y_pre), _ptr(y))
    return y_pre, y


def scatter_dense(y, coords, B, V, zero_fill, out=None):
    """Compact rows y [N', C] back to dense [B, V, C] at coords. Without
    zero_fill, rows not listed keep the contents of `out` (zeros if None)."""
    y = np.ascontiguousarray(y)
    coords = _c(coords, np.int32)
    C = y.shape[1]
    if out is None:
        out = np.zeros((B, V, C), dtype=y.dtype)
    else:
        out = np.ascontiguousarray(out).copy()
    _load().hco_scatter_dense(_ptr(y), y.dtype.itemsize, _ptr(coords), coords.shape[0], B, V, C,
                              int(zero_fill), _ptr(out))
    return out


def encoder(x_dense, mask, spiral, layers, n_threads=1):
    """A stack of sparse layers on one mask. The mask is decomposed once
    (Eq. 2); conv layers keep the centre coordinates (Eq. 5), linear and
    activation layers keep C' (Eqs. 6, 10), so every layer runs on the same
    compact row list. The first conv reads the dense input at active rows;
    later layers read the previous layer's compact output, stored in the
    layer dtype. `layers` items have .kind ('conv'|'linear'), .W, .b, .act.
    Returns (coords, row_of, offsets, n, [(y_pre, y) per layer])."""
    coords, row_of, offsets, n = mask_compact(mask)
    outs = []
    h = x_dense
    layout = LAYOUT_DENSE
    for ly in layers:
        if ly.kind == "conv":
            y_pre, y = sparse_spiral_conv(h, layout, coords, row_of, spiral, ly.W, ly.b, ly.act,
                                          n_threads=n_threads)
        else:
            if layout != LAYOUT_COMPACT:
                raise ValueError("a linear layer needs compact input")
            y_pre, y = sparse_linear(h, ly.W, ly.b, ly.act, n_threads=n_threads)
        outs.append((y_pre, y))
        h = y
        layout = LAYOUT_COMPACT
    return coords, row_of, offsets, n, outs


def mask_score(O, alpha, n_threads=1):
    """Eq. 3 on per-mask outputs O [K, N, D] (float32 or bf16 bits) and
    scores alpha [K]: returns (alpha_next fp64 [K], sim fp64 [K, K],
    S fp64 [K, K] with S[i, k] = ||O_i^T O_k||_F^2)."""
    O = np.ascontiguousarray(O)
    dt = _dtype_code(O)
    K, N, D = O.shape
    a_in = _c(alpha, np.float64)
    a_out = np.empty(K, dtype=np.float64)
    sim = np.empty((K, K), dtype=np.float64)
    S = np.empty((K, K), dtype=np.float64)
    _load().hco_mask_score(_ptr(O), dt, K, N, D, _ptr(a_in), _ptr(a_out), _ptr(sim), _ptr(S),
                           n_threads)
    return a_out, sim, S


def select_topk(alpha, kappa):
    """Indices of the kappa highest fp32 scores, highest first, ties by index."""
    alpha = _c(alpha, np.float32)
    sel = np.empty(kappa, dtype=np.int32)
    _load().hco_select_topk(_ptr(alpha), alpha.shape[0], kappa, _ptr(sel))
    return sel


def kappa_masks(masks, selected, B):
    """[B * kappa, V] frame masks: frame b * kappa + j = masks[selected[j]]."""
    masks = _c(masks, np.uint8)
    selected = _c(selected, np.int32)
    K, V = masks.shape
    kappa = selected.shape[0]
    out = np.empty((B * kappa, V), dtype=np.uint8)
    _load().hco_kappa_masks(_ptr(masks), V, _ptr(selected), kappa, B, _ptr(out))
    return out


def gather_rows(x, coords, frames_per_sample=1):
    """S' of Eq. 2: rows of the dense input x [B_in, V, C] at coords (f, v),
    frame f reading sample f // frames_per_sample."""
    x = np.ascontiguousarray(x)
    coords = _c(coords, np.int32)
    _, V, C = x.shape
    n = coords.shape[0]
    y = np.empty((n, C), dtype=x.dtype)
    _load().hco_gather_rows(_ptr(x), x.dtype.itemsize, V, C, _ptr(coords), n,
                            frames_per_sample, _ptr(y))
    return y


def sparse_conv_bwd(x, rulebook, W, y, dy, act):
    """Gradients of the sparse conv through the Eq. 4 mapping rulebook
    [L, stride] (column n < len(dy) = output row n). x: input rows
    [x_rows, C_in] (dense layout flattened to B*V rows, or compact); y: the
    stored forward output [n_rows, C_out]; dy: upstream gradient, same shape;
    all float32 or all bf16 bits. Returns (dx [x_rows, C_in], dW [L*C_in,
    C_out], dbias [C_out]), fp64."""
    x = np.ascontiguousarray(x)
    dt = _dtype_code(x)
    C_in = x.shape[-1]
    x = x.reshape(-1, C_in)
    rulebook = _c(rulebook, np.int32)
    L, stride = rulebook.shape
    W = _c(W, x.dtype)
    C_out = W.shape[1]
    y = _c(y, x.dtype)
    dy = _c(dy, x.dtype)
    n = dy.shape[0]
    dx = np.empty((x.shape[0], C_in), dtype=np.float64)
    dW = np.empty((L * C_in, C_out), dtype=np.float64)
    db = np.empty(C_out, dtype=np.float64)
    _load().hco_sparse_conv_bwd(_ptr(x), dt, x.shape[0], _ptr(rulebook), n, stride, L, C_in,
                                C_out, _ptr(W), _ptr(y), _ptr(dy), act, _ptr(dx), _ptr(dW),
                                _ptr(db))
    return dx, dW, db
