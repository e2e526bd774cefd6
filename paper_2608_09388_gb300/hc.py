"""Python binding of libhc (include/hc.h): argument marshalling only.

Each function has the name of the C entry point it calls and takes torch CUDA
tensors (device memory) plus an optional stream (default: torch's current
stream). Every step of the computation runs in libhc's CUDA kernels; there is
no host or CPU fallback. If the library has not been built, or no GPU is
present, the calls raise instead of computing anything.
"""
from __future__ import annotations

import ctypes
import os
import threading

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "_build", "libhc.so")

HC_OK, HC_ERR_INVALID_ARG, HC_ERR_UNSUPPORTED, HC_ERR_CAPACITY = 0, 1, 2, 3
HC_ERR_INVALID_INDEX, HC_ERR_TIMEOUT, HC_ERR_CUDA = 4, 5, 6
HC_F32, HC_BF16 = 0, 1
HC_ACT_NONE, HC_ACT_ELU, HC_ACT_RELU = 0, 1, 2
HC_LAYOUT_DENSE, HC_LAYOUT_COMPACT = 0, 1
HC_MAX_SPIRAL = 32
HC_STATIC_MAX_MASK_BYTES = 4096 * 4096
HC_TEST_GROUP_NORM_PATH, HC_TEST_WAIT_LIMIT_NS = 1, 2

STATUS_NAMES = {0: "HC_OK", 1: "HC_ERR_INVALID_ARG", 2: "HC_ERR_UNSUPPORTED",
                3: "HC_ERR_CAPACITY", 4: "HC_ERR_INVALID_INDEX", 5: "HC_ERR_TIMEOUT",
                6: "HC_ERR_CUDA"}

# Exported symbols, as declared in include/hc.h.
EXPORTS = ("hc_mask_compact", "hc_mask_compact_static", "hc_sparse_spiral_conv_fwd",
           "hc_conv_rulebook", "hc_mask_compact_rulebook", "hc_sparse_conv_rulebook_fwd",
           "hc_sparse_conv_rulebook_fwd_hint", "hc_sparse_linear_fwd",
           "hc_sparse_group_norm_fwd", "hc_sparse_conv_gn_fwd", "hc_mask_score_update", "hc_mask_select_topk",
           "hc_kappa_masks", "hc_gather_rows", "hc_conv_rulebook_transpose",
           "hc_sparse_conv_rulebook_bwd", "hc_scatter_dense", "hc_spiral_conv_fwd", "hc_get_device_status",
           "hc_test_set_option", "hc_last_error_string", "hc_version")


class HcError(RuntimeError):
    def __init__(self, status: int, where: str, msg: str):
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


_lib = None
_lock = threading.Lock()


def load_library(path: str | None = None):
    """Load libhc.so (built by paper_2608_09388_gb300.build). Raises if absent."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"libhc is not built ({p} missing): run __graft_entry__.build()")
        lib = ctypes.CDLL(p)
        P, I = ctypes.c_void_p, ctypes.c_int
        sig = {
            "hc_mask_compact": [P, I, I, P, P, P, P, P],
            "hc_mask_compact_static": [P, I, I, P, P, P, P, P],
            "hc_sparse_spiral_conv_fwd": [P, I, I, P, P, P, P, I, I, I, I, I, P, P, I, P, P],
            "hc_conv_rulebook": [P, P, P, P, I, I, I, I, P, P],
            "hc_mask_compact_rulebook": [P, I, I, P, I, I, P, P, P, P, P, P],
            "hc_sparse_conv_rulebook_fwd": [P, I, I, P, P, I, I, I, I, P, P, I, P, P, I, I, P,
                                            P],
            "hc_sparse_conv_rulebook_fwd_hint": [P, I, I, P, P, I, I, I, I, P, P, I, P, P, I, I,
                                                 P, ctypes.c_longlong, P],
            "hc_sparse_linear_fwd": [P, I, P, I, I, I, P, P, I, P, P],
            "hc_sparse_group_norm_fwd": [P, I, P, I, I, I, I, ctypes.c_float, P, P, I, P, P],
            "hc_sparse_conv_gn_fwd": [P, I, I, P, P, I, I, I, I, P, P, P, P, I, I,
                                      ctypes.c_float, P, P, I, P, P],
            "hc_mask_score_update": [P, I, I, I, I, P, P, P, P],
            "hc_conv_rulebook_transpose": [P, P, I, I, I, P, P, P],
            "hc_sparse_conv_rulebook_bwd": [P, I, I, P, P, I, I, I, I, P, P, P, I, P, P, P, P, P,
                                            P],
            "hc_mask_select_topk": [P, I, I, P, P],
            "hc_kappa_masks": [P, I, I, P, I, I, P, P],
            "hc_gather_rows": [P, I, I, I, I, P, P, I, I, P, P],
            "hc_scatter_dense": [P, I, P, P, P, I, I, I, I, P, P],
            "hc_spiral_conv_fwd": [P, I, P, I, I, I, I, I, P, P, I, P, P],
            "hc_get_device_status": [P],
            "hc_test_set_option": [I, ctypes.c_longlong],
            "hc_last_error_string": [],
            "hc_version": [],
        }
        for name, args in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = ctypes.c_char_p if name in ("hc_last_error_string", "hc_version") else I
        _lib = lib
        return lib


def _p(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libhc takes device tensors")
    if not t.is_contiguous():
        raise ValueError("libhc takes contiguous tensors")
    return ctypes.c_void_p(t.data_ptr())


def _p_host_ok(t):
    """A device tensor, or a pinned host tensor (read by the kernel over the
    host link under unified addressing)."""
    if t is not None and not t.is_cuda and t.is_pinned():
        if not t.is_contiguous():
            raise ValueError("libhc takes contiguous tensors")
        return ctypes.c_void_p(t.data_ptr())
    return _p(t)


def _s(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _dt(t):
    import torch
    if t.dtype == torch.float32:
        return HC_F32
    if t.dtype == torch.bfloat16:
        return HC_BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


def _check(status: int, where: str):
    if status != HC_OK:
        msg = load_library().hc_last_error_string().decode()
        raise HcError(status, where, msg)


def hc_mask_compact(mask, coords, row_of, batch_offsets, count, stream=None):
    """mask uint8 [B, V] -> coords int32 [B*V, 2], row_of int32 [B, V] (or None),
    batch_offsets int32 [B+1] (or None), count int32 [1]."""
    B, V = mask.shape
    _check(load_library().hc_mask_compact(_p(mask), B, V, _p(coords), _p(row_of),
                                          _p(batch_offsets), _p(count), _s(stream)),
           "hc_mask_compact")


def hc_mask_compact_static(mask, coords, row_of, batch_offsets, count, stream=None):
    """hc_mask_compact without any device allocation (fixed in-library
    scratch; masks up to HC_STATIC_MAX_MASK_BYTES bytes)."""
    B, V = mask.shape
    _check(load_library().hc_mask_compact_static(_p(mask), B, V, _p(coords), _p(row_of),
                                                 _p(batch_offsets), _p(count), _s(stream)),
           "hc_mask_compact_static")


def hc_sparse_spiral_conv_fwd(x, x_layout, coords, row_of, count, spiral, B, V, W, bias, act, y,
                              stream=None):
    """Sparse spiral conv; x dense [B, V, C_in] or compact [., C_in]; W [L*C_in, C_out];
    y [B*V, C_out] capacity (rows 0..N'-1 written)."""
    L = spiral.shape[1]
    C_in = x.shape[-1]
    C_out = W.shape[1]
    _check(load_library().hc_sparse_spiral_conv_fwd(
        _p(x), x_layout, _dt(x), _p(coords), _p(row_of), _p(count), _p(spiral), B, V, L, C_in,
        C_out, _p(W), _p(bias), act, _p(y), _s(stream)), "hc_sparse_spiral_conv_fwd")


def hc_conv_rulebook(coords, row_of, count, spiral, B, V, x_layout, rulebook, stream=None):
    """Eq. 4 mapping: rulebook int32 [L, B*V] of input rows per (slot, active row)."""
    L = spiral.shape[1]
    _check(load_library().hc_conv_rulebook(_p(coords), _p(row_of), _p(count), _p(spiral), B, V, L,
                                           x_layout, _p(rulebook), _s(stream)),
           "hc_conv_rulebook")


def hc_mask_compact_rulebook(mask, spiral, x_layout, coords, row_of, batch_offsets, count,
                             rulebook, stream=None):
    """hc_mask_compact then hc_conv_rulebook in one call (fused kernels where
    the frame fits): mask uint8 [B, V], spiral int32 [V, L]."""
    B, V = mask.shape
    L = spiral.shape[1]
    _check(load_library().hc_mask_compact_rulebook(
        _p(mask), B, V, _p(spiral), L, x_layout, _p(coords), _p(row_of), _p(batch_offsets),
        _p(count), _p(rulebook), _s(stream)), "hc_mask_compact_rulebook")


def hc_sparse_conv_rulebook_fwd(x, rulebook, count, W, bias, act, y, coords=None, out=None,
                                stream=None):
    """Sparse conv through a rulebook [L, capacity]: x [x_rows, C_in] (or [B, V, C_in]),
    W [L*C_in, C_out], y [capacity, C_out] or None; out [B, V, C_out] (fused scatter at
    coords) or None."""
    L, capacity = rulebook.shape
    C_in = x.shape[-1]
    x_rows = x.numel() // C_in
    C_out = W.shape[1]
    B, V = (out.shape[0], out.shape[1]) if out is not None else (0, 0)
    _check(load_library().hc_sparse_conv_rulebook_fwd(
        _p(x), _dt(x if y is None else y), x_rows, _p(rulebook), _p(count), capacity, L, C_in,
        C_out, _p(W), _p(bias), act, _p(y), _p(coords), B, V, _p(out), _s(stream)),
        "hc_sparse_conv_rulebook_fwd")


def hc_sparse_conv_rulebook_fwd_hint(x, rulebook, count, W, bias, act, y, rows_hint,
                                     coords=None, out=None, stream=None):
    """hc_sparse_conv_rulebook_fwd with a host-side estimate of N' (an int >= 0,
    0 = unknown) that only chooses the tensor-core tiling; same results."""
    L, capacity = rulebook.shape
    C_in = x.shape[-1]
    x_rows = x.numel() // C_in
    C_out = W.shape[1]
    B, V = (out.shape[0], out.shape[1]) if out is not None else (0, 0)
    _check(load_library().hc_sparse_conv_rulebook_fwd_hint(
        _p(x), _dt(x if y is None else y), x_rows, _p(rulebook), _p(count), capacity, L, C_in,
        C_out, _p(W), _p(bias), act, _p(y), _p(coords), B, V, _p(out), int(rows_hint),
        _s(stream)), "hc_sparse_conv_rulebook_fwd_hint")


def hc_sparse_linear_fwd(x, count, W, bias, act, y, stream=None):
    """Linear layer on compact rows: x [capacity, C_in], W [C_in, C_out], y [capacity, C_out]."""
    capacity, C_in = x.shape
    C_out = W.shape[1]
    _check(load_library().hc_sparse_linear_fwd(
        _p(x), _dt(x), _p(count), capacity, C_in, C_out, _p(W), _p(bias), act, _p(y),
        _s(stream)), "hc_sparse_linear_fwd")


def hc_sparse_group_norm_fwd(x, batch_offsets, G, eps, gamma, beta, act, y, stream=None):
    """Group norm of compact rows x [capacity, C], per frame (batch_offsets
    [B+1]) and group of C/G channels; y may be x."""
    capacity, C = x.shape
    B = batch_offsets.shape[0] - 1
    _check(load_library().hc_sparse_group_norm_fwd(
        _p(x), _dt(x), _p(batch_offsets), B, capacity, C, G, float(eps), _p(gamma), _p(beta),
        act, _p(y), _s(stream)), "hc_sparse_group_norm_fwd")


def hc_sparse_conv_gn_fwd(x, rulebook, count, W, bias, coords, batch_offsets, G, eps, gamma,
                          beta, act, y, stream=None):
    """Sparse conv through a rulebook [L, capacity], then group norm per frame
    (batch_offsets [B+1]) and group of C_out/G channels, then act: y
    [capacity, C_out]."""
    L, capacity = rulebook.shape
    C_in = x.shape[-1]
    x_rows = x.numel() // C_in
    C_out = W.shape[1]
    B = batch_offsets.shape[0] - 1
    _check(load_library().hc_sparse_conv_gn_fwd(
        _p(x), _dt(y), x_rows, _p(rulebook), _p(count), capacity, L, C_in, C_out, _p(W),
        _p(bias), _p(coords), _p(batch_offsets), B, G, float(eps), _p(gamma), _p(beta), act,
        _p(y), _s(stream)), "hc_sparse_conv_gn_fwd")


def hc_conv_rulebook_transpose(rulebook, count, x_rows, row_ptr, taps, stream=None):
    """Taps reading each input row (keys n*L + l, ascending) from a rulebook [L, capacity]."""
    L, capacity = rulebook.shape
    _check(load_library().hc_conv_rulebook_transpose(_p(rulebook), _p(count), capacity, L, x_rows,
                                                     _p(row_ptr), _p(taps), _s(stream)),
           "hc_conv_rulebook_transpose")


def hc_sparse_conv_rulebook_bwd(x, rulebook, count, W, y, dy, act, row_ptr=None, taps=None,
                                dx=None, dW=None, dbias=None, stream=None):
    """Gradients of the rulebook conv. x [x_rows, C_in] (or [B, V, C_in]);
    y, dy [capacity, C_out]; dx like x (or None); dW [L*C_in, C_out] and
    dbias [C_out] fp32 (or None)."""
    L, capacity = rulebook.shape
    C_in = x.shape[-1]
    x_rows = x.numel() // C_in
    C_out = W.shape[1]
    _check(load_library().hc_sparse_conv_rulebook_bwd(
        _p(x), _dt(x), x_rows, _p(rulebook), _p(count), capacity, L, C_in, C_out, _p(W), _p(y),
        _p(dy), act, _p(row_ptr), _p(taps), _p(dx), _p(dW), _p(dbias), _s(stream)),
        "hc_sparse_conv_rulebook_bwd")


def hc_mask_score_update(O, alpha_in, alpha_out, sim=None, stream=None):
    """Eq. 3 on mask outputs O [K, N, D]; alpha_in/alpha_out [K] fp32 (may
    be the same tensor); sim [K, K] fp32 or None."""
    K, N, D = O.shape
    _check(load_library().hc_mask_score_update(
        _p(O), _dt(O), K, N, D, _p(alpha_in), _p(alpha_out), _p(sim), _s(stream)),
        "hc_mask_score_update")


def hc_mask_select_topk(alpha, kappa, selected, stream=None):
    """Indices of the kappa highest scores into selected [kappa] int32."""
    _check(load_library().hc_mask_select_topk(_p(alpha), alpha.shape[0], kappa, _p(selected),
                                              _s(stream)), "hc_mask_select_topk")


def hc_kappa_masks(masks, selected, B, out, stream=None):
    """out [B*kappa, V]: frame b*kappa + j = masks[selected[j]] (masks [K, V] uint8)."""
    K, V = masks.shape
    _check(load_library().hc_kappa_masks(_p(masks), K, V, _p(selected), selected.shape[0], B,
                                         _p(out), _s(stream)), "hc_kappa_masks")


def hc_gather_rows(x, coords, count, frames_per_sample, y, stream=None):
    """S' of Eq. 2: y[n] = x[f // frames_per_sample, v] for coords[n] = (f, v);
    coords None: y[n] = x row n (x viewed as B_in * V rows), n < count. x or y
    may be a pinned host tensor: only the rows copied cross the host link."""
    B_in, V, C = x.shape
    _check(load_library().hc_gather_rows(_p_host_ok(x), _dt(x), B_in, V, C, _p(coords), _p(count),
                                         y.shape[0], frames_per_sample, _p_host_ok(y), _s(stream)),
           "hc_gather_rows")


def hc_scatter_dense(y, coords, row_of, count, B, V, zero_fill, out, stream=None):
    """Compact rows y [., C] -> dense out [B, V, C]."""
    C = y.shape[-1]
    _check(load_library().hc_scatter_dense(
        _p(y), _dt(y), _p(coords), _p(row_of), _p(count), B, V, C, int(zero_fill), _p(out),
        _s(stream)), "hc_scatter_dense")


def hc_spiral_conv_fwd(x, spiral, W, bias, act, y, stream=None):
    """Dense spiral conv over every (b, v): x [B, V, C_in] -> y [B, V, C_out]."""
    B, V, C_in = x.shape
    L = spiral.shape[1]
    C_out = W.shape[1]
    _check(load_library().hc_spiral_conv_fwd(
        _p(x), _dt(x), _p(spiral), B, V, L, C_in, C_out, _p(W), _p(bias), act, _p(y),
        _s(stream)), "hc_spiral_conv_fwd")


def hc_test_set_option(option: int, value: int):
    """Test hook (include/hc.h): force a group-norm path, or lower the
    pipelined kernels' wait limit on the current device (0 = default)."""
    _check(load_library().hc_test_set_option(int(option), int(value)), "hc_test_set_option")


def hc_get_device_status(stream=None) -> int:
    """Synchronise the stream, read and clear the device status word."""
    return int(load_library().hc_get_device_status(_s(stream)))


def hc_last_error_string() -> str:
    return load_library().hc_last_error_string().decode()


def hc_version() -> str:
    return load_library().hc_version().decode()
