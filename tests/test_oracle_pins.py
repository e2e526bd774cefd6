"""Pins for the CPU oracle: each check ties the oracle to something other than
itself (a library routine, a closed form, a hand-worked case, brute force or an
invariant the paper's definitions fix), chosen so that a plausible mistake
(a dropped term, a wrong index, a transposed operand, a wrong sign) fails at
least one of them. Planted-mistake tests at the end show that it does."""
import json
import math
import os

import numpy as np
import pytest

import oracle
from paper_2608_09388_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "octahedron.json")
ACT = {"none": oracle.ACT_NONE, "elu": oracle.ACT_ELU, "relu": oracle.ACT_RELU}


# --------------------------------------------------------------- compaction

def check_compact_vs_nonzero(mask):
    """Decomposition (Eq. 2) against numpy's row-major nonzero listing."""
    coords, row_of, offsets, n = oracle.mask_compact(mask)
    nz = np.argwhere(mask != 0).astype(np.int32)
    assert n == nz.shape[0]
    np.testing.assert_array_equal(coords, nz)
    ref_row = np.full(mask.shape, -1, dtype=np.int32)
    ref_row[nz[:, 0], nz[:, 1]] = np.arange(n, dtype=np.int32)
    np.testing.assert_array_equal(row_of, ref_row)
    ref_off = np.concatenate([[0], np.cumsum((mask != 0).sum(axis=1))]).astype(np.int32)
    np.testing.assert_array_equal(offsets, ref_off)


@pytest.mark.parametrize("B", [1, 7, 64])
@pytest.mark.parametrize("V", [1, 31, 32, 33, 655])
@pytest.mark.parametrize("density", [0.0, 0.01, 0.1, 0.5, 1.0])
def test_compact_matches_numpy_nonzero(B, V, density):
    rng = np.random.default_rng(B * 1000 + V)
    check_compact_vs_nonzero(inputs.uniform_mask(rng, B, V, density))


def test_compact_nonbinary_bytes_are_active():
    mask = np.array([[0, 2, 255, 0, 1]], dtype=np.uint8)
    coords, row_of, offsets, n = oracle.mask_compact(mask)
    assert n == 3
    np.testing.assert_array_equal(coords, [[0, 1], [0, 2], [0, 4]])


def test_compact_empty_and_full():
    z = np.zeros((3, 10), np.uint8)
    coords, row_of, offsets, n = oracle.mask_compact(z)
    assert n == 0 and (row_of == -1).all() and (offsets == 0).all()
    o = np.ones((3, 10), np.uint8)
    coords, row_of, offsets, n = oracle.mask_compact(o)
    assert n == 30
    np.testing.assert_array_equal(row_of.ravel(), np.arange(30))
    np.testing.assert_array_equal(offsets, [0, 10, 20, 30])


# ------------------------------------------------------------ golden cases

def _golden():
    with open(GOLDEN) as f:
        return json.load(f)


def _golden_case_inputs(g, case):
    sp = np.array(g["spiral_L3"], dtype=np.int32)[:, : case.get("spiral_cols", 3)].copy()
    for k, row in case.get("spiral_override", {}).items():
        sp[int(k)] = row
    x = np.array(case["x"], dtype=np.float32)
    mask = np.array(case["mask"], dtype=np.uint8)
    W = np.array(case["W"], dtype=np.float32)
    b = np.array(case["bias"], dtype=np.float32)
    return sp, x, mask, W, b


def check_golden_cases():
    g = _golden()
    for case in g["cases"]:
        sp, x, mask, W, b = _golden_case_inputs(g, case)
        coords, row_of, offsets, n = oracle.mask_compact(mask)
        if "coords" in case:
            np.testing.assert_array_equal(coords, case["coords"])
            np.testing.assert_array_equal(row_of, case["row_of"])
            np.testing.assert_array_equal(offsets, case["offsets"])
        y_pre, y = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, coords, row_of, sp, W, b,
                                             ACT[case["act"]])
        if "y" in case:
            np.testing.assert_array_equal(y_pre, np.array(case["y"], dtype=np.float64))
        if "y_expm1_of" in case:
            ref = np.vectorize(math.expm1)(np.array(case["y_expm1_of"], dtype=np.float64))
            np.testing.assert_allclose(y_pre, ref, rtol=1e-15, atol=0)
        if "y_rows" in case:
            for k, v in case["y_rows"].items():
                np.testing.assert_array_equal(y_pre[int(k)], np.array(v, dtype=np.float64))
        if "rulebook_compact" in case:
            for lay, key in ((oracle.LAYOUT_COMPACT, "rulebook_compact"),
                             (oracle.LAYOUT_DENSE, "rulebook_dense")):
                rb = oracle.conv_rulebook(coords, row_of, sp, lay, stride=n)
                np.testing.assert_array_equal(rb, case[key])
    d = g["dense_full_input"]
    sp = np.array(g["spiral_L3"], dtype=np.int32)
    y_pre, _ = oracle.dense_spiral_conv(np.array(d["x"], np.float32), sp,
                                        np.array(d["W"], np.float32), None, oracle.ACT_NONE)
    np.testing.assert_array_equal(y_pre, np.array(d["y"], dtype=np.float64))


def test_golden_octahedron():
    check_golden_cases()


# ------------------------------------------------- conv against library GEMM

def check_conv_vs_gather_matmul(seed=3, B=3, V=40, L=5, C_in=6, C_out=7, density=0.4):
    """The sparse conv written as an explicit gather (numpy fancy indexing,
    zero rows for absent taps) followed by numpy's matmul in fp64: the
    layout [L*C_in, C_out] with row l*C_in + c must agree with the loop."""
    sp, m, x, W, b = inputs.random_case(seed, B, V, L, C_in, C_out, "f32", density, neg_frac=0.2)
    coords, row_of, offsets, n = oracle.mask_compact(m)
    y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, coords, row_of, sp, W, b,
                                         oracle.ACT_NONE)
    xs = np.concatenate([x.astype(np.float64).reshape(B * V, C_in), np.zeros((1, C_in))])
    bb, vv = coords[:, 0].astype(np.int64), coords[:, 1].astype(np.int64)
    u = sp[vv]  # [n, L]
    act_nb = (u >= 0) & (m[bb[:, None], np.where(u >= 0, u, 0)] != 0)
    src = np.where(act_nb, bb[:, None] * V + np.where(u >= 0, u, 0), B * V)
    G = xs[src].reshape(n, L * C_in)  # [n, L*C_in], slot-major
    ref = np.matmul(G, W.astype(np.float64)) + b.astype(np.float64)
    np.testing.assert_allclose(y_pre, ref, rtol=1e-12, atol=1e-12)


def test_conv_vs_gather_matmul():
    check_conv_vs_gather_matmul()


def test_rulebook_gather_matmul_equals_conv():
    """Eq. 5 evaluated through the Eq. 4 rulebook with numpy (gather the rows
    the rulebook names, zero for -1, one fp64 matmul) equals the loop conv,
    for both input layouts."""
    sp, m, x, W, b = inputs.random_case(21, 3, 70, 7, 5, 6, "f32", 0.4, neg_frac=0.15)
    coords, row_of, offsets, n = oracle.mask_compact(m)
    y_ref, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, coords, row_of, sp, W, b,
                                         oracle.ACT_NONE)
    xc = x[coords[:, 0], coords[:, 1]]
    for lay, xs in ((oracle.LAYOUT_DENSE, x.reshape(-1, 5)), (oracle.LAYOUT_COMPACT, xc)):
        rb = oracle.conv_rulebook(coords, row_of, sp, lay)
        assert (rb[:, n:] == -1).all()
        xz = np.concatenate([xs.astype(np.float64), np.zeros((1, 5))])
        G = xz[np.where(rb[:, :n] >= 0, rb[:, :n], xs.shape[0])]  # [L, n, C_in]
        G = G.transpose(1, 0, 2).reshape(n, -1)
        np.testing.assert_allclose(G @ W.astype(np.float64) + b, y_ref, rtol=1e-12, atol=1e-12)


def test_conv_L1_is_matmul():
    """L = 1 (only the centre tap): the sparse conv is a plain matmul of the
    active rows (Eq. 6 special case) -- numpy matmul in fp64."""
    sp, m, x, W, b = inputs.random_case(5, 4, 50, 1, 9, 11, "f32", 0.3)
    coords, row_of, offsets, n = oracle.mask_compact(m)
    y_pre, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, coords, row_of, sp, W, b,
                                         oracle.ACT_NONE)
    xa = x[coords[:, 0], coords[:, 1]].astype(np.float64)
    np.testing.assert_allclose(y_pre, xa @ W.astype(np.float64) + b, rtol=1e-12, atol=1e-12)


def test_linear_is_matmul():
    rng = np.random.default_rng(11)
    x = rng.standard_normal((37, 13)).astype(np.float32)
    W = rng.standard_normal((13, 5)).astype(np.float32)
    b = rng.standard_normal(5).astype(np.float32)
    y_pre, _ = oracle.sparse_linear(x, W, b, oracle.ACT_NONE)
    np.testing.assert_allclose(y_pre, x.astype(np.float64) @ W.astype(np.float64) + b,
                               rtol=1e-12, atol=1e-12)
    y_pre, _ = oracle.sparse_linear(x, W, b, oracle.ACT_RELU)
    np.testing.assert_allclose(y_pre, np.maximum(x.astype(np.float64) @ W.astype(np.float64) + b, 0),
                               rtol=1e-12, atol=1e-12)


# ------------------------------------------------------------- invariants

def check_sparse_equals_dense_on_masked_input(seed=7, B=4, V=60, L=7, C_in=5, C_out=6,
                                              density=0.3, act=oracle.ACT_ELU):
    """Eq. 1 + Eq. 5: the sparse layer equals the dense layer applied to the
    masked input M o X, restricted to active rows (bit-identical in fp64:
    the dense sum only adds exact zeros)."""
    sp, m, x, W, b = inputs.random_case(seed, B, V, L, C_in, C_out, "f32", density, neg_frac=0.1)
    coords, row_of, offsets, n = oracle.mask_compact(m)
    y_sp, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, coords, row_of, sp, W, b, act)
    xm = x * m[:, :, None].astype(np.float32)
    rows = coords[:, 0].astype(np.int64) * V + coords[:, 1]
    y_de, _ = oracle.dense_spiral_conv(xm, sp, W, b, act, rows=rows)
    np.testing.assert_array_equal(y_sp, y_de)


def test_sparse_equals_dense_on_masked_input():
    check_sparse_equals_dense_on_masked_input()


def test_all_ones_mask_reproduces_dense():
    sp, m, x, W, b = inputs.random_case(8, 3, 45, 9, 4, 8, "f32", 1.0)
    coords, row_of, offsets, n = oracle.mask_compact(m)
    assert n == 3 * 45
    y_sp, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, coords, row_of, sp, W, b,
                                        oracle.ACT_ELU)
    y_de, _ = oracle.dense_spiral_conv(x, sp, W, b, oracle.ACT_ELU)
    np.testing.assert_array_equal(y_sp, y_de)


def test_empty_mask_has_no_rows():
    sp, m, x, W, b = inputs.random_case(9, 2, 30, 4, 3, 3, "f32", 0.0)
    coords, row_of, offsets, n = oracle.mask_compact(m)
    assert n == 0
    y_pre, y = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, coords, row_of, sp, W, b,
                                         oracle.ACT_ELU)
    assert y_pre.shape == (0, 3)


def test_compact_input_layout_equals_dense_layout():
    sp, m, x, W, b = inputs.random_case(10, 3, 50, 6, 4, 5, "f32", 0.35)
    coords, row_of, offsets, n = oracle.mask_compact(m)
    xc = x[coords[:, 0], coords[:, 1]]
    a, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, coords, row_of, sp, W, b, oracle.ACT_ELU)
    c, _ = oracle.sparse_spiral_conv(xc, oracle.LAYOUT_COMPACT, coords, row_of, sp, W, b,
                                     oracle.ACT_ELU)
    np.testing.assert_array_equal(a, c)


def test_brute_force_all_masks_tiny_mesh():
    """Every one of the 2^8 masks on an 8-vertex mesh: compaction against
    numpy, sparse conv against the dense layer on the masked input."""
    V, L = 8, 4
    sp, _, x, W, b = inputs.random_case(12, 1, V, L, 3, 2, "f32", 0.5, neg_frac=0.15)
    for bits in range(1 << V):
        m = np.array([[(bits >> v) & 1 for v in range(V)]], dtype=np.uint8)
        check_compact_vs_nonzero(m)
        coords, row_of, offsets, n = oracle.mask_compact(m)
        y_sp, _ = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, coords, row_of, sp, W, b,
                                            oracle.ACT_ELU)
        y_de, _ = oracle.dense_spiral_conv(x * m[:, :, None], sp, W, b, oracle.ACT_ELU,
                                           rows=coords[:, 1].astype(np.int64))
        np.testing.assert_array_equal(y_sp, y_de)


def test_stack_equals_dense_stack_remasked():
    """A 4-layer sparse stack on one mask equals the dense stack with the
    input re-masked before every layer (fp32 storage, so each layer's stored
    values agree exactly)."""
    B, V, L = 3, 64, 9
    sp, m, x, _, _ = inputs.random_case(13, B, V, L, 16, 1, "f32", 0.2)
    rng = np.random.default_rng(99)
    chans = [16, 12, 12, 8, 8]
    layers = [inputs.Layer("conv", ci, co, oracle.ACT_ELU,
                           inputs.weights(rng, L * ci, co, "f32"), inputs.bias(co))
              for ci, co in zip(chans[:-1], chans[1:])]
    coords, row_of, offsets, n, outs = oracle.encoder(x, m, sp, layers)
    h = x
    for ly in layers:
        _, hy = oracle.dense_spiral_conv(h * m[:, :, None], sp, ly.W, ly.b, ly.act)
        h = hy.reshape(B, V, -1)
    act_rows = h[coords[:, 0], coords[:, 1]]
    np.testing.assert_array_equal(outs[-1][1], act_rows)


def test_scatter_matches_numpy_assignment():
    rng = np.random.default_rng(14)
    m = inputs.uniform_mask(rng, 3, 20, 0.3)
    coords, row_of, offsets, n = oracle.mask_compact(m)
    y = rng.standard_normal((n, 4)).astype(np.float32)
    prev = rng.standard_normal((3, 20, 4)).astype(np.float32)
    out = oracle.scatter_dense(y, coords, 3, 20, zero_fill=False, out=prev)
    ref = prev.copy()
    ref[coords[:, 0], coords[:, 1]] = y
    np.testing.assert_array_equal(out, ref)
    out0 = oracle.scatter_dense(y, coords, 3, 20, zero_fill=True, out=prev)
    ref0 = np.zeros_like(prev)
    ref0[coords[:, 0], coords[:, 1]] = y
    np.testing.assert_array_equal(out0, ref0)


# ----------------------------------------------------------- bf16 storage

def check_bf16_round():
    """fp64 -> bf16 rounding against torch's float32 -> bf16 routine on values
    exactly representable in float32, and against closed-form cases that a
    round-through-float32 implementation gets wrong."""
    import torch
    rng = np.random.default_rng(15)
    vals = np.concatenate([
        rng.standard_normal(4000).astype(np.float32),
        (rng.standard_normal(1000) * 1e-39).astype(np.float32),  # subnormal range
        (rng.standard_normal(1000) * 1e38).astype(np.float32),
        np.array([0.0, -0.0, 1.0, -1.0, 3.0e38, 3.3961776e38, 1e-45], dtype=np.float32),
        # exact ties: lower 16 bits 0x8000
        (np.arange(1, 2000, dtype=np.uint32) << 16 | 0x8000).view(np.float32),
    ])
    ref = torch.from_numpy(vals).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([oracle.bf16_round(float(v)) for v in vals], dtype=np.uint16)
    finite = np.isfinite(vals)
    np.testing.assert_array_equal(got[finite], ref[finite])
    # 1 + 2^-8 is a tie -> even (1.0); a hair above must round up to 1 + 2^-7.
    assert oracle.bf16_round(1.0 + 2.0 ** -8) == 0x3F80
    assert oracle.bf16_round(1.0 + 2.0 ** -8 + 2.0 ** -30) == 0x3F81
    assert oracle.bf16_round(-(1.0 + 2.0 ** -8 + 2.0 ** -30)) == 0xBF81
    assert oracle.bf16_round(1.0 + 3 * 2.0 ** -8) == 0x3F82  # tie, odd -> up to even


def test_bf16_round():
    check_bf16_round()


def test_bf16_conv_rounds_once_from_fp64():
    sp, m, x, W, b = inputs.random_case(16, 2, 40, 5, 8, 8, "bf16", 0.5)
    coords, row_of, offsets, n = oracle.mask_compact(m)
    y_pre, y = oracle.sparse_spiral_conv(x, oracle.LAYOUT_DENSE, coords, row_of, sp, W, b,
                                         oracle.ACT_ELU)
    want = np.array([oracle.bf16_round(v) for v in y_pre.ravel()], np.uint16).reshape(y.shape)
    np.testing.assert_array_equal(y, want)
    # bf16 inputs are widened exactly: same as the f32 oracle on widened data
    xf = inputs.bf16_bits_to_f32(x)
    Wf = inputs.bf16_bits_to_f32(W)
    y32, _ = oracle.sparse_spiral_conv(xf, oracle.LAYOUT_DENSE, coords, row_of, sp, Wf, b,
                                       oracle.ACT_ELU)
    np.testing.assert_array_equal(y_pre, y32)


# ------------------------------------------------------ workload statistics

def test_workload_statistics():
    """The synthetic workloads reproduce the paper's statistics: 655 vertices,
    about 10% active at a 90% sparsity ratio (Table 4: 66 of 655)."""
    w = inputs.make_workload("encoder655_bf16")
    d = w.masks[0].mean()
    assert w.V == 655 and abs(d - 0.1) < 0.01
    sp = w.spiral
    assert (sp[:, 0] == np.arange(655)).all()
    assert ((sp >= 0) & (sp < 655)).all()
    # neighbours are distinct from the vertex and ordered by distance
    p = w.points
    d2 = ((p[sp[:, 1:]] - p[:, None, :]) ** 2).sum(-1)
    assert (np.diff(d2, axis=1) >= 0).all()
    assert (sp[:, 1:] != np.arange(655)[:, None]).all()


# ----------------------------------------------------- planted mistakes

MUTANTS = {
    "transposed weight index": ("acc[o] += xv * load_elem(W, dtype, ((int64_t)l * C_in + c) * C_out + o);",
                                "acc[o] += xv * load_elem(W, dtype, ((int64_t)c * L + l) * C_out + o);"),
    "inactive neighbour not skipped": ("if (j < 0) continue; /* neighbour not in C: tap absent */",
                                       "/* dropped */"),
    "ELU sign": ("return z > 0.0 ? z : expm1(z);", "return z > 0.0 ? z : expm1(-z);"),
    "compaction order": ("for (int64_t b = 0; b < B; ++b) {\n        offsets[b] = (int32_t)n;\n        for (int64_t v = 0; v < V; ++v) {",
                         "for (int64_t b = B - 1; b >= 0; --b) {\n        offsets[b] = (int32_t)n;\n        for (int64_t v = 0; v < V; ++v) {"),
    "bf16 rounded through float32": ("double n = nearbyint(ldexp(x, -qexp));",
                                     "double n = nearbyint(ldexp((double)(float)x, -qexp));"),
    "rulebook ignores activity": ("                if (j >= 0) e = (int32_t)(x_layout == HCO_LAYOUT_DENSE ? b * V + u : j);",
                                  "                e = (int32_t)(x_layout == HCO_LAYOUT_DENSE ? b * V + u : j);"),
    "group norm variance around zero": ("                    double d = load_elem(x, dtype, i * C + c) - mu;",
                                        "                    double d = load_elem(x, dtype, i * C + c);"),
    "group norm counts rows only": ("            double n = (double)(r1 - r0) * cpg;",
                                    "            double n = (double)(r1 - r0);"),
    "mask score without the norms' square roots": ("            double den = sqrt(S[i * K + i]) * sqrt(S[k * K + k]);",
                                                   "            double den = S[i * K + i] * S[k * K + k];"),
    "mask score averaged over K": ("        alpha_out[k] = K > 1 ? alpha_in[k] + sum / (double)(K - 1) : alpha_in[k];",
                                   "        alpha_out[k] = K > 1 ? alpha_in[k] + sum / (double)K : alpha_in[k];"),
    "mask score Gram index": ("                         load_elem(O, dtype, (k * N + n) * D + e);",
                              "                         load_elem(O, dtype, (k * N + n) * D + d);"),
    "mask score numerator not squared": ("                acc += g * g;", "                acc += fabs(g);"),
    "top-kappa ties by highest index": ("    return isnan(b) || a > b;", "    return isnan(b) || a >= b;"),
    "backward ELU derivative as exp(y)": ("    if (act == HCO_ACT_ELU) return y > 0.0 ? 1.0 : y + 1.0;",
                                          "    if (act == HCO_ACT_ELU) return y > 0.0 ? 1.0 : exp(y);"),
    "backward input gradient with a transposed weight": (
        "                    for (int o = 0; o < C_out; ++o) g += dz[o] * load_elem(W, dtype, k * C_out + o);",
        "                    for (int o = 0; o < C_out; ++o) g += dz[o] * load_elem(W, dtype, (int64_t)o * L * C_in + k);"),
    "backward absent tap read as row 0": ("            if (j < 0) continue; /* absent tap: no term, no gradient */",
                                          "            if (j < 0) j = 0;"),
    "backward bias gradient skips the activation": ("            for (int o = 0; o < C_out; ++o) dbias[o] += dz[o];",
                                                    "            for (int o = 0; o < C_out; ++o) dbias[o] += load_elem(dy, dtype, n * C_out + o);"),
    "centre tap dropped": ("for (int l = 0; l < L; ++l) {\n            int64_t u = spiral[v * L + l];\n            if (u < 0) continue; /* no neighbour in this slot */",
                           "for (int l = 1; l < L; ++l) {\n            int64_t u = spiral[v * L + l];\n            if (u < 0) continue; /* no neighbour in this slot */"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, tmp_path, monkeypatch):
    """Compile a copy of the oracle with one plausible mistake planted and
    check that the pins above reject it."""
    import ctypes
    import subprocess
    src = open(oracle._SRC).read()
    old, new = MUTANTS[name]
    assert src.count(old) >= 1, name
    mut = tmp_path / "mut.c"
    mut.write_text(src.replace(old, new, 1))  # first occurrence: the sparse operator
    so = tmp_path / "libmut.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-fopenmp", str(mut), "-o",
                    str(so), "-lm"], check=True)
    good = oracle._load()
    lib = ctypes.CDLL(str(so))
    for fn in ("hco_mask_compact", "hco_sparse_spiral_conv", "hco_dense_spiral_conv",
               "hco_sparse_linear", "hco_scatter_dense", "hco_bf16_round", "hco_conv_rulebook",
               "hco_sparse_group_norm", "hco_mask_score", "hco_select_topk", "hco_kappa_masks",
               "hco_gather_rows", "hco_sparse_conv_bwd"):
        getattr(lib, fn).argtypes = getattr(good, fn).argtypes
        getattr(lib, fn).restype = getattr(good, fn).restype
    monkeypatch.setattr(oracle, "_lib", lib)
    checks = [check_golden_cases, check_conv_vs_gather_matmul, check_group_norm_golden,
              check_group_norm_vs_numpy,
              lambda: check_compact_vs_nonzero(inputs.uniform_mask(np.random.default_rng(1), 5, 20, 0.3)),
              check_bf16_round, check_mask_score_golden, check_mask_score_vs_numpy,
              check_mask_score_d1_is_squared_cosine, check_select_topk_vs_argsort,
              check_bwd_finite_differences, check_bwd_linear_closed_form,
              check_bwd_adjoint_identity]
    caught = 0
    for chk in checks:
        try:
            chk()
        except AssertionError:
            caught += 1
    assert caught >= 1, f"planted mistake '{name}' passed every pin"


# ------------------------------------------------------------ group norm

def check_group_norm_golden():
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "group_norm.json")))
    c0, c1, c2 = g["cases"]
    y, _ = oracle.sparse_group_norm(np.array(c0["x"], np.float32), np.array(c0["offsets"]),
                                    c0["G"], eps=0.0)
    np.testing.assert_allclose(y, np.array(c0["y_over_sqrt_1_25"]) / math.sqrt(1.25), rtol=1e-14)
    y, _ = oracle.sparse_group_norm(np.array(c1["x"], np.float32), np.array(c1["offsets"]),
                                    c1["G"], eps=1.0)
    np.testing.assert_allclose(y[:2], np.array(c1["y_frame0"]) / np.sqrt(1 + 1 / np.array([1, 100])),
                               rtol=1e-14)
    np.testing.assert_array_equal(y[2], [0.0, 0.0])
    y, _ = oracle.sparse_group_norm(np.array(c2["x"], np.float32), np.array(c2["offsets"]),
                                    c2["G"], eps=0.0)
    np.testing.assert_allclose(y, np.array(c2["y"], np.float64), rtol=1e-14)


def test_group_norm_golden():
    check_group_norm_golden()


def check_group_norm_vs_numpy(seed=31):
    """Per frame and group, numpy's mean and (biased) variance of the gathered
    group values give the same normalisation; gamma, beta and ELU follow."""
    rng = np.random.default_rng(seed)
    m = inputs.uniform_mask(rng, 5, 60, 0.3)
    m[2] = 0  # an empty frame
    coords, row_of, offsets, n = oracle.mask_compact(m)
    C, G = 12, 3
    x = (rng.standard_normal((n, C)) * 2 + 0.7).astype(np.float32)
    gamma = rng.standard_normal(C).astype(np.float32)
    beta = rng.standard_normal(C).astype(np.float32)
    y, _ = oracle.sparse_group_norm(x, offsets, G, 1e-5, gamma, beta, oracle.ACT_ELU)
    ref = np.empty((n, C))
    xd = x.astype(np.float64)
    for b in range(5):
        r0, r1 = offsets[b], offsets[b + 1]
        for g in range(G):
            blk = xd[r0:r1, g * 4:(g + 1) * 4]
            if blk.size == 0:
                continue
            z = (blk - blk.mean()) / np.sqrt(blk.var() + 1e-5)
            z = z * gamma[g * 4:(g + 1) * 4] + beta[g * 4:(g + 1) * 4]
            ref[r0:r1, g * 4:(g + 1) * 4] = np.where(z > 0, z, np.expm1(np.minimum(z, 0)))
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)


def test_group_norm_vs_numpy():
    check_group_norm_vs_numpy()


def test_group_norm_is_layer_norm_at_g1_and_ignores_inactive_rows():
    """G = 1 is layer normalisation over all channels of a frame's active rows;
    inactive vertices (zeros in the dense masked tensor) do not enter the
    statistics, unlike a dense group norm over all V rows."""
    rng = np.random.default_rng(32)
    m = inputs.uniform_mask(rng, 1, 50, 0.4)
    coords, row_of, offsets, n = oracle.mask_compact(m)
    x = (rng.standard_normal((n, 8)) + 3).astype(np.float32)
    y, _ = oracle.sparse_group_norm(x, offsets, 1, 0.0)
    assert abs(y.mean()) < 1e-12 and abs(y.var() - 1.0) < 1e-12
    dense = np.zeros((50, 8))
    dense[coords[:, 1]] = x
    yd = (dense - dense.mean()) / dense.std()
    assert not np.allclose(yd[coords[:, 1]], y)


# ------------------------------------------------------------ mask score (Eq. 3)

def check_mask_score_golden():
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "mask_score.json")))
    c0, c1, c2, c3 = g["cases"]
    a, sim, _ = oracle.mask_score(np.array(c0["O"], np.float32), c0["alpha"])
    np.testing.assert_allclose(a, c0["alpha_next"], rtol=0, atol=1e-15)
    assert abs(sim[0, 1] - c0["sim01"]) < 1e-15
    a, sim, _ = oracle.mask_score(np.array(c1["O"], np.float32), c1["alpha"])
    r = 1 - 1 / math.sqrt(2)
    np.testing.assert_allclose(a, [r / 2, r / 2, r], rtol=0, atol=1e-15)
    np.testing.assert_allclose(sim, [[1, 1, 1 / math.sqrt(2)], [1, 1, 1 / math.sqrt(2)],
                                     [1 / math.sqrt(2), 1 / math.sqrt(2), 1]], atol=1e-15)
    a, _, _ = oracle.mask_score(np.array(c2["O"], np.float32), c2["alpha"])
    np.testing.assert_array_equal(a, c2["alpha_next"])
    a, _, _ = oracle.mask_score(np.array(c3["O"], np.float32), c3["alpha"])
    np.testing.assert_array_equal(a, c3["alpha_next"])


def test_mask_score_golden():
    check_mask_score_golden()


def check_mask_score_vs_numpy(seed=41, dtype="f32"):
    """The Gram matrices from numpy's matmul (fp64), their squared Frobenius
    norms and the update written out with numpy."""
    rng = np.random.default_rng(seed)
    K, N, D = 4, 97, 5
    O = (rng.standard_normal((K, N, D)) + 0.3).astype(np.float32)
    if dtype == "bf16":
        O = inputs.to_bf16_bits(O)
        Od = inputs.bf16_bits_to_f32(O).astype(np.float64)
    else:
        Od = O.astype(np.float64)
    alpha = rng.standard_normal(K)
    a, sim, S = oracle.mask_score(O, alpha, n_threads=2)
    S_ref = np.array([[np.sum((Od[i].T @ Od[k]) ** 2) for k in range(K)] for i in range(K)])
    np.testing.assert_allclose(S, S_ref, rtol=1e-12)
    nrm = np.sqrt(np.diag(S_ref))
    sim_ref = S_ref / np.outer(nrm, nrm)
    a_ref = alpha + ((1 - sim_ref).sum(axis=0) - (1 - np.diag(sim_ref))) / (K - 1)
    np.testing.assert_allclose(sim, sim_ref, rtol=1e-12)
    np.testing.assert_allclose(a, a_ref, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_mask_score_vs_numpy(dtype):
    check_mask_score_vs_numpy(dtype=dtype)


def check_mask_score_d1_is_squared_cosine(seed=42):
    """D = 1: O_i^T O_k is the dot product of two vectors, so the similarity
    is their squared cosine."""
    rng = np.random.default_rng(seed)
    v = rng.standard_normal((3, 40, 1)).astype(np.float32)
    _, sim, _ = oracle.mask_score(v, np.zeros(3))
    u = v[:, :, 0].astype(np.float64)
    cos = (u @ u.T) / np.outer(np.linalg.norm(u, axis=1), np.linalg.norm(u, axis=1))
    np.testing.assert_allclose(sim, cos ** 2, rtol=1e-12)


def test_mask_score_d1_is_squared_cosine():
    check_mask_score_d1_is_squared_cosine()


def test_mask_score_invariances():
    """The score compares feature distributions, not bases or scales: it is
    unchanged by scaling a mask's output, by an orthogonal change of feature
    basis per mask (Frobenius norms are invariant under both sides'
    orthogonal factors), and by one permutation of the rows of all masks.
    Identical outputs are fully similar (alpha unchanged); outputs on
    disjoint rows share nothing (alpha + 1)."""
    rng = np.random.default_rng(43)
    K, N, D = 3, 60, 4
    O = rng.standard_normal((K, N, D))
    alpha = rng.standard_normal(K)
    a0, _, _ = oracle.mask_score(O.astype(np.float32), alpha)
    O2 = O.copy()
    O2[1] *= -2.5
    for k in range(K):
        q, _ = np.linalg.qr(rng.standard_normal((D, D)))
        O2[k] = O2[k] @ q
    O2 = O2[:, rng.permutation(N)]
    a1, _, _ = oracle.mask_score(O2.astype(np.float32), alpha)
    np.testing.assert_allclose(a1, a0, rtol=1e-5, atol=1e-5)  # fp32 storage of the rotated data
    same = np.repeat(O[:1], K, axis=0).astype(np.float32)
    a2, _, _ = oracle.mask_score(same, alpha)
    np.testing.assert_allclose(a2, alpha, atol=1e-12)
    disj = np.zeros((K, N, D), np.float32)
    for k in range(K):
        disj[k, k * 20:(k + 1) * 20] = O[k, k * 20:(k + 1) * 20]
    a3, _, _ = oracle.mask_score(disj, alpha)
    np.testing.assert_allclose(a3, alpha + 1, atol=1e-12)


def check_select_topk_vs_argsort(seed=44):
    """Top-kappa against numpy's stable argsort of -alpha (ties by index)."""
    rng = np.random.default_rng(seed)
    for K, kappa in ((10, 3), (50, 10), (7, 7), (1, 1)):
        alpha = rng.integers(-3, 4, size=K).astype(np.float32) * 0.5  # many ties
        np.testing.assert_array_equal(oracle.select_topk(alpha, kappa),
                                      np.argsort(-alpha, kind="stable")[:kappa])


def test_select_topk_vs_argsort():
    check_select_topk_vs_argsort()


def test_select_topk_nan_ranks_last():
    """NaN scores rank below every number (numpy's argsort also puts NaN
    last); among themselves by index."""
    alpha = np.array([np.nan, 1.0, -np.inf, np.nan, 3.0, 1.0], np.float32)
    np.testing.assert_array_equal(oracle.select_topk(alpha, 6), [4, 1, 5, 2, 0, 3])
    np.testing.assert_array_equal(oracle.select_topk(alpha, 6),
                                  np.argsort(-alpha, kind="stable"))


def test_kappa_masks_and_gather_rows_vs_numpy():
    """Kept masks applied to every sample (frame b * kappa + j), and the rows
    S' of Eq. 2 gathered from the samples, against numpy indexing."""
    rng = np.random.default_rng(45)
    K, V, B, kappa, C = 6, 40, 5, 3, 7
    masks = inputs.uniform_mask(rng, K, V, 0.2)
    sel = np.array([4, 0, 2], np.int32)
    fm = oracle.kappa_masks(masks, sel, B)
    np.testing.assert_array_equal(fm, np.tile(masks[sel], (B, 1)))
    coords, _, _, n = oracle.mask_compact(fm)
    x = rng.standard_normal((B, V, C)).astype(np.float32)
    y = oracle.gather_rows(x, coords, kappa)
    np.testing.assert_array_equal(y, x[coords[:, 0] // kappa, coords[:, 1]])
    np.testing.assert_array_equal(oracle.gather_rows(x, oracle.mask_compact(masks[:B])[0]),
                                  x[np.nonzero(masks[:B])])


# ------------------------------------------------------------ backward (chain rule)

def _bwd_case(seed, act, layout=oracle.LAYOUT_DENSE, B=2, V=30, L=5, C_in=3, C_out=4):
    """A small conv with a fully seeded forward: values stay well inside
    float32's exact range for dyadic steps of 2^-12."""
    rng = np.random.default_rng(seed)
    pts = inputs.sphere_points(rng, V)
    sp = inputs.spiral_table(pts, L)
    sp[3, 2] = -1  # a missing spiral slot
    m = inputs.uniform_mask(rng, B, V, 0.6)
    coords, row_of, _, n = oracle.mask_compact(m)
    x_dense = rng.standard_normal((B, V, C_in)).astype(np.float32)
    x = x_dense if layout == oracle.LAYOUT_DENSE else oracle.gather_rows(x_dense, coords)
    W = (rng.standard_normal((L * C_in, C_out)) * 0.5).astype(np.float32)
    b = rng.standard_normal(C_out).astype(np.float32)
    g = rng.standard_normal((n, C_out)).astype(np.float32)  # upstream gradient
    rb = oracle.conv_rulebook(coords, row_of, sp, layout, stride=n)
    return dict(x=x, W=W, b=b, g=g, sp=sp, coords=coords, row_of=row_of, rb=rb, act=act,
                layout=layout)


def _loss(c, x=None, W=None, b=None):
    y, _ = oracle.sparse_spiral_conv(c["x"] if x is None else x, c["layout"], c["coords"],
                                     c["row_of"], c["sp"], c["W"] if W is None else W,
                                     c["b"] if b is None else b, c["act"])
    return float(np.sum(y * c["g"].astype(np.float64)))


def check_bwd_finite_differences(seed=51, act=oracle.ACT_ELU, layout=oracle.LAYOUT_DENSE):
    """Central differences of the fp64 forward loss sum(y * g) against the
    backward, for sampled input, weight and bias entries. Steps are 2^-12,
    exact in float32 for these magnitudes."""
    c = _bwd_case(seed, act, layout)
    _, y = oracle.sparse_spiral_conv(c["x"], c["layout"], c["coords"], c["row_of"], c["sp"],
                                     c["W"], c["b"], act)
    dx, dW, db = oracle.sparse_conv_bwd(c["x"], c["rb"], c["W"], y, c["g"], act)
    h = 2.0 ** -12
    rng = np.random.default_rng(seed + 1)
    xf = c["x"].reshape(-1)
    for idx in rng.choice(xf.size, 24, replace=False):
        xp, xm = xf.copy(), xf.copy()
        xp[idx] += h
        xm[idx] -= h
        fd = (_loss(c, x=xp.reshape(c["x"].shape)) - _loss(c, x=xm.reshape(c["x"].shape))) / (2 * h)
        assert abs(fd - dx.reshape(-1)[idx]) <= 1e-5 * max(1.0, abs(fd)), ("dx", idx, fd)
    Wf = c["W"].reshape(-1)
    for idx in rng.choice(Wf.size, 24, replace=False):
        wp, wm = Wf.copy(), Wf.copy()
        wp[idx] += h
        wm[idx] -= h
        fd = (_loss(c, W=wp.reshape(c["W"].shape)) - _loss(c, W=wm.reshape(c["W"].shape))) / (2 * h)
        assert abs(fd - dW.reshape(-1)[idx]) <= 1e-5 * max(1.0, abs(fd)), ("dW", idx, fd)
    for o in range(c["b"].size):
        bp, bm = c["b"].copy(), c["b"].copy()
        bp[o] += h
        bm[o] -= h
        fd = (_loss(c, b=bp) - _loss(c, b=bm)) / (2 * h)
        assert abs(fd - db[o]) <= 1e-5 * max(1.0, abs(fd)), ("db", o, fd)


@pytest.mark.parametrize("act", [oracle.ACT_ELU, oracle.ACT_RELU, oracle.ACT_NONE])
@pytest.mark.parametrize("layout", [oracle.LAYOUT_DENSE, oracle.LAYOUT_COMPACT])
def test_bwd_finite_differences(act, layout):
    check_bwd_finite_differences(act=act, layout=layout)


def check_bwd_linear_closed_form(seed=52):
    """L = 1 with the identity mapping is a linear layer: dW = x^T dz,
    dx = dz W^T, dbias = column sums of dz (numpy matmul, fp64)."""
    rng = np.random.default_rng(seed)
    n, C_in, C_out = 37, 6, 5
    x = rng.standard_normal((n, C_in)).astype(np.float32)
    W = rng.standard_normal((C_in, C_out)).astype(np.float32)
    y = rng.standard_normal((n, C_out)).astype(np.float32)
    g = rng.standard_normal((n, C_out)).astype(np.float32)
    rb = np.arange(n, dtype=np.int32)[None, :]
    dx, dW, db = oracle.sparse_conv_bwd(x, rb, W, y, g, oracle.ACT_ELU)
    dz = g.astype(np.float64) * np.where(y > 0, 1.0, y.astype(np.float64) + 1.0)
    np.testing.assert_allclose(dW, x.astype(np.float64).T @ dz, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dx, dz @ W.astype(np.float64).T, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(db, dz.sum(axis=0), rtol=1e-12, atol=1e-12)


def test_bwd_linear_closed_form():
    check_bwd_linear_closed_form()


def check_bwd_adjoint_identity(seed=53):
    """Without bias and activation the layer is bilinear in (x, W), so
    <y, g> = <x, dx> = <W, dW> exactly (in fp64, up to rounding order)."""
    c = _bwd_case(seed, oracle.ACT_NONE, B=3, V=60, L=7, C_in=4, C_out=6)
    y, ys = oracle.sparse_spiral_conv(c["x"], c["layout"], c["coords"], c["row_of"], c["sp"],
                                      c["W"], None, oracle.ACT_NONE)
    dx, dW, _ = oracle.sparse_conv_bwd(c["x"], c["rb"], c["W"], ys, c["g"], oracle.ACT_NONE)
    yg = float(np.sum(y * c["g"]))
    assert abs(np.sum(c["x"].reshape(dx.shape).astype(np.float64) * dx) - yg) <= 1e-10 * abs(yg) + 1e-10
    assert abs(np.sum(c["W"].astype(np.float64) * dW) - yg) <= 1e-10 * abs(yg) + 1e-10


def test_bwd_adjoint_identity():
    check_bwd_adjoint_identity()
