"""Pins of the CPU oracle against things other than itself (CPU only).

Each test checks the oracle against what the paper or the mathematics fixes:
printed values of the Appendix A.1 microcase, library routines (torch's E4M3
cast, numpy's IEEE fp32 division and fp64 sums), closed forms, invariants the
paper states (h = 1 reduces to plain MSE search; the shift 0 is always in the
window so the chosen error never exceeds the initial one; a window covering the
ladder equals the full E4M3 grid), and brute force on tiny inputs written as a
different method (nearest-value search instead of midpoint comparisons).
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
E2M1_GRID = [0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0]  # OCP FP4 E2M1 magnitudes


def to_bf16_bits(a) -> np.ndarray:
    t = torch.as_tensor(np.asarray(a, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def bits_to_f64(b: np.ndarray) -> np.ndarray:
    return torch.from_numpy(b.view(np.int16).copy()).view(torch.bfloat16).double().numpy()


def random_weights(rng, m, n, sigma=0.02):
    w = rng.standard_t(4, size=(m, n)) * sigma
    k = max(1, int(round(1e-3 * m * n)))
    idx = rng.choice(m * n, size=k, replace=False)
    w.reshape(-1)[idx] *= 20
    return to_bf16_bits(w)


def random_h(rng, n):
    return (np.exp(rng.standard_normal(n)) ** 2 * 2048).astype(np.float32)


# ---------------------------------------------------------------- formats

def test_e4m3_table_matches_torch_view_cast():
    ours = oracle.e4m3_decode_table()
    ref = torch.arange(256, dtype=torch.uint8).view(torch.float8_e4m3fn).double().numpy()
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])
    assert list(np.nonzero(nan)[0]) == [0x7F, 0xFF]


def test_e4m3_ladder_shape():
    t = oracle.e4m3_decode_table()
    ladder = t[1:127]  # bytes 0x01..0x7E: the sorted positive finite values L+ (Eq. 8)
    assert ladder.size == 126
    assert np.all(np.diff(ladder) > 0)
    assert ladder[0] == 2.0 ** -9 and ladder[-1] == 448.0
    assert t[0] == 0.0


def test_e2m1_table_is_the_ocp_grid():
    t = oracle.e2m1_decode_table()
    assert list(t[:8]) == E2M1_GRID
    assert list(t[8:]) == [-v for v in E2M1_GRID]
    # the paper's Clip range and its outer codes {+-4, +-6} (Sec. 3.1, Sec. 3.3)
    assert t.max() == 6.0 and t.min() == -6.0 and 4.0 in t


def nearest_e2m1(a: float, s: float) -> int:
    """Brute force: nearest grid value to a/s by distance a - v*s; ties to even code."""
    d = [abs(a - v * s) for v in E2M1_GRID]
    best = min(d)
    ks = [k for k in range(8) if d[k] == best]
    return ks[0] if len(ks) == 1 else [k for k in ks if k % 2 == 0][0]


def test_e2m1_rounding_against_brute_force_including_midpoints():
    s = 0.8125  # exact binary scale so midpoints are exactly representable
    vals = []
    for i in range(1, 8):
        mid = 0.5 * (E2M1_GRID[i - 1] + E2M1_GRID[i]) * s
        vals += [mid, np.nextafter(mid, 0), np.nextafter(mid, 10)]
    vals += list(np.linspace(0, 9 * s, 997)) + [6 * s, 7 * s, 100.0, 0.0]
    w = np.array(vals + [-v for v in vals])
    _, codes = oracle.quantize_at_scale(w, s)
    expect = [nearest_e2m1(abs(v), s) for v in w]
    assert list(np.abs(codes)) == expect
    # ties go to the even code: 0.25->0, 0.75->1, 1.25->1, 1.75->2, 2.5->2, 3.5->4, 5->4
    ties = np.array([0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0]) * s
    _, c = oracle.quantize_at_scale(ties, s)
    assert [E2M1_GRID[k] for k in c] == [0.0, 1.0, 1.0, 2.0, 2.0, 4.0, 4.0]


# ---------------------------------------------------------------- microcase (App. A.1)

def test_calibration_microcase_from_the_paper():
    g = json.load(open(os.path.join(GOLDEN, "microcase.json")))
    w = np.array(g["w"])
    X = np.array(g["X"])
    for row in g["rows"]:
        s = np.abs(w).max() / 6.0 if row.get("scale_exact") == "max|w|/6" else row["scale"]
        w_hat, codes = oracle.quantize_at_scale(w, s)
        np.testing.assert_allclose(w_hat, row["w_hat"], atol=0.01)
        werr = oracle.output_error(np.eye(4), w - w_hat)        # sum_j (w_j - w_hat_j)^2
        oerr = oracle.output_error(X, w - w_hat)                # ||X (w - w_hat)^T||^2, Eq. 3
        assert abs(werr - row["weight_error"]) <= 0.01, row["name"]
        assert abs(oerr - row["output_error"]) <= 0.01, row["name"]
        if "codes" in row:
            signed = [np.sign(c) * E2M1_GRID[abs(c)] for c in codes]
            assert signed == row["codes"]
    # the min-max row is printed at its exact scale: 3 decimals agree exactly
    s = 4.88 / 6.0
    w_hat, _ = oracle.quantize_at_scale(w, s)
    assert round(oracle.output_error(np.eye(4), w - w_hat), 3) == 0.573
    assert round(oracle.output_error(X, w - w_hat), 3) == 3.927


# ---------------------------------------------------------------- Hessian diagonal (Eq. 4)

def test_hessian_constant_input_closed_form():
    for c in (0.5, -1.5, 3.0):
        x = to_bf16_bits(np.full((37, 48), c))
        h = np.zeros(48)
        oracle.hessian_accumulate(x, h)
        assert np.all(h == 37 * c * c)


def test_hessian_one_hot_rows_and_chunking():
    T, n = 50, 32
    x = np.zeros((T, n))
    cols = np.arange(T) % n
    x[np.arange(T), cols] = 2.0
    bits = to_bf16_bits(x)
    h = np.zeros(n)
    oracle.hessian_accumulate(bits[:17], h)  # two chunks accumulate into one h
    oracle.hessian_accumulate(bits[17:], h)
    expect = np.bincount(cols, minlength=n) * 4.0
    assert np.array_equal(h, expect)


def test_hessian_random_against_numpy_and_strided_rows():
    rng = np.random.default_rng(3)
    x = to_bf16_bits(rng.standard_normal((300, 80)) * np.exp(rng.standard_normal(80)))
    ref = (bits_to_f64(x) ** 2).sum(axis=0)
    h = np.zeros(80)
    oracle.hessian_accumulate(x, h)
    np.testing.assert_allclose(h, ref, rtol=1e-13)
    # leading dimension: use the first 48 columns of a wider buffer
    h2 = np.zeros(48)
    oracle.hessian_accumulate(x, h2, ld=80, n=48)
    np.testing.assert_allclose(h2, ref[:48], rtol=1e-13)


# ---------------------------------------------------------------- global scale and RTN codes

def test_global_scale_is_ieee_fp32_division():
    rng = np.random.default_rng(4)
    for _ in range(200):
        w = random_weights(rng, 4, 64, sigma=float(np.exp(rng.normal(-3, 2))))
        s, amax = oracle.global_scale(w)
        assert amax == np.abs(bits_to_f64(w)).max()
        assert s == np.float32(amax) / np.float32(2688.0)   # numpy: correctly rounded fp32
    s, amax = oracle.global_scale(np.zeros((2, 16), np.uint16))
    assert amax == 0.0 and s == np.float32(1.0)


def e4m3_code_by_torch(q: np.ndarray) -> np.ndarray:
    """torch's round-to-nearest-even E4M3 cast of float32 values (overflow -> NaN byte)."""
    return torch.from_numpy(q.astype(np.float32)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()


def test_rtn_codes_against_torch_cast_on_exact_quotients():
    # amax = 2688 * 2^-10 makes s_g = 2^-10 exactly; a group whose max is 6*v*2^-10 then has
    # the exact quotient v, so torch's cast of v is the E4M3 round-to-nearest-even of Eq. 7.
    ladder = oracle.e4m3_decode_table()[0:127]
    mids = 0.5 * (ladder[:-1] + ladder[1:])
    vs = [v for v in np.concatenate([ladder[1:], mids]) if v <= 448]
    rows = []
    for v in vs:
        g = np.zeros(16)
        g[3] = 6 * v * 2.0 ** -10
        rows.append(g)
    w = np.stack(rows).reshape(len(rows), 16)
    w[0, 0] = 2688 * 2.0 ** -10                          # sets amax, s_g = 2^-10
    bits = to_bf16_bits(w)
    assert np.array_equal(bits_to_f64(bits), w)          # all values are exact in bf16
    s_g, _ = oracle.global_scale(bits)
    assert s_g == np.float32(2.0 ** -10)
    codes = oracle.rtn_codes(bits, s_g).reshape(-1)
    amax_g = np.abs(w).max(axis=1)
    expect = e4m3_code_by_torch(amax_g / (6 * 2.0 ** -10))
    expect = np.maximum(expect, 1)                        # code 0 clamps to 1
    assert np.array_equal(codes, expect)


def test_rtn_codes_against_torch_cast_on_random_groups():
    rng = np.random.default_rng(5)
    w = random_weights(rng, 64, 256)
    s_g, _ = oracle.global_scale(w)
    codes = oracle.rtn_codes(w, s_g)
    amax_g = np.abs(bits_to_f64(w)).reshape(64, 16, 16).max(axis=2)
    q = amax_g / (6.0 * float(s_g))
    expect = np.maximum(e4m3_code_by_torch(q), 1)
    expect = np.where(expect == 127, 126, expect)         # saturate instead of NaN
    assert np.array_equal(codes, expect)
    assert codes.max() == 126                             # the group holding amax hits 448


# ---------------------------------------------------------------- scale search (Algorithm 1)

def brute_force_group(g_bits, h, s_g, c0, down, up):
    """Algorithm 1 by brute force: nearest-value FP4 search, exhaustive window, tie rule
    (E, |shift|, shift).  Returns (best code, magnitude codes, errors by code)."""
    a = np.abs(bits_to_f64(g_bits))
    ladder = oracle.e4m3_decode_table()
    errs = {}
    for d in range(-down, up + 1):
        c = min(max(c0 + d, 1), 126)
        if c in errs:
            continue
        s = float(s_g) * ladder[c]
        ks = [nearest_e2m1(v, s) for v in a]
        errs[c] = (math.fsum((1.0 if h is None else float(h[j])) * (a[j] - E2M1_GRID[ks[j]] * s) ** 2
                             for j in range(16)), ks)
    best = min(errs, key=lambda c: (errs[c][0], abs(c - c0), c - c0))
    return best, errs[best][1], {c: e for c, (e, _) in errs.items()}


def test_refine_matches_brute_force_on_tiny_inputs():
    rng = np.random.default_rng(6)
    checked = 0
    for trial in range(6):
        m, n = 4, 64
        w = random_weights(rng, m, n)
        h = random_h(rng, n)
        down, up = [(4, 4), (9, 6), (2, 7), (0, 3), (5, 0), (1, 1)][trial]
        s_g, _ = oracle.global_scale(w)
        out = oracle.refine(w, h, s_g, None, down, up)
        rtn = oracle.rtn_codes(w, s_g)
        for r in range(m):
            for i in range(n // 16):
                g = w[r, 16 * i:16 * i + 16]
                best, ks, errs = brute_force_group(g, h[16 * i:16 * i + 16], s_g, int(rtn[r, i]),
                                                   down, up)
                assert math.isclose(out["e_best"][r, i], errs[best], rel_tol=1e-12)
                assert math.isclose(out["e_init"][r, i], errs[int(rtn[r, i])], rel_tol=1e-12)
                if out["near_tie"][r, i]:
                    continue
                assert out["codes"][r, i] == best
                assert out["delta"][r, i] == best - int(rtn[r, i])
                signs = (g >> 15).astype(np.uint8)
                nib = (signs << 3) | np.array(ks, np.uint8)
                assert np.array_equal(out["packed"][r, 8 * i:8 * i + 8], nib[0::2] | (nib[1::2] << 4))
                checked += 1
    assert checked > 80


def test_h_one_reduces_to_plain_mse_search():
    rng = np.random.default_rng(7)
    w = random_weights(rng, 8, 128)
    s_g, _ = oracle.global_scale(w)
    a = oracle.refine(w, None, s_g, None, 4, 4)
    b = oracle.refine(w, np.ones(128, np.float32), s_g, None, 4, 4)
    for k in ("codes", "packed", "e_best"):
        assert np.array_equal(a[k], b[k])
    rtn = oracle.rtn_codes(w, s_g)
    for r in range(8):
        for i in range(8):
            g = w[r, 16 * i:16 * i + 16]
            best, _, _ = brute_force_group(g, None, s_g, int(rtn[r, i]), 4, 4)
            if not a["near_tie"][r, i]:
                assert a["codes"][r, i] == best


def test_chosen_error_never_exceeds_initial_error():
    rng = np.random.default_rng(8)
    w = random_weights(rng, 32, 256)
    h = random_h(rng, 256)
    s_g, _ = oracle.global_scale(w)
    for down, up in ((4, 4), (9, 6), (0, 0), (16, 16)):
        out = oracle.refine(w, h, s_g, None, down, up)
        assert np.all(out["e_best"] <= out["e_init"])
        assert np.all(out["delta"] >= -down) and np.all(out["delta"] <= up)
        assert out["codes"].min() >= 1 and out["codes"].max() <= 126
    out = oracle.refine(w, h, s_g, None, 0, 0)
    assert np.array_equal(out["codes"], oracle.rtn_codes(w, s_g))   # empty window = RTN


def test_full_window_equals_full_e4m3_grid():
    rng = np.random.default_rng(9)
    w = random_weights(rng, 6, 64)
    h = random_h(rng, 64)
    s_g, _ = oracle.global_scale(w)
    small = oracle.refine(w, h, s_g, None, 4, 4)
    full = oracle.refine(w, h, s_g, None, 125, 125)
    assert np.all(full["e_best"] <= small["e_best"])
    all_codes = np.arange(1, 127, dtype=np.uint8)
    for r in range(6):
        for i in range(4):
            errs = oracle.group_errors(w[r, 16 * i:16 * i + 16], h[16 * i:16 * i + 16], s_g, all_codes)
            assert full["e_best"][r, i] == errs.min()
            if not full["near_tie"][r, i]:
                assert full["codes"][r, i] == all_codes[np.argmin(errs)]


def test_codes_invariant_under_h_power_of_two_scaling_and_row_permutation():
    rng = np.random.default_rng(10)
    w = random_weights(rng, 16, 128)
    h = random_h(rng, 128)
    s_g, _ = oracle.global_scale(w)
    base = oracle.refine(w, h, s_g, None, 4, 4)
    for k in (-7, 3, 20):
        other = oracle.refine(w, (h * np.float32(2.0 ** k)).astype(np.float32), s_g, None, 4, 4)
        assert np.array_equal(base["codes"], other["codes"])
        assert np.array_equal(base["packed"], other["packed"])
    perm = rng.permutation(16)
    other = oracle.refine(w[perm], h, s_g, None, 4, 4)
    assert np.array_equal(base["codes"][perm], other["codes"])
    assert np.array_equal(base["packed"][perm], other["packed"])


def test_init_codes_path_and_window_clipping_at_both_ends():
    rng = np.random.default_rng(11)
    w = random_weights(rng, 8, 64)
    h = random_h(rng, 64)
    s_g, _ = oracle.global_scale(w)
    rtn = oracle.rtn_codes(w, s_g)
    a = oracle.refine(w, h, s_g, None, 4, 4)
    b = oracle.refine(w, h, s_g, rtn, 4, 4)
    for k in a:
        assert np.array_equal(a[k], b[k])
    # init codes at the ladder ends: the walk clips to [1, 126]
    lo = np.ones_like(rtn)
    hi = np.full_like(rtn, 126)
    out_lo = oracle.refine(w, h, s_g, lo, 4, 4)
    out_hi = oracle.refine(w, h, s_g, hi, 4, 4)
    assert out_lo["codes"].max() <= 5 and out_lo["delta"].min() >= 0
    assert out_hi["codes"].min() >= 122 and out_hi["delta"].max() <= 0


def test_pack_matches_refine_and_decodes_to_the_quantized_weights():
    rng = np.random.default_rng(12)
    w = random_weights(rng, 8, 96)
    h = random_h(rng, 96)
    s_g, _ = oracle.global_scale(w)
    out = oracle.refine(w, h, s_g, None, 4, 4)
    packed = oracle.pack(w, s_g, out["codes"])
    assert np.array_equal(packed, out["packed"])
    # decode: nibble value * s_g * lambda(code) is the FP4 projection of w (Eq. 12)
    e2 = oracle.e2m1_decode_table()
    e4 = oracle.e4m3_decode_table()
    lo, hi = packed & 15, packed >> 4
    nib = np.empty((8, 96), np.uint8)
    nib[:, 0::2], nib[:, 1::2] = lo, hi
    scale = float(s_g) * e4[np.repeat(out["codes"], 16, axis=1)]
    wq = e2[nib] * scale
    wf = bits_to_f64(w)
    for r in range(8):
        for j in range(96):
            k = nearest_e2m1(abs(wf[r, j]), scale[r, j])
            assert abs(wq[r, j]) == E2M1_GRID[k] * scale[r, j]
            assert (nib[r, j] >> 3) == (w[r, j] >> 15)


def test_zero_groups_and_negative_zero():
    w = np.zeros((2, 32))
    w[1, 20] = 0.5                                           # second group of row 1 non-zero
    bits = to_bf16_bits(w)
    bits[0, 5] = 0x8000                                      # -0.0
    s_g, _ = oracle.global_scale(bits)
    out = oracle.refine(bits, None, s_g, None, 4, 4)
    # all-zero groups: every candidate has E = 0, the tie rule keeps the RTN code (1)
    assert out["codes"][0, 0] == 1 and out["delta"][0, 0] == 0 and out["near_tie"][0, 0] == 1
    assert out["packed"][0, 2] == 0x80                       # -0 (odd element: high nibble) keeps its sign
    assert out["codes"][1, 1] == 126 or out["e_best"][1, 1] == 0.0


# ---------------------------------------------------------------- Algorithm 2 (4over6 initialization)

def brute_force_fourover6(g_bits, s_g):
    """Algorithm 2's initialization by brute force: torch's E4M3 cast of the fp64 quotient
    (valid away from midpoints), nearest-value FP4 search, anchors in the order 4, 6."""
    a = np.abs(bits_to_f64(g_bits))
    mx = a.max()
    ladder = oracle.e4m3_decode_table()
    best = None
    for c in (4.0, 6.0):
        q = mx / (c * float(s_g))
        code = int(e4m3_code_by_torch(np.array([q]))[0])
        code = 126 if code == 127 else max(code, 1)
        s = float(s_g) * ladder[code]
        err = math.fsum((v - E2M1_GRID[nearest_e2m1(v, s)] * s) ** 2 for v in a)
        if best is None or err < best[1]:
            best = (code, err)
    return best[0]


def test_fourover6_codes_against_brute_force_and_rtn():
    rng = np.random.default_rng(13)
    w = random_weights(rng, 16, 256)
    s_g, _ = oracle.global_scale(w)
    codes, nt = oracle.fourover6_codes(w, s_g)
    rtn = oracle.rtn_codes(w, s_g)
    for r in range(16):
        for i in range(16):
            if nt[r, i]:
                continue
            assert codes[r, i] == brute_force_fourover6(w[r, 16 * i:16 * i + 16], s_g)
    # the anchor 6 is the RTN code of Eq. 7; 4over6 never has a larger MSE than RTN
    e_fo6 = oracle.refine(w, None, s_g, codes, 0, 0)["e_best"]
    e_rtn = oracle.refine(w, None, s_g, rtn, 0, 0)["e_best"]
    assert np.all(e_fo6 <= e_rtn * (1 + 1e-12))
    assert (codes != rtn).any() and (codes == rtn).any()


def test_fourover6_saturated_group_keeps_the_top_code():
    # the group holding amax: m/(6 s_g) = 448 and m/(4 s_g) = 672 both saturate to 448
    w = np.zeros((1, 32))
    w[0, 5] = 2688 * 2.0 ** -10
    w[0, 20] = 0.01
    bits = to_bf16_bits(w)
    s_g, _ = oracle.global_scale(bits)
    codes, nt = oracle.fourover6_codes(bits, s_g)
    assert codes[0, 0] == 126 and nt[0, 0] == 0


# ---------------------------------------------------------------- residual and output error (Eq. 3)

def test_dequant_residual_against_nearest_grid_value():
    """dW = W - W_hat, with W_hat found by a brute-force nearest-grid search per element (a
    different method from the oracle's decode of the packed nibbles), for RTN codes and for
    arbitrary codes (off-ladder bytes are clipped, Eq. 10); -0 stays a zero residual."""
    rng = np.random.default_rng(31)
    w = random_weights(rng, 8, 64)
    w[0, :16] = 0x8000                                   # -0
    s_g, _ = oracle.global_scale(w)
    ladder = oracle.e4m3_decode_table()
    wv = bits_to_f64(w)
    for codes in (oracle.rtn_codes(w, s_g), rng.integers(0, 256, size=(8, 4)).astype(np.uint8)):
        packed = oracle.pack(w, s_g, codes)
        dw = oracle.dequant_residual(w, s_g, codes, packed)
        for r in range(8):
            for i in range(4):
                c = min(max(int(codes[r, i]) & 0x7F, 1), 126)
                s = float(s_g) * ladder[c]
                for j in range(16):
                    v = wv[r, 16 * i + j]
                    k = nearest_e2m1(abs(v), s)
                    w_hat = math.copysign(E2M1_GRID[k] * s, v) if k else 0.0
                    assert dw[r, 16 * i + j] == v - w_hat, (r, i, j)
    assert np.all(dw[0, :16] == 0.0)


def test_output_error_closed_forms():
    """||X dW^T||_F^2: X = I gives ||dW||_F^2; one-hot rows scaled by c give
    c^2 * sum over the selected columns of the column energies; E scales with c^2."""
    rng = np.random.default_rng(32)
    m, n = 5, 24
    dW = rng.standard_normal((m, n))
    assert math.isclose(oracle.output_error(np.eye(n), dW), math.fsum((dW ** 2).ravel()), rel_tol=1e-12)
    cols = rng.integers(0, n, size=9)
    X = np.zeros((9, n))
    X[np.arange(9), cols] = 3.0
    expect = 9.0 * math.fsum(math.fsum(dW[:, j] ** 2) for j in cols)
    assert math.isclose(oracle.output_error(X, dW), expect, rel_tol=1e-12)
    Xr = rng.standard_normal((7, n))
    assert math.isclose(oracle.output_error(2.0 * Xr, dW), 4.0 * oracle.output_error(Xr, dW), rel_tol=1e-12)


# ---------------------------------------------------------------- GPTQ + H-Scale (Algorithm 3)

def test_full_hessian_diagonal_symmetry_and_closed_form():
    rng = np.random.default_rng(41)
    x = to_bf16_bits(rng.standard_normal((37, 24)) * 2.0)
    H = np.zeros((24, 24))
    oracle.hessian_full(x, H)
    h = np.zeros(24)
    oracle.hessian_accumulate(x, h)
    assert np.array_equal(np.diag(H), h)          # the diagonal is Eq. 4's h
    assert np.array_equal(H, H.T)
    onehot = np.zeros((5, 24))
    onehot[np.arange(5), [3, 3, 7, 10, 3]] = 2.0
    H1 = np.zeros((24, 24))
    oracle.hessian_full(to_bf16_bits(onehot), H1)
    expect = np.zeros((24, 24))
    expect[3, 3], expect[7, 7], expect[10, 10] = 12.0, 4.0, 4.0
    assert np.array_equal(H1, expect)


def test_gptq_factor_inverts_the_damped_hessian():
    rng = np.random.default_rng(42)
    X = rng.standard_normal((64, 32))
    X[:, 5] = 0.0                                   # a dead input channel
    H = X.T @ X
    U, dead = oracle.gptq_factor(H, damp=0.01)
    assert dead[5] and dead.sum() == 1
    Hd = H.copy()
    Hd[5, 5] = 1.0
    Hd[np.diag_indices(32)] += 0.01 * np.mean(np.diag(Hd))
    assert np.allclose(np.triu(U), U) and np.all(np.diag(U) > 0)
    assert np.allclose(Hd @ (U.T @ U), np.eye(32), atol=1e-9)


def test_gptq_one_block_equals_the_search_and_fp64_path_equals_bf16_path():
    rng = np.random.default_rng(43)
    w = random_weights(rng, 8, 64)
    h = random_h(rng, 64)
    s_g, _ = oracle.global_scale(w)
    U = np.triu(rng.standard_normal((64, 64))) + 8 * np.eye(64)
    out = oracle.gptq_hscale(w, U, h, s_g, 64, 4, 4)
    ref = oracle.refine(w, h, s_g, None, 4, 4)
    assert np.array_equal(out["codes"], ref["codes"]) and np.array_equal(out["packed"], ref["packed"])


def test_gptq_diagonal_factor_does_not_propagate():
    rng = np.random.default_rng(44)
    w = random_weights(rng, 8, 64)
    h = random_h(rng, 64)
    s_g, _ = oracle.global_scale(w)
    U = np.diag(rng.uniform(0.5, 2.0, 64))
    out = oracle.gptq_hscale(w, U, h, s_g, 16, 9, 6)
    ref = oracle.refine(w, h, s_g, None, 9, 6)
    assert np.array_equal(out["codes"], ref["codes"]) and np.array_equal(out["packed"], ref["packed"])


def brute_force_block(Wb, hb, s_g, down, up):
    """Brute-force H-Scale on real-valued rows: RTN start by torch's E4M3 cast, every code in
    the window, nearest-grid FP4 values, math.fsum errors, the tie rule of the search."""
    ladder = oracle.e4m3_decode_table()
    codes, w_hat = [], np.zeros_like(Wb)
    for r in range(Wb.shape[0]):
        row = []
        for i in range(Wb.shape[1] // 16):
            g = Wb[r, 16 * i:16 * i + 16]
            hg = hb[16 * i:16 * i + 16]
            c0 = max(1, min(126, int(e4m3_code_by_torch(np.array([np.abs(g).max() / (6 * float(s_g))]))[0])))
            best = None
            for d in range(-down, up + 1):
                c = min(max(c0 + d, 1), 126)
                s = float(s_g) * ladder[c]
                q = [E2M1_GRID[nearest_e2m1(abs(v), s)] * s for v in g]
                e = math.fsum(float(hj) * (abs(v) - qv) ** 2 for v, hj, qv in zip(g, hg, q))
                key = (e, abs(c - c0), c - c0)
                if best is None or key < best[0]:
                    best = (key, c, q)
            row.append(best[1])
            w_hat[r, 16 * i:16 * i + 16] = [math.copysign(qv, v) if qv else 0.0 for v, qv in zip(g, best[2])]
        codes.append(row)
    return np.array(codes, np.uint8), w_hat


def test_gptq_error_propagation_against_brute_force():
    """Three blocks of 16 columns: every block quantized by brute force on the running
    weights, E = (W_b - W_hat_b) / U_jj and the later columns updated element by element."""
    rng = np.random.default_rng(45)
    m, n, B = 4, 48, 16
    w = random_weights(rng, m, n)
    X = rng.standard_normal((96, n)) * np.exp(rng.standard_normal(n))
    H = X.T @ X
    h = np.diag(H).astype(np.float32)
    s_g, _ = oracle.global_scale(w)
    U, dead = oracle.gptq_factor(H)
    out = oracle.gptq_hscale(w, U, h, s_g, B, 2, 2, dead=dead)
    W = bits_to_f64(w).copy()
    for i in range(0, n, B):
        codes, w_hat = brute_force_block(W[:, i:i + B], h[i:i + B], s_g, 2, 2)
        keep = out["near_tie"][:, i // 16:(i + B) // 16] == 0
        assert np.array_equal(codes[keep], out["codes"][:, i // 16:(i + B) // 16][keep]), i
        for r in range(m):
            for j in range(i + B, n):
                W[r, j] -= math.fsum((W[r, i + k] - w_hat[r, k]) / U[i + k, i + k] * U[i + k, j]
                                     for k in range(B))
