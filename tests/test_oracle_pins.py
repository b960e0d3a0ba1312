"""Pins of the CPU oracle to facts outside itself (no GPU).

Each test ties one oracle function to something the paper or mathematics fixes: a
hand-worked example (tests/golden), a published generator output, exact rational
arithmetic on tiny inputs, a closed-form bound or a special case that reduces to a
textbook routine.  A dropped term, a flipped sign, a wrong index or a transposed
operand anywhere in the oracle fails at least one of them.
"""
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle as O

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    lines = [l.split("#")[0].strip() for l in open(os.path.join(GOLD, name))]
    return [l for l in lines if l]


def _parse_worked():
    toks = _read_golden("worked_example_g4_b4.txt")
    out, i = {}, 0
    while i < len(toks):
        head = toks[i].split()
        key = head[0]
        if key in ("x", "codes", "w", "wcodes", "T"):
            r, c = int(head[1]), int(head[2])
            rows = [[float(v) for v in toks[i + 1 + k].split()] for k in range(r)]
            out[key] = np.array(rows)
            i += 1 + r
        else:
            out[key] = [float(v) for v in head[1:]]
            i += 1
    return out


# ------------------------------------------------------------------ hash pins
def test_splitmix64_published_outputs():
    # Steele/Lea/Flood SplitMix64, reference outputs for state 0 (golden file cites them)
    for line in _read_golden("splitmix64_seed0.txt"):
        idx, hx = line.split()
        assert O.hash64(0, int(idx)) == int(hx, 16)


def test_hash_counter_and_seed_are_additive_state():
    # the (idx+1)-th output under seed s equals the 1st output under seed s + idx*golden
    g = 0x9E3779B97F4A7C15
    for s, i in [(0, 5), (123, 77), (2**63 + 5, 1 << 40)]:
        assert O.hash64(s, i) == O.hash64((s + i * g) % 2**64, 0)


# -------------------------------------------------------------- worked example
def test_worked_example_by_hand():
    ex = _parse_worked()
    bits, G = int(ex["bits"][0]), int(ex["groups"][0])
    x = ex["x"].astype(np.float32)
    d = O.shiftquant_tensor(x, bits, G, mode=0)
    assert d["status"] == 0
    np.testing.assert_array_equal(d["range"], np.array(ex["range"], np.float32))
    assert float(d["tau0"]) == ex["tau0"][0]
    np.testing.assert_array_equal(d["exp"], np.array(ex["exp"], np.uint8))
    np.testing.assert_array_equal(d["codes"], ex["codes"].astype(np.int8))
    w = O.channel_tensor(ex["w"].astype(np.float32), bits, axis=0)
    np.testing.assert_array_equal(w["codes"], ex["wcodes"].astype(np.int8))
    T = O.gemm_fwd(d["codes"], d["exp"], w["codes"], G)
    np.testing.assert_array_equal(T, ex["T"].astype(np.int64))
    Y = O.dequant(T, d["scale"], 1.0, G - 1, w["scale"])
    np.testing.assert_allclose(Y, ex["T"] / ex["y_over"][0], rtol=2e-7)


# ------------------------------------------------------------- grouping (Eq. 3)
def _floor_log2_ratio_exact(tau0, r, G):
    """Brute force: the largest e in [0, G-1] with r * 2^e <= tau0, in rationals."""
    if r == 0:
        return G - 1
    t, rr = Fraction(float(tau0)), Fraction(float(r))
    e = 0
    while e + 1 <= G - 1 and rr * 2 ** (e + 1) <= t:
        e += 1
    return e


def _boundary_ranges(rng, tau0):
    vals = [tau0, 0.0, np.float32(1e-45), np.float32(1.2e-38)]
    for k in range(0, 10):
        b = np.float32(tau0 * 2.0 ** -k)
        vals += [b, np.nextafter(b, np.float32(0)), np.nextafter(b, np.float32(np.inf))]
    vals += list((tau0 * rng.random(200) ** 6).astype(np.float32))
    vals = np.array(vals, np.float32)
    return np.minimum(vals, np.float32(tau0))


@pytest.mark.parametrize("G", [1, 2, 3, 4, 6, 8])
@pytest.mark.parametrize("tau0", [np.float32(8.0), np.float32(3.3e-3), np.float32(7.1e37),
                                  np.float32(1e-30)])
def test_grouping_matches_exact_rational_brute_force(G, tau0):
    rng = np.random.default_rng(G)
    r = _boundary_ranges(rng, tau0)
    t, e, st = O.group(r, G)
    assert st == 0 and t == tau0
    for ri, ei in zip(r, e):
        assert ei == _floor_log2_ratio_exact(tau0, ri, G), (ri, ei)


def test_grouping_threshold_invariant():
    # tau_0 2^-(e+1) < r <= tau_0 2^-e for e < G-1 and r <= tau_0 2^-(G-1) otherwise
    rng = np.random.default_rng(7)
    r = (rng.lognormal(0, 3, 5000)).astype(np.float32)
    G = 4
    t, e, _ = O.group(r, G)
    t = float(t)
    for ri, ei in zip(r.astype(float), e):
        assert ri <= t * 2.0 ** -int(ei)
        if ei < G - 1:
            assert ri > t * 2.0 ** -(int(ei) + 1)


def test_grouping_nonfinite_sets_status():
    r = np.array([1.0, np.inf, 2.0], np.float32)
    t, e, st = O.group(r, 4)
    assert st == 1 and np.isinf(t) and (e == 0).all()
    r = np.array([1.0, np.nan, np.inf], np.float32)
    t, e, st = O.group(r, 4)
    assert st == 1 and np.isnan(t)
    x = np.ones((3, 3), np.float32)
    x[1, 2] = np.nan
    rg, st = O.range_cols(x)
    assert st == 1 and np.isnan(rg[2]) and rg[0] == 1


def test_ranges_are_max_abs():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((37, 29)).astype(np.float32)
    rc, _ = O.range_cols(x)
    rr, _ = O.range_rows(x)
    np.testing.assert_array_equal(rc, np.abs(x).max(0))
    np.testing.assert_array_equal(rr, np.abs(x).max(1))


# ------------------------------------------------------- quantizer (App. D)
def _gradient_like(rng, R, C):
    scale = np.exp(rng.normal(0, 1.5, C)).astype(np.float32)
    scale[rng.random(C) < 0.02] *= 100
    return (rng.standard_normal((R, C)) * scale).astype(np.float32)


@pytest.mark.parametrize("bits", [2, 4, 6, 8])
@pytest.mark.parametrize("G", [1, 2, 4, 6])
def test_rn_error_at_most_half_group_step(bits, G):
    rng = np.random.default_rng(bits * 10 + G)
    x = _gradient_like(rng, 64, 48)
    x[:, 5] = 0
    d = O.shiftquant_tensor(x, bits, G, mode=0)
    Q = 2 ** (bits - 1) - 1
    q = d["codes"].astype(np.int64)
    assert np.abs(q).max() <= Q
    step = float(d["scale"]) * 2.0 ** -d["exp"].astype(np.float64)   # s * 2^-e per channel
    err = np.abs(x.astype(np.float64) - q * step[None, :])
    assert (err <= step[None, :] * (0.5 + 2.0 ** -15)).all()
    # the element attaining tau_0 uses the full code range
    i, j = np.unravel_index(np.argmax(np.abs(x)), x.shape)
    assert abs(int(q[i, j])) == Q
    assert (q[:, 5] == 0).all()


def test_group_steps_are_power_of_two_related():
    # App. B: s_i in {s_l, 2 s_l, ..., 2^(G-1) s_l}
    rng = np.random.default_rng(11)
    x = _gradient_like(rng, 32, 200)
    G = 4
    d = O.shiftquant_tensor(x, 6, G)
    steps = float(d["scale"]) * 2.0 ** -d["exp"].astype(np.float64)
    s_l = steps.min()
    ratios = steps / s_l
    assert set(np.unique(ratios)).issubset({1.0, 2.0, 4.0, 8.0})


def test_shiftquant_reduces_to_per_tensor_at_one_group():
    # N_G = 1 is the paper's per-tensor baseline: one scale tau_0/Q for the whole tensor,
    # i.e. per-channel quantization of the flattened tensor seen as a single channel.
    rng = np.random.default_rng(5)
    x = _gradient_like(rng, 40, 30)
    d = O.shiftquant_tensor(x, 8, 1)
    assert (d["exp"] == 0).all()
    flat = O.channel_tensor(x.reshape(-1, 1), 8, axis=0)
    np.testing.assert_array_equal(d["codes"].reshape(-1, 1), flat["codes"])
    assert d["scale"] == flat["scale"][0]


def test_zero_tensor_and_tiny_tau():
    x = np.zeros((4, 4), np.float32)
    d = O.shiftquant_tensor(x, 4, 4)
    assert d["tau0"] == 0 and d["scale"] == 0 and (d["codes"] == 0).all()
    assert (d["exp"] == 3).all()
    x[0, 0] = np.float32(1e-45)     # Q / tau_0 overflows: every code is 0
    d = O.shiftquant_tensor(x, 4, 4)
    assert d["scale"] == 0 and (d["codes"] == 0).all()


def test_sr_codes_are_neighbouring_levels_and_unbiased():
    # App. B: SR picks u(x) with probability (x - l)/(u - l); E[q] = v, Var = (v-l)(u-v)
    R = 20000
    vals = np.array([0.3, -2.75, 1.5, 5.9, -0.01, 6.0], np.float32)
    x = np.tile(vals, (R, 1))
    x[0, :] = 7.0        # pins tau_0 = 7 so that Q/tau_0 = 1 for 4 bits (v == x)
    d = O.shiftquant_tensor(x, 4, 1, mode=1, seed=1234)
    q = d["codes"][1:].astype(np.float64)
    v = vals.astype(np.float64)
    lo = np.floor(v)
    assert np.isin(q - lo[None, :], [0.0, 1.0]).all()
    n = q.shape[0]
    var = (v - lo) * (lo + 1 - v)
    mean = q.mean(0)
    assert (np.abs(mean - v) <= 5 * np.sqrt(var / n) + 1e-12).all()
    emp = q.var(0)
    assert (np.abs(emp - var) <= 0.05 * var + 1e-9).all()


def test_sr_depends_on_seed_and_position_only():
    rng = np.random.default_rng(2)
    x = _gradient_like(rng, 16, 16)
    a = O.shiftquant_tensor(x, 4, 4, mode=1, seed=9)["codes"]
    b = O.shiftquant_tensor(x, 4, 4, mode=1, seed=9)["codes"]
    c = O.shiftquant_tensor(x, 4, 4, mode=1, seed=10)["codes"]
    np.testing.assert_array_equal(a, b)
    assert (a != c).any()


def test_variance_upper_bound_of_app_b():
    # U_dq <= 4 U_fq + 2^(-2 N_G + 2) U_cq with U = sum over elements of step^2 / 4
    rng = np.random.default_rng(4)
    for G in (1, 2, 3, 4, 5):
        x = _gradient_like(rng, 8, 300)
        d = O.shiftquant_tensor(x, 4, G)
        Q = 7
        N = x.shape[0]
        step = float(d["scale"]) * 2.0 ** -d["exp"].astype(np.float64)
        U_dq = N * np.sum(step ** 2) / 4
        U_fq = N * np.sum((d["range"].astype(np.float64) / Q) ** 2) / 4
        U_cq = N * x.shape[1] * (float(d["tau0"]) / Q) ** 2 / 4
        assert U_dq <= 4 * U_fq + 2.0 ** (-2 * G + 2) * U_cq * (1 + 1e-12)


# ---------------------------------------------------- contraction (Eq. 4, App. D)
def _tiny_layer(rng, M, K, N, bits, G):
    x = _gradient_like(rng, M, K)
    w = (rng.standard_normal((K, N)) * 0.02).astype(np.float32)
    dy = _gradient_like(rng, M, N)
    return x, w, dy


def _frac_matmul(a, b):
    M, K = len(a), len(a[0])
    N = len(b[0])
    return [[sum((a[m][k] * b[k][n] for k in range(K)), Fraction(0)) for n in range(N)]
            for m in range(M)]


@pytest.mark.parametrize("bits,G", [(4, 4), (6, 4), (8, 4), (4, 1), (6, 3), (8, 6)])
def test_fwd_equals_dequantize_then_exact_matmul(bits, G):
    rng = np.random.default_rng(bits * 7 + G)
    M, K, N = 5, 7, 6
    x, w, _ = _tiny_layer(rng, M, K, N, bits, G)
    a = O.shiftquant_tensor(x, bits, G)
    b = O.channel_tensor(w, bits, axis=0)
    T = O.gemm_fwd(a["codes"], a["exp"], b["codes"], G)
    # dequantized operands as exact rationals: x_hat = q s 2^-e, w_hat = q s_W[n]
    s = Fraction(float(a["scale"]))
    xh = [[Fraction(int(a["codes"][m, k])) * s / 2 ** int(a["exp"][k]) for k in range(K)]
          for m in range(M)]
    wh = [[Fraction(int(b["codes"][k, n])) * Fraction(float(b["scale"][n]))
           for n in range(N)] for k in range(K)]
    ref = _frac_matmul(xh, wh)
    for m in range(M):
        for n in range(N):
            # Eq. 4 right-shift form: s_G s_W sum_g [partial_g >> g]  ==  T 2^-(G-1) s s_W
            exact = Fraction(int(T[m, n])) * s / 2 ** (G - 1) * Fraction(float(b["scale"][n]))
            assert exact == ref[m][n]
    Y = O.dequant(T, a["scale"], 1.0, G - 1, b["scale"])
    for m in range(M):
        for n in range(N):
            assert float(Y[m, n]) == float(np.float32(float(ref[m][n])))


@pytest.mark.parametrize("bits,G", [(4, 4), (6, 4), (8, 2)])
def test_dgrad_equals_dequantize_then_exact_matmul(bits, G):
    rng = np.random.default_rng(100 + bits * 7 + G)
    M, K, N = 6, 5, 7          # dX [M, K] = dY [M, N] W^T, W [K, N]
    _, w, dy = _tiny_layer(rng, M, K, N, bits, G)
    a = O.shiftquant_tensor(dy, bits, G, mode=1, seed=3)
    b = O.channel_tensor(w, bits, axis=1)
    T = O.gemm_dgrad(a["codes"], a["exp"], b["codes"], G)
    assert T.shape == (M, K)
    s = Fraction(float(a["scale"]))
    for m in range(M):
        for k in range(K):
            ref = sum((Fraction(int(a["codes"][m, j])) * s / 2 ** int(a["exp"][j]) *
                       Fraction(int(b["codes"][k, j])) * Fraction(float(b["scale"][k]))
                       for j in range(N)), Fraction(0))
            assert Fraction(int(T[m, k])) * s / 2 ** (G - 1) * \
                Fraction(float(b["scale"][k])) == ref


@pytest.mark.parametrize("bits,G", [(4, 4), (6, 4), (8, 4)])
def test_wgrad_equals_dequantize_then_exact_matmul(bits, G):
    rng = np.random.default_rng(200 + bits * 7 + G)
    M, K, N = 9, 5, 4          # dW [K, N] = X^T [K, M] dY [M, N]
    x, _, dy = _tiny_layer(rng, M, K, N, bits, G)
    a = O.shiftquant_tensor(x, bits, G)
    c = O.shiftquant_tensor(dy, bits, G, mode=1, seed=8)
    T = O.gemm_wgrad(a["codes"], a["exp"], c["codes"], c["exp"], G)
    assert T.shape == (K, N)
    sa, sc = Fraction(float(a["scale"])), Fraction(float(c["scale"]))
    for i in range(K):
        for j in range(N):
            ref = sum((Fraction(int(a["codes"][m, i])) * sa / 2 ** int(a["exp"][i]) *
                       Fraction(int(c["codes"][m, j])) * sc / 2 ** int(c["exp"][j])
                       for m in range(M)), Fraction(0))
            assert Fraction(int(T[i, j])) * sa * sc / 2 ** (2 * (G - 1)) == ref
    # the two-scale dequantization (App. D with both operands ShiftQuant-ed): Y is the
    # exact rational T s_X s_dY 2^-2(G-1) rounded to binary64 once (s_X s_dY is exact
    # there) and then to binary32
    Y = O.dequant(T, a["scale"], c["scale"], 2 * (G - 1))
    for i in range(K):
        for j in range(N):
            exact = Fraction(int(T[i, j])) * sa * sc / 2 ** (2 * (G - 1))
            assert float(Y[i, j]) == float(np.float32(float(exact))), (i, j)


def test_int8_per_tensor_special_case_is_plain_integer_gemm():
    # b = 8, N_G = 1: the paper's 8-bit per-tensor baseline; every shift is zero
    rng = np.random.default_rng(21)
    x, w, dy = _tiny_layer(rng, 33, 17, 11, 8, 1)
    a = O.shiftquant_tensor(x, 8, 1)
    g = O.shiftquant_tensor(dy, 8, 1)
    wf = O.channel_tensor(w, 8, axis=0)
    wd = O.channel_tensor(w, 8, axis=1)
    A, Gc = a["codes"].astype(np.int64), g["codes"].astype(np.int64)
    np.testing.assert_array_equal(O.gemm_fwd(a["codes"], a["exp"], wf["codes"], 1),
                                  A @ wf["codes"].astype(np.int64))
    np.testing.assert_array_equal(O.gemm_dgrad(g["codes"], g["exp"], wd["codes"], 1),
                                  Gc @ wd["codes"].astype(np.int64).T)
    np.testing.assert_array_equal(O.gemm_wgrad(a["codes"], a["exp"], g["codes"], g["exp"], 1),
                                  A.T @ Gc)


def test_shift_is_per_inner_index_group():
    # one channel moved to another group changes exactly its own term by a power of two
    qA = np.array([[3, -2, 5]], np.int8)
    qW = np.array([[1], [4], [-1]], np.int8)
    e0 = np.array([0, 1, 2], np.uint8)
    e1 = np.array([0, 2, 2], np.uint8)
    T0 = int(O.gemm_fwd(qA, e0, qW, 3)[0, 0])
    T1 = int(O.gemm_fwd(qA, e1, qW, 3)[0, 0])
    assert T0 == 3 * 1 * 4 + (-2) * 4 * 2 + 5 * (-1) * 1
    assert T0 - T1 == (-2) * 4 * (2 - 1)


def test_row_sampling_matches_full():
    rng = np.random.default_rng(31)
    x, w, dy = _tiny_layer(rng, 20, 12, 9, 6, 4)
    a = O.shiftquant_tensor(x, 6, 4)
    g = O.shiftquant_tensor(dy, 6, 4, mode=1, seed=1)
    wf = O.channel_tensor(w, 6, axis=0)
    wd = O.channel_tensor(w, 6, axis=1)
    rows = [0, 7, 19]
    np.testing.assert_array_equal(O.gemm_fwd(a["codes"], a["exp"], wf["codes"], 4, rows),
                                  O.gemm_fwd(a["codes"], a["exp"], wf["codes"], 4)[rows])
    np.testing.assert_array_equal(O.gemm_dgrad(g["codes"], g["exp"], wd["codes"], 4, rows),
                                  O.gemm_dgrad(g["codes"], g["exp"], wd["codes"], 4)[rows])
    r2 = [1, 11]
    np.testing.assert_array_equal(
        O.gemm_wgrad(a["codes"], a["exp"], g["codes"], g["exp"], 4, r2),
        O.gemm_wgrad(a["codes"], a["exp"], g["codes"], g["exp"], 4)[r2])


def test_worked_ties_round_to_even():
    toks = _read_golden("worked_example_ties.txt")
    x = np.array([[float(v) for v in toks[3].split()], [float(v) for v in toks[4].split()]],
                 np.float32)
    exp = np.array([int(v) for v in toks[5].split()[1:]], np.uint8)
    codes = np.array([[int(v) for v in toks[7].split()], [int(v) for v in toks[8].split()]],
                     np.int8)
    d = O.shiftquant_tensor(x, 4, 4, mode=0)
    np.testing.assert_array_equal(d["exp"], exp)
    np.testing.assert_array_equal(d["codes"], codes)


def test_dequant_by_hand():
    # Y = T s_a s_b 2^-shift col_scale[j]: 3 * 0.5 * 0.25 / 4 = 0.09375 and, with a column
    # scale of 3, -5 * 0.5 * 0.25 / 4 * 3 = -0.46875 (all exact)
    T = np.array([[3, -5]], np.int64)
    Y = O.dequant(T, np.float32(0.5), np.float32(0.25), 2)
    assert Y.tolist() == [[0.09375, -0.15625]]
    Y = O.dequant(T, np.float32(0.5), np.float32(0.25), 2, np.array([1.0, 3.0], np.float32))
    assert Y.tolist() == [[0.09375, -0.46875]]


# ------------------------------------------------ per-channel weights (Sec. 5.1)
def test_per_row_weight_worked_example():
    toks = _read_golden("worked_example_per_row_b4.txt")
    bits = int(toks[0].split()[1])
    w = np.array([[float(v) for v in toks[2 + k].split()] for k in range(3)], np.float32)
    rng = np.array([float(v) for v in toks[5].split()[1:]], np.float32)
    num = [np.float32(float(v)) for v in toks[6].split()[1:]]
    den = np.float32(float(toks[7].split()[1]))
    codes = np.array([[int(v) for v in toks[9 + k].split()] for k in range(3)], np.int8)
    d = O.channel_tensor(w, bits, axis=1)
    assert d["status"] == 0
    np.testing.assert_array_equal(d["range"], rng)
    np.testing.assert_array_equal(d["codes"], codes)
    # the scales are binary32 quotients range / Q (numpy's IEEE division)
    np.testing.assert_array_equal(d["scale"], np.array([n / den for n in num], np.float32))


@pytest.mark.parametrize("axis", [0, 1])
@pytest.mark.parametrize("bits", [4, 6, 8])
def test_rn_error_per_channel_weights(axis, bits):
    # per channel (a column for axis 0, a row for axis 1): |w - q s| <= s (1/2 + 2^-15),
    # s = range / Q, and the element of largest magnitude of a channel maps to +-Q
    rng = np.random.default_rng(40 + 3 * bits + axis)
    R, C = 23, 17
    w = (rng.standard_normal((R, C)) * np.exp(rng.normal(0, 1, (R, 1)))
         * np.exp(rng.normal(0, 1, (1, C)))).astype(np.float32)
    w[4, :] = 0
    w[:, 6] = 0
    d = O.channel_tensor(w, bits, axis=axis)
    Q = 2 ** (bits - 1) - 1
    q = d["codes"].astype(np.int64)
    assert np.abs(q).max() <= Q
    wt = w if axis == 0 else w.T          # channels along the columns of wt
    qt = q if axis == 0 else q.T
    rg = np.abs(wt.astype(np.float64)).max(0)
    np.testing.assert_array_equal(d["range"], rg.astype(np.float32))
    s = d["scale"].astype(np.float64)
    err = np.abs(wt.astype(np.float64) - qt * s[None, :])
    assert (err <= s[None, :] * (0.5 + 2.0 ** -15) + 0.0).all()
    for ch in range(wt.shape[1]):
        if rg[ch] == 0:
            assert s[ch] == 0 and (qt[:, ch] == 0).all()
        else:
            i = int(np.argmax(np.abs(wt[:, ch])))
            assert abs(int(qt[i, ch])) == Q


# ------------------------------------------------------- SR draw (App. B, R6)
def _parse_sr_golden():
    toks = _read_golden("sr_draws_seed0.txt")
    cases = []
    for i in range(0, len(toks), 3):
        head, xs, cs = toks[i].split(), toks[i + 1].split(), toks[i + 2].split()
        assert head[0] == "case" and xs[0] == "x24" and cs[0] == "codes"
        x = np.array([int(v) * 2.0 ** -24 for v in xs[1:]], np.float64).reshape(2, 2)
        assert (x.astype(np.float32).astype(np.float64) == x).all()   # exact in binary32
        cases.append((head[1], int(head[2], 16), x.astype(np.float32),
                      np.array([int(v) for v in cs[1:]], np.int8).reshape(2, 2)))
    return cases


def test_sr_draws_match_published_generator_outputs():
    cases = _parse_sr_golden()
    assert len(cases) == 6
    for name, seed, x, codes in cases:
        d = O.shiftquant_tensor(x, 4, 1, mode=1, seed=seed)
        assert float(d["tau0"]) == 7.0 and (d["exp"] == 0).all()
        np.testing.assert_array_equal(d["codes"], codes, err_msg=name)


# --------------------------------- packed sub-byte storage (Sec. 5.2; R17, R18)
def _golden_packed():
    d = {}
    for line in _read_golden("packed_storage.txt"):
        k, *v = line.split()
        d[k] = v
    return d


def test_packed_codes_and_group_maps_by_hand():
    d = _golden_packed()
    q = np.array([[int(v) for v in d["codes0"]], [int(v) for v in d["codes1"]]], np.int8)
    want = np.array([[int(v, 16) for v in d["packed0"]], [int(v, 16) for v in d["packed1"]]],
                    np.uint8)
    np.testing.assert_array_equal(O.pack4(q), want)
    np.testing.assert_array_equal(O.unpack4(want, 7), q)
    for G, key in ((4, "map4"), (8, "map8"), (2, "map2")):
        e = np.array([int(v) for v in d[key]], np.uint8)
        b = np.array([int(v, 16) for v in d[key + "_bytes"]], np.uint8)
        np.testing.assert_array_equal(O.pack_groups(e, G), b)
        np.testing.assert_array_equal(O.unpack_groups(b, e.size, G), e)


@pytest.mark.parametrize("C", [1, 2, 7, 64, 129])
def test_packing_round_trips_and_halves_the_bytes(C):
    rng = np.random.default_rng(C)
    q = rng.integers(-8, 8, (5, C)).astype(np.int8)
    b = O.pack4(q)
    assert b.shape == (5, (C + 1) // 2)
    np.testing.assert_array_equal(O.unpack4(b, C), q)
    for G in (1, 2, 3, 4, 5, 8):
        e = rng.integers(0, G, C).astype(np.uint8)
        np.testing.assert_array_equal(O.unpack_groups(O.pack_groups(e, G), C, G), e)
    # the 2-bit map of N_G = 4 (Sec. 5.2): four channels per byte
    assert O.pack_groups(np.zeros(C, np.uint8), 4).size == (C + 3) // 4
