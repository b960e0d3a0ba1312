"""Pins of the oracle's fully-quantized L1 BatchNorm (Sec. 4, App. C; readings R12-R16 of the
oracle source) to facts outside it, on CPU:

* on inputs that every quantizer of the layer represents exactly (codes, mean, sigma, gamma
  and beta all on their grids) the oracle's forward is the textbook L1 batch normalization
  y = gamma (x - mean) / mean|x - mean| + beta, evaluated here in binary64;
* its backward matches central finite differences of that textbook forward (with the
  incoming gradient on its own grid, so stochastic rounding is exact);
* translation invariance of batch normalization: per channel the input gradient sums to 0;
* the mean rounds half to even onto the code grid, a constant channel outputs beta.
"""
import numpy as np
import pytest

import oracle as O


def _textbook(x, gamma, beta):
    """L1 batch normalization in binary64 (R12: sigma = mean |x - mean| per channel)."""
    x = x.astype(np.float64)
    mu = x.mean(0)
    sig = np.abs(x - mu).mean(0)
    return gamma.astype(np.float64) * (x - mu) / sig + beta.astype(np.float64)


def _deviations(rng, total, lim, fixed=None):
    """32 positive integer deviations <= lim summing to `total` (the first one fixed if given),
    spread by random transfers."""
    n = 32
    a = np.full(n, total // n, np.int64)
    a[: total % n] += 1
    if fixed is not None:
        rest = total - fixed
        a[1:] = rest // (n - 1)
        a[1: 1 + rest % (n - 1)] += 1
        a[0] = fixed
    lo = 1 if fixed is None else 1
    for _ in range(400):
        i, j = rng.integers(lo if fixed is None else 1, n, 2)
        d = int(rng.integers(1, 6))
        if i != j and a[i] - d >= 1 and a[j] + d <= lim:
            a[i] -= d
            a[j] += d
    assert a.sum() == total and a.min() >= 1 and a.max() <= lim
    return a


def _on_grid_case(seed):
    """x = q s with s = 2^-3, bits 8, N_G = 1, tau_0 = 127 s (channel 0 holds +-127); per
    channel an integer code mean m and 32 pairs of deviations +-a with sum a = 8 k, so that
    sigma = mean |d| s = k 2^-5 lies on the sigma grid of sigma_max = 127 2^-5; gamma = j 2^-6
    and beta = i 2^-7 on their 8-bit grids."""
    rng = np.random.default_rng(seed)
    R, C = 64, 6
    ks = [127, 40, 63, 100, 17, 90]
    q = np.zeros((R, C), np.int64)
    for c, k in enumerate(ks):
        m = 0 if c == 0 else int(rng.integers(-20, 21))
        a = _deviations(rng, 8 * k, 127 - abs(m), fixed=127 if c == 0 else None)
        q[:, c] = rng.permutation(np.concatenate([m + a, m - a]))
    x = (q * 0.125).astype(np.float32)
    gamma = (rng.integers(-127, 128, C) * 2.0 ** -6).astype(np.float32)
    gamma[0] = 127 * 2.0 ** -6
    beta = (rng.integers(-127, 128, C) * 2.0 ** -7).astype(np.float32)
    beta[1] = -127 * 2.0 ** -7
    return x, gamma, beta


def _check_on_grid(f, x, gamma, beta):
    # the premise: every quantizer of the layer is lossless on this input
    np.testing.assert_array_equal(f["q"].astype(np.float64) * 0.125, x)
    assert (f["m"] == np.round(x.astype(np.float64).mean(0) / 0.125)).all()
    np.testing.assert_array_equal(f["sigma_q"], f["sigma"])
    np.testing.assert_array_equal(f["gamma_q"], gamma)
    np.testing.assert_array_equal(f["beta_q"], beta)


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_l1bn_forward_on_grid_is_the_textbook_layer(seed):
    x, gamma, beta = _on_grid_case(seed)
    xm = x.astype(np.float64).mean(0)
    assert np.allclose(xm / 0.125, np.round(xm / 0.125))       # integer code means
    f = O.l1bn_forward(x, gamma, beta, 8, 1)
    assert f["status"] == 0
    _check_on_grid(f, x, gamma, beta)
    want = _textbook(x, gamma, beta)
    np.testing.assert_allclose(f["y"], want, rtol=5e-7, atol=5e-7 * np.abs(want).max())


@pytest.mark.parametrize("seed", [4, 5])
def test_l1bn_backward_matches_finite_differences(seed):
    x, gamma, beta = _on_grid_case(seed)
    R, C = x.shape
    rng = np.random.default_rng(seed)
    t = 2.0 ** -4
    gy = (rng.integers(-127, 128, (R, C)) * t).astype(np.float32)
    gy[0, 0] = 127 * t                                          # tau_0 = 127 t: exact codes
    f = O.l1bn_forward(x, gamma, beta, 8, 1)
    _check_on_grid(f, x, gamma, beta)
    b = O.l1bn_backward(gy, f, 8, 1, seed=77)
    np.testing.assert_array_equal(b["p"].astype(np.float64) * t, gy)   # SR exact on grid
    g64 = gy.astype(np.float64)

    def loss(xx, gg=gamma, bb=beta):
        return float((_textbook(xx, gg, bb) * g64).sum())

    h = 1e-3   # far below the smallest |x - mean| (one code step, 0.125): no kink crossed
    x64 = x.astype(np.float64)
    for (r, c) in [(0, 0), (5, 1), (17, 2), (33, 3), (63, 5), (40, 4)]:
        xp, xm = x64.copy(), x64.copy()
        xp[r, c] += h
        xm[r, c] -= h
        num = (loss(xp) - loss(xm)) / (2 * h)
        scale = np.abs(b["dx"][:, c]).max()
        assert abs(b["dx"][r, c] - num) <= 1e-5 * scale + 1e-9, (r, c, b["dx"][r, c], num)
    for c in range(C):
        e = np.zeros(C)
        e[c] = 1e-3
        num_g = (loss(x64, gamma + e, beta) - loss(x64, gamma - e, beta)) / 2e-3
        num_b = (loss(x64, gamma, beta + e) - loss(x64, gamma, beta - e)) / 2e-3
        assert abs(b["dgamma"][c] - num_g) <= 1e-5 * abs(num_g) + 1e-6
        assert abs(b["dbeta"][c] - num_b) <= 1e-6 * abs(num_b) + 1e-9


def test_l1bn_input_gradient_sums_to_zero_per_channel():
    # shifting a channel by a constant leaves x-hat unchanged, so the gradient of any loss
    # sums to 0 over the channel (exactly, up to binary32 rounding)
    rng = np.random.default_rng(11)
    R, C = 700, 33
    x = (rng.standard_normal((R, C)) * np.exp(rng.normal(0, 1, C)) + rng.normal(0, 2, C)) \
        .astype(np.float32)
    gamma = rng.normal(1, 0.3, C).astype(np.float32)
    beta = rng.normal(0, 0.3, C).astype(np.float32)
    gy = (rng.laplace(0, 1, (R, C)) * np.exp(rng.normal(0, 1.5, C))).astype(np.float32)
    f = O.l1bn_forward(x, gamma, beta, 8, 4)
    b = O.l1bn_backward(gy, f, 8, 4, seed=5)
    tot = np.abs(b["dx"]).sum(0)
    assert (np.abs(b["dx"].astype(np.float64).sum(0)) <= 1e-5 * tot + 1e-30).all()
    # and the statistics are the integer ones of the codes
    q = f["q"].astype(np.int64)
    np.testing.assert_array_equal(f["S1"], q.sum(0))
    d = q - f["m"].astype(np.int64)[None, :]
    np.testing.assert_array_equal(f["S"], np.abs(d).sum(0))
    np.testing.assert_array_equal(f["Z"], np.sign(d).sum(0))


def test_l1bn_mean_rounds_half_to_even_and_constant_channel_gives_beta():
    # bits 8, N_G = 1, tau_0 = 127 (channel 0 holds +-127), so codes equal x
    x = np.array([[127, 2, 3, -2, 5],
                  [-127, 3, 4, -3, 5]], np.float32)
    gamma = np.array([1, 1, 1, 1, 1], np.float32)
    beta = np.array([0, 0, 0, 0.5, -0.25], np.float32)
    f = O.l1bn_forward(x, gamma, beta, 8, 1)
    np.testing.assert_array_equal(f["q"], x.astype(np.int8))
    # means 0, 2.5 -> 2, 3.5 -> 4, -2.5 -> -2, 5
    np.testing.assert_array_equal(f["m"], [0, 2, 4, -2, 5])
    # channel 4 is constant: sigma 0, its output is beta^q and it passes no gradient
    assert f["sigma"][4] == 0 and f["sigma_q"][4] == 0
    np.testing.assert_array_equal(f["y"][:, 4], f["beta_q"][4])
    gy = np.array([[1, 1, 1, 1, 1], [-1, 2, 3, 4, 5]], np.float32)
    b = O.l1bn_backward(gy, f, 8, 1)
    assert (b["dx"][:, 4] == 0).all()
