"""GPU parity of the range pass, the grouping and the quantizer against the oracle:
bit-exact ranges, tau_0, exponents, scales and codes (both roundings, every granularity,
ragged and padded shapes, the degenerate inputs)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2411_10948_gb300 import layer as L
from paper_2411_10948_gb300 import native as N
from parity_util import compare_shift, decode, f32_bits, folded, to_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2411_10948_gb300 import build
    build.build_library()
    N.load()


def gradient_like(rng, R, C, sigma=1.5, frac=0.02, factor=100.0):
    s = np.exp(rng.normal(0, sigma, C)).astype(np.float32)
    s[rng.random(C) < frac] *= factor
    return (rng.standard_normal((R, C)) * s).astype(np.float32)


def gpu_shift(x_np, bits, G, mode, seed, ld=None, transposed=True):
    x = to_gpu(x_np, ld)
    R, C = x_np.shape
    q = L.ShiftTensor.alloc(R, C, bits, G, "cuda", transposed)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    L.shift_quantize(x, q, bits, G, mode, seed, status)
    torch.cuda.synchronize()
    return q, int(status.item())


SHAPES = [(1, 1), (3, 5), (64, 64), (65, 130), (200, 257), (1000, 96), (37, 1031)]


@pytest.mark.parametrize("shape", SHAPES)
@pytest.mark.parametrize("padded", [False, True])
def test_calibrate_and_quantize_rn(shape, padded):
    rng = np.random.default_rng(shape[0] * 31 + shape[1])
    x = gradient_like(rng, *shape)
    ld = shape[1] + 3 if padded else None
    for bits, G in ((4, 4), (6, 4), (8, 4), (2, 1), (5, 8)):
        q, st = gpu_shift(x, bits, G, N.SQ_ROUND_NEAREST_EVEN, 0, ld)
        assert st == 0
        compare_shift(q, O.shiftquant_tensor(x, bits, G, mode=0), f"{shape} b{bits} G{G}")


@pytest.mark.parametrize("shape", [(5, 7), (128, 300), (513, 64)])
@pytest.mark.parametrize("seed", [0, 1, 2**63 + 12345])
def test_quantize_sr(shape, seed):
    rng = np.random.default_rng(7 + shape[1])
    x = gradient_like(rng, *shape, sigma=2.0)
    for bits, G in ((4, 4), (6, 4), (8, 2)):
        q, st = gpu_shift(x, bits, G, N.SQ_ROUND_STOCHASTIC, seed)
        assert st == 0
        compare_shift(q, O.shiftquant_tensor(x, bits, G, mode=1, seed=seed), f"SR b{bits}")


def test_boundary_channels_zero_channels_and_denormals():
    # channels exactly at tau_0 2^-k and one ulp either side, all-zero and denormal channels
    tau = np.float32(3.0)
    cols = []
    for k in range(6):
        b = np.float32(tau * 2.0 ** -k)
        cols += [b, np.nextafter(b, np.float32(0)), np.nextafter(b, np.float32(10))]
    cols += [0.0, np.float32(1e-45), np.float32(3e-39), tau]
    c = np.minimum(np.array(cols, np.float32), tau)
    x = np.tile(c, (9, 1))
    x[1::2] *= -0.5
    x[3] = 0
    for G in (1, 3, 4, 8):
        q, st = gpu_shift(x, 4, G, N.SQ_ROUND_NEAREST_EVEN, 0)
        assert st == 0
        compare_shift(q, O.shiftquant_tensor(x, 4, G, mode=0), f"boundaries G{G}")


def test_all_zero_and_tiny_tensors():
    for x in (np.zeros((17, 33), np.float32), np.full((4, 4), 1e-45, np.float32)):
        q, st = gpu_shift(x, 4, 4, N.SQ_ROUND_NEAREST_EVEN, 0)
        assert st == 0
        o = O.shiftquant_tensor(x, 4, 4)
        compare_shift(q, o, "degenerate")
        assert q.scale.item() == 0 and (decode(q.codes) == 0).all()


def test_single_outlier_channel():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((300, 200)).astype(np.float32)
    x[:, 17] *= 1e4
    q, _ = gpu_shift(x, 4, 4, N.SQ_ROUND_STOCHASTIC, 5)
    o = O.shiftquant_tensor(x, 4, 4, mode=1, seed=5)
    compare_shift(q, o, "outlier")
    assert int(q.exp[17].item()) == 0 and (q.exp.cpu().numpy()[np.arange(200) != 17] == 3).all()


@pytest.mark.parametrize("bad", [np.nan, np.inf, -np.inf])
def test_nonfinite_input_sets_status(bad):
    x = np.ones((20, 30), np.float32)
    x[7, 11] = bad
    q, st = gpu_shift(x, 4, 4, N.SQ_ROUND_NEAREST_EVEN, 0)
    assert st & N.SQ_DEV_NONFINITE
    o = O.shiftquant_tensor(x, 4, 4)
    assert o["status"] == 1
    t = q.tau0.item()
    assert (np.isnan(t) and np.isnan(o["tau0"])) or (np.isinf(t) and np.isinf(o["tau0"]))
    assert (q.exp.cpu().numpy() == 0).all()
    assert q.scale.item() == 0 and (decode(q.codes) == 0).all()


def test_empty_tensors():
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for R, C in ((0, 5), (5, 0), (0, 0)):
        x = torch.zeros((R, C), device="cuda")
        q = L.ShiftTensor.alloc(R, C, 4, 4, "cuda")
        q.tau0.fill_(7)
        q.scale.fill_(7)
        L.shift_quantize(x, q, 4, 4, 0, 0, status)
        torch.cuda.synchronize()
        assert q.tau0.item() == 0 and q.scale.item() == 0
    assert status.item() == 0


@pytest.mark.parametrize("shape", [(1, 1), (70, 33), (300, 257), (2304, 256)])
@pytest.mark.parametrize("bits,G", [(4, 4), (6, 4), (8, 4), (4, 7)])
def test_weight_quantization_with_fold(shape, bits, G):
    rng = np.random.default_rng(shape[0] + bits)
    K, Nn = shape
    w = (rng.standard_normal((K, Nn)) * 0.02).astype(np.float32)
    w[:, 0] = 0          # a zero out-channel
    ex = rng.integers(0, G, K).astype(np.uint8)     # exponents of the activation (by row)
    eg = rng.integers(0, G, Nn).astype(np.uint8)    # exponents of the gradient (by column)
    wg = torch.from_numpy(w).cuda()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    f = L.ChannelTensor(L.empty_codes(Nn, K, bits, G, "cuda"), torch.zeros(Nn, device="cuda"),
                        torch.zeros(Nn, device="cuda"))
    d = L.ChannelTensor(L.empty_codes(K, Nn, bits, G, "cuda"), torch.zeros(K, device="cuda"),
                        torch.zeros(K, device="cuda"))
    L.weight_quantize_fwd(wg, f, torch.from_numpy(ex).cuda(), bits, G, status)
    L.weight_quantize_dgrad(wg, d, torch.from_numpy(eg).cuda(), bits, G, status)
    torch.cuda.synchronize()
    assert status.item() == 0
    of = O.channel_tensor(w, bits, axis=0)
    od = O.channel_tensor(w, bits, axis=1)
    np.testing.assert_array_equal(f32_bits(f.range.cpu().numpy()), f32_bits(of["range"]))
    np.testing.assert_array_equal(f32_bits(f.scale.cpu().numpy()), f32_bits(of["scale"]))
    np.testing.assert_array_equal(decode(f.codes), folded(of["codes"], ex, G, axis=0).T)
    np.testing.assert_array_equal(f32_bits(d.range.cpu().numpy()), f32_bits(od["range"]))
    np.testing.assert_array_equal(f32_bits(d.scale.cpu().numpy()), f32_bits(od["scale"]))
    np.testing.assert_array_equal(decode(d.codes), folded(od["codes"], eg, G, axis=1))
