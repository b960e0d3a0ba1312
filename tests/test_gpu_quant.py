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


def both_roles(w_np, bits, G, ex, eg, ld=None):
    """Both weight roles by shiftquant_calibrate_weight + shiftquant_quantize_weight."""
    K, Nn = w_np.shape
    wg = to_gpu(w_np, ld) if w_np.size else torch.zeros((K, Nn), device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    f = L.ChannelTensor(L.empty_codes(Nn, K, bits, G, "cuda"), torch.zeros(max(Nn, 1), device="cuda")[:Nn],
                        torch.full((max(Nn, 1),), 7.0, device="cuda")[:Nn])
    d = L.ChannelTensor(L.empty_codes(K, Nn, bits, G, "cuda"), torch.zeros(max(K, 1), device="cuda")[:K],
                        torch.full((max(K, 1),), 7.0, device="cuda")[:K])
    L.weight_quantize_both(wg, f, d, None if ex is None else torch.from_numpy(ex).cuda(),
                           None if eg is None else torch.from_numpy(eg).cuda(), bits, G, status)
    torch.cuda.synchronize()
    return f, d, int(status.item())


@pytest.mark.parametrize("shape", [(1, 1), (70, 33), (300, 257), (2304, 256), (129, 1031),
                                   (64, 600), (1000, 96), (700, 4100), (3, 2049)])
@pytest.mark.parametrize("bits,G", [(4, 4), (6, 4), (8, 4), (4, 7)])
@pytest.mark.parametrize("fold", [True, False])
def test_weight_both_roles_from_one_pass(shape, bits, G, fold):
    """The fused weight quantizer (one range pass, one quantize pass for both roles) gives
    the oracle's per-column and per-row ranges, scales and folded codes bit for bit."""
    rng = np.random.default_rng(shape[0] * 7 + shape[1] + bits)
    K, Nn = shape
    w = (rng.standard_normal((K, Nn)) * np.exp(rng.normal(0, 1, Nn)) * 0.02).astype(np.float32)
    w[:, 0] = 0                      # a zero out-channel
    w[K // 2, :] = 0                 # a zero in-channel
    ex = rng.integers(0, G, K).astype(np.uint8) if fold else None
    eg = rng.integers(0, G, Nn).astype(np.uint8) if fold else None
    # with the fold: dense rows; without: rows padded to an odd length (scalar loads)
    f, d, st = both_roles(w, bits, G, ex, eg, ld=None if fold else Nn + 1)
    assert st == 0
    of = O.channel_tensor(w, bits, axis=0)
    od = O.channel_tensor(w, bits, axis=1)
    zx = np.full(K, G - 1, np.uint8) if ex is None else ex    # no fold: shift 2^0
    zg = np.full(Nn, G - 1, np.uint8) if eg is None else eg
    np.testing.assert_array_equal(f32_bits(f.range.cpu().numpy()), f32_bits(of["range"]))
    np.testing.assert_array_equal(f32_bits(f.scale.cpu().numpy()), f32_bits(of["scale"]))
    np.testing.assert_array_equal(decode(f.codes), folded(of["codes"], zx, G, axis=0).T)
    np.testing.assert_array_equal(f32_bits(d.range.cpu().numpy()), f32_bits(od["range"]))
    np.testing.assert_array_equal(f32_bits(d.scale.cpu().numpy()), f32_bits(od["scale"]))
    np.testing.assert_array_equal(decode(d.codes), folded(od["codes"], zg, G, axis=1))


@pytest.mark.parametrize("bad", [np.nan, np.inf])
@pytest.mark.parametrize("C,col", [(300, 200), (1300, 1200)])   # narrow and wide range passes
def test_weight_both_roles_nonfinite(bad, C, col):
    w = np.full((40, C), 0.01, np.float32)
    w[13, col] = bad
    f, d, st = both_roles(w, 4, 4, None, None)
    assert st & N.SQ_DEV_NONFINITE
    fr, dr = f.range.cpu().numpy(), d.range.cpu().numpy()
    assert not np.isfinite(fr[col]) and not np.isfinite(dr[13])
    assert np.isfinite(np.delete(fr, col)).all() and np.isfinite(np.delete(dr, 13)).all()


def test_weight_both_roles_empty():
    for K, Nn in ((0, 5), (5, 0)):
        f, d, st = both_roles(np.zeros((K, Nn), np.float32), 4, 4, None, None)
        assert st == 0
        assert (f.range.cpu().numpy() == 0).all() and (f.scale.cpu().numpy() == 0).all()
        assert (d.range.cpu().numpy() == 0).all() and (d.scale.cpu().numpy() == 0).all()


@pytest.mark.parametrize("mode", [N.SQ_ROUND_NEAREST_EVEN, N.SQ_ROUND_STOCHASTIC])
@pytest.mark.parametrize("bits", [4, 6])
def test_row_shards_quantize_as_the_whole_tensor(mode, bits):
    # a tensor split by rows over two "ranks" (here two shards on one GPU, the all-reduce
    # of their ranges an element-wise maximum): shard ranges, the exchange, the grouping
    # alone (shiftquant_group) and the quantizer with the shifted generator give exactly the
    # whole tensor's ranges, tau_0, exponents, scale, codes and transposed codes
    rng = np.random.default_rng(bits * 10 + mode)
    R, C, G, seed = 3000, 700, 4, 0x1234ABCD
    x = to_gpu(gradient_like(rng, R, C))
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    whole = L.ShiftTensor.alloc(R, C, bits, G, "cuda")
    L.shift_quantize(x, whole, bits, G, mode, seed, st)
    bounds = [(0, 1201), (1201, R)]
    shards = [L.ShiftTensor.alloc(r1 - r0, C, bits, G, "cuda") for r0, r1 in bounds]
    parts = []
    for (r0, r1), q in zip(bounds, shards):
        N.shiftquant_calibrate(x[r0:r1], N.SQ_GRAN_PER_COL, G, q.range, None, None, st)
        parts.append(q.range.clone())
    both = torch.maximum(parts[0], parts[1])
    for (r0, r1), q in zip(bounds, shards):
        L.shard_shift_quantize(x[r0:r1], q, bits, G, mode, seed, r0, st, lambda t: t.copy_(both))
    torch.cuda.synchronize()
    assert st.item() == 0
    want_codes, want_t = decode(whole.codes), decode(whole.codes_t)
    for (r0, r1), q in zip(bounds, shards):
        np.testing.assert_array_equal(f32_bits(q.range.cpu().numpy()), f32_bits(whole.range.cpu().numpy()))
        assert f32_bits([q.tau0.item()])[0] == f32_bits([whole.tau0.item()])[0]
        np.testing.assert_array_equal(q.exp.cpu().numpy(), whole.exp.cpu().numpy())
        assert f32_bits([q.scale.item()])[0] == f32_bits([whole.scale.item()])[0]
        np.testing.assert_array_equal(decode(q.codes), want_codes[r0:r1])
        np.testing.assert_array_equal(decode(q.codes_t), want_t[:, r0:r1])


def test_group_entry_matches_the_range_pass_grouping():
    # shiftquant_group on the range pass's own output reproduces its tau_0 and exponents,
    # including all-zero and outlier channels; zero channels alone give tau_0 = 0
    rng = np.random.default_rng(5)
    x = gradient_like(rng, 500, 333)
    x[:, 7] = 0.0
    xg = to_gpu(x)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    for G in (1, 3, 4, 8):
        q = L.ShiftTensor.alloc(500, 333, 4, G, "cuda")
        N.shiftquant_calibrate(xg, N.SQ_GRAN_SHIFT, G, q.range, q.tau0, q.exp, st)
        tau = torch.zeros(1, device="cuda")
        e = torch.empty(333, dtype=torch.uint8, device="cuda")
        N.shiftquant_group(q.range, G, tau, e, st)
        torch.cuda.synchronize()
        assert tau.item() == q.tau0.item()
        np.testing.assert_array_equal(e.cpu().numpy(), q.exp.cpu().numpy())
        t_o, e_o, _ = O.group(q.range.cpu().numpy(), G)
        np.testing.assert_array_equal(e.cpu().numpy(), e_o)
    z = torch.zeros(16, device="cuda")
    N.shiftquant_group(z, 4, tau, e[:16], st)
    torch.cuda.synchronize()
    assert tau.item() == 0.0 and (e[:16].cpu().numpy() == 3).all() and st.item() == 0
