"""GPU parity of the fully-quantized L1 batch normalization (shiftquant_l1bn_forward /
_backward) against the oracle (Sec. 4, App. C): the input's int8 codes, y, dx, dgamma and
dbeta bit for bit -- every channel sum is an exact integer and every other step one
binary32 operation in the oracle's order.  Shapes span several column blocks and row slabs,
ragged channel counts (scalar paths), one row, a constant channel, and a ResNet-sized
activation."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2411_10948_gb300 import native as N
from parity_util import f32_bits, to_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2411_10948_gb300 import build
    build.build_library()
    N.load()


def _inputs(rng, R, C):
    x = (rng.standard_normal((R, C)) * np.exp(rng.normal(0, 1, C)) + rng.normal(0, 1, C)) \
        .astype(np.float32)
    x[:, rng.random(C) < 0.05] *= 30.0
    gamma = rng.normal(1, 0.3, C).astype(np.float32)
    beta = rng.normal(0, 0.3, C).astype(np.float32)
    dy = (rng.laplace(0, 1, (R, C)) * np.exp(rng.normal(0, 1.5, C))).astype(np.float32)
    return x, gamma, beta, dy


def _run(x, gamma, beta, dy, bits, G, seed):
    R, C = x.shape
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    state = torch.zeros(N.shiftquant_l1bn_state_bytes(R, C), dtype=torch.uint8, device="cuda")
    y = torch.full((R, C), 9.0, device="cuda")
    dx = torch.full((R, C), 9.0, device="cuda")
    dg = torch.zeros(C, device="cuda")
    db = torch.zeros(C, device="cuda")
    vec = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    N.shiftquant_l1bn_forward(to_gpu(x), vec(gamma), vec(beta), bits, G, y, state, st)
    N.shiftquant_l1bn_backward(to_gpu(dy), bits, G, seed, state, dx, dg, db, st)
    torch.cuda.synchronize()
    q = state[: R * C].view(torch.int8).reshape(R, C).cpu().numpy()
    return q, y.cpu().numpy(), dx.cpu().numpy(), dg.cpu().numpy(), db.cpu().numpy(), st.item()


@pytest.mark.parametrize("R,C,bits,G", [(12544, 256, 8, 4), (1000, 77, 8, 4), (3000, 130, 6, 3),
                                        (1, 9, 8, 4), (64, 4, 4, 1), (200, 1000, 8, 8),
                                        (20000, 64, 8, 4), (3001, 16, 8, 4), (777, 3, 8, 4),
                                        (5000, 600, 8, 4), (300, 1100, 8, 4), (1500, 1027, 6, 4),
                                        (200704, 64, 8, 4)])
def test_l1bn_matches_oracle_bit_for_bit(R, C, bits, G):
    rng = np.random.default_rng(R + C)
    x, gamma, beta, dy = _inputs(rng, R, C)
    if C > 3:
        x[:, 3] = 1.25            # a constant channel: sigma 0, output beta^q, no gradient
    seed = 0xFACE + R
    q, y, dx, dg, db, st = _run(x, gamma, beta, dy, bits, G, seed)
    assert st == 0
    f = O.l1bn_forward(x, gamma, beta, bits, G)
    b = O.l1bn_backward(dy, f, bits, G, seed)
    np.testing.assert_array_equal(q, f["q"])
    np.testing.assert_array_equal(f32_bits(y), f32_bits(f["y"]), err_msg="y")
    np.testing.assert_array_equal(f32_bits(dg), f32_bits(b["dgamma"]), err_msg="dgamma")
    np.testing.assert_array_equal(f32_bits(db), f32_bits(b["dbeta"]), err_msg="dbeta")
    np.testing.assert_array_equal(f32_bits(dx), f32_bits(b["dx"]), err_msg="dx")


def test_l1bn_launch_forms():
    # at most 1024 channels: one cooperative launch per call; wider: the chain of kernels
    # (the shapes above cover both, and both must match the oracle bit for bit)
    for C in (3, 64, 256, 1024):
        assert N.shiftquant_l1bn_kernel_launches(C) == 1
        assert N.shiftquant_l1bn_kernel_launches(C, True) == 1
    assert N.shiftquant_l1bn_kernel_launches(1025) == 9
    assert N.shiftquant_l1bn_kernel_launches(1100, True) == 7
    assert N.shiftquant_l1bn_kernel_launches(0) == 0


def test_l1bn_repeated_calls_on_one_state_stay_exact():
    # the single-launch form zeroes its barrier counter and range slots per call: a second
    # forward and backward on the same state (a training loop) give the same bits
    rng = np.random.default_rng(11)
    x, gamma, beta, dy = _inputs(rng, 4000, 96)
    R, C = x.shape
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    state = torch.full((N.shiftquant_l1bn_state_bytes(R, C),), 0x5A, dtype=torch.uint8, device="cuda")
    outs = []
    for _ in range(2):
        y = torch.empty((R, C), device="cuda")
        dx = torch.empty((R, C), device="cuda")
        dg = torch.empty(C, device="cuda")
        db = torch.empty(C, device="cuda")
        N.shiftquant_l1bn_forward(to_gpu(x), torch.from_numpy(gamma).cuda(), torch.from_numpy(beta).cuda(),
                                  8, 4, y, state, st)
        N.shiftquant_l1bn_backward(to_gpu(dy), 8, 4, 9, state, dx, dg, db, st)
        torch.cuda.synchronize()
        outs.append([t.cpu().numpy() for t in (y, dx, dg, db)])
    assert st.item() == 0
    f = O.l1bn_forward(x, gamma, beta, 8, 4)
    b = O.l1bn_backward(dy, f, 8, 4, 9)
    for got in outs:
        np.testing.assert_array_equal(f32_bits(got[0]), f32_bits(f["y"]))
        np.testing.assert_array_equal(f32_bits(got[1]), f32_bits(b["dx"]))
        np.testing.assert_array_equal(f32_bits(got[2]), f32_bits(b["dgamma"]))
        np.testing.assert_array_equal(f32_bits(got[3]), f32_bits(b["dbeta"]))


def test_l1bn_nonfinite_input_sets_status():
    rng = np.random.default_rng(3)
    x, gamma, beta, dy = _inputs(rng, 100, 20)
    x[7, 2] = np.nan
    *_, st = _run(x, gamma, beta, dy, 8, 4, 1)
    assert st & N.SQ_DEV_NONFINITE


def test_l1bn_rejects_bad_arguments():
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    x = torch.zeros((4, 8), device="cuda")
    g = torch.ones(8, device="cuda")
    small = torch.zeros(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(N.ShiftQuantError):
        N.shiftquant_l1bn_forward(x, g, g, 8, 4, x, small, st)          # state too small
    state = torch.zeros(N.shiftquant_l1bn_state_bytes(4, 8), dtype=torch.uint8, device="cuda")
    with pytest.raises(N.ShiftQuantError):
        N.shiftquant_l1bn_forward(x, g, g, 9, 4, x, state, st)          # bits
