"""The device-side timeout path on the GPU, in the form that faults nothing: a GEMM launch
whose producer issues no operand copy (shiftquant_selftest_wait_timeout), so a bounded
wait runs out because nothing ever arrives.  The launch must record SQ_DEV_TIMEOUT, return
within a few seconds, and leave the context usable for a normal launch right after."""
import time

import numpy as np
import pytest
import torch

import oracle as O
from paper_2411_10948_gb300 import layer as L
from paper_2411_10948_gb300 import native as N
from parity_util import assert_close_f32, to_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2411_10948_gb300 import build
    build.build_library()
    N.load()


def test_a_wait_that_runs_out_reports_timeout_and_the_context_stays_usable():
    M, K, Nn, bits, G = 128, 256, 256, 4, 4
    a = L.empty_codes(M, K, bits, G, "cuda")
    b = L.empty_codes(Nn, K, bits, G, "cuda")
    one = torch.ones(1, device="cuda")
    ones = torch.ones(Nn, device="cuda")
    y = torch.full((M, Nn), 3.0, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    N.shiftquant_selftest_wait_timeout(a, one, b, ones, M, Nn, K, bits, G, y, st)
    torch.cuda.synchronize()   # the launch returns by itself
    dt = time.perf_counter() - t0
    assert st.item() & N.SQ_DEV_TIMEOUT, st.item()
    assert dt < 30.0, dt
    assert (y == 3.0).all()    # nothing was written
    # a normal layer step right after, on the same context, matches the oracle
    rng = np.random.default_rng(9)
    x = rng.standard_normal((300, 200)).astype(np.float32)
    w = (rng.standard_normal((200, 96)) * 0.02).astype(np.float32)
    dy = rng.laplace(0, 1, (300, 96)).astype(np.float32)
    lay = L.QuantLinear(300, 200, 96, 4, 4, "cuda")
    lay.step(to_gpu(x), to_gpu(w), to_gpu(dy), 5)
    torch.cuda.synchronize()
    assert lay.status.item() == 0
    ox = O.shiftquant_tensor(x, 4, 4, 0)
    wf = O.channel_tensor(w, 4, 0)
    want = O.dequant(O.gemm_fwd(ox["codes"], ox["exp"], wf["codes"], 4), ox["scale"], 1.0, 3,
                     wf["scale"])
    assert_close_f32(lay.y.cpu().numpy(), want, "Y after the timeout")


def test_selftest_refuses_empty_or_large_launches():
    one = torch.ones(1, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    a = L.empty_codes(8, 64, 4, 4, "cuda")
    y = torch.zeros((8, 8), device="cuda")
    for M, Nn, K in ((0, 8, 64), (8, 8, 0), (5000, 8, 64)):
        with pytest.raises(N.ShiftQuantError):
            N.shiftquant_selftest_wait_timeout(a, one, a, one, M, Nn, K, 4, 4, y, st)


def test_a_grid_barrier_that_runs_out_reports_timeout_and_the_context_stays_usable():
    # the single-launch L1 batch normalization's grid barrier: one block never arrives, so
    # every block's bounded wait runs out (about 1 s), records SQ_DEV_TIMEOUT and returns;
    # an L1 batch normalization right after matches the oracle
    scratch = torch.zeros(64, dtype=torch.int32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    N.shiftquant_selftest_grid_barrier_timeout(scratch, st)
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert st.item() & N.SQ_DEV_TIMEOUT, st.item()
    assert dt < 30.0, dt
    rng = np.random.default_rng(5)
    R, C = 500, 48
    x = rng.standard_normal((R, C)).astype(np.float32)
    gamma = np.ones(C, np.float32)
    beta = np.zeros(C, np.float32)
    st2 = torch.zeros(1, dtype=torch.int32, device="cuda")
    state = torch.zeros(N.shiftquant_l1bn_state_bytes(R, C), dtype=torch.uint8, device="cuda")
    y = torch.empty((R, C), device="cuda")
    N.shiftquant_l1bn_forward(to_gpu(x), torch.from_numpy(gamma).cuda(), torch.from_numpy(beta).cuda(),
                              8, 4, y, state, st2)
    torch.cuda.synchronize()
    assert st2.item() == 0
    f = O.l1bn_forward(x, gamma, beta, 8, 4)
    np.testing.assert_array_equal(y.cpu().numpy().view(np.uint32), f["y"].view(np.uint32))
