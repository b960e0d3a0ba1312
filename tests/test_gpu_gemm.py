"""GPU parity of the three ShiftMM GEMMs against the oracle: integer accumulators bit-exact,
fp32 outputs within 1e-6 relative; plus worst-case magnitudes that push every chunk of
the exact FP32 accumulation to its bound, split-K against unsplit, and empty shapes."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2411_10948_gb300 import layer as L
from paper_2411_10948_gb300 import native as N
from parity_util import assert_close_f32, compare_shift, decode, f32_bits, folded, oracle_layer, \
    to_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2411_10948_gb300 import build
    build.build_library()
    N.load()


def layer_inputs(rng, M, K, Nn):
    sx = np.exp(rng.normal(0, 1.0, K)).astype(np.float32)
    sx[rng.random(K) < 0.02] *= 50
    x = (rng.standard_normal((M, K)) * sx).astype(np.float32)
    w = (rng.standard_normal((K, Nn)) * 0.02).astype(np.float32)
    sg = np.exp(rng.normal(0, 2.0, Nn)).astype(np.float32)
    sg[rng.random(Nn) < 0.01] *= 1000
    dy = (rng.laplace(0, 1, (M, Nn)) * sg).astype(np.float32)
    return x, w, dy


def run_and_compare(x, w, dy, bits, G, seed=11, use_workspace=True, fused=False,
                    transposed=True):
    M, K = x.shape
    Nn = w.shape[1]
    lay = L.QuantLinear(M, K, Nn, bits, G, "cuda", with_acc=True, use_workspace=use_workspace,
                        transposed=transposed)
    if fused:
        lay.quantize_activation(to_gpu(x))
        lay.quantize_gradient(to_gpu(dy), seed)
        lay.quantize_weights(to_gpu(w))
        lay.gemms()
    else:
        lay.step(to_gpu(x), to_gpu(w), to_gpu(dy), seed)
    torch.cuda.synchronize()
    assert lay.status.item() == 0
    o = oracle_layer(x, w, dy, bits, G, seed)
    compare_shift(lay.x, o["x"], "X")
    compare_shift(lay.g, o["g"], "dY")
    np.testing.assert_array_equal(decode(lay.wf.codes), folded(o["wf"]["codes"], o["x"]["exp"], G, 0).T)
    np.testing.assert_array_equal(decode(lay.wd.codes), folded(o["wd"]["codes"], o["g"]["exp"], G, 1))
    np.testing.assert_array_equal(lay.acc["fwd"].cpu().numpy(), o["T_fwd"], err_msg="T fwd")
    np.testing.assert_array_equal(lay.acc["dgrad"].cpu().numpy(), o["T_dgrad"], err_msg="T dgrad")
    np.testing.assert_array_equal(lay.acc["wgrad"].cpu().numpy(), o["T_wgrad"], err_msg="T wgrad")
    assert_close_f32(lay.y.cpu().numpy(), o["y"], "Y")
    assert_close_f32(lay.dx.cpu().numpy(), o["dx"], "dX")
    assert_close_f32(lay.dw.cpu().numpy(), o["dw"], "dW")
    return lay


@pytest.mark.parametrize("M,K,Nn", [(1, 1, 1), (5, 3, 7), (128, 128, 256), (130, 70, 300),
                                    (257, 520, 260), (300, 1000, 513)])
@pytest.mark.parametrize("bits", [4, 6, 8])
def test_layer_chain_matches_oracle(M, K, Nn, bits):
    rng = np.random.default_rng(M * 7 + K * 3 + Nn + bits)
    run_and_compare(*layer_inputs(rng, M, K, Nn), bits, 4)


@pytest.mark.parametrize("M,K,Nn,bits", [(1900, 1800, 1700, 6), (3300, 3500, 3400, 4),
                                         (2000, 1800, 1700, 8)])
def test_pair_tiles_with_ragged_tails_match_oracle(M, K, Nn, bits):
    # layer launches that run on CTA pairs (256 x 256 tiles): M = 1900 leaves the second CTA
    # of the last pair entirely past M, and the column tails (1700, 1800, 3400, 3500) end
    # inside one CTA's half of B; 8-bit adds multi-chunk K loops sized from the exponents
    assert N.shiftquant_gemm_layer_cta_pairs(M, K, Nn, bits, 4) == 1
    rng = np.random.default_rng(M + K + Nn + bits)
    run_and_compare(*layer_inputs(rng, M, K, Nn), bits, 4, fused=True)


@pytest.mark.parametrize("M,K,Nn", [(1, 1, 1), (5, 3, 7), (130, 70, 300), (300, 1000, 513),
                                    (4096, 64, 96), (2000, 700, 256), (1900, 1800, 1700)])
@pytest.mark.parametrize("bits", [6, 8, 4])
def test_weight_gradient_reads_the_codes_in_place(M, K, Nn, bits):
    # no transposed copies: the weight gradient of the layer launch reads X's [M, K] and dY's
    # [M, N] codes as MN-major operands (the tensor core transposes them from shared memory);
    # ragged tails in both the output (K, N) and the inner (token) index, single tiles and
    # CTA pairs (1900 x 1800 x 1700)
    rng = np.random.default_rng(M + 3 * K + Nn + bits)
    lay = run_and_compare(*layer_inputs(rng, M, K, Nn), bits, 4, fused=True, transposed=False)
    assert lay.x.codes_t is None and lay.g.codes_t is None


def test_layout_advice_keeps_copies_only_where_the_tensor_core_sets_the_pace():
    # shiftquant_gemm_layer_wgrad_in_place: in place where the launch is bound by split-K
    # reductions or epilogues, transposed copies for full waves of long pair-tile units
    adv = N.shiftquant_gemm_layer_wgrad_in_place
    assert adv(12544, 2304, 256, 4, 4) == 1        # single tiles
    assert adv(12608, 768, 3072, 6, 4) == 1        # split-K weight gradient
    assert adv(16384, 4096, 11008, 6, 4) == 0      # 688 unsplit units of 256 K blocks
    assert adv(4096, 4096, 4096, 6, 4) == 0
    assert adv(16, 16, 16, 9, 4) == -1
    lay = L.QuantLinear(12544, 2304, 256, 4, 4, "cuda", transposed=None)
    assert lay.x.codes_t is None and lay.g.codes_t is None
    lay = L.QuantLinear(4096, 4096, 4096, 6, 4, "cuda", transposed=None)
    assert lay.x.codes_t is not None and lay.g.codes_t is not None


@pytest.mark.parametrize("bits", [6, 4])
def test_weight_gradient_in_place_equals_the_transposed_copies(bits):
    # the same launch on the codes in place and on transposed copies: equal dW bit for bit,
    # through the separate-GEMM step as well (its weight gradient becomes a layer launch)
    rng = np.random.default_rng(60 + bits)
    x, w, dy = layer_inputs(rng, 3000, 640, 384)
    a = run_and_compare(x, w, dy, bits, 4, fused=True, transposed=False)
    b = run_and_compare(x, w, dy, bits, 4, fused=True, transposed=True)
    c = run_and_compare(x, w, dy, bits, 4, fused=False, transposed=False)
    for t in (b, c):
        np.testing.assert_array_equal(a.dw.cpu().numpy(), t.dw.cpu().numpy())


def test_tile_mode_query():
    # conv3x3's short K loops stay on single tiles; the large linear layer runs on pairs
    assert N.shiftquant_gemm_layer_cta_pairs(12544, 2304, 256, 4, 4) == 0
    assert N.shiftquant_gemm_layer_cta_pairs(16384, 4096, 11008, 6, 4) == 1
    assert N.shiftquant_gemm_layer_cta_pairs(0, 0, 0, 6, 4) == -1
    assert N.shiftquant_gemm_layer_cta_pairs(16, 16, 16, 9, 4) == -1


@pytest.mark.parametrize("bits,G", [(6, 4), (8, 4), (8, 5), (4, 7), (5, 5), (3, 8)])
def test_multi_chunk_inner_dims(bits, G):
    # K long enough that the exact-FP32 chunking splits the K loop several times
    rng = np.random.default_rng(bits * 13 + G)
    run_and_compare(*layer_inputs(rng, 200, 5000, 300), bits, G)


def test_split_k_equals_unsplit():
    rng = np.random.default_rng(99)
    x, w, dy = layer_inputs(rng, 4096, 64, 96)      # wgrad: 1 output tile, K = 4096 tokens
    a = run_and_compare(x, w, dy, 6, 4, use_workspace=True)
    assert a.ws is not None, "expected the wgrad to split K across SMs"
    b = run_and_compare(x, w, dy, 6, 4, use_workspace=False)
    np.testing.assert_array_equal(a.dw.cpu().numpy(), b.dw.cpu().numpy())


def _encode(vals: np.ndarray, bits: int, G: int) -> torch.Tensor:
    """Code tensor (padded rows) holding the given integers in the library's storage type."""
    R, C = vals.shape
    t = L.empty_codes(R, C, bits, G, "cuda")
    v = torch.from_numpy(vals.astype(np.float32)).cuda()
    if t.dtype == torch.uint8:
        t.copy_(v.to(torch.float8_e4m3fn).view(torch.uint8))
    else:
        t.copy_(v.to(torch.bfloat16))
    assert (decode(t) == vals).all()
    return t


@pytest.mark.parametrize("bits,G,K", [(4, 4, 50000), (6, 4, 6628), (8, 4, 1000), (8, 5, 700),
                                      (6, 8, 3000)])
def test_worst_case_magnitudes_stay_exact(bits, G, K):
    # every product at (or one step below) the largest magnitude, same sign within a row,
    # with odd products mixed in: partial sums reach the chunk bound and an accumulator
    # that dropped low-order bits would lose the odd terms
    Q = 2 ** (bits - 1) - 1
    M, Nn = 130, 260
    rng = np.random.default_rng(K)
    A = np.full((M, K), Q, np.int64)
    A[1::2] *= -1                                   # alternate row signs
    A[5] = rng.integers(-Q, Q + 1, K)               # one random row
    kk = np.arange(K)[None, :]
    nn = np.arange(Nn)[:, None]
    B = np.where((kk + nn) % 3 == 0, Q, Q << (G - 1)).astype(np.int64)
    B[7] = rng.integers(-Q, Q + 1, K) << rng.integers(0, G, K)
    a, b = _encode(A, bits, G), _encode(B, bits, G)
    one = torch.ones(1, device="cuda")
    ones = torch.ones(Nn, device="cuda")
    y = torch.zeros((M, Nn), device="cuda")
    acc = torch.zeros((M, Nn), dtype=torch.int64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    N.shiftquant_gemm_fwd(a, one, b, ones, M, Nn, K, bits, G, y, acc, None, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    T = A @ B.T
    np.testing.assert_array_equal(acc.cpu().numpy(), T)
    assert_close_f32(y.cpu().numpy(), T.astype(np.float64) * 2.0 ** -(G - 1), "Y")


@pytest.mark.parametrize("bits,T", [(8, 4000), (6, 20000), (4, 9000)])
def test_worst_case_wgrad(bits, T):
    Q = 2 ** (bits - 1) - 1
    G = 4
    Ci, Co = 140, 270
    rng = np.random.default_rng(T)
    X = np.full((Ci, T), Q, np.int64)
    X[::3] = rng.integers(-Q, Q + 1, (len(X[::3]), T))
    Y = np.full((Co, T), Q, np.int64)
    Y[:, ::5] = 1
    ex = rng.integers(0, G, Ci).astype(np.uint8)
    ey = rng.integers(0, G, Co).astype(np.uint8)
    a, b = _encode(X, bits, G), _encode(Y, bits, G)
    one = torch.ones(1, device="cuda")
    dw = torch.zeros((Ci, Co), device="cuda")
    acc = torch.zeros((Ci, Co), dtype=torch.int64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    N.shiftquant_gemm_wgrad(a, one, torch.from_numpy(ex).cuda(), b, one,
                            torch.from_numpy(ey).cuda(), Ci, Co, T, bits, G, dw, acc, None, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    raw = X @ Y.T
    sh = (2 * (G - 1) - ex.astype(np.int64)[:, None] - ey.astype(np.int64)[None, :])
    np.testing.assert_array_equal(acc.cpu().numpy(), raw << sh)
    assert_close_f32(dw.cpu().numpy(), raw * 2.0 ** -(ex[:, None] + ey[None, :]).astype(np.float64),
                     "dW")


@pytest.mark.parametrize("which,bits,G,K", [(0, 8, 4, 20000), (1, 8, 4, 21000), (0, 8, 5, 10000),
                                            (1, 6, 4, 330000)])
def test_int64_accumulation_beyond_the_int32_range(which, bits, G, K):
    # max|T| = Q^2 2^(G-1) K passes 2^31: the K loop splits into int32-exact parts whose sums
    # add in int64 in the workspace.  Same-sign worst-case products drive T past 2^31, odd
    # products are mixed in, and T is compared with the exact integer product.
    Q = 2 ** (bits - 1) - 1
    M, Nn = 130, 260
    rng = np.random.default_rng(K + which)
    A = np.full((M, K), Q, np.int64)
    A[1::2] *= -1
    A[5] = rng.integers(-Q, Q + 1, K)
    kk = np.arange(K)[None, :]
    nn = np.arange(Nn)[:, None]
    B = np.where((kk + nn) % 7 == 0, Q - 1, Q << (G - 1)).astype(np.int64)
    B[7] = rng.integers(-Q, Q + 1, K) << rng.integers(0, G, K)
    # the reference product in binary64 BLAS: every partial sum is an integer below 2^53,
    # so it is exact whatever the summation order
    T = np.rint(A.astype(np.float64) @ B.T.astype(np.float64)).astype(np.int64)
    assert np.abs(T).max() > 2**31 and Q * Q * (1 << (G - 1)) * K > 2**31
    a, b = _encode(A, bits, G), _encode(B, bits, G)
    one = torch.ones(1, device="cuda")
    ones = torch.ones(Nn, device="cuda")
    y = torch.zeros((M, Nn), device="cuda")
    acc = torch.zeros((M, Nn), dtype=torch.int64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    need = N.shiftquant_gemm_workspace_bytes(which, M, Nn, K, bits, G)
    assert need >= M * Nn * 8
    ws = torch.zeros(need // 4, dtype=torch.int32, device="cuda")
    fn = N.shiftquant_gemm_fwd if which == 0 else N.shiftquant_gemm_dgrad
    # without the workspace the call is refused before any launch
    with pytest.raises(N.ShiftQuantError) as e:
        fn(a, one, b, ones, M, Nn, K, bits, G, y, acc, None, st)
    assert e.value.status == N.SQ_EUNSUPPORTED and "int64" in str(e.value)
    fn(a, one, b, ones, M, Nn, K, bits, G, y, acc, ws, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    np.testing.assert_array_equal(acc.cpu().numpy(), T)
    assert_close_f32(y.cpu().numpy(), T.astype(np.float64) * 2.0 ** -(G - 1), "Y")


def test_int64_weight_gradient_beyond_the_int32_range():
    # 8 bits over 160000 tokens: Q^2 T > 2^31, the token loop splits into int32-exact parts
    bits, G, T = 8, 4, 160000
    Q = 2 ** (bits - 1) - 1
    Ci, Co = 96, 136
    rng = np.random.default_rng(3)
    X = np.full((Ci, T), Q, np.int64)
    X[::5] = rng.integers(-Q, Q + 1, (len(X[::5]), T))
    Y = np.full((Co, T), Q, np.int64)
    Y[:, ::9] = 1
    ex = rng.integers(0, G, Ci).astype(np.uint8)
    ey = rng.integers(0, G, Co).astype(np.uint8)
    a, b = _encode(X, bits, G), _encode(Y, bits, G)
    raw = (torch.from_numpy(X).double() @ torch.from_numpy(Y).double().T).numpy()
    raw = np.rint(raw).astype(np.int64)   # every partial sum is below 2^53: exact in binary64
    assert np.abs(raw).max() > 2**31
    one = torch.ones(1, device="cuda")
    dw = torch.zeros((Ci, Co), device="cuda")
    acc = torch.zeros((Ci, Co), dtype=torch.int64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    need = N.shiftquant_gemm_workspace_bytes(2, Ci, Co, T, bits, G)
    ws = torch.zeros(need // 4, dtype=torch.int32, device="cuda")
    N.shiftquant_gemm_wgrad(a, one, torch.from_numpy(ex).cuda(), b, one,
                            torch.from_numpy(ey).cuda(), Ci, Co, T, bits, G, dw, acc, ws, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    sh = (2 * (G - 1) - ex.astype(np.int64)[:, None] - ey.astype(np.int64)[None, :])
    np.testing.assert_array_equal(acc.cpu().numpy(), raw << sh)
    assert_close_f32(dw.cpu().numpy(), raw * 2.0 ** -(ex[:, None] + ey[None, :]).astype(np.float64),
                     "dW")


def test_layer_launch_with_an_int64_gemm_matches_oracle():
    # the layer launch mixes a forward GEMM past the int32 range (8 bits, K = 17000: int64
    # splits) with the loss-propagation and weight-gradient GEMMs of ordinary ranges
    rng = np.random.default_rng(17)
    run_and_compare(*layer_inputs(rng, 256, 17000, 256), 8, 4, fused=True)


def test_empty_and_zero_inner_dims():
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    one = torch.ones(1, device="cuda")
    codes = L.empty_codes(8, 16, 4, 4, "cuda")
    y = torch.full((8, 8), 5.0, device="cuda")
    acc = torch.full((8, 8), 5, dtype=torch.int64, device="cuda")
    # K = 0: T = 0, Y = 0
    N.shiftquant_gemm_fwd(codes[:, :0], one, codes[:, :0], torch.ones(8, device="cuda"), 8, 8, 0,
                          4, 4, y, acc, None, st)
    torch.cuda.synchronize()
    assert (y == 0).all() and (acc == 0).all() and st.item() == 0
    # M = 0 / N = 0: nothing happens
    N.shiftquant_gemm_fwd(codes, one, codes, torch.ones(8, device="cuda"), 0, 8, 16, 4, 4,
                          y[:0], None, None, st)
    N.shiftquant_gemm_dgrad(codes, one, codes, torch.ones(8, device="cuda"), 8, 0, 16, 4, 4,
                            y[:, :0], None, None, st)
    torch.cuda.synchronize()
    assert st.item() == 0


def test_zero_gradient_gives_zero_outputs():
    rng = np.random.default_rng(1)
    x, w, dy = layer_inputs(rng, 100, 64, 80)
    dy[:] = 0
    lay = run_and_compare(x, w, dy, 4, 4)
    assert (lay.dx == 0).all() and (lay.dw == 0).all()


def test_concurrent_step_equals_serial_step():
    # the five-stream step (as captured in the benchmark's CUDA graph) computes exactly
    # what the serial step computes
    rng = np.random.default_rng(77)
    x, w, dy = layer_inputs(rng, 4096, 320, 192)
    ser = L.QuantLinear(4096, 320, 192, 4, 4, "cuda", with_acc=True)
    con = L.QuantLinear(4096, 320, 192, 4, 4, "cuda", with_acc=True)
    xg, wg, dyg = to_gpu(x), to_gpu(w), to_gpu(dy)
    ser.step(xg, wg, dyg, 5)
    streams = [torch.cuda.Stream() for _ in range(5)]
    graph = L.CapturedStep(lambda: con.step_concurrent(xg, wg, dyg, 5, streams))
    graph.replay()
    graph.replay()
    torch.cuda.synchronize()
    assert ser.status.item() == 0 and con.status.item() == 0
    for k in ("fwd", "dgrad", "wgrad"):
        np.testing.assert_array_equal(ser.acc[k].cpu().numpy(), con.acc[k].cpu().numpy())
    for a, b in ((ser.y, con.y), (ser.dx, con.dx), (ser.dw, con.dw)):
        np.testing.assert_array_equal(a.cpu().numpy(), b.cpu().numpy())


def test_c_host_steps_equal_device_steps():
    # shiftquant_layer_step_host_split (copies in on a copy-in stream, the layer's whole step
    # on the layer's stream, copies back on a copy-out stream, inside one C call) driven by
    # layer.HostSteps on two alternating buffer sets: every step's host outputs equal a
    # device-resident step on the same inputs and seed
    shapes = [(3000, 640, 384), (3000, 384, 640)]
    bits, G, seed, steps = 6, 4, 0x5EED, 5
    pipe = L.HostSteps(shapes, bits, G, "cuda")
    host_in, host_out = [], []
    for i in range(steps):
        rng = np.random.default_rng(100 + i)
        host_in.append([tuple(torch.from_numpy(a).pin_memory() for a in layer_inputs(rng, *sh))
                        for sh in shapes])
        host_out.append([tuple(torch.empty(shp, dtype=torch.float32).pin_memory()
                               for shp in ((M, Nn), (M, K), (K, Nn)))
                         for (M, K, Nn) in shapes])
    pipe.run(host_in, host_out, seed=seed).synchronize()
    assert pipe.status_ok()
    ref = [L.QuantLinear(M, K, Nn, bits, G, "cuda") for (M, K, Nn) in shapes]
    for i in range(steps):
        for li, lay in enumerate(ref):
            x, w, dy = (t.cuda() for t in host_in[i][li])
            lay.step(x, w, dy, seed + i)
            torch.cuda.synchronize()
            assert lay.status.item() == 0
            for got, want in zip(host_out[i][li], (lay.y, lay.dx, lay.dw)):
                np.testing.assert_array_equal(got.numpy(), want.cpu().numpy())


@pytest.mark.parametrize("bits,transposed", [(4, True), (4, False), (6, False)])
def test_c_layer_step_matches_oracle(bits, transposed):
    # shiftquant_layer_step on device inputs: the whole step against the oracle's layer; with
    # transposed=False the step writes no transposed copies and dW reads the codes in place
    rng = np.random.default_rng(77 + bits)
    M, K, Nn, G, seed = 1000, 320, 288, 4, 0xABC
    x, w, dy = layer_inputs(rng, M, K, Nn)
    lay = L.QuantLinear(M, K, Nn, bits, G, "cuda", transposed=transposed)
    N.shiftquant_layer_step(lay.step_args(to_gpu(x), to_gpu(w), to_gpu(dy)), seed)
    torch.cuda.synchronize()
    assert lay.status.item() == 0
    ox = O.shiftquant_tensor(x, bits, G, 0)
    og = O.shiftquant_tensor(dy, bits, G, 1, seed)
    wf = O.channel_tensor(w, bits, 0)
    wd = O.channel_tensor(w, bits, 1)
    want = (O.dequant(O.gemm_fwd(ox["codes"], ox["exp"], wf["codes"], G), ox["scale"], 1.0,
                      G - 1, wf["scale"]),
            O.dequant(O.gemm_dgrad(og["codes"], og["exp"], wd["codes"], G), og["scale"], 1.0,
                      G - 1, wd["scale"]),
            O.dequant(O.gemm_wgrad(ox["codes"], ox["exp"], og["codes"], og["exp"], G),
                      ox["scale"], og["scale"], 2 * (G - 1)))
    for got, ref, what in zip((lay.y, lay.dx, lay.dw), want, ("Y", "dX", "dW")):
        assert_close_f32(got.cpu().numpy(), ref, what)


@pytest.mark.parametrize("M,K,Nn", [(5, 3, 7), (300, 1000, 513), (4096, 64, 96), (2000, 700, 256)])
@pytest.mark.parametrize("bits", [4, 6, 8])
def test_layer_gemms_in_one_launch_match_oracle(M, K, Nn, bits):
    # shiftquant_gemm_layer: the three GEMMs share one persistent launch (and one workspace)
    rng = np.random.default_rng(M + K + Nn + bits)
    run_and_compare(*layer_inputs(rng, M, K, Nn), bits, 4, fused=True)


def test_layer_gemms_equal_separate_launches():
    rng = np.random.default_rng(5)
    x, w, dy = layer_inputs(rng, 3000, 640, 384)
    a = run_and_compare(x, w, dy, 6, 4, fused=True)
    b = run_and_compare(x, w, dy, 6, 4, fused=False)
    for t, u in ((a.y, b.y), (a.dx, b.dx), (a.dw, b.dw)):
        np.testing.assert_array_equal(t.cpu().numpy(), u.cpu().numpy())


@pytest.mark.parametrize("M,K,Nn,bits", [(12544, 2304, 256, 4), (4096, 64, 96, 6),
                                         (3000, 640, 384, 6), (12608, 768, 3072, 6)])
def test_layer_launch_count_query_matches_the_launch(M, K, Nn, bits):
    # shiftquant_gemm_layer_kernel_launches predicts the kernels one layer call launches (the
    # GEMM launch and one output pass per split GEMM); count them in a profiler trace
    from torch.profiler import ProfilerActivity, profile
    rng = np.random.default_rng(M + Nn)
    x, w, dy = layer_inputs(rng, M, K, Nn)
    lay = L.QuantLinear(M, K, Nn, bits, 4, "cuda")
    lay.quantize_activation(to_gpu(x))
    lay.quantize_gradient(to_gpu(dy), 3)
    lay.quantize_weights(to_gpu(w))
    torch.cuda.synchronize()
    with profile(activities=[ProfilerActivity.CUDA]):   # the first session may record nothing
        torch.zeros(1, device="cuda").add_(1)
        torch.cuda.synchronize()
    with profile(activities=[ProfilerActivity.CUDA]) as prof:
        lay.gemms()
        torch.cuda.synchronize()
    names = [e.name for e in prof.events()]
    ours = [n for n in names if "shiftmm_kernel" in n or "splitk_finalize_kernel" in n]
    if not ours:
        pytest.skip("the profiler recorded no kernels on this machine")
    assert lay.status.item() == 0
    want = N.shiftquant_gemm_layer_kernel_launches(M, K, Nn, bits, 4, lay.ws_layer.numel() * 4)
    assert len(ours) == want, ours
    assert N.shiftquant_gemm_layer_kernel_launches(M, K, Nn, bits, 4, 0) == 1


@pytest.mark.parametrize("mask", [1, 2, 4, 5, 6])
def test_layer_launch_subsets_match_the_full_launch(mask):
    # gemm_mask runs a subset of the layer's GEMMs (bit 0 forward, 1 loss propagation,
    # 2 weight gradient); max_ctas caps the grid: each output equals the full launch's, and
    # the outputs left out stay untouched
    rng = np.random.default_rng(40 + mask)
    x, w, dy = layer_inputs(rng, 2000, 700, 256)
    full = L.QuantLinear(2000, 700, 256, 4, 4, "cuda")
    part = L.QuantLinear(2000, 700, 256, 4, 4, "cuda")
    for lay in (full, part):
        lay.quantize_activation(to_gpu(x))
        lay.quantize_gradient(to_gpu(dy), 9)
        lay.quantize_weights(to_gpu(w))
    full.gemms()
    for t in (part.y, part.dx, part.dw):
        t.fill_(-3.0)
    part.gemms(gemm_mask=mask, max_ctas=37)
    torch.cuda.synchronize()
    assert full.status.item() == 0 and part.status.item() == 0
    for bit, a, b in ((1, full.y, part.y), (2, full.dx, part.dx), (4, full.dw, part.dw)):
        if mask & bit:
            np.testing.assert_array_equal(a.cpu().numpy(), b.cpu().numpy())
        else:
            assert (b == -3.0).all()


def test_step_with_a_separate_loss_propagation_launch_equals_the_fused_step():
    rng = np.random.default_rng(41)
    x, w, dy = layer_inputs(rng, 4096, 320, 192)
    fused = L.QuantLinear(4096, 320, 192, 6, 4, "cuda", with_acc=True)
    split = L.QuantLinear(4096, 320, 192, 6, 4, "cuda", with_acc=True)
    xg, wg, dyg = to_gpu(x), to_gpu(w), to_gpu(dy)
    streams = [torch.cuda.Stream() for _ in range(5)]
    g1 = L.CapturedStep(lambda: fused.step_concurrent(xg, wg, dyg, 5, streams))
    g2 = L.CapturedStep(lambda: split.step_concurrent(xg, wg, dyg, 5, streams, dgrad_ctas=40))
    g1.replay()
    g2.replay()
    torch.cuda.synchronize()
    assert fused.status.item() == 0 and split.status.item() == 0
    for k in ("fwd", "dgrad", "wgrad"):
        np.testing.assert_array_equal(fused.acc[k].cpu().numpy(), split.acc[k].cpu().numpy())
    for a, b in ((fused.y, split.y), (fused.dx, split.dx), (fused.dw, split.dw)):
        np.testing.assert_array_equal(a.cpu().numpy(), b.cpu().numpy())


@pytest.mark.parametrize("bits,G,K", [(8, 4, 5000), (6, 4, 9000), (4, 4, 30000), (8, 3, 3000)])
def test_layer_chunks_from_exponents_stay_exact(bits, G, K):
    # The layer launch sizes its exact FP32 chunks from the inner channels' exponents.
    # Codes at the largest magnitude with one sign per row, a few channels in group 0 (the
    # largest fold) among many in the last group, and odd products mixed in: every chunk's
    # partial sums reach the bound, and an off-by-one chunk would round away odd terms.
    Q = 2 ** (bits - 1) - 1
    M, Nn = 130, 260
    rng = np.random.default_rng(K + bits)
    e = np.full(K, G - 1, np.int64)
    e[::17] = 0
    e[5::41] = 1
    A = np.full((M, K), Q, np.int64)
    A[1::2] *= -1
    A[3] = rng.integers(-Q, Q + 1, K)
    Bq = np.where((np.arange(K)[None, :] + np.arange(Nn)[:, None]) % 3 == 0, Q, Q - 1)
    Bq[9] = rng.integers(-Q, Q + 1, K)
    Bf = Bq.astype(np.int64) << (G - 1 - e)[None, :]
    a, b = _encode(A, bits, G), _encode(Bf, bits, G)
    xe = torch.from_numpy(e.astype(np.uint8)).cuda()
    one = torch.ones(1, device="cuda")
    ones = torch.ones(Nn, device="cuda")
    y = torch.zeros((M, Nn), device="cuda")
    acc = torch.zeros((M, Nn), dtype=torch.int64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    N.shiftquant_gemm_layer(a, None, one, xe, None, None, None, None, b, ones, None, None,
                            M, K, Nn, bits, G, y, None, None, acc_y=acc, dev_status=st,
                            gemm_mask=1)
    torch.cuda.synchronize()
    assert st.item() == 0
    T = A @ Bf.T
    np.testing.assert_array_equal(acc.cpu().numpy(), T)
    assert_close_f32(y.cpu().numpy(), T.astype(np.float64) * 2.0 ** -(G - 1), "Y")


@pytest.mark.parametrize("bits", [4, 6, 8])
def test_token_shards_weight_gradient_is_exact(bits):
    # data parallel over tokens, exactly: two shards quantized with the range exchange
    # (layer.shard_shift_quantize), each shard's int32 weight-gradient sums
    # (shiftquant_gemm_wgrad_partial), their sum standing in for the all-reduce, and one
    # dequantizing pass (shiftquant_gemm_wgrad_finish) give the whole batch's dW and T
    rng = np.random.default_rng(40 + bits)
    M, K, Nn, G, seed = 3000, 320, 256, 4, 77
    x, w, dy = layer_inputs(rng, M, K, Nn)
    xg, dyg = to_gpu(x), to_gpu(dy)
    whole = L.QuantLinear(M, K, Nn, bits, G, "cuda", with_acc=True)
    whole.quantize_activation(xg)
    whole.quantize_gradient(dyg, seed)
    whole.wgrad()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    bounds = [(0, 1337), (1337, M)]
    qx = [L.ShiftTensor.alloc(r1 - r0, K, bits, G, "cuda") for r0, r1 in bounds]
    qg = [L.ShiftTensor.alloc(r1 - r0, Nn, bits, G, "cuda") for r0, r1 in bounds]
    for t, qs in ((xg, qx), (dyg, qg)):
        parts = []
        for (r0, r1), q in zip(bounds, qs):
            N.shiftquant_calibrate(t[r0:r1], N.SQ_GRAN_PER_COL, G, q.range, None, None, st)
            parts.append(q.range.clone())
        both = torch.maximum(parts[0], parts[1])
        mode, sd = (N.SQ_ROUND_NEAREST_EVEN, 0) if t is xg else (N.SQ_ROUND_STOCHASTIC, seed)
        for (r0, r1), q in zip(bounds, qs):
            L.shard_shift_quantize(t[r0:r1], q, bits, G, mode, sd, r0, st,
                                   lambda r, both=both: r.copy_(both))
    sums = []
    for (r0, r1), a, b in zip(bounds, qx, qg):
        tt = torch.full((K, Nn), -1, dtype=torch.int32, device="cuda")
        N.shiftquant_gemm_wgrad_partial(a.codes_t, a.scale, a.exp, b.codes_t, b.scale, b.exp, K, Nn,
                                        r1 - r0, M, bits, G, tt, st)
        sums.append(tt)
    total = sums[0] + sums[1]
    dw = torch.empty((K, Nn), dtype=torch.float32, device="cuda")
    acc = torch.empty((K, Nn), dtype=torch.int64, device="cuda")
    N.shiftquant_gemm_wgrad_finish(total, K, Nn, bits, G, qx[0].scale, qx[0].exp, qg[0].scale,
                                   qg[0].exp, dw, acc, st)
    torch.cuda.synchronize()
    assert st.item() == 0 and whole.status.item() == 0
    np.testing.assert_array_equal(acc.cpu().numpy(), whole.acc["wgrad"].cpu().numpy())
    np.testing.assert_array_equal(f32_bits(dw.cpu().numpy()), f32_bits(whole.dw.cpu().numpy()))


@pytest.mark.parametrize("M,K,Nn,bits", [(4096, 512, 768, 6), (1000, 300, 250, 4),
                                         (200, 2304, 256, 4), (3000, 4096, 1024, 6)])
def test_fused_output_ranges_equal_a_range_pass_of_the_outputs(M, K, Nn, bits):
    # y_range / dx_range of the layer launch (formed in the epilogue, or in the split-K output
    # pass for a GEMM with few tiles) against the oracle's range pass over the GPU's own fp32
    # Y and dX, bit for bit; ragged tiles, single and pair tile modes
    rng = np.random.default_rng(M + K + Nn)
    x, w, dy = layer_inputs(rng, M, K, Nn)
    G = 4
    lay = L.QuantLinear(M, K, Nn, bits, G, "cuda")
    lay.quantize_activation(to_gpu(x))
    lay.quantize_gradient(to_gpu(dy), 5)
    lay.quantize_weights(to_gpu(w))
    yr = torch.full((Nn,), 7.0, device="cuda")      # stale values: the call zeroes them first
    dxr = torch.full((K,), 7.0, device="cuda")
    lay.gemms(y_range=yr, dx_range=dxr)
    torch.cuda.synchronize()
    assert lay.status.item() == 0
    for out, got, what in ((lay.y, yr, "Y"), (lay.dx, dxr, "dX")):
        want, st = O.range_cols(out.cpu().numpy())
        assert st == 0
        np.testing.assert_array_equal(f32_bits(got.cpu().numpy()), f32_bits(want), err_msg=what)


@pytest.mark.parametrize("bits", [4, 6])
def test_chain_with_fused_ranges_equals_separate_range_passes(bits):
    # a three-layer chain trained forward then backward: the fused range outputs replace the
    # range passes of the inner activations and gradients and change no bit of any result
    M, dims, G, seed = 1500, (320, 512, 384, 256), 4, 0x77
    rng = np.random.default_rng(bits)
    x0 = to_gpu(rng.standard_normal((M, dims[0])).astype(np.float32))
    ws = [to_gpu((rng.standard_normal((dims[i], dims[i + 1])) * 0.05).astype(np.float32))
          for i in range(3)]
    dy = to_gpu((rng.laplace(0, 1, (M, dims[-1])) * np.exp(rng.normal(0, 2, dims[-1])))
                .astype(np.float32))
    out = []
    for fused in (True, False):
        ch = L.LinearChain(M, dims, bits, G, "cuda", fused_ranges=fused)
        ch.step(x0, ws, dy, seed)
        torch.cuda.synchronize()
        assert ch.status_ok()
        out.append(ch)
    a, b = out
    for la, lb in zip(a.layers, b.layers):
        for t, u in ((la.y, lb.y), (la.dx, lb.dx), (la.dw, lb.dw), (la.x.exp, lb.x.exp),
                     (la.g.exp, lb.g.exp), (la.x.tau0, lb.x.tau0), (la.g.tau0, lb.g.tau0)):
            np.testing.assert_array_equal(t.cpu().numpy(), u.cpu().numpy())
        np.testing.assert_array_equal(decode(la.x.codes), decode(lb.x.codes))
        np.testing.assert_array_equal(decode(la.g.codes), decode(lb.g.codes))
    # the inner tensors really were grouped from the fused ranges
    for l in range(2):
        want, _ = O.range_cols(a.layers[l].y.cpu().numpy())
        np.testing.assert_array_equal(f32_bits(a.y_range[l].cpu().numpy()), f32_bits(want))


def test_c_host_step_on_one_stream_equals_device_step():
    # shiftquant_layer_step_host: copies in, the step and copies back in one stream's order
    M, K, Nn = 1000, 384, 640
    bits, G, seed = 4, 4, 0xBEEF
    rng = np.random.default_rng(7)
    x, w, dy = (torch.from_numpy(a).pin_memory() for a in layer_inputs(rng, M, K, Nn))
    outs = [torch.empty(shp, dtype=torch.float32).pin_memory() for shp in ((M, Nn), (M, K), (K, Nn))]
    lay = L.QuantLinear(M, K, Nn, bits, G, "cuda", with_inputs=True)
    ev = torch.cuda.Event()
    ev.record()
    N.shiftquant_layer_step_host(lay.step_args(), x, w, dy, *outs, seed, inputs_queued=ev)
    torch.cuda.synchronize()
    assert lay.status.item() == 0
    ref = L.QuantLinear(M, K, Nn, bits, G, "cuda")
    ref.step(x.cuda(), w.cuda(), dy.cuda(), seed)
    torch.cuda.synchronize()
    for got, want in zip(outs, (ref.y, ref.dx, ref.dw)):
        np.testing.assert_array_equal(got.numpy(), want.cpu().numpy())
