"""Parity at the benchmark's full sizes, in the launch configuration the benchmark times
(the five-stream step captured in a CUDA graph, each layer's X and dY codes with or
without transposed copies as the library advises, as the benchmark builds them), for every
workload: the quantizer outputs of every tensor compared in full (ranges, tau_0,
exponents, scales, codes and, where kept, transposed codes, bit-exact), and the three GEMMs
on sampled output rows (integer accumulators bit-exact, fp32 outputs within 1e-6
relative)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2411_10948_gb300 import layer as L
from paper_2411_10948_gb300 import native as N
from paper_2411_10948_gb300 import workloads as W
from parity_util import assert_close_f32, decode, f32_bits

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

SEED = 3
SR_SEED = 0x5EED


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2411_10948_gb300 import build
    build.build_library()
    N.load()


def _compare_codes_chunked(gpu_codes, ora_codes, what, transpose=False, chunk=4096):
    """Decode the GPU codes block by block (host memory stays bounded) and compare."""
    R = gpu_codes.shape[0]
    for r in range(0, R, chunk):
        got = decode(gpu_codes[r:r + chunk])
        want = (ora_codes[:, r:r + chunk].T if transpose else ora_codes[r:r + chunk]).astype(np.int64)
        if not np.array_equal(got, want):
            bad = np.argwhere(got != want)[0]
            raise AssertionError(f"{what}: first mismatch at {(r + bad[0], bad[1])}: "
                                 f"{got[tuple(bad)]} vs {want[tuple(bad)]}")


def _compare_shift(q, o, what):
    np.testing.assert_array_equal(f32_bits(q.range.cpu().numpy()), f32_bits(o["range"]), what)
    assert f32_bits([q.tau0.item()])[0] == f32_bits([o["tau0"]])[0], what
    np.testing.assert_array_equal(q.exp.cpu().numpy(), o["exp"], what)
    assert f32_bits([q.scale.item()])[0] == f32_bits([o["scale"]])[0], what
    _compare_codes_chunked(q.codes, o["codes"], what + " codes")
    if q.codes_t is not None:
        _compare_codes_chunked(q.codes_t, o["codes"], what + " transposed codes", transpose=True)


@pytest.mark.parametrize("name", ["wgrad_small", "conv3x3", "vit_mlp", "vit_block",
                                  "large_linear", "large_linear_8bit"])
def test_workload_full_size(name):
    wl = W.workload(name)
    rng = np.random.default_rng(17)
    for li, spec in enumerate(wl.layers):
        x, w, dy = W.np_layer_inputs(spec, SEED, li)
        G, bits = spec.n_groups, spec.bits
        lay = L.QuantLinear(spec.M, spec.K, spec.N, bits, G, "cuda", with_acc=True, transposed=None)
        want_t = N.shiftquant_gemm_layer_wgrad_in_place(spec.M, spec.K, spec.N, bits, G) != 1
        assert (lay.x.codes_t is not None) == want_t
        xg, wg, dyg = (torch.from_numpy(a).cuda() for a in (x, w, dy))
        streams = [torch.cuda.Stream() for _ in range(5)]
        graph = L.CapturedStep(lambda: lay.step_concurrent(xg, wg, dyg, SR_SEED, streams))
        graph.replay()
        torch.cuda.synchronize()
        assert lay.status.item() == 0, f"{name}/{spec.name}: device status {lay.status.item()}"

        ox = O.shiftquant_tensor(x, bits, G, 0)
        _compare_shift(lay.x, ox, f"{name}/{spec.name} X")
        og = O.shiftquant_tensor(dy, bits, G, 1, SR_SEED)
        _compare_shift(lay.g, og, f"{name}/{spec.name} dY")
        wf = O.channel_tensor(w, bits, 0)
        wd = O.channel_tensor(w, bits, 1)
        np.testing.assert_array_equal(f32_bits(lay.wf.scale.cpu().numpy()), f32_bits(wf["scale"]))
        np.testing.assert_array_equal(f32_bits(lay.wd.scale.cpu().numpy()), f32_bits(wd["scale"]))
        fold_f = (1 << (G - 1 - ox["exp"].astype(np.int64)))[:, None]
        np.testing.assert_array_equal(decode(lay.wf.codes), (wf["codes"].astype(np.int64) * fold_f).T)
        fold_d = (1 << (G - 1 - og["exp"].astype(np.int64)))[None, :]
        np.testing.assert_array_equal(decode(lay.wd.codes), wd["codes"].astype(np.int64) * fold_d)

        # GEMMs on sampled rows: the first and last row tiles' edges plus random rows
        rows = np.unique(np.concatenate([[0, 127, 128, spec.M - 1],
                                         rng.choice(spec.M, 40, replace=False)]))
        chans = np.unique(np.concatenate([[0, spec.K - 1], rng.choice(spec.K, 24, replace=False)]))
        T_f = O.gemm_fwd(ox["codes"], ox["exp"], wf["codes"], G, rows)
        T_d = O.gemm_dgrad(og["codes"], og["exp"], wd["codes"], G, rows)
        T_w = O.gemm_wgrad(ox["codes"], ox["exp"], og["codes"], og["exp"], G, chans)
        np.testing.assert_array_equal(lay.acc["fwd"][rows].cpu().numpy(), T_f)
        np.testing.assert_array_equal(lay.acc["dgrad"][rows].cpu().numpy(), T_d)
        np.testing.assert_array_equal(lay.acc["wgrad"][chans].cpu().numpy(), T_w)
        assert_close_f32(lay.y[rows].cpu().numpy(),
                         O.dequant(T_f, ox["scale"], 1.0, G - 1, wf["scale"]), f"{name} Y")
        assert_close_f32(lay.dx[rows].cpu().numpy(),
                         O.dequant(T_d, og["scale"], 1.0, G - 1, wd["scale"]), f"{name} dX")
        assert_close_f32(lay.dw[chans].cpu().numpy(),
                         O.dequant(T_w, ox["scale"], og["scale"], 2 * (G - 1)), f"{name} dW")
        del lay, graph, xg, wg, dyg
        torch.cuda.empty_cache()
