"""Helpers for the GPU-vs-oracle parity tests: run the oracle chain of one quantized layer
on numpy inputs, run the CUDA path on the same inputs, and compare element by element."""
from __future__ import annotations

import numpy as np
import torch

import oracle as O

# fp32 outputs: the GPU epilogue rounds int->fp32, the scale product and the final
# multiply (three roundings, <= 3 * 2^-24 relative) against the oracle's single rounding
# of the binary64 product: within 1e-6 relative
RTOL = 1e-6
ATOL = 1e-35


def to_gpu(a: np.ndarray, ld: int | None = None) -> torch.Tensor:
    """Copy a 2-D float32 array to the device, optionally with a padded leading dim."""
    R, C = a.shape
    if ld is None or ld == C:
        return torch.from_numpy(np.ascontiguousarray(a)).cuda()
    buf = torch.zeros((R, ld), dtype=torch.float32, device="cuda")
    buf[:, :C] = torch.from_numpy(np.ascontiguousarray(a)).cuda()
    return buf[:, :C]


def decode(t: torch.Tensor) -> np.ndarray:
    """Integer values of a code tensor (E4M3 bytes or BF16)."""
    v = t.view(torch.float8_e4m3fn).float() if t.dtype == torch.uint8 else t.float()
    a = v.cpu().numpy().astype(np.float64)
    assert np.all(a == np.round(a)), "a stored code is not an integer"
    return a.astype(np.int64)


def f32_bits(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, np.float32)).view(np.uint32)


def oracle_layer(x, w, dy, bits, G, seed, rows=None, wrows=None):
    """Oracle chain of one layer.  rows/wrows restrict the GEMM outputs that are computed
    (rows of Y and dX, rows = input channels of dW)."""
    ox = O.shiftquant_tensor(x, bits, G, mode=0)
    og = O.shiftquant_tensor(dy, bits, G, mode=1, seed=seed)
    owf = O.channel_tensor(w, bits, axis=0)
    owd = O.channel_tensor(w, bits, axis=1)
    T_f = O.gemm_fwd(ox["codes"], ox["exp"], owf["codes"], G, rows)
    T_d = O.gemm_dgrad(og["codes"], og["exp"], owd["codes"], G, rows)
    T_w = O.gemm_wgrad(ox["codes"], ox["exp"], og["codes"], og["exp"], G, wrows)
    return {
        "x": ox, "g": og, "wf": owf, "wd": owd,
        "T_fwd": T_f, "T_dgrad": T_d, "T_wgrad": T_w,
        "y": O.dequant(T_f, ox["scale"], 1.0, G - 1, owf["scale"]),
        "dx": O.dequant(T_d, og["scale"], 1.0, G - 1, owd["scale"]),
        "dw": O.dequant(T_w, ox["scale"], og["scale"], 2 * (G - 1)),
    }


def assert_close_f32(got: np.ndarray, ref: np.ndarray, what: str):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    err = np.abs(got - ref)
    bad = err > RTOL * np.abs(ref) + ATOL
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {int(bad.sum())} elements beyond {RTOL} relative, first at "
                             f"{tuple(i)}: got {got[tuple(i)]!r} want {ref[tuple(i)]!r}")


def compare_shift(gpu_q, ora: dict, what: str, check_t: bool = True):
    """Bit-exact comparison of a ShiftTensor against the oracle's dict."""
    np.testing.assert_array_equal(f32_bits(gpu_q.range.cpu().numpy()), f32_bits(ora["range"]),
                                  err_msg=f"{what}: ranges")
    assert f32_bits([gpu_q.tau0.item()])[0] == f32_bits([ora["tau0"]])[0], f"{what}: tau0"
    np.testing.assert_array_equal(gpu_q.exp.cpu().numpy(), ora["exp"], err_msg=f"{what}: exps")
    assert f32_bits([gpu_q.scale.item()])[0] == f32_bits([ora["scale"]])[0], f"{what}: scale"
    np.testing.assert_array_equal(decode(gpu_q.codes), ora["codes"].astype(np.int64),
                                  err_msg=f"{what}: codes")
    if check_t and gpu_q.codes_t is not None:
        np.testing.assert_array_equal(decode(gpu_q.codes_t), ora["codes"].astype(np.int64).T,
                                      err_msg=f"{what}: transposed codes")


def folded(codes: np.ndarray, exps: np.ndarray, G: int, axis: int) -> np.ndarray:
    """Weight codes times 2^(G-1-e) along the GEMM inner index (axis 0: rows, 1: columns)."""
    f = (1 << (G - 1 - exps.astype(np.int64)))
    return codes.astype(np.int64) * (f[:, None] if axis == 0 else f[None, :])
