"""ShiftQuant CPU oracle (test infrastructure only).

A ctypes front end over ``shiftquant_oracle.c``, the plain C restatement of the
paper's definitions (arXiv 2411.10948: Sec. 3.1 grouping, Eq. 3 thresholds, Eq. 4 and
App. D contraction, App. B stochastic rounding, Sec. 5.1 roles).  Only the tests, the
smoke check and the benchmark's CPU-baseline leg may import this package; the CUDA
library never does, and this package imports nothing from the CUDA side.

Every function takes and returns numpy arrays.  Codes are int8 (the paper's signed
integer format, |q| <= 2^(b-1) - 1), exponents uint8 (the group index e of each
channel, 0 = the group holding tau_0), integer accumulators int64.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "shiftquant_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libsqoracle.so")
_lock = threading.Lock()
_lib = None

# the flags that keep the arithmetic strict IEEE binary32 on x86-64 and aarch64 alike
CFLAGS = ["-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fno-fast-math",
          "-fPIC", "-shared"]


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/_build/libsqoracle.so`` (gcc, no GPU needed)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or \
            os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", *CFLAGS, _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        i64, i32, u64, f32 = ctypes.c_int64, ctypes.c_int, ctypes.c_uint64, ctypes.c_float
        vp = ctypes.c_void_p
        lib.sqo_max_threads.argtypes = []
        lib.sqo_max_threads.restype = i32
        lib.sqo_hash.argtypes = [u64, u64]
        lib.sqo_hash.restype = u64
        lib.sqo_range_cols.argtypes = [vp, i64, i64, i64, vp]
        lib.sqo_range_rows.argtypes = [vp, i64, i64, i64, vp]
        lib.sqo_group.argtypes = [vp, i64, i32, vp, vp]
        lib.sqo_quantize_shift.argtypes = [vp, i64, i64, i64, i32, i32, f32, vp, i32, u64,
                                           i64, vp, vp]
        lib.sqo_quantize_channel.argtypes = [vp, i64, i64, i64, i32, i32, vp, i32, u64, vp,
                                             vp]
        lib.sqo_gemm_fwd.argtypes = [vp, vp, vp, i64, i64, i64, i32, vp, i64, vp]
        lib.sqo_gemm_dgrad.argtypes = [vp, vp, vp, i64, i64, i64, i32, vp, i64, vp]
        lib.sqo_gemm_wgrad.argtypes = [vp, vp, vp, vp, i64, i64, i64, i32, vp, i64, vp]
        lib.sqo_dequant.argtypes = [vp, i64, i64, f32, f32, i32, vp, vp]
        lib.sqo_pack4.argtypes = [vp, i64, i64, vp]
        lib.sqo_unpack4.argtypes = [vp, i64, i64, vp]
        lib.sqo_pack_groups.argtypes = [vp, i64, i32, vp]
        lib.sqo_unpack_groups.argtypes = [vp, i64, i32, vp]
        for name in ("sqo_pack4", "sqo_unpack4", "sqo_pack_groups", "sqo_unpack_groups"):
            getattr(lib, name).restype = None
        lib.sqo_l1bn_forward.argtypes = [vp, i64, i64, i32, i32, vp, vp, vp, vp, vp, vp]
        lib.sqo_l1bn_backward.argtypes = [vp, i64, i64, i32, i32, u64, vp, vp, vp, vp, vp, vp,
                                          vp]
        for name in ("sqo_range_cols", "sqo_range_rows", "sqo_group", "sqo_quantize_shift",
                     "sqo_quantize_channel", "sqo_l1bn_forward", "sqo_l1bn_backward"):
            getattr(lib, name).restype = i32
        for name in ("sqo_gemm_fwd", "sqo_gemm_dgrad", "sqo_gemm_wgrad", "sqo_dequant"):
            getattr(lib, name).restype = None
        _lib = lib
        return lib


def _p(a: np.ndarray):
    return ctypes.c_void_p(a.ctypes.data) if a is not None else None


def _f32(x) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    assert x.ndim == 2
    return x


def _rows(rows):
    if rows is None:
        return None, 0
    r = np.ascontiguousarray(rows, dtype=np.int64)
    return r, int(r.size)


def max_threads() -> int:
    """Threads the oracle's OpenMP loops use."""
    return int(_load().sqo_max_threads())


# ---------------------------------------------------------------- hash (SR draws)
def hash64(seed: int, idx: int) -> int:
    """SplitMix64 output for counter ``idx`` under ``seed`` (the SR random source)."""
    return int(_load().sqo_hash(seed & (2**64 - 1), idx & (2**64 - 1)))


# ---------------------------------------------------------------- Sec. 3.1 ranges
def range_cols(x) -> tuple[np.ndarray, int]:
    """Per-column max|x| and the non-finite status (1 if any NaN/Inf)."""
    x = _f32(x)
    out = np.empty(x.shape[1], np.float32)
    st = _load().sqo_range_cols(_p(x), x.shape[0], x.shape[1], x.shape[1], _p(out))
    return out, int(st)


def range_rows(x) -> tuple[np.ndarray, int]:
    """Per-row max|x| and the non-finite status."""
    x = _f32(x)
    out = np.empty(x.shape[0], np.float32)
    st = _load().sqo_range_rows(_p(x), x.shape[0], x.shape[1], x.shape[1], _p(out))
    return out, int(st)


# ------------------------------------------------------------------- Eq. 3 groups
def group(ranges, n_groups: int) -> tuple[np.float32, np.ndarray, int]:
    """tau_0 and the per-channel group exponents e (Eq. 3, power-of-two thresholds)."""
    r = np.ascontiguousarray(ranges, dtype=np.float32)
    e = np.empty(r.size, np.uint8)
    tau = np.zeros(1, np.float32)
    st = _load().sqo_group(_p(r), r.size, n_groups, _p(tau), _p(e))
    return np.float32(tau[0]), e, int(st)


# --------------------------------------------------------- App. D quantization
def quantize_shift(x, bits: int, n_groups: int, tau0, exps, mode: int = 0,
                   seed: int = 0, row0: int = 0) -> tuple[np.ndarray, np.float32]:
    """ShiftQuant codes (int8 [R, C]) and the tensor scale s = tau_0 / Q.  x holds rows
    row0.. of the logical tensor (stochastic rounding draws by the logical index)."""
    x = _f32(x)
    e = np.ascontiguousarray(exps, dtype=np.uint8)
    q = np.empty(x.shape, np.int8)
    s = np.zeros(1, np.float32)
    _load().sqo_quantize_shift(_p(x), x.shape[0], x.shape[1], x.shape[1], bits, n_groups,
                               np.float32(tau0), _p(e), mode, seed & (2**64 - 1), row0, _p(q),
                               _p(s))
    return q, np.float32(s[0])


def quantize_channel(x, bits: int, axis: int, ranges, mode: int = 0,
                     seed: int = 0) -> tuple[np.ndarray, np.ndarray]:
    """Per-channel codes; axis 0 = one scale per column, axis 1 = one per row."""
    x = _f32(x)
    r = np.ascontiguousarray(ranges, dtype=np.float32)
    q = np.empty(x.shape, np.int8)
    s = np.empty(x.shape[1] if axis == 0 else x.shape[0], np.float32)
    _load().sqo_quantize_channel(_p(x), x.shape[0], x.shape[1], x.shape[1], bits, axis,
                                 _p(r), mode, seed & (2**64 - 1), _p(q), _p(s))
    return q, s


# ------------------------------------------------------- Eq. 4 contractions
def gemm_fwd(qA, eA, qW, n_groups: int, rows=None) -> np.ndarray:
    """T = sum_g (qA[:, P^g] qW[P^g, :]) << (G-1-g); qA [M, K], qW [K, N] -> int64."""
    qA = np.ascontiguousarray(qA, np.int8)
    qW = np.ascontiguousarray(qW, np.int8)
    e = np.ascontiguousarray(eA, np.uint8)
    M, K = qA.shape
    N = qW.shape[1]
    r, nr = _rows(rows)
    T = np.empty((nr if r is not None else M, N), np.int64)
    _load().sqo_gemm_fwd(_p(qA), _p(e), _p(qW), M, N, K, n_groups, _p(r), nr, _p(T))
    return T


def gemm_dgrad(qY, eY, qW, n_groups: int, rows=None) -> np.ndarray:
    """T = sum_g (qY[:, P^g] qW[:, P^g]^T) << (G-1-g); qY [M, N], qW [K, N] -> [M, K]."""
    qY = np.ascontiguousarray(qY, np.int8)
    qW = np.ascontiguousarray(qW, np.int8)
    e = np.ascontiguousarray(eY, np.uint8)
    M, N = qY.shape
    K = qW.shape[0]
    r, nr = _rows(rows)
    T = np.empty((nr if r is not None else M, K), np.int64)
    _load().sqo_gemm_dgrad(_p(qY), _p(e), _p(qW), M, N, K, n_groups, _p(r), nr, _p(T))
    return T


def gemm_wgrad(qX, eX, qY, eY, n_groups: int, rows=None) -> np.ndarray:
    """T[i, j] = (sum_m qX[m, i] qY[m, j]) << ((G-1-eX_i) + (G-1-eY_j)) -> [K, N]."""
    qX = np.ascontiguousarray(qX, np.int8)
    qY = np.ascontiguousarray(qY, np.int8)
    ex = np.ascontiguousarray(eX, np.uint8)
    ey = np.ascontiguousarray(eY, np.uint8)
    M, K = qX.shape
    N = qY.shape[1]
    r, nr = _rows(rows)
    T = np.empty((nr if r is not None else K, N), np.int64)
    _load().sqo_gemm_wgrad(_p(qX), _p(ex), _p(qY), _p(ey), M, K, N, n_groups, _p(r), nr,
                           _p(T))
    return T


def dequant(T, s_a, s_b, shift: int, col_scale=None) -> np.ndarray:
    """Y = fp32( T * s_a * s_b * 2^-shift * col_scale[j] ) evaluated in binary64."""
    T = np.ascontiguousarray(T, np.int64)
    cs = None if col_scale is None else np.ascontiguousarray(col_scale, np.float32)
    Y = np.empty(T.shape, np.float32)
    _load().sqo_dequant(_p(T), T.shape[0], T.shape[1], np.float32(s_a), np.float32(s_b),
                        shift, _p(cs), _p(Y))
    return Y


# ------------------------------------------------ composite: one quantized layer
def shiftquant_tensor(x, bits: int, n_groups: int, mode: int = 0, seed: int = 0) -> dict:
    """Range pass, grouping and quantization of an activation or gradient [R, C]."""
    rng, st1 = range_cols(x)
    tau0, e, st2 = group(rng, n_groups)
    q, s = quantize_shift(x, bits, n_groups, tau0, e, mode, seed)
    return {"range": rng, "tau0": tau0, "exp": e, "codes": q, "scale": s,
            "status": st1 | st2}


def channel_tensor(w, bits: int, axis: int, mode: int = 0, seed: int = 0) -> dict:
    """Per-channel quantization of a weight [K, N]; axis 0 per column, 1 per row."""
    rng, st = (range_cols(w) if axis == 0 else range_rows(w))
    q, s = quantize_channel(w, bits, axis, rng, mode, seed)
    return {"range": rng, "codes": q, "scale": s, "status": st}


# --------------------------------------- Sec. 4, App. C: fully-quantized L1 BatchNorm
def l1bn_forward(x, gamma, beta, bits: int = 8, n_groups: int = 4) -> dict:
    """Forward of the fully-quantized L1 BatchNorm over x [R, C] (readings R12-R16 of the
    C source): codes q, output y, integer stats (sum q, sum |q - m|, sum sign(q - m)) and
    per-channel values (s, m, sigma, sigma^q, gamma^q, beta^q)."""
    x = _f32(x)
    R, C = x.shape
    g = np.ascontiguousarray(gamma, np.float32)
    b = np.ascontiguousarray(beta, np.float32)
    q = np.empty((R, C), np.int8)
    y = np.empty((R, C), np.float32)
    stats = np.empty((3, C), np.int64)
    chan = np.empty((6, C), np.float32)
    st = _load().sqo_l1bn_forward(_p(x), R, C, bits, n_groups, _p(g), _p(b), _p(q), _p(y),
                                  _p(stats), _p(chan))
    names = ("s", "m", "sigma", "sigma_q", "gamma_q", "beta_q")
    return {"q": q, "y": y, "S1": stats[0], "S": stats[1], "Z": stats[2], "stats": stats,
            "chan": chan, **{k: chan[i] for i, k in enumerate(names)}, "status": int(st)}


def l1bn_backward(gy, fwd: dict, bits: int = 8, n_groups: int = 4, seed: int = 0) -> dict:
    """Backward of the fully-quantized L1 BatchNorm (R15) from gy [R, C] and the forward's
    result: gradient codes p, dx, dgamma, dbeta."""
    gy = _f32(gy)
    R, C = gy.shape
    p = np.empty((R, C), np.int8)
    dx = np.empty((R, C), np.float32)
    dg = np.empty(C, np.float32)
    db = np.empty(C, np.float32)
    st = _load().sqo_l1bn_backward(_p(gy), R, C, bits, n_groups, seed & (2**64 - 1),
                                   _p(np.ascontiguousarray(fwd["q"])),
                                   _p(np.ascontiguousarray(fwd["stats"])),
                                   _p(np.ascontiguousarray(fwd["chan"])), _p(p), _p(dx), _p(dg),
                                   _p(db))
    return {"p": p, "dx": dx, "dgamma": dg, "dbeta": db, "status": int(st)}


# ------------------------------------------- Sec. 5.2: packed sub-byte storage (R17, R18)
def pack4(q) -> np.ndarray:
    """Codes of at most 4 bits [R, C] -> bytes [R, ceil(C/2)], two's-complement nibbles,
    element 2b in the low nibble of byte b."""
    q = np.ascontiguousarray(q, np.int8)
    R, C = q.shape
    out = np.empty((R, (C + 1) // 2), np.uint8)
    _load().sqo_pack4(_p(q), R, C, _p(out))
    return out


def unpack4(b, cols: int) -> np.ndarray:
    b = np.ascontiguousarray(b, np.uint8)
    q = np.empty((b.shape[0], cols), np.int8)
    _load().sqo_unpack4(_p(b), b.shape[0], cols, _p(q))
    return q


def group_field_bits(n_groups: int) -> int:
    return 1 if n_groups <= 2 else (2 if n_groups <= 4 else 4)


def pack_groups(e, n_groups: int) -> np.ndarray:
    """The grouping map in 1/2/4-bit fields, 8/w channels per byte (low bits first)."""
    e = np.ascontiguousarray(e, np.uint8)
    per = 8 // group_field_bits(n_groups)
    out = np.empty((e.size + per - 1) // per, np.uint8)
    _load().sqo_pack_groups(_p(e), e.size, n_groups, _p(out))
    return out


def unpack_groups(b, channels: int, n_groups: int) -> np.ndarray:
    b = np.ascontiguousarray(b, np.uint8)
    e = np.empty(channels, np.uint8)
    _load().sqo_unpack_groups(_p(b), channels, n_groups, _p(e))
    return e
