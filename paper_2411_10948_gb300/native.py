"""ctypes binding of libshiftquant.so: one Python function per C entry point, same names,
argument marshalling only (tensor -> data pointer, current stream -> cudaStream_t).

Every computation runs in the CUDA library.  If the library is missing the import of a
function raises: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

SQ_OK = 0
SQ_EINVAL = -1
SQ_EALIGN = -2
SQ_EUNSUPPORTED = -3
SQ_ECUDA = -4
SQ_DEV_NONFINITE = 1
SQ_DEV_TIMEOUT = 2
SQ_DEV_INTERNAL = 4
SQ_ROUND_NEAREST_EVEN = 0
SQ_ROUND_STOCHASTIC = 1
SQ_GRAN_SHIFT = 0
SQ_GRAN_PER_COL = 1
SQ_GRAN_PER_ROW = 2
SQ_CODE_E4M3 = 0
SQ_CODE_BF16 = 1

# every symbol declared in include/shiftquant.h
EXPORTS = (
    "shiftquant_code_type", "shiftquant_code_bytes", "shiftquant_calibrate",
    "shiftquant_group", "shiftquant_quantize", "shiftquant_calibrate_weight",
    "shiftquant_quantize_weight", "shiftquant_gemm_fwd", "shiftquant_gemm_dgrad",
    "shiftquant_gemm_wgrad", "shiftquant_gemm_wgrad_partial", "shiftquant_gemm_wgrad_finish",
    "shiftquant_gemm_wgrad_static", "shiftquant_gemm_workspace_bytes",
    "shiftquant_gemm_layer", "shiftquant_gemm_layer_workspace_bytes",
    "shiftquant_gemm_layer_workspace_bytes_grouped",
    "shiftquant_gemm_layer_kernel_launches", "shiftquant_gemm_layer_cta_pairs",
    "shiftquant_gemm_layer_wgrad_in_place",
    "shiftquant_layer_step", "shiftquant_layer_step_host", "shiftquant_layer_step_host_split",
    "shiftquant_selftest_wait_timeout",
    "shiftquant_l1bn_state_bytes", "shiftquant_l1bn_forward", "shiftquant_l1bn_backward",
    "shiftquant_l1bn_kernel_launches", "shiftquant_selftest_grid_barrier_timeout",
    "shiftquant_group_order", "shiftquant_group_order_width", "shiftquant_quantize_ordered",
    "shiftquant_pack_codes", "shiftquant_unpack_codes", "shiftquant_packed_groups_bytes",
    "shiftquant_pack_groups", "shiftquant_unpack_groups",
    "shiftquant_status_string", "shiftquant_last_error",
)

_lib = None


class SqLayerGemms(ctypes.Structure):
    """Mirror of the C struct sq_layer_gemms (include/shiftquant.h)."""
    _fields_ = [
        ("x_codes", ctypes.c_void_p), ("ld_x", ctypes.c_int64),
        ("xt_codes", ctypes.c_void_p), ("ld_xt", ctypes.c_int64),
        ("x_scale", ctypes.c_void_p), ("x_exp", ctypes.c_void_p),
        ("g_codes", ctypes.c_void_p), ("ld_g", ctypes.c_int64),
        ("gt_codes", ctypes.c_void_p), ("ld_gt", ctypes.c_int64),
        ("g_scale", ctypes.c_void_p), ("g_exp", ctypes.c_void_p),
        ("wf_codes", ctypes.c_void_p), ("ld_wf", ctypes.c_int64), ("wf_scale", ctypes.c_void_p),
        ("wd_codes", ctypes.c_void_p), ("ld_wd", ctypes.c_int64), ("wd_scale", ctypes.c_void_p),
        ("M", ctypes.c_int64), ("K", ctypes.c_int64), ("N", ctypes.c_int64),
        ("bits", ctypes.c_int), ("n_groups", ctypes.c_int),
        ("y", ctypes.c_void_p), ("ld_y", ctypes.c_int64),
        ("dx", ctypes.c_void_p), ("ld_dx", ctypes.c_int64),
        ("dw", ctypes.c_void_p), ("ld_dw", ctypes.c_int64),
        ("acc_y", ctypes.c_void_p), ("ld_acc_y", ctypes.c_int64),
        ("acc_dx", ctypes.c_void_p), ("ld_acc_dx", ctypes.c_int64),
        ("acc_dw", ctypes.c_void_p), ("ld_acc_dw", ctypes.c_int64),
        ("gemm_mask", ctypes.c_int), ("max_ctas", ctypes.c_int),
        ("y_range", ctypes.c_void_p), ("dx_range", ctypes.c_void_p),
        ("x_seg", ctypes.c_void_p), ("g_seg", ctypes.c_void_p),
    ]


class SqLayerStep(ctypes.Structure):
    """Mirror of the C struct sq_layer_step (include/shiftquant.h)."""
    _fields_ = [
        ("M", ctypes.c_int64), ("K", ctypes.c_int64), ("N", ctypes.c_int64),
        ("bits", ctypes.c_int), ("n_groups", ctypes.c_int),
        ("x", ctypes.c_void_p), ("w", ctypes.c_void_p), ("dy", ctypes.c_void_p),
        ("x_codes", ctypes.c_void_p), ("ld_x", ctypes.c_int64),
        ("xt_codes", ctypes.c_void_p), ("ld_xt", ctypes.c_int64),
        ("x_range", ctypes.c_void_p), ("x_tau0", ctypes.c_void_p),
        ("x_scale", ctypes.c_void_p), ("x_exp", ctypes.c_void_p),
        ("g_codes", ctypes.c_void_p), ("ld_g", ctypes.c_int64),
        ("gt_codes", ctypes.c_void_p), ("ld_gt", ctypes.c_int64),
        ("g_range", ctypes.c_void_p), ("g_tau0", ctypes.c_void_p),
        ("g_scale", ctypes.c_void_p), ("g_exp", ctypes.c_void_p),
        ("wf_codes", ctypes.c_void_p), ("ld_wf", ctypes.c_int64),
        ("wf_range", ctypes.c_void_p), ("wf_scale", ctypes.c_void_p),
        ("wd_codes", ctypes.c_void_p), ("ld_wd", ctypes.c_int64),
        ("wd_range", ctypes.c_void_p), ("wd_scale", ctypes.c_void_p),
        ("y", ctypes.c_void_p), ("dx", ctypes.c_void_p), ("dw", ctypes.c_void_p),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t),
        ("dev_status", ctypes.c_void_p),
    ]


class ShiftQuantError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{message} (status {status})")
        self.status = status


def library_path() -> str:
    return _build.LIB


def load(path: str | None = None) -> ctypes.CDLL:
    """Load libshiftquant.so (built in-tree by build.build_library)."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or _build.LIB
    if not os.path.exists(p):
        raise ImportError(f"libshiftquant.so is not built ({p}); run "
                          "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(p)
    i32, i64, u64, vp, sz = (ctypes.c_int, ctypes.c_int64, ctypes.c_uint64, ctypes.c_void_p,
                             ctypes.c_size_t)
    lib.shiftquant_code_type.argtypes = [i32, i32]
    lib.shiftquant_code_type.restype = i32
    lib.shiftquant_code_bytes.argtypes = [i32, i32]
    lib.shiftquant_code_bytes.restype = i32
    lib.shiftquant_calibrate.argtypes = [vp, i64, i64, i64, i32, i32, vp, vp, vp, vp, vp]
    lib.shiftquant_calibrate.restype = i32
    lib.shiftquant_group.argtypes = [vp, i64, i32, vp, vp, vp, vp]
    lib.shiftquant_group.restype = i32
    lib.shiftquant_calibrate_weight.argtypes = [vp, i64, i64, i64, vp, vp, vp, vp]
    lib.shiftquant_calibrate_weight.restype = i32
    lib.shiftquant_quantize_weight.argtypes = [vp, i64, i64, i64, i32, i32, vp, vp, vp, vp, vp,
                                               i64, vp, vp, i64, vp, vp]
    lib.shiftquant_quantize_weight.restype = i32
    lib.shiftquant_gemm_wgrad_partial.argtypes = [vp, i64, vp, vp, vp, i64, vp, vp, i64, i64, i64,
                                                  i64, i32, i32, vp, vp, vp]
    lib.shiftquant_gemm_wgrad_partial.restype = i32
    lib.shiftquant_gemm_wgrad_finish.argtypes = [vp, i64, i64, i32, i32, vp, vp, vp, vp, vp, i64,
                                                 vp, i64, vp, vp]
    lib.shiftquant_gemm_wgrad_finish.restype = i32
    lib.shiftquant_quantize.argtypes = [vp, i64, i64, i64, i32, i32, i32, vp, vp, vp, i32, u64,
                                        i64, vp, i64, vp, i64, vp, vp]
    lib.shiftquant_quantize.restype = i32
    gemm = [vp, i64, vp, vp, i64, vp, i64, i64, i64, i32, i32, vp, i64, vp, i64, vp, sz, vp, vp]
    lib.shiftquant_gemm_fwd.argtypes = gemm
    lib.shiftquant_gemm_fwd.restype = i32
    lib.shiftquant_gemm_dgrad.argtypes = gemm
    lib.shiftquant_gemm_dgrad.restype = i32
    lib.shiftquant_gemm_wgrad.argtypes = [vp, i64, vp, vp, vp, i64, vp, vp, i64, i64, i64, i32,
                                          i32, vp, i64, vp, i64, vp, sz, vp, vp]
    lib.shiftquant_gemm_wgrad.restype = i32
    lib.shiftquant_gemm_wgrad_static.argtypes = [vp, i64, vp, vp, vp, i64, vp, vp, i64, i64, i64,
                                                 i32, i32, vp, i64, vp, i64, vp, vp]
    lib.shiftquant_gemm_wgrad_static.restype = i32
    lib.shiftquant_gemm_layer.argtypes = [ctypes.POINTER(SqLayerGemms), vp, sz, vp, vp]
    lib.shiftquant_gemm_layer.restype = i32
    lib.shiftquant_gemm_layer_workspace_bytes.argtypes = [i64, i64, i64, i32, i32]
    lib.shiftquant_gemm_layer_workspace_bytes.restype = sz
    lib.shiftquant_gemm_layer_workspace_bytes_grouped.argtypes = [i64, i64, i64, i32, i32]
    lib.shiftquant_gemm_layer_workspace_bytes_grouped.restype = sz
    lib.shiftquant_gemm_layer_kernel_launches.argtypes = [i64, i64, i64, i32, i32, sz, i32]
    lib.shiftquant_gemm_layer_kernel_launches.restype = i32
    lib.shiftquant_gemm_layer_cta_pairs.argtypes = [i64, i64, i64, i32, i32, i32]
    lib.shiftquant_gemm_layer_cta_pairs.restype = i32
    lib.shiftquant_gemm_layer_wgrad_in_place.argtypes = [i64, i64, i64, i32, i32]
    lib.shiftquant_gemm_layer_wgrad_in_place.restype = i32
    lib.shiftquant_gemm_workspace_bytes.argtypes = [i32, i64, i64, i64, i32, i32]
    lib.shiftquant_gemm_workspace_bytes.restype = sz
    lib.shiftquant_layer_step.argtypes = [ctypes.POINTER(SqLayerStep), u64, vp]
    lib.shiftquant_layer_step.restype = i32
    lib.shiftquant_layer_step_host.argtypes = [ctypes.POINTER(SqLayerStep), vp, vp, vp, vp, vp,
                                               vp, u64, vp, vp]
    lib.shiftquant_layer_step_host.restype = i32
    lib.shiftquant_layer_step_host_split.argtypes = [ctypes.POINTER(SqLayerStep), vp, vp, vp, vp,
                                                     vp, vp, u64, vp, vp, vp, vp, vp, vp, vp]
    lib.shiftquant_layer_step_host_split.restype = i32
    lib.shiftquant_selftest_wait_timeout.argtypes = [vp, i64, vp, vp, i64, vp, i64, i64, i64,
                                                     i32, i32, vp, i64, vp, vp]
    lib.shiftquant_selftest_wait_timeout.restype = i32
    lib.shiftquant_l1bn_state_bytes.argtypes = [i64, i64]
    lib.shiftquant_l1bn_state_bytes.restype = sz
    lib.shiftquant_l1bn_kernel_launches.argtypes = [i64, i32]
    lib.shiftquant_l1bn_kernel_launches.restype = i32
    lib.shiftquant_selftest_grid_barrier_timeout.argtypes = [vp, vp, vp]
    lib.shiftquant_selftest_grid_barrier_timeout.restype = i32
    lib.shiftquant_l1bn_forward.argtypes = [vp, i64, i64, i64, vp, vp, i32, i32, vp, i64, vp, sz,
                                            vp, vp]
    lib.shiftquant_l1bn_forward.restype = i32
    lib.shiftquant_l1bn_backward.argtypes = [vp, i64, i64, i64, i32, i32, u64, vp, sz, vp, i64,
                                             vp, vp, vp, vp]
    lib.shiftquant_l1bn_backward.restype = i32
    lib.shiftquant_group_order.argtypes = [vp, i64, i32, i32, vp, vp, vp]
    lib.shiftquant_group_order.restype = i32
    lib.shiftquant_group_order_width.argtypes = [i64, i32, i32]
    lib.shiftquant_group_order_width.restype = i64
    lib.shiftquant_quantize_ordered.argtypes = [vp, i64, i64, i64, i32, i32, i32, vp, vp, i32, u64,
                                                i64, vp, vp, vp, i64, vp, i64, vp, vp]
    lib.shiftquant_quantize_ordered.restype = i32
    lib.shiftquant_pack_codes.argtypes = [vp, i64, i64, i64, i32, i32, vp, i64, vp, vp]
    lib.shiftquant_pack_codes.restype = i32
    lib.shiftquant_unpack_codes.argtypes = [vp, i64, i64, i64, i32, i32, vp, i64, vp]
    lib.shiftquant_unpack_codes.restype = i32
    lib.shiftquant_packed_groups_bytes.argtypes = [i64, i32]
    lib.shiftquant_packed_groups_bytes.restype = i64
    lib.shiftquant_pack_groups.argtypes = [vp, i64, i32, vp, vp]
    lib.shiftquant_pack_groups.restype = i32
    lib.shiftquant_unpack_groups.argtypes = [vp, i64, i32, vp, vp]
    lib.shiftquant_unpack_groups.restype = i32
    lib.shiftquant_status_string.argtypes = [i32]
    lib.shiftquant_status_string.restype = ctypes.c_char_p
    lib.shiftquant_last_error.argtypes = []
    lib.shiftquant_last_error.restype = ctypes.c_char_p
    if path is None:
        _lib = lib
    return lib


def _check(status: int) -> None:
    if status != SQ_OK:
        lib = load()
        msg = lib.shiftquant_last_error().decode() or lib.shiftquant_status_string(status).decode()
        raise ShiftQuantError(status, msg)


def _ptr(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ld(t) -> int:
    assert t.dim() == 2 and t.stride(1) == 1, "matrices must be row-major with unit column stride"
    return t.stride(0)


# ------------------------------------------------------------------ entry points
def shiftquant_code_type(bits: int, n_groups: int) -> int:
    r = load().shiftquant_code_type(bits, n_groups)
    if r < 0:
        _check(r)
    return r


def shiftquant_code_bytes(bits: int, n_groups: int) -> int:
    r = load().shiftquant_code_bytes(bits, n_groups)
    if r < 0:
        _check(r)
    return r


def code_dtype(bits: int, n_groups: int) -> torch.dtype:
    """torch dtype of the code storage: uint8 bytes holding E4M3, or bfloat16."""
    return torch.uint8 if shiftquant_code_type(bits, n_groups) == SQ_CODE_E4M3 else torch.bfloat16


def shiftquant_calibrate(x, gran, n_groups, range_out, tau0_out, exp_out, dev_status,
                         stream=None) -> None:
    _check(load().shiftquant_calibrate(_ptr(x), x.shape[0], x.shape[1], _ld(x), gran, n_groups,
                                       _ptr(range_out), _ptr(tau0_out), _ptr(exp_out),
                                       _ptr(dev_status), _stream(stream)))


def shiftquant_group(range_, n_groups, tau0_out, exp_out, dev_status, stream=None) -> None:
    """tau_0 and the group exponents from a given range vector (see the header)."""
    _check(load().shiftquant_group(_ptr(range_), range_.numel(), n_groups, _ptr(tau0_out),
                                   _ptr(exp_out), _ptr(dev_status), _stream(stream)))


def shiftquant_quantize(x, gran, bits, n_groups, range_or_tau0, exp, fold_exp, mode, seed,
                        codes, codes_t, scale_out, stream=None, row0=0) -> None:
    _check(load().shiftquant_quantize(
        _ptr(x), x.shape[0], x.shape[1], _ld(x), gran, bits, n_groups, _ptr(range_or_tau0),
        _ptr(exp), _ptr(fold_exp), mode, seed & (2**64 - 1), row0, _ptr(codes),
        _ld(codes) if codes is not None else 0, _ptr(codes_t),
        _ld(codes_t) if codes_t is not None else 0, _ptr(scale_out), _stream(stream)))


def shiftquant_calibrate_weight(w, range_out_ch, range_in_ch, dev_status, stream=None) -> None:
    """Both weight ranges (per out-channel and per in-channel) from one read of w [K, N]."""
    _check(load().shiftquant_calibrate_weight(_ptr(w), w.shape[0], w.shape[1], _ld(w),
                                              _ptr(range_out_ch), _ptr(range_in_ch),
                                              _ptr(dev_status), _stream(stream)))


def shiftquant_quantize_weight(w, bits, n_groups, range_out_ch, range_in_ch, fold_fwd,
                               fold_dgrad, codes_fwd, scale_fwd, codes_dgrad, scale_dgrad,
                               stream=None) -> None:
    """Both weight roles from one read of w [K, N]: codes_fwd [N, K] (per out-channel,
    transposed) and codes_dgrad [K, N] (per in-channel)."""
    _check(load().shiftquant_quantize_weight(
        _ptr(w), w.shape[0], w.shape[1], _ld(w), bits, n_groups, _ptr(range_out_ch),
        _ptr(range_in_ch), _ptr(fold_fwd), _ptr(fold_dgrad), _ptr(codes_fwd),
        _ld(codes_fwd) if codes_fwd is not None else 0, _ptr(scale_fwd), _ptr(codes_dgrad),
        _ld(codes_dgrad) if codes_dgrad is not None else 0, _ptr(scale_dgrad),
        _stream(stream)))


def _gemm(fn, a, a_scale, b, b_scale, M, N, K, bits, n_groups, y, acc, workspace, dev_status,
          stream):
    _check(fn(_ptr(a), _ld(a), _ptr(a_scale), _ptr(b), _ld(b), _ptr(b_scale), M, N, K, bits,
              n_groups, _ptr(y), _ld(y), _ptr(acc), _ld(acc) if acc is not None else 0,
              _ptr(workspace), workspace.numel() * workspace.element_size()
              if workspace is not None else 0, _ptr(dev_status), _stream(stream)))


def shiftquant_gemm_fwd(a_codes, a_scale, b_codes, b_scale, M, N, K, bits, n_groups, y,
                        acc=None, workspace=None, dev_status=None, stream=None) -> None:
    _gemm(load().shiftquant_gemm_fwd, a_codes, a_scale, b_codes, b_scale, M, N, K, bits,
          n_groups, y, acc, workspace, dev_status, stream)


def shiftquant_gemm_dgrad(a_codes, a_scale, b_codes, b_scale, M, N_out, K_in, bits, n_groups,
                          dx, acc=None, workspace=None, dev_status=None, stream=None) -> None:
    _gemm(load().shiftquant_gemm_dgrad, a_codes, a_scale, b_codes, b_scale, M, N_out, K_in,
          bits, n_groups, dx, acc, workspace, dev_status, stream)


def shiftquant_gemm_wgrad(xt_codes, x_scale, x_exp, gt_codes, g_scale, g_exp, Ci, Co, T, bits,
                          n_groups, dw, acc=None, workspace=None, dev_status=None,
                          stream=None) -> None:
    _check(load().shiftquant_gemm_wgrad(
        _ptr(xt_codes), _ld(xt_codes), _ptr(x_scale), _ptr(x_exp), _ptr(gt_codes), _ld(gt_codes),
        _ptr(g_scale), _ptr(g_exp), Ci, Co, T, bits, n_groups, _ptr(dw), _ld(dw), _ptr(acc),
        _ld(acc) if acc is not None else 0, _ptr(workspace),
        workspace.numel() * workspace.element_size() if workspace is not None else 0,
        _ptr(dev_status), _stream(stream)))


def shiftquant_gemm_wgrad_static(xt_codes, x_scale, x_exp, gt_codes, g_scale, g_exp, Ci, Co, T,
                                 bits, n_groups, dw, acc=None, dev_status=None,
                                 stream=None) -> None:
    """Weight gradient with the library's own static split-K scratch (no allocation)."""
    _check(load().shiftquant_gemm_wgrad_static(
        _ptr(xt_codes), _ld(xt_codes), _ptr(x_scale), _ptr(x_exp), _ptr(gt_codes), _ld(gt_codes),
        _ptr(g_scale), _ptr(g_exp), Ci, Co, T, bits, n_groups, _ptr(dw), _ld(dw), _ptr(acc),
        _ld(acc) if acc is not None else 0, _ptr(dev_status), _stream(stream)))


def shiftquant_gemm_workspace_bytes(which: int, M: int, N: int, K: int, bits: int,
                                    n_groups: int) -> int:
    return int(load().shiftquant_gemm_workspace_bytes(which, M, N, K, bits, n_groups))


def _addr(t):
    return t.data_ptr() if t is not None else None


def _ld_opt(t) -> int:
    """Leading dimension of an optional matrix (0 when absent)."""
    return _ld(t) if t is not None else 0


def shiftquant_gemm_layer(x_codes, xt_codes, x_scale, x_exp, g_codes, gt_codes, g_scale, g_exp,
                          wf_codes, wf_scale, wd_codes, wd_scale, M, K, N, bits, n_groups, y, dx,
                          dw, acc_y=None, acc_dx=None, acc_dw=None, workspace=None,
                          dev_status=None, stream=None, gemm_mask=0, max_ctas=0, y_range=None,
                          dx_range=None, x_seg=None, g_seg=None) -> None:
    """Forward, loss-propagation and weight-gradient GEMMs of one layer in one launch
    (gemm_mask: bit 0 forward, 1 loss propagation, 2 weight gradient; 0 = all); y_range and
    dx_range optionally receive the per-column max |Y| and max |dX| from the epilogue."""
    a = SqLayerGemms(
        x_codes=_addr(x_codes), ld_x=_ld_opt(x_codes), xt_codes=_addr(xt_codes),
        ld_xt=_ld_opt(xt_codes), x_scale=_addr(x_scale), x_exp=_addr(x_exp),
        g_codes=_addr(g_codes), ld_g=_ld_opt(g_codes), gt_codes=_addr(gt_codes),
        ld_gt=_ld_opt(gt_codes), g_scale=_addr(g_scale), g_exp=_addr(g_exp),
        wf_codes=_addr(wf_codes), ld_wf=_ld_opt(wf_codes), wf_scale=_addr(wf_scale),
        wd_codes=_addr(wd_codes), ld_wd=_ld_opt(wd_codes), wd_scale=_addr(wd_scale),
        M=M, K=K, N=N, bits=bits, n_groups=n_groups,
        y=_addr(y), ld_y=_ld_opt(y), dx=_addr(dx), ld_dx=_ld_opt(dx), dw=_addr(dw),
        ld_dw=_ld_opt(dw), acc_y=_addr(acc_y), ld_acc_y=_ld_opt(acc_y),
        acc_dx=_addr(acc_dx), ld_acc_dx=_ld_opt(acc_dx),
        acc_dw=_addr(acc_dw), ld_acc_dw=_ld_opt(acc_dw),
        gemm_mask=gemm_mask, max_ctas=max_ctas, y_range=_addr(y_range),
        dx_range=_addr(dx_range), x_seg=_addr(x_seg), g_seg=_addr(g_seg))
    _check(load().shiftquant_gemm_layer(
        ctypes.byref(a), _ptr(workspace),
        workspace.numel() * workspace.element_size() if workspace is not None else 0,
        _ptr(dev_status), _stream(stream)))


def shiftquant_gemm_wgrad_partial(xt_codes, x_scale, x_exp, gt_codes, g_scale, g_exp, Ci, Co, T,
                                  total_tokens, bits, n_groups, t_out, dev_status,
                                  stream=None) -> None:
    """One token shard's int32 weight-gradient sums (see the header)."""
    _check(load().shiftquant_gemm_wgrad_partial(
        _ptr(xt_codes), _ld(xt_codes), _ptr(x_scale), _ptr(x_exp), _ptr(gt_codes),
        _ld(gt_codes), _ptr(g_scale), _ptr(g_exp), Ci, Co, T, total_tokens, bits, n_groups,
        _ptr(t_out), _ptr(dev_status), _stream(stream)))


def shiftquant_gemm_wgrad_finish(t, Ci, Co, bits, n_groups, x_scale, x_exp, g_scale, g_exp, dw,
                                 acc_out, dev_status, stream=None) -> None:
    """dW from the summed int32 sums of every shard (see the header)."""
    _check(load().shiftquant_gemm_wgrad_finish(
        _ptr(t), Ci, Co, bits, n_groups, _ptr(x_scale), _ptr(x_exp), _ptr(g_scale), _ptr(g_exp),
        _ptr(dw), _ld(dw), _ptr(acc_out), _ld(acc_out) if acc_out is not None else 0,
        _ptr(dev_status), _stream(stream)))


def shiftquant_gemm_layer_workspace_bytes(M: int, K: int, N: int, bits: int, n_groups: int,
                                          grouped: bool = False) -> int:
    fn = (load().shiftquant_gemm_layer_workspace_bytes_grouped if grouped
          else load().shiftquant_gemm_layer_workspace_bytes)
    return int(fn(M, K, N, bits, n_groups))


def shiftquant_gemm_layer_kernel_launches(M: int, K: int, N: int, bits: int, n_groups: int,
                                          workspace_bytes: int, gemm_mask: int = 0) -> int:
    return int(load().shiftquant_gemm_layer_kernel_launches(M, K, N, bits, n_groups,
                                                            workspace_bytes, gemm_mask))


def shiftquant_gemm_layer_cta_pairs(M: int, K: int, N: int, bits: int, n_groups: int,
                                    gemm_mask: int = 0) -> int:
    """1: the layer launch runs on 2-CTA clusters (256 x 256 tiles); 0: single-CTA tiles."""
    return int(load().shiftquant_gemm_layer_cta_pairs(M, K, N, bits, n_groups, gemm_mask))


def shiftquant_gemm_layer_wgrad_in_place(M: int, K: int, N: int, bits: int,
                                         n_groups: int) -> int:
    """1: the layer launch's weight gradient reads X's and dY's codes in place as fast as
    transposed copies (skip the copies); 0: keep the copies; -1: invalid or no device."""
    return int(load().shiftquant_gemm_layer_wgrad_in_place(M, K, N, bits, n_groups))


def layer_step_args(M, K, N, bits, n_groups, x, w, dy, x_codes, xt_codes, x_range, x_tau0,
                    x_scale, x_exp, g_codes, gt_codes, g_range, g_tau0, g_scale, g_exp,
                    wf_codes, wf_range, wf_scale, wd_codes, wd_range, wd_scale, y, dx, dw,
                    workspace, dev_status) -> SqLayerStep:
    """The C struct sq_layer_step over these device tensors (inputs and outputs dense)."""
    for t, shape in ((x, (M, K)), (w, (K, N)), (dy, (M, N)), (y, (M, N)), (dx, (M, K)),
                     (dw, (K, N))):
        assert tuple(t.shape) == shape and t.is_contiguous(), "dense fp32 matrices expected"
    return SqLayerStep(
        M=M, K=K, N=N, bits=bits, n_groups=n_groups, x=_addr(x), w=_addr(w), dy=_addr(dy),
        x_codes=_addr(x_codes), ld_x=_ld(x_codes), xt_codes=_addr(xt_codes),
        ld_xt=_ld_opt(xt_codes),
        x_range=_addr(x_range), x_tau0=_addr(x_tau0), x_scale=_addr(x_scale), x_exp=_addr(x_exp),
        g_codes=_addr(g_codes), ld_g=_ld(g_codes), gt_codes=_addr(gt_codes),
        ld_gt=_ld_opt(gt_codes),
        g_range=_addr(g_range), g_tau0=_addr(g_tau0), g_scale=_addr(g_scale), g_exp=_addr(g_exp),
        wf_codes=_addr(wf_codes), ld_wf=_ld(wf_codes), wf_range=_addr(wf_range),
        wf_scale=_addr(wf_scale), wd_codes=_addr(wd_codes), ld_wd=_ld(wd_codes),
        wd_range=_addr(wd_range), wd_scale=_addr(wd_scale), y=_addr(y), dx=_addr(dx),
        dw=_addr(dw), workspace=_addr(workspace),
        workspace_bytes=workspace.numel() * workspace.element_size() if workspace is not None else 0,
        dev_status=_addr(dev_status))


def shiftquant_layer_step(args: SqLayerStep, seed: int, stream=None) -> None:
    """One layer's whole training step on the device (see the header)."""
    _check(load().shiftquant_layer_step(ctypes.byref(args), seed & (2**64 - 1), _stream(stream)))


def _host_ptr(t):
    if t is None:
        return None
    assert t.device.type == "cpu" and t.is_contiguous() and t.dtype == torch.float32
    return ctypes.c_void_p(t.data_ptr())


def shiftquant_layer_step_host(args: SqLayerStep, x_host, w_host, dy_host, y_host, dx_host,
                               dw_host, seed: int, stream=None, inputs_queued=None) -> None:
    """The step fed from host tensors and returned to them (pinned for asynchronous copies);
    any of them may be None.  inputs_queued: an optional torch.cuda.Event (already created)
    recorded after the input copies (see the header)."""
    ev = ctypes.c_void_p(inputs_queued.cuda_event) if inputs_queued is not None else None
    _check(load().shiftquant_layer_step_host(
        ctypes.byref(args), _host_ptr(x_host), _host_ptr(w_host), _host_ptr(dy_host),
        _host_ptr(y_host), _host_ptr(dx_host), _host_ptr(dw_host), seed & (2**64 - 1), ev,
        _stream(stream)))


def _event(ev):
    return ctypes.c_void_p(ev.cuda_event) if ev is not None else None


def shiftquant_layer_step_host_split(args: SqLayerStep, x_host, w_host, dy_host, y_host,
                                     dx_host, dw_host, seed: int, copy_in_stream, stream,
                                     copy_out_stream, buffers_free, inputs_in, step_done,
                                     outputs_out) -> None:
    """The host-fed step with its copies on their own streams (see the header); the events
    are torch.cuda.Event objects that already exist (buffers_free may be None)."""
    _check(load().shiftquant_layer_step_host_split(
        ctypes.byref(args), _host_ptr(x_host), _host_ptr(w_host), _host_ptr(dy_host),
        _host_ptr(y_host), _host_ptr(dx_host), _host_ptr(dw_host), seed & (2**64 - 1),
        _stream(copy_in_stream), _stream(stream), _stream(copy_out_stream), _event(buffers_free),
        _event(inputs_in), _event(step_done), _event(outputs_out)))


def shiftquant_selftest_wait_timeout(a_codes, a_scale, b_codes, b_scale, M, N, K, bits, n_groups,
                                     y, dev_status, stream=None) -> None:
    """A GEMM launch whose waits run out on purpose (see the header): SQ_DEV_TIMEOUT."""
    _check(load().shiftquant_selftest_wait_timeout(
        _ptr(a_codes), _ld(a_codes), _ptr(a_scale), _ptr(b_codes), _ld(b_codes), _ptr(b_scale),
        M, N, K, bits, n_groups, _ptr(y), _ld(y), _ptr(dev_status), _stream(stream)))


def shiftquant_l1bn_state_bytes(rows: int, channels: int) -> int:
    return int(load().shiftquant_l1bn_state_bytes(rows, channels))


def shiftquant_selftest_grid_barrier_timeout(scratch, dev_status, stream=None) -> None:
    """Failure-path self-test: a grid barrier whose bounded waits run out (about 1 s)."""
    _check(load().shiftquant_selftest_grid_barrier_timeout(_ptr(scratch), _ptr(dev_status),
                                                           _stream(stream)))


def shiftquant_l1bn_kernel_launches(channels: int, backward: bool = False) -> int:
    """Kernels one L1 batch-norm call launches: 1 in the single-launch form, else 9 / 7."""
    return int(load().shiftquant_l1bn_kernel_launches(channels, 1 if backward else 0))


def shiftquant_l1bn_forward(x, gamma, beta, bits, n_groups, y, state, dev_status,
                            stream=None) -> None:
    """Fully-quantized L1 batch normalization, forward (see the header)."""
    _check(load().shiftquant_l1bn_forward(
        _ptr(x), x.shape[0], x.shape[1], _ld(x), _ptr(gamma), _ptr(beta), bits, n_groups,
        _ptr(y), _ld(y), _ptr(state), state.numel() * state.element_size(), _ptr(dev_status),
        _stream(stream)))


def shiftquant_l1bn_backward(dy, bits, n_groups, seed, state, dx, dgamma, dbeta, dev_status,
                             stream=None) -> None:
    """Fully-quantized L1 batch normalization, backward (see the header)."""
    _check(load().shiftquant_l1bn_backward(
        _ptr(dy), dy.shape[0], dy.shape[1], _ld(dy), bits, n_groups, seed & (2**64 - 1),
        _ptr(state), state.numel() * state.element_size(), _ptr(dx), _ld(dx), _ptr(dgamma),
        _ptr(dbeta), _ptr(dev_status), _stream(stream)))


def shiftquant_group_order_width(channels: int, bits: int, n_groups: int) -> int:
    return int(load().shiftquant_group_order_width(channels, bits, n_groups))


def shiftquant_group_order(exp, bits, n_groups, pos_out, seg_out, stream=None) -> None:
    """Stable group order of a GEMM inner index from its exponents (see the header)."""
    _check(load().shiftquant_group_order(_ptr(exp), exp.numel(), bits, n_groups, _ptr(pos_out),
                                         _ptr(seg_out), _stream(stream)))


def shiftquant_quantize_ordered(x, gran, bits, n_groups, range_or_tau0, exp, mode, seed, pos, seg,
                                codes, codes_t, scale_out, stream=None, row0=0) -> None:
    """shiftquant_quantize writing the GEMM inner index in group order (see the header)."""
    _check(load().shiftquant_quantize_ordered(
        _ptr(x), x.shape[0], x.shape[1], _ld(x), gran, bits, n_groups, _ptr(range_or_tau0),
        _ptr(exp), mode, seed & (2**64 - 1), row0, _ptr(pos), _ptr(seg), _ptr(codes),
        _ld(codes) if codes is not None else 0, _ptr(codes_t),
        _ld(codes_t) if codes_t is not None else 0, _ptr(scale_out), _stream(stream)))


def shiftquant_pack_codes(codes, bits, n_groups, packed, dev_status, stream=None) -> None:
    """4-bit codes [R, C] -> packed bytes [R, >= ceil(C/2)] (see the header)."""
    _check(load().shiftquant_pack_codes(_ptr(codes), codes.shape[0], codes.shape[1], _ld(codes),
                                        bits, n_groups, _ptr(packed), _ld(packed),
                                        _ptr(dev_status), _stream(stream)))


def shiftquant_unpack_codes(packed, cols, bits, n_groups, codes, stream=None) -> None:
    _check(load().shiftquant_unpack_codes(_ptr(packed), _ld(packed), packed.shape[0], cols, bits,
                                          n_groups, _ptr(codes), _ld(codes), _stream(stream)))


def shiftquant_packed_groups_bytes(channels: int, n_groups: int) -> int:
    return int(load().shiftquant_packed_groups_bytes(channels, n_groups))


def shiftquant_pack_groups(exp, n_groups, packed, stream=None) -> None:
    _check(load().shiftquant_pack_groups(_ptr(exp), exp.numel(), n_groups, _ptr(packed),
                                         _stream(stream)))


def shiftquant_unpack_groups(packed, channels, n_groups, exp, stream=None) -> None:
    _check(load().shiftquant_unpack_groups(_ptr(packed), channels, n_groups, _ptr(exp),
                                           _stream(stream)))
