"""The C ABI library builds for sm_103a, loads, exports every declared symbol and rejects
bad arguments on the host before launching anything (no GPU needed)."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2411_10948_gb300 import build, native

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "shiftquant.h")


@pytest.fixture(scope="module")
def lib():
    build.build_library()
    return native.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(shiftquant_\w+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("shiftquant_calibrate", "shiftquant_quantize", "shiftquant_gemm_fwd",
              "shiftquant_gemm_dgrad", "shiftquant_gemm_wgrad"):
        assert n in names
    assert set(names) == set(native.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", build.LIB], capture_output=True,
                         text=True).stdout
    exported = set(re.findall(r"\bT (shiftquant_\w+)", out))
    assert set(declared_functions()) <= exported


def test_header_compiles_as_plain_c(tmp_path):
    src = tmp_path / "t.c"
    src.write_text('#include "shiftquant.h"\nint main(void){return SQ_OK;}\n')
    subprocess.check_call(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.dirname(HEADER),
                           "-c", str(src), "-o", str(tmp_path / "t.o")])


def test_code_type_rules(lib):
    # E4M3 holds |q| <= 15 and the shifted weight codes up to 448, else BF16
    assert native.shiftquant_code_type(4, 4) == native.SQ_CODE_E4M3      # 7 * 8 = 56
    assert native.shiftquant_code_type(4, 7) == native.SQ_CODE_E4M3      # 7 * 64 = 448
    assert native.shiftquant_code_type(4, 8) == native.SQ_CODE_BF16      # 7 * 128 > 448
    assert native.shiftquant_code_type(5, 5) == native.SQ_CODE_E4M3      # 15 * 16 = 240
    assert native.shiftquant_code_type(5, 6) == native.SQ_CODE_BF16      # 15 * 32 = 480
    assert native.shiftquant_code_type(6, 4) == native.SQ_CODE_BF16
    assert native.shiftquant_code_type(8, 1) == native.SQ_CODE_BF16
    assert native.shiftquant_code_bytes(4, 4) == 1
    assert native.shiftquant_code_bytes(8, 4) == 2
    for bad in ((1, 4), (9, 4), (4, 0), (4, 9)):
        assert lib.shiftquant_code_type(*bad) == native.SQ_EINVAL
    assert "bits" in lib.shiftquant_last_error().decode()


def test_host_validation_rejects_before_launch(lib):
    st = ctypes.c_void_p(16)   # never dereferenced: every call below fails validation first
    # negative sizes
    assert lib.shiftquant_calibrate(st, -1, 4, 4, 0, 4, st, st, st, st, None) == native.SQ_EINVAL
    # bad granularity and missing outputs
    assert lib.shiftquant_calibrate(st, 4, 4, 4, 7, 4, st, st, st, st, None) == native.SQ_EINVAL
    assert lib.shiftquant_calibrate(st, 4, 4, 4, 0, 4, st, None, st, st, None) == native.SQ_EINVAL
    # ld < cols
    assert lib.shiftquant_calibrate(st, 4, 8, 4, 0, 4, st, st, st, st, None) == native.SQ_EINVAL
    # both weight roles: negative sizes, ld < cols, missing outputs, bad bits
    assert lib.shiftquant_calibrate_weight(st, -1, 4, 4, st, st, st, None) == native.SQ_EINVAL
    assert lib.shiftquant_calibrate_weight(st, 4, 8, 4, st, st, st, None) == native.SQ_EINVAL
    assert lib.shiftquant_calibrate_weight(st, 4, 4, 4, st, None, st, None) == native.SQ_EINVAL
    assert lib.shiftquant_calibrate_weight(st, 4, 4, 4, st, st, None, None) == native.SQ_EINVAL
    assert lib.shiftquant_quantize_weight(st, 4, 4, 4, 9, 4, st, st, None, None, st, 16, st, st,
                                          16, st, None) == native.SQ_EINVAL
    assert lib.shiftquant_quantize_weight(st, 4, 4, 4, 4, 4, st, st, None, None, None, 16, st,
                                          st, 16, st, None) == native.SQ_EINVAL
    assert lib.shiftquant_quantize_weight(st, 4, 4, 4, 4, 4, st, st, None, None, st, 2, st, st,
                                          16, st, None) == native.SQ_EINVAL   # ld_fwd < rows
    assert lib.shiftquant_quantize_weight(st, 4, 4, 4, 4, 4, st, st, None, None, st, 16, st, st,
                                          2, st, None) == native.SQ_EINVAL    # ld_dgrad < cols
    assert lib.shiftquant_quantize_weight(st, -4, 4, 4, 4, 4, st, st, None, None, st, 16, st, st,
                                          16, st, None) == native.SQ_EINVAL
    # quantize: bits, rounding mode, SHIFT with fold_exp, no outputs
    args = dict(x=st, rows=4, cols=4, ld=4, gran=0, bits=4, g=4, rt=st, exp=st, fold=None,
                mode=0, seed=0, row0=0, codes=st, ldc=16, codes_t=None, ldt=0, scale=st,
                s=None)

    def q(**kw):
        a = dict(args, **kw)
        return lib.shiftquant_quantize(a["x"], a["rows"], a["cols"], a["ld"], a["gran"],
                                       a["bits"], a["g"], a["rt"], a["exp"], a["fold"], a["mode"],
                                       a["seed"], a["row0"], a["codes"], a["ldc"], a["codes_t"],
                                       a["ldt"], a["scale"], a["s"])
    assert q(bits=9) == native.SQ_EINVAL
    assert q(mode=5) == native.SQ_EINVAL
    assert q(fold=st) == native.SQ_EINVAL
    assert q(codes=None) == native.SQ_EINVAL
    assert q(ldc=2) == native.SQ_EINVAL
    assert q(row0=-1) == native.SQ_EINVAL
    # gemm: misaligned operand and leading dimension (TMA needs 16-byte rows)
    a16, a_odd = ctypes.c_void_p(256), ctypes.c_void_p(257)
    g = lib.shiftquant_gemm_fwd
    assert g(a_odd, 64, st, a16, 64, st, 8, 8, 64, 4, 4, st, 8, None, 0, None, 0, st,
             None) == native.SQ_EALIGN
    assert g(a16, 65, st, a16, 80, st, 8, 8, 64, 4, 4, st, 8, None, 0, None, 0, st,
             None) == native.SQ_EALIGN
    # gemm: missing status word, negative sizes, bad bits
    assert g(a16, 64, st, a16, 64, st, 8, 8, 64, 4, 4, st, 8, None, 0, None, 0, None,
             None) == native.SQ_EINVAL
    assert g(a16, 64, st, a16, 64, st, -8, 8, 64, 4, 4, st, 8, None, 0, None, 0, st,
             None) == native.SQ_EINVAL
    assert g(a16, 64, st, a16, 64, st, 8, 8, 64, 1, 4, st, 8, None, 0, None, 0, st,
             None) == native.SQ_EINVAL


def test_exact_range_limits_reject_before_launch(lib):
    st = ctypes.c_void_p(16)
    a16 = ctypes.c_void_p(256)
    g = lib.shiftquant_gemm_fwd
    # 8-bit, N_G = 6: one 64-wide K block of products 127 * 127 * 32 can pass 2^24, the exact
    # FP32 range of the tensor cores' sums, whatever K
    r = g(a16, 64, st, a16, 64, st, 8, 8, 64, 8, 6, st, 8, None, 0, None, 0, st, None)
    assert r == native.SQ_EUNSUPPORTED
    assert "exact FP32" in lib.shiftquant_last_error().decode()
    # the sharded weight gradient adds int32 sums across ranks: 8 bits over more than 133144
    # tokens in all is refused (a single-device call accumulates in int64 instead)
    p = lib.shiftquant_gemm_wgrad_partial
    r = p(a16, 140000, st, st, a16, 140000, st, st, 8, 8, 70000, 140000, 8, 4, a16, st, None)
    assert r == native.SQ_EUNSUPPORTED
    assert "int32" in lib.shiftquant_last_error().decode()


@pytest.mark.skipif(__import__("torch").cuda.is_available(),
                    reason="passes fake device pointers; only meaningful without a device")
def test_empty_shapes_accept_null_pointers_of_empty_buffers(lib):
    # torch hands NULL data pointers for empty tensors: an empty shape must never be
    # rejected for them (without a device the call ends in SQ_ECUDA or SQ_OK instead)
    fake = ctypes.c_void_p(4096)
    for R, C in ((0, 5), (5, 0), (0, 0)):
        rng = fake if C else None
        ex = fake if C else None
        r = lib.shiftquant_calibrate(None, R, C, max(C, 1), 0, 4, rng, fake, ex, fake, None)
        assert r != native.SQ_EINVAL, (R, C, lib.shiftquant_last_error())
        r = lib.shiftquant_quantize(None, R, C, max(C, 1), 0, 4, 4, fake, ex, None, 0, 0, 0,
                                    fake if R and C else None, 16, None, 0, fake, None)
        assert r != native.SQ_EINVAL, (R, C, lib.shiftquant_last_error())
        for gran in (1, 2):
            ch = C if gran == 1 else R
            r = lib.shiftquant_calibrate(None, R, C, max(C, 1), gran, 4,
                                         fake if ch else None, None, None, fake, None)
            assert r != native.SQ_EINVAL, (gran, R, C, lib.shiftquant_last_error())
            r = lib.shiftquant_quantize(None, R, C, max(C, 1), gran, 4, 4,
                                        fake if ch else None, None, None, 0, 0, 0, None, 0,
                                        None, 0, fake if ch else None, None)
            assert r != native.SQ_EINVAL, (gran, R, C, lib.shiftquant_last_error())


@pytest.mark.parametrize("cname,pyname", [("sq_layer_gemms", "SqLayerGemms"),
                                           ("sq_layer_step", "SqLayerStep")])
def test_layer_struct_layout_matches_the_binding(tmp_path, cname, pyname):
    # the ctypes mirrors of the C structs must have their size and field offsets
    import ctypes
    from paper_2411_10948_gb300 import native as nat
    SqLayerGemms = getattr(nat, pyname)
    fields = [f for f, _ in SqLayerGemms._fields_]
    src = tmp_path / "layout.c"
    src.write_text('#include <stddef.h>\n#include <stdio.h>\n#include "shiftquant.h"\nint main(void) {\n'
                   f'  printf("%zu\\n", sizeof({cname}));\n' +
                   "".join(f'  printf("%zu\\n", offsetof({cname}, {f}));\n' for f in fields) +
                   "  return 0;\n}\n")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)],
                   check=True)
    out = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True,
                                          check=True).stdout.split()]
    assert out[0] == ctypes.sizeof(SqLayerGemms)
    assert out[1:] == [getattr(SqLayerGemms, f).offset for f in fields]


def test_sharding_entries_reject_bad_arguments_before_launch(lib):
    # shiftquant_group, shiftquant_gemm_wgrad_partial / _finish: host checks only, no device
    st = ctypes.c_void_p(4096)          # stand-in device pointers: never dereferenced here
    odd = ctypes.c_void_p(4096 + 4)     # not 16-byte aligned
    g = lib.shiftquant_group
    assert g(st, 16, 0, st, st, st, None) == native.SQ_EINVAL      # n_groups
    assert g(st, -1, 4, st, st, st, None) == native.SQ_EINVAL      # channels
    assert g(None, 16, 4, st, st, st, None) == native.SQ_EINVAL    # range
    assert g(st, 16, 4, None, st, st, None) == native.SQ_EINVAL    # tau0_out
    assert g(st, 16, 4, st, st, None, None) == native.SQ_EINVAL    # dev_status
    p = lambda **k: lib.shiftquant_gemm_wgrad_partial(
        st, 64, st, st, st, 64, st, st, k.get("Ci", 32), k.get("Co", 32), k.get("T", 64),
        k.get("total", 128), k.get("bits", 4), 4, k.get("t", st), st, None)
    assert p(bits=1) == native.SQ_EINVAL
    assert p(T=-1) == native.SQ_EINVAL
    assert p(total=32) == native.SQ_EINVAL                          # total_tokens < T
    assert p(t=odd) == native.SQ_EALIGN
    assert p(Co=30) == native.SQ_EALIGN                             # Co % 4
    assert p(bits=8, total=1 << 20) == native.SQ_EUNSUPPORTED      # beyond exact int32
    assert p(Ci=0) == native.SQ_OK and p(Co=0) == native.SQ_OK     # empty: nothing to do
    f = lambda **k: lib.shiftquant_gemm_wgrad_finish(
        k.get("t", st), 32, k.get("Co", 32), 4, 4, st, st, st, st, k.get("dw", st),
        k.get("ld", 32), None, 0, st, None)
    assert f(t=odd) == native.SQ_EALIGN
    assert f(Co=30) == native.SQ_EALIGN
    assert f(dw=None) == native.SQ_EINVAL
    assert f(ld=16) == native.SQ_EINVAL


def test_static_weight_gradient_rejects_oversized_outputs_before_anything_else(lib):
    # the 2^20-output limit of the library's static scratch is checked first and without
    # forming Ci * Co (huge sizes must not wrap past it)
    st = ctypes.c_void_p(16)
    a16 = ctypes.c_void_p(256)
    f = lib.shiftquant_gemm_wgrad_static
    for ci, co in ((2**40, 2**40), (2**62, 4), (4, 2**62), ((1 << 20) + 1, 1), (1025, 1024)):
        r = f(a16, 64, st, st, a16, 64, st, st, ci, co, 64, 4, 4, st, co, None, 0, st, None)
        assert r == native.SQ_EUNSUPPORTED, (ci, co)
        assert "static scratch" in lib.shiftquant_last_error().decode()


def test_layer_step_validates_before_anything_runs(lib):
    # a NULL struct, a missing status word, bad bits or a missing buffer fail on the host
    from paper_2411_10948_gb300.native import SqLayerStep
    assert lib.shiftquant_layer_step(None, 0, None) == native.SQ_EINVAL
    fake = 4096
    a = SqLayerStep(M=64, K=64, N=64, bits=4, n_groups=4, dev_status=None)
    for f, _ in SqLayerStep._fields_:
        if f not in ("M", "K", "N", "bits", "n_groups", "workspace", "workspace_bytes",
                     "dev_status") and not f.startswith("ld_"):
            setattr(a, f, fake)
    assert lib.shiftquant_layer_step(ctypes.byref(a), 0, None) == native.SQ_EINVAL
    a.dev_status = fake
    a.bits = 9
    assert lib.shiftquant_layer_step(ctypes.byref(a), 0, None) == native.SQ_EINVAL
    a.bits = 4
    a.dy = None
    assert lib.shiftquant_layer_step(ctypes.byref(a), 0, None) == native.SQ_EINVAL
    assert lib.shiftquant_layer_step_host(ctypes.byref(a), None, None, None, None, None, None, 0,
                                          None, None) == native.SQ_EINVAL
    assert "NULL" in lib.shiftquant_last_error().decode()
    assert lib.shiftquant_layer_step_host_split(ctypes.byref(a), None, None, None, None, None,
                                                None, 0, None, None, None, None, fake, fake,
                                                fake) == native.SQ_EINVAL
    a.dy = fake
    # every buffer given: the three events are still required
    assert lib.shiftquant_layer_step_host_split(ctypes.byref(a), None, None, None, None, None,
                                                None, 0, None, None, None, None, None, fake,
                                                fake) == native.SQ_EINVAL
    assert "inputs_in" in lib.shiftquant_last_error().decode()


def test_layer_launch_refuses_in_place_weight_gradient_on_group_ordered_codes(lib):
    # without a transposed copy the weight gradient reads the codes in place, which a
    # group-ordered operand (channels permuted) cannot serve: refused on the host
    from paper_2411_10948_gb300.native import SqLayerGemms
    fake = 4096
    a = SqLayerGemms(M=64, K=64, N=64, bits=8, n_groups=4, x_codes=fake, ld_x=64,
                     xt_codes=None, g_codes=fake, ld_g=64, gt_codes=fake, ld_gt=64,
                     x_seg=fake)
    st = ctypes.c_void_p(fake)
    assert lib.shiftquant_gemm_layer(ctypes.byref(a), None, 0, st, None) == native.SQ_EINVAL
    assert "transposed copy" in lib.shiftquant_last_error().decode()
    a.x_seg, a.g_seg, a.xt_codes, a.gt_codes = None, fake, fake, None
    assert lib.shiftquant_gemm_layer(ctypes.byref(a), None, 0, st, None) == native.SQ_EINVAL


def test_grid_barrier_selftest_validates_before_launch(lib):
    st = ctypes.c_void_p(4096)
    assert lib.shiftquant_selftest_grid_barrier_timeout(None, st, None) == native.SQ_EINVAL
    assert lib.shiftquant_selftest_grid_barrier_timeout(ctypes.c_void_p(4100), st, None) == native.SQ_EINVAL
    assert lib.shiftquant_selftest_grid_barrier_timeout(ctypes.c_void_p(4096), None, None) == native.SQ_EINVAL
