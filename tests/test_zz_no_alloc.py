"""The allocation-free weight-gradient entry point against the regular one.

shiftquant_gemm_wgrad_static is for callers that cannot allocate device memory, such as
a plug-in inside a framework that owns every device allocation, or a deployment whose
device memory is fixed when the library loads.  Its split-K scratch is an array inside
the library instead of a caller workspace.  Two calls in a row through the C ABI must
agree with shiftquant_gemm_wgrad given a caller-allocated workspace: integer
accumulators bit-exact, fp32 outputs within the parity tolerance.
"""
import numpy as np
import pytest
import torch

from paper_2411_10948_gb300 import layer as L
from paper_2411_10948_gb300 import native as N
from parity_util import assert_close_f32, to_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2411_10948_gb300 import build
    build.build_library()
    N.load()


def _quantized_layer(T, Ci, Co, bits, seed):
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal((T, Ci)) * np.exp(rng.normal(0, 1, Ci))).astype(np.float32)
    dy = (rng.laplace(0, 1, (T, Co)) * np.exp(rng.normal(0, 2, Co))).astype(np.float32)
    lay = L.QuantLinear(T, Ci, Co, bits, 4, "cuda", with_acc=False, use_workspace=False)
    lay.quantize_activation(to_gpu(x))
    lay.quantize_gradient(to_gpu(dy), seed=seed)
    return lay


@pytest.mark.parametrize("T,Ci,Co,bits", [(8192, 512, 256, 4), (6000, 384, 640, 6)])
def test_static_scratch_wgrad_matches_workspace_wgrad(T, Ci, Co, bits):
    lay = _quantized_layer(T, Ci, Co, bits, seed=T + Ci)
    need = N.shiftquant_gemm_workspace_bytes(2, Ci, Co, T, bits, 4)
    assert need > 0, "this shape is meant to split its token axis across SMs"
    ws = torch.zeros(need // 4, dtype=torch.int32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    dw_ref = torch.zeros((Ci, Co), device="cuda")
    acc_ref = torch.zeros((Ci, Co), dtype=torch.int64, device="cuda")
    N.shiftquant_gemm_wgrad(lay.x.codes_t, lay.x.scale, lay.x.exp, lay.g.codes_t, lay.g.scale,
                            lay.g.exp, Ci, Co, T, bits, 4, dw_ref, acc_ref, ws, status)
    torch.cuda.synchronize()
    assert status.item() == 0
    for _ in range(2):   # the array keeps the previous call's sums: each call must clear it
        dw = torch.full((Ci, Co), 7.0, device="cuda")
        acc = torch.full((Ci, Co), 7, dtype=torch.int64, device="cuda")
        N.shiftquant_gemm_wgrad_static(lay.x.codes_t, lay.x.scale, lay.x.exp, lay.g.codes_t,
                                       lay.g.scale, lay.g.exp, Ci, Co, T, bits, 4, dw, acc,
                                       status)
        torch.cuda.synchronize()
        assert status.item() == 0
        np.testing.assert_array_equal(acc.cpu().numpy(), acc_ref.cpu().numpy())
        assert_close_f32(dw.cpu().numpy(), dw_ref.cpu().numpy(), "dW (static scratch)")


def test_static_scratch_rejects_outputs_beyond_its_size():
    lay = _quantized_layer(256, 64, 64, 4, seed=1)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    dw = torch.zeros((64, 64), device="cuda")
    with pytest.raises(N.ShiftQuantError) as e:
        # 2048 x 1024 outputs need 8 MiB of int32 partial sums: more than the 4 MiB array
        N.shiftquant_gemm_wgrad_static(lay.x.codes_t, lay.x.scale, lay.x.exp, lay.g.codes_t,
                                       lay.g.scale, lay.g.exp, 2048, 1024, 256, 4, 4, dw, None,
                                       status)
    assert e.value.status == N.SQ_EUNSUPPORTED
    assert "static scratch" in str(e.value)
