"""GPU parity of the group-ordered contraction (Sec. 3.2's per-group products, fused into
one launch): the stable group order, the quantizer writing the GEMM inner index in that
order (codes equal to the plain ones, moved; padding zero), and the layer GEMMs over
group-ordered operands -- integer accumulators bit-exact against the oracle's Eq. 4 result,
fp32 outputs within 1e-6 relative -- including every channel in the top group (where the
folded layout needs its shortest chunks), 8-bit codes with N_G up to 8 (beyond the folded
layout's exact range) and a K loop past the int32 range."""
import numpy as np
import pytest
import torch

from paper_2411_10948_gb300 import layer as L
from paper_2411_10948_gb300 import native as N
from parity_util import assert_close_f32, decode, oracle_layer, to_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2411_10948_gb300 import build
    build.build_library()
    N.load()


def _expected_order(e, G, bk):
    e = np.minimum(e.astype(np.int64), G - 1)
    counts = np.bincount(e, minlength=G)
    starts = np.zeros(G + 1, np.int64)
    for g in range(G):
        starts[g + 1] = starts[g] + (counts[g] + bk - 1) // bk * bk
    pos = np.empty(len(e), np.int64)
    for g in range(G):
        idx = np.nonzero(e == g)[0]           # ascending: the order within a group is stable
        pos[idx] = starts[g] + np.arange(len(idx))
    return pos, starts, counts


@pytest.mark.parametrize("C,G,bits", [(4096, 4, 8), (1000, 8, 8), (77, 3, 4), (5000, 4, 6), (1, 4, 8)])
def test_group_order_is_the_stable_group_sort(C, G, bits):
    rng = np.random.default_rng(C + G)
    e = rng.integers(0, G, C).astype(np.uint8)
    if C > 10:
        e[e == 1] = 2                          # an empty group
    pos = torch.zeros(C, dtype=torch.int32, device="cuda")
    seg = torch.zeros(2 * G + 1, dtype=torch.int32, device="cuda")
    N.shiftquant_group_order(torch.from_numpy(e).cuda(), bits, G, pos, seg)
    torch.cuda.synchronize()
    bk = 128 // N.shiftquant_code_bytes(bits, G)
    want_pos, starts, counts = _expected_order(e, G, bk)
    np.testing.assert_array_equal(pos.cpu().numpy(), want_pos)
    sg = seg.cpu().numpy()
    np.testing.assert_array_equal(sg[: G + 1], starts)
    np.testing.assert_array_equal(sg[G + 1:], counts)
    assert sg[G] <= N.shiftquant_group_order_width(C, bits, G)


def _garbage(t):
    # stale contents (0x7F bytes: NaN in E4M3, a large BF16) that the order's padding must not keep
    t.view(torch.uint8).fill_(0x7F)
    return t


@pytest.mark.parametrize("bits,G", [(8, 4), (4, 4)])
def test_ordered_quantizer_moves_the_plain_codes(bits, G):
    rng = np.random.default_rng(bits)
    M, K, Nn = 300, 700, 260
    x = (rng.standard_normal((M, K)) * np.exp(rng.normal(0, 1.5, K))).astype(np.float32)
    w = (rng.standard_normal((K, Nn)) * 0.02).astype(np.float32)
    plain = L.QuantLinear(M, K, Nn, bits, G, "cuda")
    grp = L.QuantLinear(M, K, Nn, bits, G, "cuda", grouped=True)
    for t in (grp.x.codes, grp.wf.codes, grp.wd.codes):
        _garbage(t)
    xg, wg = to_gpu(x), to_gpu(w)
    plain.quantize_activation(xg)
    plain.quantize_gradient(xg[:, :Nn].contiguous(), 3)
    grp.quantize_activation(xg)
    grp.quantize_gradient(xg[:, :Nn].contiguous(), 3)
    # weights unfolded in both, to compare the placement alone
    for lay in (plain, grp):
        N.shiftquant_calibrate(wg, N.SQ_GRAN_PER_COL, G, lay.wf.range, None, None, lay.status)
        N.shiftquant_calibrate(wg, N.SQ_GRAN_PER_ROW, G, lay.wd.range, None, None, lay.status)
    N.shiftquant_quantize(wg, N.SQ_GRAN_PER_COL, bits, G, plain.wf.range, None, None, 0, 0, None,
                          plain.wf.codes, plain.wf.scale)
    N.shiftquant_quantize(wg, N.SQ_GRAN_PER_ROW, bits, G, plain.wd.range, None, None, 0, 0,
                          plain.wd.codes, None, plain.wd.scale)
    grp.quantize_weights(wg)
    torch.cuda.synchronize()
    assert grp.status.item() == 0 and plain.status.item() == 0
    for q, pos, seg, ref in ((grp.x.codes, grp.x_pos, grp.x_seg, plain.x.codes),
                             (grp.g.codes, grp.g_pos, grp.g_seg, plain.g.codes),
                             (grp.wf.codes, grp.x_pos, grp.x_seg, plain.wf.codes),
                             (grp.wd.codes, grp.g_pos, grp.g_seg, plain.wd.codes)):
        p = pos.cpu().numpy().astype(np.int64)
        sg = seg.cpu().numpy()
        got = decode(q[:, : sg[G]])            # past the used width nothing is written or read
        want = decode(ref)
        np.testing.assert_array_equal(got[:, p], want)
        pad = np.ones(got.shape[1], bool)
        pad[p] = False
        assert (got[:, pad] == 0).all()
    np.testing.assert_array_equal(decode(grp.x.codes_t), decode(plain.x.codes_t))


def _layer_inputs(rng, M, K, Nn, flat=False):
    if flat:   # every channel's range within a factor 2 of the largest: all in group 0
        x = rng.standard_normal((M, K)).astype(np.float32)
        dy = rng.standard_normal((M, Nn)).astype(np.float32)
    else:
        sx = np.exp(rng.normal(0, 1.0, K)).astype(np.float32)
        sx[rng.random(K) < 0.02] *= 50
        x = (rng.standard_normal((M, K)) * sx).astype(np.float32)
        sg = np.exp(rng.normal(0, 2.0, Nn)).astype(np.float32)
        dy = (rng.laplace(0, 1, (M, Nn)) * sg).astype(np.float32)
    w = (rng.standard_normal((K, Nn)) * 0.02).astype(np.float32)
    return x, w, dy


@pytest.mark.parametrize("M,K,Nn,bits,G,flat", [(2000, 700, 384, 8, 4, False),
                                                (2000, 768, 512, 8, 4, True),
                                                (1500, 640, 300, 8, 8, False),
                                                (1000, 500, 260, 8, 6, True),
                                                (3000, 1024, 512, 6, 4, False),
                                                (4096, 640, 256, 4, 4, False),
                                                (300, 3000, 256, 8, 8, False)])
def test_grouped_layer_matches_oracle(M, K, Nn, bits, G, flat):
    rng = np.random.default_rng(M + K + Nn + G)
    x, w, dy = _layer_inputs(rng, M, K, Nn, flat)
    lay = L.QuantLinear(M, K, Nn, bits, G, "cuda", with_acc=True, grouped=True)
    lay.step(to_gpu(x), to_gpu(w), to_gpu(dy), 11)
    torch.cuda.synchronize()
    assert lay.status.item() == 0
    o = oracle_layer(x, w, dy, bits, G, 11)
    if flat:
        assert (o["x"]["exp"] == 0).all() and (o["g"]["exp"] == 0).all()
    np.testing.assert_array_equal(lay.acc["fwd"].cpu().numpy(), o["T_fwd"], err_msg="T fwd")
    np.testing.assert_array_equal(lay.acc["dgrad"].cpu().numpy(), o["T_dgrad"], err_msg="T dgrad")
    np.testing.assert_array_equal(lay.acc["wgrad"].cpu().numpy(), o["T_wgrad"], err_msg="T wgrad")
    assert_close_f32(lay.y.cpu().numpy(), o["y"], "Y")
    assert_close_f32(lay.dx.cpu().numpy(), o["dx"], "dX")
    assert_close_f32(lay.dw.cpu().numpy(), o["dw"], "dW")


def test_folded_layout_refuses_what_the_group_order_runs():
    # 8 bits with N_G = 8: a 64-wide K block of folded products (127 * 127 * 128 each) can pass
    # the exact FP32 range, so the folded layout is refused; the group order runs it (above)
    lay = L.QuantLinear(256, 256, 256, 8, 8, "cuda")
    x = torch.randn(256, 256, device="cuda")
    lay.quantize_activation(x)
    lay.quantize_gradient(x, 1)
    lay.quantize_weights(x * 0.02)
    with pytest.raises(N.ShiftQuantError) as e:
        lay.gemms()
    assert e.value.status == N.SQ_EUNSUPPORTED
