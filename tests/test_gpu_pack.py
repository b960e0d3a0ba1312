"""GPU parity of packed sub-byte storage (Sec. 5.2) against the oracle's format: the
library's 4-bit ShiftQuant codes packed two per byte equal the oracle's packing of the
oracle's codes byte for byte, unpacking restores the codes, and the grouping map packs into
the oracle's 1/2/4-bit fields; ragged rows (odd widths, tails shorter than a thread's
sixteen codes) and unaligned leading dimensions take the scalar paths."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2411_10948_gb300 import layer as L
from paper_2411_10948_gb300 import native as N
from parity_util import decode, to_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2411_10948_gb300 import build
    build.build_library()
    N.load()


@pytest.mark.parametrize("R,C,bits,G,ldp_extra", [(12544, 2304, 4, 4, 0), (300, 77, 4, 4, 3),
                                                  (64, 33, 3, 2, 0), (129, 1000, 4, 8, 0),
                                                  (5, 1, 2, 1, 0), (2304, 12544, 4, 4, 0),
                                                  (40, 528, 4, 4, 8)])
def test_packed_codes_match_oracle_and_round_trip(R, C, bits, G, ldp_extra):
    rng = np.random.default_rng(R + C)
    x = (rng.standard_normal((R, C)) * np.exp(rng.normal(0, 1.5, C))).astype(np.float32)
    q = L.ShiftTensor.alloc(R, C, bits, G, "cuda", transposed=False)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    L.shift_quantize(to_gpu(x), q, bits, G, N.SQ_ROUND_STOCHASTIC, 5, st)
    W = (C + 1) // 2 + ldp_extra
    packed = torch.full((R, W), 0xAA, dtype=torch.uint8, device="cuda")
    N.shiftquant_pack_codes(q.codes, bits, G, packed[:, : (C + 1) // 2] if ldp_extra == 0 else packed,
                            st)
    back = L.empty_codes(R, C, bits, G, "cuda")
    back.view(torch.uint8).fill_(0x55)
    N.shiftquant_unpack_codes(packed, C, bits, G, back)
    torch.cuda.synchronize()
    assert st.item() == 0
    oq = O.shiftquant_tensor(x, bits, G, mode=1, seed=5)["codes"]
    np.testing.assert_array_equal(decode(q.codes), oq)                    # the codes packed
    np.testing.assert_array_equal(packed[:, : (C + 1) // 2].cpu().numpy(), O.pack4(oq))
    np.testing.assert_array_equal(decode(back), oq)


def test_packing_a_shifted_code_sets_the_status():
    t = L.empty_codes(4, 16, 4, 4, "cuda")
    t.copy_(torch.full((4, 16), 56.0, device="cuda").to(torch.float8_e4m3fn).view(torch.uint8))
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    packed = torch.zeros((4, 8), dtype=torch.uint8, device="cuda")
    N.shiftquant_pack_codes(t, 4, 4, packed, st)
    torch.cuda.synchronize()
    assert st.item() & N.SQ_DEV_INTERNAL


@pytest.mark.parametrize("C,G", [(2304, 4), (77, 4), (1000, 8), (33, 2), (9, 1)])
def test_packed_group_map_matches_oracle(C, G):
    rng = np.random.default_rng(C + G)
    e = rng.integers(0, G, C).astype(np.uint8)
    nb = N.shiftquant_packed_groups_bytes(C, G)
    packed = torch.zeros(nb, dtype=torch.uint8, device="cuda")
    N.shiftquant_pack_groups(torch.from_numpy(e).cuda(), G, packed)
    back = torch.zeros(C, dtype=torch.uint8, device="cuda")
    N.shiftquant_unpack_groups(packed, C, G, back)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(packed.cpu().numpy(), O.pack_groups(e, G))
    np.testing.assert_array_equal(back.cpu().numpy(), e)
