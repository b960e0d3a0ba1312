"""Tensors split by rows (tokens) across ranks, on CPU with two `gloo` ranks and the oracle as
each rank's compute.  Quantization: each rank takes its shard's per-column ranges,
all-reduces them with MAX, groups, and quantizes telling the quantizer the shard's first
row (row0: stochastic rounding draws by the logical index); every rank's ranges, tau_0, exponents, codes and scale must
equal the whole tensor's.  Weight gradient: the ranks' integer sums, all-reduced with SUM
and dequantized once, must equal the whole batch's.  The CUDA path is exercised the same
way on one GPU by tests/test_gpu_quant.py and tests/test_gpu_gemm.py."""
import multiprocessing as mp
import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _tensor():
    rng = np.random.default_rng(7)
    R, C = 300, 96
    x = (rng.standard_normal((R, C)) * np.exp(rng.normal(0.0, 1.5, C))).astype(np.float32)
    x[:, 5] *= 100.0
    x[:, 9] = 0.0
    return x


def _shard_main(rank, world, port, bits, G, mode, seed, bounds, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import torch
    import torch.distributed as dist
    import oracle as O
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        x = _tensor()
        r0, r1 = bounds[rank], bounds[rank + 1]
        shard = x[r0:r1]
        local, _ = O.range_cols(shard)
        t = torch.from_numpy(local.copy())
        dist.all_reduce(t, op=dist.ReduceOp.MAX)   # the exchange
        rng = t.numpy()
        tau0, e, _ = O.group(rng, G)
        q, s = O.quantize_shift(shard, bits, G, tau0, e, mode, seed, row0=r0)
        whole = O.shiftquant_tensor(x, bits, G, mode, seed)
        ok = (np.array_equal(rng.view(np.uint32), whole["range"].view(np.uint32))
              and np.float32(tau0).view(np.uint32) == np.float32(whole["tau0"]).view(np.uint32)
              and np.array_equal(e, whole["exp"])
              and np.array_equal(q, whole["codes"][r0:r1])
              and np.float32(s).view(np.uint32) == np.float32(whole["scale"]).view(np.uint32))
        out.put((rank, bool(ok)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("bits,mode", [(4, 0), (4, 1), (8, 1)])
def test_two_gloo_ranks_quantize_their_shards_as_the_whole_tensor(bits, mode):
    world, G, seed, bounds = 2, 4, 0xC0FFEE, [0, 131, 300]
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_shard_main, args=(r, world, port, bits, G, mode, seed, bounds, out))
             for r in range(world)]
    for p in procs:
        p.start()
    got = sorted(out.get(timeout=180) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert got == [(0, True), (1, True)]


def test_row_offset_draws_the_whole_tensors_numbers():
    # rows row0.. of a tensor quantized alone with row0 draw what the whole tensor draws for
    # them: the stochastic codes of every shard equal the whole tensor's rows, and without the
    # offset they do not
    sys.path.insert(0, ROOT)
    import oracle as O
    x = _tensor()
    G, bits, seed = 4, 4, 0xDEADBEEF12345678
    whole = O.shiftquant_tensor(x, bits, G, 1, seed)
    for r0, r1 in ((0, 1), (1, 40), (131, 300), (299, 300)):
        q, _ = O.quantize_shift(x[r0:r1], bits, G, whole["tau0"], whole["exp"], 1, seed, row0=r0)
        np.testing.assert_array_equal(q, whole["codes"][r0:r1])
    q, _ = O.quantize_shift(x[131:300], bits, G, whole["tau0"], whole["exp"], 1, seed)
    assert (q != whole["codes"][131:300]).any()


def _wgrad_main(rank, world, port, bits, G, seed, bounds, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import torch
    import torch.distributed as dist
    import oracle as O
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        x = _tensor()
        dy = _tensor()[:, ::-1].copy() * np.float32(0.5)
        r0, r1 = bounds[rank], bounds[rank + 1]
        q = {}
        for name, t, mode, sd in (("x", x, 0, 0), ("g", dy, 1, seed)):
            local, _ = O.range_cols(t[r0:r1])
            rt = torch.from_numpy(local.copy())
            dist.all_reduce(rt, op=dist.ReduceOp.MAX)
            tau0, e, _ = O.group(rt.numpy(), G)
            codes, s = O.quantize_shift(t[r0:r1], bits, G, tau0, e, mode, sd, row0=r0)
            q[name] = (codes, e, s)
        # the shard's weight-gradient sums (canonical, int64), summed over the ranks
        T = torch.from_numpy(O.gemm_wgrad(q["x"][0], q["x"][1], q["g"][0], q["g"][1], G))
        dist.all_reduce(T, op=dist.ReduceOp.SUM)
        dw = O.dequant(T.numpy(), q["x"][2], q["g"][2], 2 * (G - 1))
        ox = O.shiftquant_tensor(x, bits, G, 0, 0)
        og = O.shiftquant_tensor(dy, bits, G, 1, seed)
        T_whole = O.gemm_wgrad(ox["codes"], ox["exp"], og["codes"], og["exp"], G)
        dw_whole = O.dequant(T_whole, ox["scale"], og["scale"], 2 * (G - 1))
        ok = np.array_equal(T.numpy(), T_whole) and np.array_equal(dw.view(np.uint32),
                                                                   dw_whole.view(np.uint32))
        out.put((rank, bool(ok)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("bits", [4, 8])
def test_two_gloo_ranks_sum_the_weight_gradient_exactly(bits):
    # each rank's integer weight-gradient sums over its own tokens, all-reduced with SUM and
    # dequantized once, equal the whole batch's dW bit for bit
    world, G, seed, bounds = 2, 4, 0xBEEF, [0, 131, 300]
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_wgrad_main, args=(r, world, port, bits, G, seed, bounds, out))
             for r in range(world)]
    for p in procs:
        p.start()
    got = sorted(out.get(timeout=180) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert got == [(0, True), (1, True)]
