"""One ShiftQuant-quantized linear layer Y = X W on the GPU: the buffers it needs and the
sequence of C-ABI calls for its three training GEMMs, with the operand roles of the
paper's setup (Sec. 5.1): ShiftQuant on activations and gradients, per-out-channel
weights in the forward GEMM, per-in-channel weights in loss propagation.

torch only allocates device memory here; every arithmetic step is a libshiftquant call.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import native as N


def round_up(n: int, m: int) -> int:
    return (n + m - 1) // m * m


def code_ld(cols: int, bits: int, n_groups: int) -> int:
    """Leading dimension (elements) that keeps every code row 16-byte aligned for TMA."""
    return max(round_up(cols, 16 // N.shiftquant_code_bytes(bits, n_groups)), 16)


def empty_codes(rows: int, cols: int, bits: int, n_groups: int, device) -> torch.Tensor:
    """[rows, cols] view of a code buffer whose rows are padded to a 16-byte multiple."""
    ld = code_ld(cols, bits, n_groups)
    buf = torch.zeros((max(rows, 1), ld), dtype=N.code_dtype(bits, n_groups), device=device)
    return buf[:rows, :cols]


@dataclass
class ShiftTensor:
    """A ShiftQuant-quantized [R, C] tensor: codes (and their transpose), group exponents,
    the channel ranges, tau_0 and the tensor scale s = tau_0 / Q."""
    codes: torch.Tensor
    codes_t: torch.Tensor | None
    exp: torch.Tensor
    range: torch.Tensor
    tau0: torch.Tensor
    scale: torch.Tensor

    @staticmethod
    def alloc(R, C, bits, n_groups, device, transposed=True) -> "ShiftTensor":
        return ShiftTensor(
            codes=empty_codes(R, C, bits, n_groups, device),
            codes_t=empty_codes(C, R, bits, n_groups, device) if transposed else None,
            exp=torch.zeros(max(C, 1), dtype=torch.uint8, device=device)[:C],
            range=torch.zeros(max(C, 1), dtype=torch.float32, device=device)[:C],
            tau0=torch.zeros(1, dtype=torch.float32, device=device),
            scale=torch.zeros(1, dtype=torch.float32, device=device))


@dataclass
class ChannelTensor:
    """A per-channel quantized weight in the layout one GEMM reads, with its scales."""
    codes: torch.Tensor
    range: torch.Tensor
    scale: torch.Tensor


def shift_quantize(x, q: ShiftTensor, bits, n_groups, mode, seed, status, stream=None):
    """Range pass, grouping and quantization of x [R, C] into q (three launches)."""
    N.shiftquant_calibrate(x, N.SQ_GRAN_SHIFT, n_groups, q.range, q.tau0, q.exp, status, stream)
    N.shiftquant_quantize(x, N.SQ_GRAN_SHIFT, bits, n_groups, q.tau0, q.exp, None, mode, seed,
                          q.codes, q.codes_t, q.scale, stream)


def shard_shift_quantize(x, q: ShiftTensor, bits, n_groups, mode, seed, row0, status,
                         all_reduce_max, stream=None):
    """ShiftQuant of one row (token) shard x [R_local, C] of a tensor split across ranks,
    equal bit for bit to the whole tensor's rows: the shard's per-column ranges, their
    element-wise maximum over all shards (all_reduce_max(tensor) in place -- for instance
    torch.distributed.all_reduce with ReduceOp.MAX: the one exchange the path needs), the
    grouping from that, and the quantizer told the shard's first row (row0 in the whole
    tensor), so that stochastic rounding draws the whole tensor's numbers."""
    N.shiftquant_calibrate(x, N.SQ_GRAN_PER_COL, n_groups, q.range, None, None, status, stream)
    all_reduce_max(q.range)
    N.shiftquant_group(q.range, n_groups, q.tau0, q.exp, status, stream)
    N.shiftquant_quantize(x, N.SQ_GRAN_SHIFT, bits, n_groups, q.tau0, q.exp, None, mode,
                          seed, q.codes, q.codes_t, q.scale, stream, row0=row0)


def weight_quantize_fwd(w, out: ChannelTensor, fold_exp, bits, n_groups, status, stream=None):
    """W [K, N] per-out-channel, written transposed [N, K] with 2^(G-1-e_k) folded in."""
    N.shiftquant_calibrate(w, N.SQ_GRAN_PER_COL, n_groups, out.range, None, None, status, stream)
    N.shiftquant_quantize(w, N.SQ_GRAN_PER_COL, bits, n_groups, out.range, None, fold_exp,
                          N.SQ_ROUND_NEAREST_EVEN, 0, None, out.codes, out.scale, stream)


def weight_quantize_dgrad(w, out: ChannelTensor, fold_exp, bits, n_groups, status, stream=None):
    """W [K, N] per-in-channel, natural layout, 2^(G-1-e_j) of dY's channel j folded in."""
    N.shiftquant_calibrate(w, N.SQ_GRAN_PER_ROW, n_groups, out.range, None, None, status, stream)
    N.shiftquant_quantize(w, N.SQ_GRAN_PER_ROW, bits, n_groups, out.range, None, fold_exp,
                          N.SQ_ROUND_NEAREST_EVEN, 0, out.codes, None, out.scale, stream)


def weight_quantize_both(w, wf: ChannelTensor, wd: ChannelTensor, x_exp, g_exp, bits, n_groups,
                         status, stream=None):
    """Both roles of W [K, N] in two passes over it: the ranges of both from one read, then
    both code sets from one read (the same codes as weight_quantize_fwd and _dgrad)."""
    N.shiftquant_calibrate_weight(w, wf.range, wd.range, status, stream)
    N.shiftquant_quantize_weight(w, bits, n_groups, wf.range, wd.range, x_exp, g_exp, wf.codes,
                                 wf.scale, wd.codes, wd.scale, stream)


class QuantLinear:
    """Buffers and calls of one quantized linear layer: X [M, K], W [K, N], dY [M, N]."""

    def __init__(self, M, K, N_, bits, n_groups, device="cuda", with_acc=False,
                 use_workspace=True, with_inputs=False, grouped=False, transposed=True):
        """transposed=False: X and dY keep no transposed code copies; the weight gradient
        reads their codes in place (MN-major operands of the layer launch).  None: the
        library's advice for this shape (shiftquant_gemm_layer_wgrad_in_place).  A grouped
        layer needs the copies (its forward operands are channel-permuted)."""
        if grouped and transposed is False:
            raise ValueError("a group-ordered layer needs the transposed code copies")
        if transposed is None:
            transposed = grouped or N.shiftquant_gemm_layer_wgrad_in_place(
                M, K, N_, bits, n_groups) != 1
        self.M, self.K, self.N, self.bits, self.G = M, K, N_, bits, n_groups
        self.grouped = grouped
        dev = torch.device(device)
        # device input buffers for shiftquant_layer_step(_host), when asked for
        self.inputs = None
        if with_inputs:
            self.inputs = (torch.zeros((M, K), dtype=torch.float32, device=dev),
                           torch.zeros((K, N_), dtype=torch.float32, device=dev),
                           torch.zeros((M, N_), dtype=torch.float32, device=dev))
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.x = ShiftTensor.alloc(M, K, bits, n_groups, dev, transposed)
        self.g = ShiftTensor.alloc(M, N_, bits, n_groups, dev, transposed)
        # grouped: the forward and loss-propagation operands hold their inner index in group
        # order (Sec. 3.2's per-group products as one launch) over the padded width
        self.x_pos = self.x_seg = self.g_pos = self.g_seg = None
        kw = N.shiftquant_group_order_width(K, bits, n_groups) if grouped else K
        nw = N.shiftquant_group_order_width(N_, bits, n_groups) if grouped else N_
        if grouped:
            self.x.codes = empty_codes(M, kw, bits, n_groups, dev)
            self.g.codes = empty_codes(M, nw, bits, n_groups, dev)
            self.x_pos = torch.zeros(max(K, 1), dtype=torch.int32, device=dev)[:K]
            self.g_pos = torch.zeros(max(N_, 1), dtype=torch.int32, device=dev)[:N_]
            self.x_seg = torch.zeros(2 * n_groups + 1, dtype=torch.int32, device=dev)
            self.g_seg = torch.zeros(2 * n_groups + 1, dtype=torch.int32, device=dev)
        self.wf = ChannelTensor(empty_codes(N_, kw, bits, n_groups, dev),
                                torch.zeros(N_, dtype=torch.float32, device=dev),
                                torch.zeros(N_, dtype=torch.float32, device=dev))
        self.wd = ChannelTensor(empty_codes(K, nw, bits, n_groups, dev),
                                torch.zeros(K, dtype=torch.float32, device=dev),
                                torch.zeros(K, dtype=torch.float32, device=dev))
        self.y = torch.zeros((M, N_), dtype=torch.float32, device=dev)
        self.dx = torch.zeros((M, K), dtype=torch.float32, device=dev)
        self.dw = torch.zeros((K, N_), dtype=torch.float32, device=dev)
        self.acc = None
        if with_acc:
            self.acc = {"fwd": torch.zeros((M, N_), dtype=torch.int64, device=dev),
                        "dgrad": torch.zeros((M, K), dtype=torch.int64, device=dev),
                        "wgrad": torch.zeros((K, N_), dtype=torch.int64, device=dev)}
        # one split-K workspace per GEMM, so the three may run concurrently
        self.ws_fwd = self.ws_dgrad = self.ws_wgrad = None
        if use_workspace:
            def ws(which, m, n, k):
                need = N.shiftquant_gemm_workspace_bytes(which, m, n, k, bits, n_groups)
                return torch.zeros(need // 4, dtype=torch.int32, device=dev) if need else None
            self.ws_fwd = ws(0, M, N_, K)
            self.ws_dgrad = ws(1, M, K, N_)
            self.ws_wgrad = ws(2, K, N_, M)
        self.ws = self.ws_fwd if self.ws_fwd is not None else (
            self.ws_dgrad if self.ws_dgrad is not None else self.ws_wgrad)
        self.ws_layer = None
        if use_workspace:
            need = N.shiftquant_gemm_layer_workspace_bytes(M, K, N_, bits, n_groups,
                                                           grouped=grouped)
            if need:
                self.ws_layer = torch.zeros(need // 4, dtype=torch.int32, device=dev)

    # --- the hot path, step by step --------------------------------------------------
    def _shift_quantize(self, t, q, pos, seg, mode, seed, stream):
        if not self.grouped:
            shift_quantize(t, q, self.bits, self.G, mode, seed, self.status, stream)
            return
        N.shiftquant_calibrate(t, N.SQ_GRAN_SHIFT, self.G, q.range, q.tau0, q.exp, self.status,
                               stream)
        N.shiftquant_group_order(q.exp, self.bits, self.G, pos, seg, stream)
        N.shiftquant_quantize_ordered(t, N.SQ_GRAN_SHIFT, self.bits, self.G, q.tau0, q.exp, mode,
                                      seed, pos, seg, q.codes, q.codes_t, q.scale, stream)

    def quantize_activation(self, x, stream=None):
        self._shift_quantize(x, self.x, self.x_pos, self.x_seg, N.SQ_ROUND_NEAREST_EVEN, 0,
                             stream)

    def quantize_gradient(self, dy, seed, stream=None):
        self._shift_quantize(dy, self.g, self.g_pos, self.g_seg, N.SQ_ROUND_STOCHASTIC, seed,
                             stream)

    def quantize_weights(self, w, stream=None):
        if not self.grouped:
            weight_quantize_both(w, self.wf, self.wd, self.x.exp, self.g.exp, self.bits, self.G,
                                 self.status, stream)
            return
        # group-ordered weights carry no folded shift: each segment is shifted whole
        st, b, G = self.status, self.bits, self.G
        N.shiftquant_calibrate(w, N.SQ_GRAN_PER_COL, G, self.wf.range, None, None, st, stream)
        N.shiftquant_quantize_ordered(w, N.SQ_GRAN_PER_COL, b, G, self.wf.range, None,
                                      N.SQ_ROUND_NEAREST_EVEN, 0, self.x_pos, self.x_seg, None,
                                      self.wf.codes, self.wf.scale, stream)
        N.shiftquant_calibrate(w, N.SQ_GRAN_PER_ROW, G, self.wd.range, None, None, st, stream)
        N.shiftquant_quantize_ordered(w, N.SQ_GRAN_PER_ROW, b, G, self.wd.range, None,
                                      N.SQ_ROUND_NEAREST_EVEN, 0, self.g_pos, self.g_seg,
                                      self.wd.codes, None, self.wd.scale, stream)

    def forward(self, stream=None):
        N.shiftquant_gemm_fwd(self.x.codes, self.x.scale, self.wf.codes, self.wf.scale, self.M,
                              self.N, self.K, self.bits, self.G, self.y,
                              self.acc["fwd"] if self.acc else None, self.ws_fwd, self.status,
                              stream)

    def dgrad(self, stream=None):
        N.shiftquant_gemm_dgrad(self.g.codes, self.g.scale, self.wd.codes, self.wd.scale, self.M,
                                self.K, self.N, self.bits, self.G, self.dx,
                                self.acc["dgrad"] if self.acc else None, self.ws_dgrad,
                                self.status, stream)

    def wgrad(self, stream=None):
        if self.x.codes_t is None or self.g.codes_t is None:
            # codes in place: the layer launch with the weight gradient alone
            self.gemms(stream, gemm_mask=4)
            return
        N.shiftquant_gemm_wgrad(self.x.codes_t, self.x.scale, self.x.exp, self.g.codes_t,
                                self.g.scale, self.g.exp, self.K, self.N, self.M, self.bits,
                                self.G, self.dw, self.acc["wgrad"] if self.acc else None,
                                self.ws_wgrad, self.status, stream)

    def gemms(self, stream=None, gemm_mask=0, max_ctas=0, use_workspace=True, y_range=None,
              dx_range=None):
        """The three GEMMs in one persistent launch (shiftquant_gemm_layer); gemm_mask picks
        a subset (bit 0 forward, 1 loss propagation, 2 weight gradient), max_ctas caps the
        CTAs.  A launch running beside another on a different stream must not share its
        workspace: pass use_workspace=False to one of them."""
        acc = self.acc or {}
        N.shiftquant_gemm_layer(self.x.codes, self.x.codes_t, self.x.scale, self.x.exp,
                                self.g.codes, self.g.codes_t, self.g.scale, self.g.exp,
                                self.wf.codes, self.wf.scale, self.wd.codes, self.wd.scale,
                                self.M, self.K, self.N, self.bits, self.G, self.y, self.dx,
                                self.dw, acc.get("fwd"), acc.get("dgrad"), acc.get("wgrad"),
                                self.ws_layer if use_workspace else None, self.status, stream,
                                gemm_mask=gemm_mask, max_ctas=max_ctas, y_range=y_range,
                                dx_range=dx_range, x_seg=self.x_seg, g_seg=self.g_seg)

    def step(self, x, w, dy, seed, stream=None):
        """One training step of the layer: every quantizer pass and all three GEMMs."""
        self.quantize_activation(x, stream)
        self.quantize_gradient(dy, seed, stream)
        self.quantize_weights(w, stream)
        if self.grouped:   # group-ordered operands: the layer launch carries the segment tables
            self.gemms(stream)
            return
        self.forward(stream)
        self.dgrad(stream)
        self.wgrad(stream)

    def step_concurrent(self, x, w, dy, seed, streams, gemm_events=None, dgrad_ctas=0,
                        start_event=None):
        """The same step with its independent quantizer work on three streams forked from the
        current one -- the activation chain, the gradient chain and the weight (its range
        pass right away, its quantization for both roles once both other operands'
        exponents exist) -- joined back before the three GEMMs run as one launch on the
        current stream.
        Capturable in a CUDA graph, which then runs the independent work concurrently.
        gemm_events: optional (start, end) CUDA events recorded around the GEMM call (for
        timing inside a captured graph they must be created with external=True);
        start_event: optional event recorded on the current stream before anything else
        (with gemm_events[0]: the quantizer phase of the step).
        dgrad_ctas > 0: the loss-propagation GEMM (which needs only dY's and W's codes) runs
        as its own launch of at most that many CTAs on the gradient stream as soon as its
        operands exist, beside the activation chain; the forward and weight-gradient GEMMs
        follow as one launch."""
        main = torch.cuda.current_stream()
        if start_event is not None:
            start_event.record(main)
        s_x, s_g, s_w = streams[:3]
        for s in (s_x, s_g, s_w):
            s.wait_stream(main)
        ev = {k: torch.cuda.Event() for k in ("x_cal", "g_cal")}
        b, G, st = self.bits, self.G, self.status
        for s_, q, t, mode, sd, cal in ((s_x, self.x, x, N.SQ_ROUND_NEAREST_EVEN, 0, "x_cal"),
                                        (s_g, self.g, dy, N.SQ_ROUND_STOCHASTIC, seed, "g_cal")):
            with torch.cuda.stream(s_):
                N.shiftquant_calibrate(t, N.SQ_GRAN_SHIFT, G, q.range, q.tau0, q.exp, st, s_)
                ev[cal].record(s_)
                N.shiftquant_quantize(t, N.SQ_GRAN_SHIFT, b, G, q.tau0, q.exp, None, mode, sd,
                                      q.codes, q.codes_t, q.scale, s_)
        with torch.cuda.stream(s_w):
            N.shiftquant_calibrate_weight(w, self.wf.range, self.wd.range, st, s_w)
            s_w.wait_event(ev["x_cal"])
            s_w.wait_event(ev["g_cal"])
            N.shiftquant_quantize_weight(w, b, G, self.wf.range, self.wd.range, self.x.exp,
                                         self.g.exp, self.wf.codes, self.wf.scale, self.wd.codes,
                                         self.wd.scale, s_w)
        if dgrad_ctas > 0:
            with torch.cuda.stream(s_g):
                s_g.wait_stream(s_w)
                self.gemms(s_g, gemm_mask=2, max_ctas=dgrad_ctas, use_workspace=False)
            for s in (s_x, s_w):
                main.wait_stream(s)
            if gemm_events is not None:
                gemm_events[0].record(main)
            self.gemms(main, gemm_mask=5)
            if gemm_events is not None:
                gemm_events[1].record(main)
            main.wait_stream(s_g)
            return
        for s in (s_x, s_g, s_w):
            main.wait_stream(s)
        if gemm_events is not None:
            gemm_events[0].record(main)
        self.gemms(main)
        if gemm_events is not None:
            gemm_events[1].record(main)

    def step_args(self, x=None, w=None, dy=None):
        """The C struct sq_layer_step over this layer's buffers, with x, w, dy (dense device
        tensors) as the inputs, or the layer's own input buffers (with_inputs=True)."""
        if x is None:
            assert self.inputs is not None, "QuantLinear(with_inputs=True) or explicit inputs"
            x, w, dy = self.inputs
        return N.layer_step_args(
            self.M, self.K, self.N, self.bits, self.G, x, w, dy, self.x.codes, self.x.codes_t,
            self.x.range, self.x.tau0, self.x.scale, self.x.exp, self.g.codes, self.g.codes_t,
            self.g.range, self.g.tau0, self.g.scale, self.g.exp, self.wf.codes, self.wf.range,
            self.wf.scale, self.wd.codes, self.wd.range, self.wd.scale, self.y, self.dx, self.dw,
            self.ws_layer, self.status)

    @property
    def gemm_ops(self) -> int:
        return 3 * 2 * self.M * self.N * self.K


class LinearChain:
    """Quantized linear layers applied one after another, X_{l+1} = Y_l (nothing between the
    layers), trained by a forward pass over the layers and a backward pass in reverse with
    dY_l = dX_{l+1}.  dims = (d_0, d_1, ..., d_L): layer l maps d_l to d_{l+1} over M tokens.

    fused_ranges=True: the range pass of every inner activation Y_l and inner gradient dX_l
    is formed in the epilogue of the GEMM that writes it (the y_range / dx_range outputs of
    shiftquant_gemm_layer), and its consumer groups from that vector (shiftquant_group) and
    quantizes: no pass over the tensor before its quantization.  fused_ranges=False runs the
    usual range pass (shiftquant_calibrate) instead.  Both give the same bits."""

    def __init__(self, M, dims, bits, n_groups, device="cuda", fused_ranges=True):
        dev = torch.device(device)
        self.M, self.dims, self.bits, self.G = M, list(dims), bits, n_groups
        self.fused = fused_ranges
        self.layers = [QuantLinear(M, dims[i], dims[i + 1], bits, n_groups, dev,
                                   transposed=None)
                       for i in range(len(dims) - 1)]
        self.y_range = [torch.zeros(d, dtype=torch.float32, device=dev) for d in dims[1:]]
        self.dx_range = [torch.zeros(d, dtype=torch.float32, device=dev) for d in dims[:-1]]

    def _quantize_input(self, t, q, range_vec, mode, seed, status, stream):
        if range_vec is not None:
            N.shiftquant_group(range_vec, self.G, q.tau0, q.exp, status, stream)
        else:
            N.shiftquant_calibrate(t, N.SQ_GRAN_SHIFT, self.G, q.range, q.tau0, q.exp, status,
                                   stream)
        N.shiftquant_quantize(t, N.SQ_GRAN_SHIFT, self.bits, self.G, q.tau0, q.exp, None, mode,
                              seed, q.codes, q.codes_t, q.scale, stream)

    def step(self, x0, weights, dy_last, seed, stream=None):
        """One training step: forward through every layer from x0 [M, d_0], then backward
        from dy_last [M, d_L]; weights[l] is W_l [d_l, d_{l+1}].  Layer l's gradient rounds
        stochastically under seed + l."""
        Lz = self.layers
        last = len(Lz) - 1
        for l, lay in enumerate(Lz):
            x = x0 if l == 0 else Lz[l - 1].y
            rng = self.y_range[l - 1] if (self.fused and l > 0) else None
            self._quantize_input(x, lay.x, rng, N.SQ_ROUND_NEAREST_EVEN, 0, lay.status, stream)
            weight_quantize_fwd(weights[l], lay.wf, lay.x.exp, self.bits, self.G, lay.status,
                                stream)
            lay.gemms(stream, gemm_mask=1,
                      y_range=self.y_range[l] if (self.fused and l < last) else None)
        for l in range(last, -1, -1):
            lay = Lz[l]
            dy = dy_last if l == last else Lz[l + 1].dx
            rng = self.dx_range[l + 1] if (self.fused and l < last) else None
            self._quantize_input(dy, lay.g, rng, N.SQ_ROUND_STOCHASTIC, seed + l, lay.status,
                                 stream)
            weight_quantize_dgrad(weights[l], lay.wd, lay.g.exp, self.bits, self.G, lay.status,
                                  stream)
            lay.gemms(stream, gemm_mask=6,
                      dx_range=self.dx_range[l] if (self.fused and l > 0) else None)

    def status_ok(self) -> bool:
        return all(int(l.status.item()) == 0 for l in self.layers)

    @property
    def gemm_ops(self) -> int:
        return sum(l.gemm_ops for l in self.layers)


class CapturedStep:
    """A sequence of library calls captured once into a CUDA graph and replayed with one
    launch, so a step of many short kernels pays no per-call CPU cost.  Buffers are the
    ones the calls referenced at capture time: refill them in place between replays.
    Every kernel runs again on each replay; scalar arguments (such as the SR seed) keep
    their captured values."""

    def __init__(self, fn, warmup: int = 1):
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            for _ in range(warmup):
                fn()
        torch.cuda.current_stream().wait_stream(s)
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            fn()

    def replay(self) -> None:
        self.graph.replay()


class HostSteps:
    """Training steps fed from host memory and returned to it through the C entry point
    shiftquant_layer_step_host_split: for every layer of a step, one call copies X, W and
    dY in on the copy-in stream, runs the layer's whole step on the layer's own stream and
    copies Y, dX and dW back on the copy-out stream, the three joined by events.  Two sets
    of device buffers take the steps in turn; a set's copies in wait for its previous
    copies back.  With one stream for every copy in and one for every copy back, each
    direction of the host link works through its copies in step order while earlier steps
    compute, so the link, not the GPU, sets the pace (a copy engine serves its copies in
    queue order: copies in queued behind another call's copies back would wait for them).

    shapes: (M, K, N) per layer."""

    def __init__(self, shapes, bits, n_groups, device="cuda", slots=2):
        dev = torch.device(device)
        self.shapes = list(shapes)
        self.copy_in = torch.cuda.Stream(device=dev)
        self.copy_out = torch.cuda.Stream(device=dev)
        self.slots = []
        for _ in range(slots):
            layers = [QuantLinear(M, K, N_, bits, n_groups, dev, with_inputs=True,
                                  transposed=None)
                      for (M, K, N_) in self.shapes]
            # per layer: inputs in, step done, outputs out (recorded once here so that the
            # CUDA events exist before the library records them)
            events = [{k: torch.cuda.Event() for k in ("in", "done", "out")} for _ in layers]
            for evs in events:
                for ev in evs.values():
                    ev.record()
            self.slots.append({"layers": layers, "args": [l.step_args() for l in layers],
                               "streams": [torch.cuda.Stream(device=dev) for _ in layers],
                               "events": events})

    def run(self, host_inputs, host_outputs, seed=0x5EED) -> torch.cuda.Event:
        """Queue one step per entry: host_inputs[i] = (x, w, dy) per layer, host_outputs[i] =
        (y, dx, dw) per layer, page-locked float32 host tensors (an entry may be None to
        skip that copy).  Step i draws its stochastic rounding under seed + i.  Returns an
        event on the current stream after the last copy back (synchronize on it before
        reading the host outputs)."""
        cur = torch.cuda.current_stream()
        streams = [self.copy_in, self.copy_out] + [st for sl in self.slots for st in sl["streams"]]
        for st in streams:
            st.wait_stream(cur)
        for i, (hin, hout) in enumerate(zip(host_inputs, host_outputs)):
            sl = self.slots[i % len(self.slots)]
            for args, st, ev, (x, w, dy), (y, dx, dw) in zip(sl["args"], sl["streams"],
                                                             sl["events"], hin, hout):
                N.shiftquant_layer_step_host_split(args, x, w, dy, y, dx, dw, seed + i,
                                                   self.copy_in, st, self.copy_out,
                                                   buffers_free=ev["out"], inputs_in=ev["in"],
                                                   step_done=ev["done"], outputs_out=ev["out"])
        for st in streams:
            cur.wait_stream(st)
        end = torch.cuda.Event(enable_timing=True)
        end.record(cur)
        return end

    def status_ok(self) -> bool:
        return all(int(l.status.item()) == 0 for sl in self.slots for l in sl["layers"])
