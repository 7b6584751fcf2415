"""Device buffers and the call sequence of one MoE layer step over the C ABI.

PyTorch supplies device memory and the stream; every stage runs in the
library's kernels through ``abi``.  Forward: route -> (LatentMoE down-
projection) -> dispatch -> grouped SwiGLU experts -> combine -> (up-
projection).  Backward runs the inverses in reverse order (Sec. 4.1 footnote:
the three forward transfers and their three inverses).
"""
from __future__ import annotations

import torch

from . import abi


def _dt(dtype: str):
    return torch.bfloat16 if dtype == "bf16" else torch.float32


class MoeLayer:
    """All buffers of one layer step for one shape, allocated once on ``device``.

    ``router="softmax"`` routes with softmax + renormalised top-K;
    ``router="sigmoid"`` with sigmoid scores, a selection-only expert bias and
    the sequence-level balance loss (coefficient ``aux_coef``; its gradient
    enters the backward pass scaled by ``aux_grad``), Sec. 5.2.
    ``shared_F > 0`` adds the ungated shared expert of that width (Sec. 5.2),
    whose output is added to the layer output.
    ``gather=True`` lets GEMM-1 and its weight gradient read the dispatched
    rows straight from x by token_of_row (no x_perm copy; the GEMM's producer
    copies the rows with 16-byte cp.async copies); the default ``False``
    writes x_perm in the dispatch and reads it back with tiled TMA copies,
    which is 2.4-2.7x faster on GB300 (one producer warp's row copies cannot
    keep the tensor cores fed).
    ``payload="fp8"`` dispatches the hidden rows as FP8 E4M3 codes with one
    power-of-two scale per row (b_x = 1) and dequantizes them on arrival;
    the gradient passes the quantization unchanged.  ``payload="nvfp4"``
    sends E2M1 codes with one E4M3 scale per 16 elements and one power-of-two
    scale per row (b_x = 1/2 plus the scales) the same way.
    """

    def __init__(self, S, GBS, K, D, E, F, dtype="bf16", H=0, device="cuda", router="softmax", aux_coef=1e-4,
                 aux_grad=1.0, shared_F=0, gather=False, payload="bf16"):
        if router not in ("softmax", "sigmoid"):
            raise ValueError(f"unknown router {router!r}")
        self.router = router
        self.gather = bool(gather)
        if payload not in ("bf16", "fp8", "nvfp4") or (payload != "bf16" and (gather or dtype != "bf16")):
            raise ValueError(f"payload {payload!r} with gather={gather}, dtype={dtype}")
        self.payload = payload
        self.aux_coef = float(aux_coef)
        self.aux_grad = float(aux_grad)
        self.shape = abi.MoeShape.of(S, GBS, K, D, E, F, dtype, H)
        self.T = T = S * GBS
        self.TK = TK = T * K
        self.K, self.D, self.E, self.F, self.H = K, D, E, F, H
        self.Din = H if H else D
        self.dtype = dtype
        dt = _dt(dtype)
        dev = torch.device(device)
        f32, i32 = torch.float32, torch.int32
        e = lambda *s, d=dt: torch.empty(*s, dtype=d, device=dev)  # noqa: E731
        Din = self.Din
        # weights; a LatentMoE layer with the softmax router keeps w_down [D, H]
        # and w_router [E, H] in one [D + E, H] array, which its backward reads
        # as one operand (moe_latent_route_bwd)
        self.latent_fused = bool(H) and router == "softmax" and dtype == "bf16" and (D + E) % 8 == 0
        self.w_down_router = e(D + E, H) if self.latent_fused else None
        self.w_router = self.w_down_router[D:] if self.latent_fused else e(E, Din)
        self.w1 = e(E, 2 * F, D)
        self.w2 = e(E, D, F)
        self.bias = None
        self.expert_bias = torch.zeros(E, dtype=f32, device=dev) if router == "sigmoid" else None
        self.shared_F = Fs = int(shared_F)
        self.w_s1 = e(Fs, self.Din) if Fs else None
        self.w_s2 = e(self.Din, Fs) if Fs else None
        self.w_down = (self.w_down_router[:D] if self.latent_fused else e(D, H)) if H else None
        self.w_upp = e(H, D) if H else None
        # forward
        self.x = e(T, Din)
        self.logits = e(T, E, d=f32)
        self.topk_idx = e(T, K, d=i32)
        self.topk_prob = e(T, K, d=f32)
        self.aux_f = e(GBS, E, d=f32) if router == "sigmoid" else None
        self.aux_loss = e(4, d=f32) if router == "sigmoid" else None
        self.x_lat = e(T, D) if H else None
        self.expert_offsets = e(E + 1, d=i32)
        self.row_of_slot = e(TK, d=i32)
        self.token_of_row = e(TK, d=i32)
        self.x_perm = None if self.gather else e(TK, D)
        self.x_perm_q = e(TK, D, d=torch.uint8) if payload == "fp8" else None
        self.x_scale_perm = e(TK, d=f32) if payload == "fp8" else None
        self.x_perm_q4 = e(TK, D // 2, d=torch.uint8) if payload == "nvfp4" else None
        self.x_bscale_perm = e(TK, D // 16, d=torch.uint8) if payload == "nvfp4" else None
        self.x_rscale_perm = e(TK, d=f32) if payload == "nvfp4" else None
        self.prob_perm = e(TK, d=f32)
        self.h = e(TK, 2 * F)
        self.act = e(TK, F)
        self.y_perm = e(TK, D)
        self.y_lat = e(T, D) if H else None
        self.y = e(T, Din)
        self.h_s = e(T, Fs) if Fs else None
        self.act_s = e(T, Fs) if Fs else None
        self.dh_s = e(T, Fs) if Fs else None
        self.dw_s1 = e(Fs, Din, d=f32) if Fs else None
        self.dw_s2 = e(Din, Fs, d=f32) if Fs else None
        # backward
        self.dy = e(T, Din)
        self.dy_lat = e(T, D) if H else None
        self.dy_perm = e(TK, D)
        self.dprob_perm = e(TK, d=f32)
        self.dx_perm = e(TK, D)
        self.dw1 = e(E, 2 * F, D, d=f32)
        self.dw2 = e(E, D, F, d=f32)
        # fused LatentMoE tail: [dx_lat | bf16 dlogits] in one [T, D + E] array
        self.dx_cat = e(T, D + E) if self.latent_fused else None
        self.dx_lat = (self.dx_cat[:, :D] if self.latent_fused else e(T, D)) if H else None
        self.dprob = e(T, K, d=f32)
        self.dx = e(T, Din)
        self.dlogits = e(T, E, d=f32)
        self.dw_router = e(E, Din, d=f32)
        self.dw_down = e(D, H, d=f32) if H else None
        self.dw_upp = e(H, D, d=f32) if H else None
        self.ws = torch.empty(abi.moe_workspace_size(self.shape), dtype=torch.uint8, device=dev)

    # ------------------------------------------------------------------
    def load(self, inputs: dict, stream=None) -> None:
        """Copy one ``synth.make_inputs`` dict into the device buffers and pack w1."""
        self.x.copy_(inputs["x"], non_blocking=True)
        self.dy.copy_(inputs["dy"], non_blocking=True)
        self.w_router.copy_(inputs["w_router"], non_blocking=True)
        self.w2.copy_(inputs["w2"], non_blocking=True)
        wg = inputs["w_gate"].to(self.x.device, non_blocking=True)
        wu = inputs["w_up"].to(self.x.device, non_blocking=True)
        abi.moe_pack_w1(self.shape, wg, wu, self.w1, stream)
        if self.H:
            self.w_down.copy_(inputs["w_down"], non_blocking=True)
            self.w_upp.copy_(inputs["w_upp"], non_blocking=True)
        if inputs.get("bias") is not None:
            self.bias = inputs["bias"].to(self.x.device, non_blocking=True).contiguous()
        else:
            self.bias = None
        if self.shared_F:
            self.w_s1.copy_(inputs["w_s1"], non_blocking=True)
            self.w_s2.copy_(inputs["w_s2"], non_blocking=True)
        if self.router == "sigmoid" and inputs.get("expert_bias") is not None:
            self.expert_bias.copy_(inputs["expert_bias"], non_blocking=True)

    # ------------------------------------------------------------------
    def forward(self, stream=None):
        s = self.shape
        if self.router == "sigmoid":
            abi.moe_route_sigmoid(s, self.x, self.w_router, self.expert_bias, self.aux_coef, self.logits,
                                  self.topk_idx, self.topk_prob, self.aux_f, self.aux_loss, self.ws, stream)
        else:
            abi.moe_route(s, self.x, self.w_router, self.bias, self.logits, self.topk_idx, self.topk_prob, self.ws,
                          stream)
        xd = self.x
        if self.H:
            abi.moe_latent_proj(s, self.H, self.D, self.x, self.w_down, self.x_lat, self.ws, stream)
            xd = self.x_lat
        if self.payload == "fp8":
            abi.moe_dispatch_fp8(s, xd, self.topk_idx, self.topk_prob, self.expert_offsets, self.row_of_slot,
                                 self.token_of_row, self.x_perm_q, self.x_scale_perm, self.prob_perm, self.ws, stream)
            abi.moe_dequant_rows(s, self.x_perm_q, self.x_scale_perm, self.x_perm, stream)
        elif self.payload == "nvfp4":
            abi.moe_dispatch_nvfp4(s, xd, self.topk_idx, self.topk_prob, self.expert_offsets, self.row_of_slot,
                                   self.token_of_row, self.x_perm_q4, self.x_bscale_perm, self.x_rscale_perm,
                                   self.prob_perm, self.ws, stream)
            abi.moe_dequant_nvfp4(s, self.x_perm_q4, self.x_bscale_perm, self.x_rscale_perm, self.x_perm, stream)
        else:
            abi.moe_dispatch(s, xd, self.topk_idx, self.topk_prob, self.expert_offsets, self.row_of_slot,
                             self.token_of_row, self.x_perm, self.prob_perm, self.ws, stream)
        if self.gather:
            abi.moe_expert_ffn_gather(s, xd, self.token_of_row, self.expert_offsets, self.w1, self.w2, self.h,
                                      self.act, self.y_perm, self.ws, stream)
        else:
            abi.moe_expert_ffn(s, self.x_perm, self.expert_offsets, self.w1, self.w2, self.h, self.act,
                               self.y_perm, self.ws, stream)
        if self.H:
            abi.moe_combine(s, self.y_perm, self.prob_perm, self.row_of_slot, self.y_lat, stream)
            abi.moe_latent_proj(s, self.D, self.H, self.y_lat, self.w_upp, self.y, self.ws, stream)
        else:
            abi.moe_combine(s, self.y_perm, self.prob_perm, self.row_of_slot, self.y, stream)
        if self.shared_F:
            abi.moe_shared_expert(s, self.shared_F, self.x, self.w_s1, self.w_s2, self.h_s, self.act_s, self.y,
                                  stream)
        return self.y

    def backward(self, stream=None):
        s = self.shape
        dyd = self.dy
        if self.H:
            abi.moe_latent_proj_bwd(s, self.D, self.H, self.dy, self.y_lat, self.w_upp, self.dy_lat, False,
                                    self.dw_upp, self.ws, stream)
            dyd = self.dy_lat
        abi.moe_combine_bwd(s, dyd, self.y_perm, self.prob_perm, self.row_of_slot, self.dy_perm, self.dprob_perm,
                            stream)
        if self.gather:
            xd = self.x_lat if self.H else self.x
            abi.moe_expert_ffn_bwd_gather(s, self.dy_perm, xd, self.token_of_row, self.h, self.act,
                                          self.expert_offsets, self.w1, self.w2, self.dx_perm, self.dw1, self.dw2,
                                          self.ws, stream)
        else:
            abi.moe_expert_ffn_bwd(s, self.dy_perm, self.x_perm, self.h, self.act, self.expert_offsets, self.w1,
                                   self.w2, self.dx_perm, self.dw1, self.dw2, self.ws, stream)
        if self.latent_fused:
            # dispatch backward, dlogits, dw_down, dw_router and dx from one product over [dx_lat | dz]
            abi.moe_latent_route_bwd(s, self.dx_perm, self.dprob_perm, self.row_of_slot, self.x, self.w_down_router,
                                     self.topk_idx, self.topk_prob, self.dx_cat, self.dx, self.dprob, self.dlogits,
                                     self.dw_down, self.dw_router, self.ws, stream)
        elif self.H:
            abi.moe_dispatch_bwd(s, self.dx_perm, self.dprob_perm, self.row_of_slot, self.dx_lat, self.dprob, stream)
            abi.moe_latent_proj_bwd(s, self.H, self.D, self.dx_lat, self.x, self.w_down, self.dx, False,
                                    self.dw_down, self.ws, stream)
        elif self.router == "softmax":
            # one pass: dispatch backward, dlogits and dx += dlogits . w_router
            abi.moe_dispatch_route_bwd(s, self.dx_perm, self.dprob_perm, self.row_of_slot, self.x, self.w_router,
                                       self.topk_idx, self.topk_prob, self.dx, self.dprob, self.dlogits,
                                       self.dw_router, self.ws, stream)
        else:
            abi.moe_dispatch_bwd(s, self.dx_perm, self.dprob_perm, self.row_of_slot, self.dx, self.dprob, stream)
        if self.router == "sigmoid":
            abi.moe_route_sigmoid_bwd(s, self.x, self.w_router, self.logits, self.topk_idx, self.topk_prob,
                                      self.dprob, self.aux_f, self.aux_coef, self.aux_grad, self.dx, self.dw_router,
                                      self.dlogits, self.ws, stream)
        elif self.H and not self.latent_fused:
            abi.moe_route_bwd(s, self.x, self.w_router, self.topk_idx, self.topk_prob, self.dprob, self.dx,
                              self.dw_router, self.dlogits, self.ws, stream)
        if self.shared_F:
            abi.moe_shared_expert_bwd(s, self.shared_F, self.dy, self.x, self.h_s, self.act_s, self.w_s1, self.w_s2,
                                      self.dh_s, self.dx, self.dw_s1, self.dw_s2, stream)
        return self.dx

    def step(self, stream=None):
        self.forward(stream)
        self.backward(stream)

    def capture(self):
        """Record one step (forward + backward) as a CUDA graph.  Every entry
        point only enqueues kernels on the current stream, with buffers and
        workspace allocated up front, so the step is capturable; replay() then
        runs the same launches without per-launch host work.  Run one eager
        step first (it sets up per-kernel attributes)."""
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.step()
        return g

    # ------------------------------------------------------------------
    # Steps on batches in pinned host memory, copies overlapped with compute
    _IO = ("x", "dy", "y", "dx")

    def _bind(self, bufs: dict) -> None:
        for k in self._IO:
            setattr(self, k, bufs[k])

    def prepare_host_pipeline(self, graphs: bool = True) -> None:
        """Allocate a second set of the step's host-facing buffers (x, dy, y,
        dx) and, with ``graphs``, capture one CUDA graph per set (each after one
        eager step).  Called once, before ``run_host``; ``x`` and ``dy`` keep
        the values they hold."""
        first = {k: getattr(self, k) for k in self._IO}
        second = {k: torch.empty_like(v) for k, v in first.items()}
        second["x"].copy_(first["x"])
        second["dy"].copy_(first["dy"])
        self._sets = [first, second]
        self._graphs = None
        if graphs:
            self._graphs = []
            for bufs in self._sets:
                self._bind(bufs)
                self.step()
                self._graphs.append(self.capture())
        self._bind(first)
        self._h2d = torch.cuda.Stream(device=self.x.device)
        self._d2h = torch.cuda.Stream(device=self.x.device)
        torch.cuda.synchronize(self.x.device)

    def run_host(self, batches) -> None:
        """One forward + backward step per batch ``(x, dy, y, dx)`` of pinned
        host tensors: x and dy are the step's inputs, y and dx receive its
        outputs.  Step i + 1's inputs are copied in on one copy stream while
        step i computes, and step i's outputs are copied out on another while
        step i + 1 computes, the two device buffer sets alternating.  Every
        copy is ordered after the work already on the current stream, and the
        current stream waits for the last output copy before this returns
        (asynchronously: synchronise the stream before reading y and dx)."""
        if not hasattr(self, "_sets"):
            raise RuntimeError("call prepare_host_pipeline() first")
        batches = list(batches)
        n = len(batches)
        cs = torch.cuda.current_stream(self.x.device)
        h2d, d2h = self._h2d, self._d2h
        ready = [torch.cuda.Event(), torch.cuda.Event()]     # a set's inputs are on the device
        done = [torch.cuda.Event(), torch.cuda.Event()]      # a set's step finished
        drained = [torch.cuda.Event(), torch.cuda.Event()]   # a set's outputs are on the host
        h2d.wait_stream(cs)

        def load(i):
            b, bufs = i % 2, self._sets[i % 2]
            with torch.cuda.stream(h2d):
                if i >= 2:
                    h2d.wait_event(done[b])                  # step i - 2 no longer reads this set
                bufs["x"].copy_(batches[i][0], non_blocking=True)
                bufs["dy"].copy_(batches[i][1], non_blocking=True)
                ready[b].record(h2d)

        if n:
            load(0)
        for i in range(n):
            b, bufs = i % 2, self._sets[i % 2]
            if i + 1 < n:
                load(i + 1)
            cs.wait_event(ready[b])
            if i >= 2:
                cs.wait_event(drained[b])                    # step i - 2's outputs have left this set
            if self._graphs is not None:
                self._graphs[b].replay()
            else:
                self._bind(bufs)
                self.step()
            done[b].record(cs)
            with torch.cuda.stream(d2h):
                d2h.wait_event(done[b])
                batches[i][2].copy_(bufs["y"], non_blocking=True)
                batches[i][3].copy_(bufs["dx"], non_blocking=True)
                drained[b].record(d2h)
        cs.wait_stream(d2h)
        cs.wait_stream(h2d)
        self._bind(self._sets[0])

    # ------------------------------------------------------------------
    def unpack_w1_like(self, t: torch.Tensor):
        """Split a packed [E, 2F, D] tensor (w1 or dw1) into gate and up [E, F, D]."""
        v = t.view(self.E, self.F // 64, 2, 64, self.D)
        return v[:, :, 0].reshape(self.E, self.F, self.D), v[:, :, 1].reshape(self.E, self.F, self.D)

    def unpack_h(self, h: torch.Tensor):
        """Split a packed [rows, 2F] tensor (h or dH) into its gate and up halves [rows, F]."""
        v = h.view(h.shape[0], self.F // 64, 2, 64)
        return v[:, :, 0].reshape(h.shape[0], self.F), v[:, :, 1].reshape(h.shape[0], self.F)
