"""One MoE expert layer step through the C ABI.

PyTorch only allocates device memory and provides the stream; every step of
the layer runs in the library's kernels (see _lib.py for the entry points).
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import torch

from . import _lib as L


@dataclasses.dataclass
class LayerShape:
    T: int
    d: int
    E: int
    k: int
    F: int

    @property
    def rows_cap(self) -> int:
        return L.moe_perm_rows_max(self.T, self.k, self.E)


class MoELayerBuffers:
    """Device buffers of one layer step (activations, grouped layout, grads).

    gather=False (default): moe_permute writes X_perm and the GEMMs read it with tile
    loads. gather=True: the grouped operand is read from x through token_of_row by the
    GEMMs' 4-row TMA gathers (moe_permute_map and the *_gather calls), so X_perm is not
    allocated; the results are identical, but on GB300 the gathers make the two GEMMs
    that read X_perm about 3.3x slower (32 gathers of 4 x 128 bytes per 128-row k-block
    against one tile load), far more than the separate gather pass costs.

    fused_combine=True: the combine runs in the down GEMM's epilogue
    (moe_grouped_ffn_fwd_combine, fp32 atomics into y_acc; the last bits of y can
    change from run to run); O is then stored only when a backward follows."""

    def __init__(self, shape: LayerShape, device="cuda", backward: bool = True,
                 gather: bool = False, fused_combine: bool = False):
        s = shape
        self.shape = s
        self.gather = gather
        self.fused_combine = fused_combine
        if fused_combine and gather:
            raise ValueError("fused_combine reads X_perm: use it with gather=False")
        self.x = None  # the forward's input, kept for the backward
        R = s.rows_cap
        dev = torch.device(device)
        bf16, f32, i32 = torch.bfloat16, torch.float32, torch.int32
        self.ws_bytes = max(L.moe_workspace_size(s.T, s.d, s.E, s.k, s.F), 256)
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=dev)
        self.logits = torch.empty(s.T, s.E, dtype=f32, device=dev)
        self.topk_idx = torch.empty(s.T, s.k, dtype=i32, device=dev)
        self.topk_gate = torch.empty(s.T, s.k, dtype=f32, device=dev)
        self.counts = torch.empty(s.E, dtype=i32, device=dev)
        self.group_offsets = torch.empty(s.E + 1, dtype=i32, device=dev)
        self.group_counts = torch.empty(s.E, dtype=i32, device=dev)
        self.row_of_assignment = torch.empty(s.T, s.k, dtype=i32, device=dev)
        if gather:
            self.token_of_row = torch.empty(R, dtype=i32, device=dev)
            self.x_perm = None
        else:
            self.token_of_row = None
            self.x_perm = torch.empty(R, s.d, dtype=bf16, device=dev)
        self.ab = torch.empty(R, 2 * s.F, dtype=bf16, device=dev)
        self.h = torch.empty(R, s.F, dtype=bf16, device=dev)
        self.out_perm = (torch.empty(R, s.d, dtype=bf16, device=dev)
                         if backward or not fused_combine else None)
        self.y_acc = torch.empty(s.T, s.d, dtype=f32, device=dev) if fused_combine else None
        self.y = torch.empty(s.T, s.d, dtype=bf16, device=dev)
        if backward:
            self.d_out_perm = torch.empty(R, s.d, dtype=bf16, device=dev)
            self.d_gate = torch.empty(s.T, s.k, dtype=f32, device=dev)
            self.d_ab = torch.empty(R, 2 * s.F, dtype=bf16, device=dev)
            self.dx_perm = torch.empty(R, s.d, dtype=bf16, device=dev)
            self.dw_gate_up = torch.empty(s.E, 2 * s.F, s.d, dtype=bf16, device=dev)
            self.dw_down = torch.empty(s.E, s.d, s.F, dtype=bf16, device=dev)
            self.d_logits = torch.empty(s.T, s.k, dtype=f32, device=dev)
            self.dw_router = torch.empty(s.d, s.E, dtype=f32, device=dev)
            self.dx = torch.empty(s.T, s.d, dtype=bf16, device=dev)
            # second stream: the router backward and the unpermute-sum run beside
            # the grouped GEMMs (whose CTAs leave registers and threads free)
            self.side = torch.cuda.Stream(device=dev) if dev.type == "cuda" else None


def route(b: MoELayerBuffers, x, w_router, bias, active_mask=None, logits_in=None,
          keep_logits: bool = False, stream=None):
    s = b.shape
    L.moe_route(x, w_router, bias, active_mask, s.T, s.d, s.E, s.k, logits_in,
                b.logits if keep_logits else None, b.topk_idx, b.topk_gate, b.counts, b.ws,
                b.ws_bytes, stream)


def forward(b: MoELayerBuffers, x, w_router, bias, w_gate_up, w_down, active_mask=None,
            logits_in=None, keep_logits: bool = False, stream=None):
    """route -> permute -> grouped SwiGLU FFN -> combine (in the down GEMM's epilogue
    when b.fused_combine). Returns b.y."""
    s = b.shape
    R = s.rows_cap
    route(b, x, w_router, bias, active_mask, logits_in, keep_logits, stream)
    b.x = x
    if b.gather:
        L.moe_permute_map(b.topk_idx, b.counts, s.T, s.E, s.k, R, b.group_offsets,
                          b.group_counts, b.row_of_assignment, b.token_of_row, b.ws, b.ws_bytes,
                          stream)
        L.moe_grouped_ffn_fwd_gather(x, b.token_of_row, s.T, b.group_offsets, s.E, s.d, s.F, R,
                                     w_gate_up, w_down, b.ab, b.h, b.out_perm, b.ws, b.ws_bytes,
                                     stream)
    else:
        L.moe_permute(x, b.topk_idx, b.counts, s.T, s.d, s.E, s.k, R, b.group_offsets,
                      b.group_counts, b.row_of_assignment, b.x_perm, b.ws, b.ws_bytes, stream)
        if b.fused_combine:
            L.moe_grouped_ffn_fwd_combine(b.x_perm, b.group_offsets, s.E, s.d, s.F, R, w_gate_up,
                                          w_down, b.row_of_assignment, b.topk_gate, s.T, s.k,
                                          b.ab, b.h, b.out_perm, b.y_acc, b.y, b.ws, b.ws_bytes,
                                          stream)
            return b.y
        L.moe_grouped_ffn_fwd(b.x_perm, b.group_offsets, s.E, s.d, s.F, R, w_gate_up, w_down,
                              b.ab, b.h, b.out_perm, b.ws, b.ws_bytes, stream)
    L.moe_unpermute_combine(b.out_perm, b.row_of_assignment, b.topk_gate, s.T, s.d, s.k, b.y,
                            stream)
    return b.y


def backward(b: MoELayerBuffers, dy, w_router, w_gate_up, w_down, stream=None,
             overlap: bool = False, active_mask=None):
    """combine bwd -> grouped FFN dgrad (with the gate gradient and the router's term of dx)
    -> router bwd -> permute bwd -> grouped FFN wgrad.

    active_mask: the LAEP mask the forward routed with (None: all experts live). Pruned
    experts' weight gradients are not written (their buffers keep what they held); live
    experts without tokens get exact zeros.

    With overlap, the router backward and the unpermute-sum (after the dgrad GEMMs) run on
    a second stream while the main stream computes the weight gradients; the main stream
    waits for them at the end. The
    default is one stream: on GB300 at T=65536, d_model=7168 the step is power-capped,
    and running those memory-bound kernels beside the GEMMs slowed the GEMMs by more
    than it hid (96.1-96.7 against 97.0-97.3 ms per step).
    Returns (dx, dw_gate_up, dw_down, dw_router)."""
    s = b.shape
    R = s.rows_cap
    main = torch.cuda.current_stream() if stream is None else stream
    side = b.side if overlap else main
    # d_out_perm = g * dy; the gate gradient comes from the dH GEMM (below), so the combine
    # backward does not read out_perm
    L.moe_unpermute_combine_bwd(dy, None, b.row_of_assignment, b.topk_gate,
                                b.group_offsets, b.group_counts, s.T, s.d, s.E, s.k,
                                b.d_out_perm, None, main)
    # dH (+ the gate gradient into b.d_gate), dX with the router's term of dx added to the
    # grouped rows in its epilogue
    L.moe_grouped_ffn_bwd_dgrad(b.d_out_perm, b.ab, b.group_offsets, s.E, s.d, s.F, R,
                                w_gate_up, w_down, b.topk_gate, None, b.row_of_assignment,
                                w_router, s.T, s.k, b.d_gate, b.d_ab, b.dx_perm, b.ws,
                                b.ws_bytes, main)
    if overlap:
        ev = torch.cuda.Event()
        ev.record(main)
        side.wait_event(ev)
    L.moe_route_bwd(b.x, b.topk_idx, b.topk_gate, b.d_gate, s.T, s.d, s.E, s.k, b.d_logits,
                    b.dw_router, b.ws, b.ws_bytes, side)
    L.moe_permute_bwd(b.dx_perm, b.row_of_assignment, b.topk_idx, None, None, s.T, s.d, s.E,
                      s.k, b.dx, b.ws, b.ws_bytes, side)
    if b.gather:
        L.moe_grouped_ffn_bwd_wgrad_gather(b.d_out_perm, b.x, b.token_of_row, s.T, b.h, b.d_ab,
                                           b.group_offsets, active_mask, s.E, s.d, s.F, R,
                                           b.dw_gate_up, b.dw_down, b.ws, b.ws_bytes, main)
    else:
        L.moe_grouped_ffn_bwd_wgrad(b.d_out_perm, b.x_perm, b.h, b.d_ab, b.group_offsets,
                                    active_mask, s.E, s.d, s.F, R, b.dw_gate_up, b.dw_down, b.ws,
                                    b.ws_bytes, main)
    if overlap:
        ev = torch.cuda.Event()
        ev.record(side)
        main.wait_event(ev)
    return b.dx, b.dw_gate_up, b.dw_down, b.dw_router


def prune_from_counts(counts_host, S: int, k: int, *, prune_count: int = -1,
                      alpha: float = 0.0, beta: float = 0.0):
    """LAEP decision on a host histogram; returns (mask uint8 tensor on CPU, n_pruned)."""
    mask, n = L.laep_prune_mask([int(c) for c in counts_host], S, k, alpha, beta, prune_count)
    return torch.tensor(mask, dtype=torch.uint8), n
