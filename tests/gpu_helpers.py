"""Shared helpers of the GPU parity tests: run the CUDA path through the C ABI
and the oracle on the same seeded inputs, compare with the stated bars."""
import numpy as np
import torch

from oracle import moe_oracle as O
from paper_2601_14327_gb300 import _lib as L
from paper_2601_14327_gb300 import layer
from paper_2601_14327_gb300 import synth

# max|gpu - oracle| / max|oracle| per tensor, for bf16 data with fp32 accumulation
REL_TOL = 2e-2


def rel_err(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.max(np.abs(ref))
    if den == 0:
        return float(np.max(np.abs(got)))
    return float(np.max(np.abs(got - ref)) / den)


def assert_close(name, got, ref, tol=REL_TOL):
    e = rel_err(got, ref)
    assert e <= tol, f"{name}: max-abs-err/max|ref| = {e:.3e} > {tol}"
    return e


def to_np(t):
    return t.detach().float().cpu().numpy() if t.dtype in (torch.bfloat16, torch.float16) \
        else t.detach().cpu().numpy()


def case_inputs(T, d, E, k, F, bias="zipf", zipf_s=1.2, seed=0, weight_std=0.02):
    """Seeded inputs on the CPU (both sides use the same bytes)."""
    return synth.make_layer_inputs(T, d, E, k, F, bias=bias, zipf_s=zipf_s, seed=seed,
                                   backward=True, weight_std=weight_std)


def oracle_inputs(inp):
    return {n: (v.double().numpy() if v.is_floating_point() else v.numpy()) for n, v in inp.items()}


def run_gpu_layer(inp, E, k, mask=None, logits_in=None, backward=True, fused_combine=False):
    """Full step through the C ABI; returns the buffers object."""
    T, d = inp["x"].shape
    F = inp["w_down"].shape[2]
    dev = "cuda"
    g = {n: v.to(dev) for n, v in inp.items()}
    b = layer.MoELayerBuffers(layer.LayerShape(T, d, E, k, F), dev, backward=backward,
                              fused_combine=fused_combine)
    m = None if mask is None else torch.as_tensor(mask, dtype=torch.uint8).to(dev)
    li = None if logits_in is None else torch.as_tensor(logits_in, dtype=torch.float32).to(dev)
    layer.forward(b, g["x"], g["w_router"], g["bias"], g["w_gate_up"], g["w_down"], m, li,
                  keep_logits=True)
    if backward:
        layer.backward(b, g["dy"], g["w_router"], g["w_gate_up"], g["w_down"])
    torch.cuda.synchronize()
    return b


def unblock_ab(ab_flat, F):
    """[rows, 2F] matrix from the 32-row blocked layout of the saved pre-activations:
    element (r, c) sits at ((r/32)*(2F/8) + c/8)*256 + (r%32)*8 + c%8."""
    a = np.asarray(ab_flat).reshape(-1)
    nblk = a.size // (32 * 2 * F)
    a = a[:nblk * 32 * 2 * F].reshape(nblk, 2 * F // 8, 32, 8)
    return a.transpose(0, 2, 1, 3).reshape(nblk * 32, 2 * F)


def topk_margin(z32, k):
    """Smallest gap among the k+1 largest logits per token: above the rounding of
    the logits, the ordered top-k is unique (inf gaps past the last expert)."""
    z = np.sort(np.asarray(z32, np.float64), axis=1)[:, ::-1][:, :k + 1]
    if z.shape[1] <= k:
        z = np.concatenate([z, np.full((z.shape[0], 1), -np.inf)], axis=1)
    return (z[:, :-1] - z[:, 1:]).min(axis=1)


def dx_perm_ref(ref, w_router, T, k):
    """The oracle's per-assignment rows of dx_perm [T*k, d]: dX plus the router's term
    d_logits[t,j] * W_r[:, e_j], which the dX GEMM's epilogue adds (moe_permute_bwd then
    sums the rows without a router term)."""
    wr = np.asarray(w_router, np.float64)
    rows = ref["dX"] + ref["d_logits"][:, :, None] * wr.T[ref["topk_idx"]]
    return rows.reshape(T * k, -1)
