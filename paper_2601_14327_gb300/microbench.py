"""Times single entry points of the library on synthetic inputs (CUDA events).

    python -m paper_2601_14327_gb300.microbench route --T 16384 --d 4096 --E 64 --k 8
    python -m paper_2601_14327_gb300.microbench permute --T 16384 --d 4096 --E 64 --k 8

Holds only what the chosen call needs on the device, so a profiler capture of one
kernel stays small. Prints one JSON line per call with the mean time per call.
"""
from __future__ import annotations

import argparse
import json
import math

import torch

from . import _lib as L
from . import synth


def _time(fn, iters, warmup):
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(iters):
        fn()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / iters


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("call", choices=["route", "permute", "combine", "permute_bwd",
                                     "permute_bwd_norouter", "route_bwd"])
    ap.add_argument("--T", type=int, default=16384)
    ap.add_argument("--d", type=int, default=4096)
    ap.add_argument("--E", type=int, default=64)
    ap.add_argument("--k", type=int, default=8)
    ap.add_argument("--iters", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    a = ap.parse_args()
    dev = "cuda"
    T, d, E, k = a.T, a.d, a.E, a.k
    gen = torch.Generator(device=dev)
    gen.manual_seed(7)
    x = torch.randn(T, d, generator=gen, device=dev).to(torch.bfloat16)
    w = torch.randn(d, E, generator=gen, device=dev) / math.sqrt(d)
    bias = synth.gate_bias(E, "zipf", 1.2, gen, dev)
    ws_bytes = L.moe_workspace_size(T, d, E, k, 128)
    ws = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=dev)
    idx = torch.empty(T, k, dtype=torch.int32, device=dev)
    gate = torch.empty(T, k, dtype=torch.float32, device=dev)
    counts = torch.empty(E, dtype=torch.int32, device=dev)

    def route():
        L.moe_route(x, w, bias, None, T, d, E, k, None, None, idx, gate, counts, ws, ws_bytes)

    out = {"call": a.call, "T": T, "d": d, "E": E, "k": k}
    if a.call == "route":
        ms = _time(route, a.iters, a.warmup)
        nbytes = 2 * T * d + 4 * d * E + 8 * T * k  # x, router weight, indices and gates
        out.update(ms=round(ms, 4), gbs=round(nbytes / (ms / 1e3) / 1e9, 1))
    else:
        route()
        R = L.moe_perm_rows_max(T, k, E)
        goff = torch.empty(E + 1, dtype=torch.int32, device=dev)
        gcnt = torch.empty(E, dtype=torch.int32, device=dev)
        row = torch.empty(T, k, dtype=torch.int32, device=dev)
        xp = torch.empty(R, d, dtype=torch.bfloat16, device=dev)

        def permute():
            L.moe_permute(x, idx, None, T, d, E, k, R, goff, gcnt, row, xp, ws, ws_bytes)

        if a.call == "permute":
            ms = _time(permute, a.iters, a.warmup)
            nbytes = 2 * T * d + 2 * T * k * d
        elif a.call.startswith("permute_bwd"):
            permute()
            dl = torch.randn(T, k, generator=gen, device=dev) * 0.1
            dx = torch.empty(T, d, dtype=torch.bfloat16, device=dev)
            router = a.call == "permute_bwd"
            ms = _time(lambda: L.moe_permute_bwd(xp, row, idx, dl if router else None,
                                                 w if router else None, T, d, E, k, dx, ws,
                                                 ws_bytes), a.iters, a.warmup)
            nbytes = 2 * T * k * d + 2 * T * d
        elif a.call == "route_bwd":
            dg = torch.randn(T, k, generator=gen, device=dev)
            dl = torch.empty(T, k, dtype=torch.float32, device=dev)
            dw = torch.empty(d, E, dtype=torch.float32, device=dev)
            ms = _time(lambda: L.moe_route_bwd(x, idx, gate, dg, T, d, E, k, dl, dw, ws,
                                               ws_bytes), a.iters, a.warmup)
            nbytes = 2 * T * d
        else:
            permute()
            y = torch.empty(T, d, dtype=torch.bfloat16, device=dev)
            ms = _time(lambda: L.moe_unpermute_combine(xp, row, gate, T, d, k, y), a.iters,
                       a.warmup)
            nbytes = 2 * T * k * d + 2 * T * d
        out.update(ms=round(ms, 4), gbs=round(nbytes / (ms / 1e3) / 1e9, 1))
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
