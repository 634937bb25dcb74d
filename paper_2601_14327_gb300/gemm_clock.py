"""Grouped GEMMs against cuBLAS per SM clock, at the same power draw.

Each pair of grouped GEMMs of one fwd+bwd layer step (forward gate/up + down, dgrad dH + dX,
wgrad dW_down + dW_gate_up) runs back to back for a few seconds on the LAEP-pruned workload
(T=16384, d_model=4096, 48 of 64 experts live, top-8, d_ff=2048), and so does a cuBLAS bf16
GEMM of 8192^3, while nvidia-smi samples the SM clock and the power draw. On a power-capped
GPU the clock follows the load, so TFLOP/s per MHz is the figure that compares kernels.

    python -m paper_2601_14327_gb300.gemm_clock [--seconds 3]
"""
import argparse
import json
import statistics
import subprocess
import threading
import time

import torch

from . import _lib as L
from . import layer, synth


def _sampled(fn, seconds):
    proc = subprocess.Popen(["nvidia-smi", "-i", str(torch.cuda.current_device()),
                             "--query-gpu=clocks.sm,power.draw", "--format=csv,noheader,nounits",
                             "-lms", "50"], stdout=subprocess.PIPE, text=True)
    lines = []
    th = threading.Thread(target=lambda: [lines.append((time.monotonic(), l)) for l in proc.stdout],
                          daemon=True)
    th.start()
    time.sleep(0.3)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n, t0 = 0, time.monotonic()
    a.record()
    while time.monotonic() - t0 < seconds:
        for _ in range(10):
            fn()
        n += 10
        torch.cuda.synchronize()
    b.record()
    torch.cuda.synchronize()
    t1 = time.monotonic()
    proc.terminate()
    th.join(timeout=2)
    # samples from the second half of the loop (the clock has settled)
    vals = [tuple(float(v) for v in l.split(",")) for t, l in lines
            if (t0 + t1) / 2 <= t <= t1 and l.count(",") == 1]
    mhz = statistics.median(v[0] for v in vals) if vals else float("nan")
    watts = statistics.median(v[1] for v in vals) if vals else float("nan")
    return a.elapsed_time(b) / n, mhz, watts


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--seconds", type=float, default=3.0)
    args = ap.parse_args()
    dev = "cuda"
    c = synth.CONFIGS[2]
    inp = synth.make_config_inputs(2, device=dev)
    T, d, E, k, F = c.T, c.d, c.E, c.k, c.F
    shape = layer.LayerShape(T, d, E, k, F)
    b = layer.MoELayerBuffers(shape, dev)
    layer.route(b, inp["x"], inp["w_router"], inp["bias"])
    mask, _ = layer.prune_from_counts(b.counts.cpu().tolist(), T, k, prune_count=c.prune_lowest)
    mask = mask.to(dev)
    layer.forward(b, inp["x"], inp["w_router"], inp["bias"], inp["w_gate_up"], inp["w_down"], mask)
    layer.backward(b, inp["dy"], inp["w_router"], inp["w_gate_up"], inp["w_down"])
    torch.cuda.synchronize()
    R = shape.rows_cap
    A = T * k
    two = 2.0 * A * d * F  # FLOPs of a d x F contraction over the real assignments
    runs = {
        "forward (gate/up + down)": (lambda: L.moe_grouped_ffn_fwd(
            b.x_perm, b.group_offsets, E, d, F, R, inp["w_gate_up"], inp["w_down"], b.ab, b.h,
            b.out_perm, b.ws, b.ws_bytes), 3 * two),
        "dgrad (dH + dX)": (lambda: L.moe_grouped_ffn_bwd_dgrad(
            b.d_out_perm, b.ab, b.group_offsets, E, d, F, R, inp["w_gate_up"], inp["w_down"],
            b.d_ab, b.dx_perm), 3 * two),
        "wgrad (dW_down + dW_gate_up)": (lambda: L.moe_grouped_ffn_bwd_wgrad(
            b.d_out_perm, b.x_perm, b.h, b.d_ab, b.group_offsets, E, d, F, R, b.dw_gate_up,
            b.dw_down), 3 * two),
    }
    n = 8192
    ma = torch.randn(n, n, device=dev, dtype=torch.bfloat16)
    mb = torch.randn(n, n, device=dev, dtype=torch.bfloat16)
    mc = torch.empty(n, n, device=dev, dtype=torch.bfloat16)
    torch.matmul(ma, mb, out=mc)  # library warm-up outside the sampled loop
    runs["cuBLAS bf16 8192^3"] = (lambda: torch.matmul(ma, mb, out=mc), 2.0 * n ** 3)
    for name, (fn, flops) in runs.items():
        fn()
        ms, mhz, watts = _sampled(fn, args.seconds)
        tf = flops / (ms / 1e3) / 1e12
        print(json.dumps({"loop": name, "ms": round(ms, 4), "tflops": round(tf, 1),
                          "sm_mhz": mhz, "watts": watts,
                          "gflops_per_mhz": round(tf / mhz * 1e3, 1)}), flush=True)


if __name__ == "__main__":
    main()
