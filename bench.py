#!/usr/bin/env python
"""Benchmark of one MoE expert-layer training step (forward + backward) on GB300.

A step is one pass of the whole hot path over one batch: route (fp32 logits,
top-k over the experts LAEP kept, gates, histogram) -> permute -> grouped
SwiGLU FFN forward -> combine -> combine backward -> grouped FFN backward
(dgrad + wgrad) -> router backward -> permute backward. The LAEP pruning
decision itself runs once before the timed steps, as in the paper (one prune
once the loads are stable), on the histogram of a first routing pass.

Default workload: the largest one, T=65536 tokens, d_model=7168, 256 experts of
which the 85 least-loaded are pruned and removed from the weights (171 kept),
top-8, d_ff=2048, Zipf(1.0) gate bias, bf16 data with an fp32 router, seeded
synthetic inputs; its line also times the unpruned layer (all 256 experts) for
the pruned-vs-unpruned ratio. `--config N` selects another workload.

Prints ONE JSON line (rank 0). `--impl reference` times the CPU oracle on a
bounded token sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

NCPU = os.cpu_count() or 1
for _v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, str(NCPU))

import numpy as np  # noqa: E402
import torch  # noqa: E402

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2601_14327_gb300 import _lib as L  # noqa: E402
from paper_2601_14327_gb300 import layer, synth  # noqa: E402

METRIC = "MoE layer fwd+bwd tokens/s; grouped-GEMM TFLOPS as % of GB300 bf16 peak"
GEMMS = ["gemm_gate_up", "gemm_down", "gemm_dgrad_down", "gemm_dgrad_gate_up",
         "gemm_wgrad_down", "gemm_wgrad_gate_up"]


def committed_traffic(workload, kernel):
    """DRAM bytes per launch of `kernel` at `workload` from the committed ncu record
    (profiles/dram_traffic_<workload>.json), or None when the sources that kernel is built
    from changed since the counters were taken (or no record exists)."""
    path = os.path.join(ROOT, "profiles", f"dram_traffic_{workload}.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        rec = json.load(f).get("kernels", {}).get(kernel)
    if rec is None:
        return None
    return rec["bytes_per_launch"] if sources_digest(rec["sources"]) == rec["sources_sha256"] else None


def sources_digest(sources):
    """SHA-256 over the code of the given source files with comments removed (string and
    character literals kept), so that a comment edit does not invalidate a capture."""
    import hashlib
    import re
    token = re.compile(r'//[^\n]*|/\*.*?\*/|"(?:\\.|[^"\\\n])*"|\'(?:\\.|[^\'\\\n])*\'',
                       re.S)
    h = hashlib.sha256()
    for src in sources:
        with open(os.path.join(ROOT, src), encoding="utf-8") as f:
            text = f.read()
        code = token.sub(lambda m: m.group(0) if m.group(0)[0] in "\"'" else " ", text)
        h.update(re.sub(r"\s+", " ", code).encode())
    return h.hexdigest()


HBM_NOMINAL_GBS = 8000.0  # GB300 HBM3e, nominal (~8 TB/s); the measured copy peak is below it
BF16_NOMINAL_TFLOPS = 2250.0  # GB300 dense bf16 tensor peak, nominal (no 2:4 sparsity)
SUSTAINED_REGION_S = 1.0  # timed regions at least this long use the sustained bf16 peak


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        clk = (p.get("clocks_under_load") or {}).get("sm_mhz_median")
        return {"hbm_gbs": p["hbm_gbs"], "bf16_tflops": p["bf16_tflops"],
                "bf16_tflops_sustained": p.get("bf16_tflops_sustained", p["bf16_tflops"]),
                "sustained_sm_mhz": clk, "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "sustained_sm_mhz": None, "source": "fallback"}


def per_clock_frac(tflops, sm_mhz, peaks):
    """TFLOP/s per MHz of SM clock against the sustained cuBLAS run's TFLOP/s per MHz at its
    own median clock: the fraction of the reference's work per clock, which clock
    differences between the two measurements do not inflate (None without both clocks)."""
    ref_mhz = peaks.get("sustained_sm_mhz")
    if not sm_mhz or not ref_mhz:
        return None
    return round((tflops / sm_mhz) / (peaks["bf16_tflops_sustained"] / ref_mhz), 4)


def tensor_peak(peaks, region_s):
    """bf16 denominator for kernels timed inside a region of `region_s` seconds, and its
    name. A region of a second or more runs at the clock the power cap settles at, so it is
    compared with the sustained cuBLAS rate (a seconds-long loop under the cap); a shorter
    region with the burst rate (cuBLAS timed alone)."""
    if region_s >= SUSTAINED_REGION_S:
        return (peaks["bf16_tflops_sustained"],
                f"bf16_tflops_sustained of MEASURED_PEAKS.json ({peaks['source']}): timed region "
                f"{region_s:.2f} s >= {SUSTAINED_REGION_S:g} s")
    return (peaks["bf16_tflops"],
            f"bf16_tflops (burst) of MEASURED_PEAKS.json ({peaks['source']}): timed region "
            f"{region_s:.2f} s < {SUSTAINED_REGION_S:g} s")


# --------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples during the timed region (median SM clock under load). Samples
    are kept with their arrival time; those between mark_start() and mark_end() (the
    timed region) are the ones reported, when there are any."""

    Q = ("clocks.sm,clocks.max.sm,utilization.gpu,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []
        self.t0 = self.t1 = None

    def mark_start(self):
        self.t0 = time.monotonic()

    def mark_end(self):
        self.t1 = time.monotonic()

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.monotonic(), line.strip()))

    def wait_first(self, timeout=5.0):
        """Blocks until the sampler has delivered a line (or `timeout` seconds)."""
        t_end = time.monotonic() + timeout
        while self.proc is not None and not self.lines and time.monotonic() < t_end:
            time.sleep(0.02)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, mx, reasons, loaded = [], None, set(), []
        lines = self.lines
        if self.t0 is not None and self.t1 is not None:
            inside = [(t, ln) for t, ln in lines if self.t0 <= t <= self.t1]
            lines = inside or lines
        for _, ln in lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 8:
                continue
            try:
                s, m, u = float(f[0]), float(f[1]), float(f[2])
            except ValueError:
                continue
            sm.append(s)
            mx = m
            if u >= 50:
                loaded.append(s)
            for n, v in zip(names, f[4:8]):
                if v.lower() in ("active", "1"):
                    reasons.add(n)
        use = loaded or sm
        return {"sm_mhz": statistics.median(use) if use else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm), "samples_under_load": len(loaded)}


# ------------------------------------------------------------------- workload

class Workload:
    """Inputs, the one-time LAEP prune, and the buffers of one layer step."""

    def __init__(self, cfg_id: int, device: str, compact_override=None, tokens=None,
                 experts=None, no_prune=False, bias=None, gather=False, overlap=False,
                 backward=None, fused_combine=False):
        c = synth.CONFIGS[cfg_id]
        if tokens or experts or no_prune or bias:  # a variant of the workload (profiling)
            import dataclasses
            c = dataclasses.replace(c, name=c.name + f"_variant_T{tokens or c.T}_E{experts or c.E}"
                                    f"_{bias or c.bias}", T=tokens or c.T, E=experts or c.E,
                                    bias=bias or c.bias,
                                    prune_lowest=0 if no_prune else c.prune_lowest)
        self.cfg = c
        self.cfg_id = cfg_id
        self.device = device
        inp = synth.make_layer_inputs(c.T, c.d, c.E, c.k, c.F, bias=c.bias, zipf_s=c.zipf_s,
                                      seed=synth.seed_for(cfg_id), device=device)
        self.inp = inp
        T, d, E, k, F = c.T, c.d, c.E, c.k, c.F
        self.mask = None
        self.keep = None
        self.counts0 = None
        self.n_pruned = 0
        compact = c.compact if compact_override is None else compact_override
        if c.prune_lowest:
            # first routing pass over all experts -> histogram -> LAEP decision
            b0 = layer.MoELayerBuffers(layer.LayerShape(T, d, E, k, F), device, backward=False)
            layer.route(b0, inp["x"], inp["w_router"], inp["bias"])
            counts = b0.counts.cpu().tolist()
            self.counts0 = counts
            del b0
            mask, self.n_pruned = layer.prune_from_counts(counts, T, k,
                                                          prune_count=c.prune_lowest)
            if compact:
                keep = torch.nonzero(mask).flatten().to(device)
                self.keep = keep.cpu().numpy()
                inp["w_router"] = inp["w_router"].index_select(1, keep).contiguous()
                inp["bias"] = inp["bias"].index_select(0, keep).contiguous()
                inp["w_gate_up"] = inp["w_gate_up"].index_select(0, keep).contiguous()
                inp["w_down"] = inp["w_down"].index_select(0, keep).contiguous()
                E = int(keep.numel())
            else:
                self.mask = mask.to(device)
        self.shape = layer.LayerShape(T, d, E, k, F)
        self.E_live = E - (self.n_pruned if self.mask is not None else 0)
        # the forward-only workloads time the forward pass (backward=True forces both)
        self.backward = c.backward if backward is None else bool(backward)
        self.bufs = layer.MoELayerBuffers(self.shape, device, backward=self.backward,
                                          gather=gather, fused_combine=fused_combine)

        self.graph = None
        self.overlap = overlap

    def step(self, x=None, dy=None):
        if self.graph is not None and x is None and dy is None:
            self.graph.replay()
            return
        self.eager_step(x, dy)

    def eager_step(self, x=None, dy=None):
        i, b = self.inp, self.bufs
        layer.forward(b, i["x"] if x is None else x, i["w_router"], i["bias"], i["w_gate_up"],
                      i["w_down"], self.mask)
        if self.backward:
            layer.backward(b, i["dy"] if dy is None else dy, i["w_router"], i["w_gate_up"],
                           i["w_down"], overlap=self.overlap, active_mask=self.mask)

    def make_graph(self, x=None, dy=None):
        """A CUDA graph of one whole step (both streams) on inputs x, dy. The library's calls
        allocate nothing and never synchronize, so they capture as they are; what they set up
        once (tensor-map encoder, occupancy, attributes) ran in eager warm-up steps before."""
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.eager_step(x, dy)
        torch.cuda.synchronize()
        return g

    def capture(self):
        """Later steps without explicit inputs replay a graph of the step."""
        self.graph = self.make_graph()

    def live_counts(self):
        """Rows per live expert (pruned experts of a mask excluded: they get no tile and
        no weight-gradient write)."""
        counts = self.bufs.counts.cpu().tolist()
        if self.mask is None:
            return counts
        m = self.mask.cpu().tolist()
        return [c for c, keep in zip(counts, m) if keep]

    def gemm_flops(self):
        """Algorithmic FLOPs per GEMM call (real assignments only; one call per step)."""
        s = self.shape
        A = s.T * s.k
        two = 2.0 * A * s.d * s.F
        return {"gemm_gate_up": 2 * two, "gemm_down": two, "gemm_dgrad_down": two,
                "gemm_dgrad_gate_up": 2 * two, "gemm_wgrad_down": two,
                "gemm_wgrad_gate_up": 2 * two}


# ------------------------------------------------------------------ the arms

def dist_setup(n_gpus):
    """One process per GPU (torchrun sets RANK/LOCAL_RANK/WORLD_SIZE). Each rank runs
    an independent replica of the layer step: the path has no exchange, so the only
    collectives are the barrier and the max over ranks of the timed region."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
            dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        else:
            dist.init_process_group("gloo")
    elif torch.cuda.is_available():
        torch.cuda.set_device(0)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world):
    """Largest value of x over the ranks (the slowest replica sets the job time)."""
    if world > 1:
        import torch.distributed as dist
        dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
        t = torch.tensor([x], dtype=torch.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())
    return x


def replica_throughput(world, tokens_per_rank, steps, ms_max):
    """Whole-job tokens/s of `world` replicas, timed by the slowest one."""
    return world * tokens_per_rank * steps / (ms_max / 1e3)


def oracle_sample(h, k, backward=True):
    """Runs the CPU oracle's whole layer on a sample prepared by sample_inputs (forward, and
    backward unless the workload is forward-only); returns the seconds it took."""
    from oracle import moe_oracle as O
    t0 = time.perf_counter()
    O.moe_layer(h["x"], h["w_router"], h["bias"], h["mask"], k, h["w_gate_up"], h["w_down"],
                dy=h["dy"] if backward else None)
    return time.perf_counter() - t0


def sample_inputs(inp, mask, k, n_tok):
    """float32 host inputs of a bounded oracle sample: the first n_tok tokens, and of the
    experts only those the sample's tokens are routed to (the router's columns, bias and
    expert weights of that subset, in expert order). Every token's k selected experts are in
    the subset and the order of expert ids is kept, so the top-k, the gates and every output
    and gradient of these tokens are the full layer's; the weights of the experts no sampled
    token reaches (up to 22.5 GB at T=65536, d=7168, 256 experts) stay on the device.
    Returns (inputs, number of experts in the subset)."""
    from oracle import moe_oracle as O
    x = inp["x"][:n_tok].float().cpu().numpy()
    wr = inp["w_router"].float().cpu().numpy()
    b = inp["bias"].float().cpu().numpy()
    m = None if mask is None else mask.cpu().numpy()
    idx, _ = O.route_topk(O.router_logits(x, wr, b, m), k)
    used = np.unique(idx)
    sel = torch.as_tensor(used, dtype=torch.long, device=inp["w_gate_up"].device)
    out = {"x": x, "w_router": np.ascontiguousarray(wr[:, used]), "bias": b[used],
           "mask": None,  # the subset holds only experts tokens were routed to: all live
           "w_gate_up": inp["w_gate_up"].index_select(0, sel).float().cpu().numpy(),
           "w_down": inp["w_down"].index_select(0, sel).float().cpu().numpy()}
    if "dy" in inp:
        out["dy"] = inp["dy"][:n_tok].float().cpu().numpy()
    return out, int(used.size)


# tokens of the oracle sample per workload: the CPU baseline of the main arm (10-30 s of host
# time on 16 cores), and one step of the reference arm at 30 steps (fewer at more steps)
CPU_TOKENS = {0: 512, 1: 1024, 2: 4096, 3: 1024, 4: 16}
REF_TOKENS_30 = {0: 512, 1: 256, 2: 64, 3: 32, 4: 3}


def timed_steps(wl, steps, world, local, per_kernel_timing=True, flush=None):
    """K timed steps between barrier+synchronize; returns (max-over-ranks ms, per-kernel
    CUDA-event table, clock samples). With `flush` (a buffer larger than L2) the buffer is
    rewritten before every step and only the steps are timed (an event pair per step)."""
    stream = torch.cuda.current_stream()
    clocks = ClockSampler(local)
    L.moe_timing_enable(per_kernel_timing)
    L.moe_timing_read(reset=True)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps if flush is not None else 1)]
    clocks.start()
    clocks.wait_first()  # the sampler is running before the timed region opens
    barrier(world)
    torch.cuda.synchronize()
    clocks.mark_start()
    if flush is None:
        ev[0][0].record(stream)
        for _ in range(steps):
            wl.step()
        ev[0][1].record(stream)
    else:
        for i in range(steps):
            flush.zero_()
            ev[i][0].record(stream)
            wl.step()
            ev[i][1].record(stream)
    torch.cuda.synchronize()
    clocks.mark_end()
    barrier(world)
    clk = clocks.stop()
    L.moe_timing_enable(False)
    per_kernel = L.moe_timing_read(reset=True)
    assert L.moe_device_error(clear=True) == 0, "device error during the timed steps"
    ms = sum(a.elapsed_time(b) for a, b in ev)
    return max_over_ranks(ms, world), per_kernel, clk


def group_bound_seconds(shape, counts, peaks, tflops_peak):
    """Per GEMM: the sum over experts of max(FLOPs_e / tensor peak, bytes_e / HBM peak),
    each expert's group taken alone at full machine speed. Under skewed loads a light
    expert's GEMM is bound by its weight (or weight-gradient) bytes, not its FLOPs, so
    this, not the FLOP roofline, is what a grouped GEMM can reach on these loads. `counts`
    holds the live experts' rows; pruned experts get no tile and no write."""
    d, F = shape.d, shape.F
    P = tflops_peak * 1e12
    BW = peaks["hbm_gbs"] * 1e9
    out = dict.fromkeys(GEMMS, 0.0)
    for m in counts:
        m = int(m)
        fl = {  # FLOPs, bytes (activations read/written, weights or weight gradients)
            "gemm_gate_up": (4 * m * d * F, 2 * m * d + 4 * F * d + 4 * m * F + 2 * m * F),
            "gemm_down": (2 * m * F * d, 2 * m * F + 2 * d * F + 2 * m * d),
            "gemm_dgrad_down": (2 * m * d * F, 2 * m * d + 2 * d * F + 8 * m * F),
            "gemm_dgrad_gate_up": (4 * m * F * d, 4 * m * F + 4 * F * d + 2 * m * d),
            "gemm_wgrad_down": (2 * m * d * F, 2 * m * d + 2 * m * F + 2 * d * F),
            "gemm_wgrad_gate_up": (4 * m * F * d, 4 * m * F + 2 * m * d + 4 * F * d),
        }
        for n, (f, b) in fl.items():
            if m == 0 and not n.startswith("gemm_wgrad"):
                continue  # no rows: no tile (a live expert's zero weight gradient is written)
            out[n] += max(f / P, b / BW)
    return out


# kernels of the second stream: timed in a pass of their own with the second stream off,
# because beside the persistent GEMMs their CUDA events also count the time they queue
SIDE_KERNELS = ("route_bwd_dz", "route_bwd_dw", "route_bwd_reduce", "transpose_router",
                "permute_bwd")


def route_tc_flops(s):
    """Tensor-core FLOPs of the router's two contractions (logits x.W_r and dW_r = x^T.dZ):
    the fp32 operand is carried as three bf16 terms, so 3 x 2 x T x d x NP, with NP the
    experts rounded up to 16 (the MMA's N)."""
    NP = (s.E + 15) // 16 * 16
    return 3 * 2 * s.T * s.d * NP


def kernel_report(wl, per_kernel, steps, peaks, tflops_peak, counts, sm_mhz=None,
                  alone=None, alone_steps=1):
    """Per-kernel live CUDA-event times with achieved rates against the roofline. Entries of
    `alone` (a pass with the second stream off) replace the second-stream kernels'."""
    s = wl.shape
    A = s.T * s.k
    flops = wl.gemm_flops()
    bound = group_bound_seconds(s, counts, peaks, tflops_peak)
    hbm = {  # algorithmic bytes per launch of the HBM-bound kernels
        "perm_gather": 2 * s.T * s.d + 2 * A * s.d,
        "combine": 2 * A * s.d + 2 * s.T * s.d,
        "combine_bwd": 2 * s.T * s.d + 4 * A * s.d,
        "combine_bwd_dout": 2 * s.T * s.d + 2 * A * s.d,
        "combine_bwd_dgate": 2 * s.T * s.d + 2 * A * s.d,
        "permute_bwd": 2 * A * s.d + 2 * s.T * s.d,
        "route_bwd_dw": 2 * s.T * s.d + 4 * s.d * s.E,
        "route_logits": 2 * s.T * s.d + 4 * s.d * s.E + 4 * s.T * s.E,
    }
    tc_route = {"route_logits": route_tc_flops(s), "route_bwd_dw": route_tc_flops(s)}
    tot = sum(v[1] for v in per_kernel.values())
    out = {}
    for n, (c, ms) in per_kernel.items():
        e = {"launches": c, "ms_per_step": round(ms / steps, 4), "share": round(ms / tot, 4)}
        if alone and n in SIDE_KERNELS and n in alone:
            c, ms = alone[n]
            e.update(ms_per_step_alone=round(ms / alone_steps, 4),
                     timed="alone (second stream off); ms_per_step is the overlapped pass, "
                           "queueing behind the GEMMs included")
            ms_launch = ms / c
        else:
            ms_launch = ms / c
        per_launch_s = ms_launch / 1e3
        if n in flops:
            # one call of each GEMM per step; on large layers an activation GEMM is two
            # launches (CTA-pair kernel + the one-SM kernel for odd last row blocks)
            per_call_s = ms / steps / 1e3
            tf = flops[n] / per_call_s / 1e12
            e.update(tflops=round(tf, 1), frac=round(tf / tflops_peak, 4),
                     frac_nominal=round(tf / BF16_NOMINAL_TFLOPS, 4),
                     group_bound_frac=round(bound[n] / per_call_s, 4))
            if sm_mhz:
                e["gflops_per_mhz"] = round(tf * 1e3 / sm_mhz, 1)
                e["frac_per_clock"] = per_clock_frac(tf, sm_mhz, peaks)
        elif n in hbm:
            gbs = hbm[n] / per_launch_s / 1e9
            e.update(gbs=round(gbs, 1), frac=round(gbs / peaks["hbm_gbs"], 4),
                     frac_nominal=round(gbs / HBM_NOMINAL_GBS, 4))
            if n in tc_route:
                tf = tc_route[n] / per_launch_s / 1e12
                e.update(tc_tflops=round(tf, 1), tc_frac=round(tf / tflops_peak, 4))
        out[n] = e
    return out


PARAMS_NOTE = ("paper context (Table 5, 824 AI chips, BF16, expert parallelism): LAEP lifts "
               "pre-training from 62.14 to 92.60 TFLOPS per chip (+49%) and cuts parameters "
               "1515B -> 1010B (-33.3%); on one GPU with fixed top-k the FLOPs are unchanged, so "
               "only weight bytes, dW writes and ragged tiles differ")


def laep_comparison(args, world, local, pruned_tps, wl_pruned):
    """Same workload without pruning (all experts live), timed the same way."""
    steps = max(3, min(args.steps, 10))
    # live experts: the compacted count, or the unmasked ones when pruning is a mask
    pruned_params = 3 * wl_pruned.E_live * wl_pruned.shape.d * wl_pruned.shape.F
    c = wl_pruned.cfg
    wl_u = Workload(args.config, "cuda", no_prune=True, gather=bool(args.gather),
                    overlap=bool(args.overlap), fused_combine=bool(args.fused_combine))
    for _ in range(args.warmup):
        wl_u.step()
    if args.graph:
        wl_u.capture()
        for _ in range(args.warmup):
            wl_u.step()
    ms_u, _, _ = timed_steps(wl_u, steps, world, local, per_kernel_timing=not args.graph)
    tps_u = replica_throughput(world, wl_u.shape.T, steps, ms_u)
    unpruned_params = 3 * wl_u.shape.E * wl_u.shape.d * wl_u.shape.F
    del wl_u
    torch.cuda.empty_cache()
    return {"experts_unpruned": c.E, "experts_pruned": wl_pruned.E_live,
            "pruning": ("compacted (pruned experts' weights removed)" if wl_pruned.mask is None
                        else "mask (pruned experts get no token and no tile; their weight "
                             "gradients are not written)"),
            "unpruned_tokens_per_s": round(tps_u, 1), "pruned_tokens_per_s": round(pruned_tps, 1),
            "speedup": round(pruned_tps / tps_u, 4),
            "expert_params_unpruned": unpruned_params, "expert_params_pruned": pruned_params,
            "expert_param_reduction": round(1 - pruned_params / unpruned_params, 4),
            "unpruned_steps": steps, "context": PARAMS_NOTE}


def workload_config(args, c, T, E_held, E_live, n_pruned, backward, world):
    """The `config` object of both arms' lines. E_held = experts whose weights the timed
    layer holds (after compaction), E_live = experts tokens can be routed to."""
    return {"workload": c.name, "T": T, "d_model": c.d, "experts": c.E, "experts_live": E_live,
            "top_k": c.k, "d_ff": c.F, "gate_bias": c.bias, "pruned": n_pruned,
            "pass": "forward+backward" if backward else "forward",
            "l2": ("256 MB buffer rewritten before every timed step" if args.flush_l2
                   else "no flush (inputs larger than L2: x %.0f MB, expert weights %.2f GB)"
                   % (2 * T * c.d / 1e6, 6 * E_held * c.d * c.F / 1e9)),
            "parallelism": "replicas" if world > 1 else "1 GPU",
            "dispatch": ("TMA gathers from x (X_perm not materialized)" if args.gather
                         else "materialized X_perm"),
            "combine": ("in the down GEMM's epilogue (fp32 atomics)" if args.fused_combine
                        else "separate kernel")}


def run_ours(args):
    world, rank, local = dist_setup(args.gpus)
    L.load()
    peaks = measured_peaks()
    wl = Workload(args.config, "cuda", tokens=args.tokens, experts=args.experts,
                  no_prune=args.no_prune, bias=args.bias, gather=bool(args.gather),
                  overlap=bool(args.overlap), fused_combine=bool(args.fused_combine))
    s = wl.shape
    torch.cuda.synchronize()
    for _ in range(args.warmup):
        wl.step()
    torch.cuda.synchronize()
    assert L.moe_device_error(clear=True) == 0, "device error during warm-up"

    stream = torch.cuda.current_stream()
    # a 256 MB buffer rewritten before every timed step evicts the step's data from L2
    flush = (torch.empty(256 << 20, dtype=torch.uint8, device="cuda") if args.flush_l2
             else None)
    if args.graph:
        # per-kernel CUDA-event table from eager steps, the timed steps replay a graph
        ms_eager, per_kernel, clk_eager = timed_steps(wl, args.steps, world, local,
                                                      per_kernel_timing=True, flush=flush)
        wl.capture()
        for _ in range(args.warmup):
            wl.step()
        ms_total, _, clk = timed_steps(wl, args.steps, world, local, per_kernel_timing=False,
                                       flush=flush)
    else:
        ms_total, per_kernel, clk = timed_steps(wl, args.steps, world, local, flush=flush)
        ms_eager, clk_eager = ms_total, clk
    ms_step = ms_total / args.steps
    tokens_per_s = replica_throughput(world, s.T, args.steps, ms_total)
    launches = sum(n for n, _ in per_kernel.values())

    # the second-stream kernels at their own rates: a few eager steps with that stream off
    alone, alone_steps = None, 0
    if wl.backward and wl.overlap:
        alone_steps = min(args.steps, 5)
        graph, wl.graph, wl.overlap = wl.graph, None, False
        _, alone, _ = timed_steps(wl, alone_steps, world, local, per_kernel_timing=True)
        wl.graph, wl.overlap = graph, True

    # dominant kernel and its roofline; the peak follows the length of the region the
    # kernels were timed in (the eager pass, as long as the timed one)
    tflops_peak, peak_source = tensor_peak(peaks, ms_eager / 1e3)
    gemm_ms = {n: per_kernel[n][1] / args.steps for n in GEMMS if n in per_kernel}  # per call
    flops = wl.gemm_flops()
    dom = max(gemm_ms, key=lambda n: per_kernel[n][1])
    dom_tflops = flops[dom] / (gemm_ms[dom] / 1e3) / 1e12
    all_gemm_ms = sum(per_kernel[n][1] for n in gemm_ms) / args.steps
    all_gemm_tflops = sum(flops[n] for n in gemm_ms) / (all_gemm_ms / 1e3) / 1e12
    live_counts = wl.live_counts()
    kernel_table = kernel_report(wl, per_kernel, args.steps, peaks, tflops_peak, live_counts,
                                 sm_mhz=clk_eager.get("sm_mhz"), alone=alone,
                                 alone_steps=alone_steps)
    gb = group_bound_seconds(wl.shape, live_counts, peaks, tflops_peak)
    gemm_bound_frac = sum(gb[n] for n in gemm_ms) / (all_gemm_ms / 1e3)

    # end to end through the public API: every step uploads its inputs from pinned host
    # memory and downloads its results (x, dy in; y, dx out; forward-only workloads: x in,
    # y out). An upload stream, a download stream and NSLOT device slots pipeline the
    # copies with the compute: step i+NSLOT's inputs and step i's results move while the
    # steps in between compute, so a copy that stalls for a while (host-side stalls of
    # ~20 ms were seen now and then on the Grace host) does not stop the compute stream;
    # the first uploads and the last downloads are inside the timed region.
    e2e = None
    if not args.no_e2e:
        NSLOT = 4
        in_names = ["x", "dy"] if wl.backward else ["x"]
        out_names = ["y", "dx"] if wl.backward else ["y"]
        host_in = {n: wl.inp[n].cpu().pin_memory() for n in in_names}
        dev_in = [{n: torch.empty_like(wl.inp[n]) for n in in_names} for _ in range(NSLOT)]
        dev_out = ([{n: getattr(wl.bufs, n) for n in out_names}] +  # results rotate slots
                   [{n: torch.empty_like(getattr(wl.bufs, n)) for n in out_names}
                    for _ in range(NSLOT - 1)])
        host_out = [{n: torch.empty_like(dev_out[0][n], device="cpu").pin_memory()
                     for n in out_names} for _ in range(NSLOT)]
        for j in range(NSLOT):
            for n in in_names:
                dev_in[j][n].copy_(host_in[n])

        def use_slot(j):
            for n in out_names:
                setattr(wl.bufs, n, dev_out[j][n])

        def inputs(j):
            return dev_in[j]["x"], dev_in[j].get("dy")

        graphs = []
        for j in range(NSLOT):
            use_slot(j)
            wl.eager_step(*inputs(j))
            graphs.append(wl.make_graph(*inputs(j)) if args.graph else None)
        # uploads and downloads on separate streams: the two directions overlap
        up, down = torch.cuda.Stream(), torch.cuda.Stream()
        in_ready = [torch.cuda.Event() for _ in range(NSLOT)]
        step_done = [torch.cuda.Event() for _ in range(NSLOT)]
        out_copied = [torch.cuda.Event() for _ in range(NSLOT)]
        for j in range(NSLOT):  # the copy path warmed up like the steps (untimed)
            for n in out_names:
                host_out[j][n].copy_(dev_out[j][n])

        def upload(j):
            with torch.cuda.stream(up):
                for n in in_names:
                    dev_in[j][n].copy_(host_in[n], non_blocking=True)
                in_ready[j].record(up)

        def run(i, n):
            j = i % NSLOT
            stream.wait_event(in_ready[j])
            if i >= NSLOT:
                stream.wait_event(out_copied[j])  # results of step i-NSLOT have left slot j
            if graphs[j] is not None:
                graphs[j].replay()
            else:
                use_slot(j)
                wl.eager_step(*inputs(j))
            step_done[j].record(stream)
            with torch.cuda.stream(down):
                down.wait_event(step_done[j])
                for name in out_names:
                    host_out[j][name].copy_(dev_out[j][name], non_blocking=True)
                out_copied[j].record(down)
            if i + NSLOT < n:
                up.wait_event(step_done[j])  # step i no longer reads slot j's inputs
                upload(j)

        def pipeline(n):
            """n steps, each with its uploads and downloads; returns on the host at once."""
            start = stream.record_event()
            up.wait_event(start)
            down.wait_event(start)
            for j in range(min(NSLOT, n)):
                upload(j)
            for i in range(n):
                run(i, n)
            for j in range(min(NSLOT, n)):
                stream.wait_event(out_copied[j])

        # untimed warm-up of the whole pipeline, copies included: the host link's first
        # copies after an idle spell were seen to take 15-25 ms instead of ~1.4 ms
        pipeline(max(args.warmup, 1))
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier(world)
        torch.cuda.synchronize()
        ev0.record(stream)
        pipeline(args.steps)
        ev1.record(stream)
        torch.cuda.synchronize()
        barrier(world)
        use_slot(0)
        e_ms = max_over_ranks(ev0.elapsed_time(ev1), world)
        nb = lambda ts: sum(t.numel() * t.element_size() for t in ts)
        e2e = {"value": round(replica_throughput(world, s.T, args.steps, e_ms), 1),
               "unit": "tokens/s",
               "h2d_bytes_per_step": nb(host_in.values()),
               "d2h_bytes_per_step": nb(host_out[0].values()),
               "note": f"{', '.join(in_names)} uploaded and {', '.join(out_names)} downloaded "
                       f"every step (an upload and a download stream, {NSLOT} device slots), "
                       "overlapped with the neighbouring steps' compute"}

    # pruned vs unpruned, after the end-to-end run (it allocates a second workload)
    laep = None
    if (wl.cfg.prune_lowest and args.tokens is None and args.experts is None and not args.no_prune
            and args.bias is None and not args.no_laep):
        laep = laep_comparison(args, world, local, tokens_per_s, wl)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n_tok = min(args.cpu_tokens or CPU_TOKENS[args.config], s.T)
        hin, n_exp = sample_inputs(wl.inp, wl.mask, s.k, n_tok)
        secs = oracle_sample(hin, s.k, backward=wl.backward)
        del hin
        cpu = {"value": round(n_tok / secs, 3), "unit": "tokens/s",
               "cores": int(os.environ.get("OPENBLAS_NUM_THREADS", NCPU)), "kind": "oracle",
               "sample": f"first {n_tok} of {s.T} tokens of the same layer step "
                         f"({'fwd+bwd' if wl.backward else 'forward'}), with the {n_exp} of "
                         f"{s.E} experts they are routed to (same routing, mask and weights), "
                         f"fp64 numpy oracle, {secs:.1f} s wall"}

    c = wl.cfg
    default_workload = (args.tokens is None and args.experts is None and not args.no_prune
                        and args.bias is None)
    out = {
        "metric": METRIC, "value": round(tokens_per_s, 1), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; random-init expert weights)",
        "config": workload_config(args, c, s.T, s.E, wl.E_live, wl.n_pruned, wl.backward,
                                  world),
        "grouped_gemm": {"tflops": round(all_gemm_tflops, 1),
                         "frac_of_peak": round(all_gemm_tflops / tflops_peak, 4),
                         "peak_tflops": tflops_peak, "peak_source": peak_source,
                         "frac_nominal": round(all_gemm_tflops / BF16_NOMINAL_TFLOPS, 4),
                         "nominal_tflops": BF16_NOMINAL_TFLOPS,
                         "gflops_per_mhz": (round(all_gemm_tflops * 1e3 / clk_eager["sm_mhz"], 1)
                                            if clk_eager.get("sm_mhz") else None),
                         "sm_mhz": clk_eager.get("sm_mhz"),
                         "frac_per_clock": per_clock_frac(all_gemm_tflops, clk_eager.get("sm_mhz"),
                                                          peaks),
                         "ms_per_step": round(all_gemm_ms, 4),
                         "group_bound_frac": round(gemm_bound_frac, 4),
                         "group_bound": "sum over live experts of max(FLOPs/tensor peak, "
                                        "bytes/HBM peak) over the measured time"},
        "roofline": {"kernel": dom, "bound": "tensor", "achieved": round(dom_tflops, 1),
                     "peak": tflops_peak, "unit": "TFLOP/s", "frac": round(dom_tflops / tflops_peak, 4),
                     "frac_nominal": round(dom_tflops / BF16_NOMINAL_TFLOPS, 4),
                     "frac_per_clock": per_clock_frac(dom_tflops, clk_eager.get("sm_mhz"), peaks),
                     "frac_per_clock_note": "TFLOP/s per MHz of SM clock over the sustained cuBLAS "
                                            "run's TFLOP/s per MHz at its median clock "
                                            "(clocks_under_load of MEASURED_PEAKS.json)",
                     "traffic": committed_traffic(c.name, dom) if default_workload else None,
                     "peak_source": peak_source,
                     "achieved_from": f"algorithmic FLOPs of one call / its CUDA-event time "
                                      f"per step (the sum of its launches) over {args.steps} "
                                      f"eager steps"},
        "timed_as": "CUDA graph replay of the whole step" if args.graph else "eager launches",
        "kernels": kernel_table,
        "laep": laep,
        "gpu_launches": launches,
        "clocks": clk,
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def layer_calls(wl):
    """One entry point of the layer step each, on the workload's buffers (as a step makes
    them): `--call NAME` times one of them alone."""
    i, b, s = wl.inp, wl.bufs, wl.shape
    R = s.rows_cap
    if isinstance(wl, RouterWorkload):
        return {
            "route": lambda: layer.route(b, i["x"], i["w_router"], i["bias"]),
            "route_bwd": lambda: L.moe_route_bwd(b.x, b.topk_idx, b.topk_gate, b.d_gate, s.T,
                                                 s.d, s.E, s.k, b.d_logits, b.dw_router, b.ws,
                                                 b.ws_bytes),
        }
    return {
        "route": lambda: layer.route(b, i["x"], i["w_router"], i["bias"], wl.mask),
        "permute": lambda: L.moe_permute(i["x"], b.topk_idx, b.counts, s.T, s.d, s.E, s.k, R,
                                         b.group_offsets, b.group_counts, b.row_of_assignment,
                                         b.x_perm, b.ws, b.ws_bytes),
        "ffn_fwd": lambda: L.moe_grouped_ffn_fwd(b.x_perm, b.group_offsets, s.E, s.d, s.F, R,
                                                 i["w_gate_up"], i["w_down"], b.ab, b.h,
                                                 b.out_perm, b.ws, b.ws_bytes),
        "combine": lambda: L.moe_unpermute_combine(b.out_perm, b.row_of_assignment, b.topk_gate,
                                                   s.T, s.d, s.k, b.y),
        "combine_bwd": lambda: L.moe_unpermute_combine_bwd(
            i["dy"], None, b.row_of_assignment, b.topk_gate, b.group_offsets,
            b.group_counts, s.T, s.d, s.E, s.k, b.d_out_perm, None),
        "ffn_bwd_dgrad": lambda: L.moe_grouped_ffn_bwd_dgrad(
            b.d_out_perm, b.ab, b.group_offsets, s.E, s.d, s.F, R, i["w_gate_up"], i["w_down"],
            b.topk_gate, None, b.row_of_assignment, i["w_router"], s.T, s.k, b.d_gate, b.d_ab,
            b.dx_perm, b.ws, b.ws_bytes),
        "ffn_bwd_wgrad": lambda: L.moe_grouped_ffn_bwd_wgrad(
            b.d_out_perm, b.x_perm, b.h, b.d_ab, b.group_offsets, wl.mask, s.E, s.d, s.F, R,
            b.dw_gate_up, b.dw_down, b.ws, b.ws_bytes),
        "route_bwd": lambda: L.moe_route_bwd(b.x, b.topk_idx, b.topk_gate, b.d_gate, s.T, s.d,
                                             s.E, s.k, b.d_logits, b.dw_router, b.ws,
                                             b.ws_bytes),
        "permute_bwd": lambda: L.moe_permute_bwd(b.dx_perm, b.row_of_assignment, b.topk_idx,
                                                 None, None, s.T, s.d, s.E, s.k, b.dx, b.ws,
                                                 b.ws_bytes),
    }


CALL_NAMES = ["route", "permute", "ffn_fwd", "combine", "combine_bwd", "ffn_bwd_dgrad",
              "ffn_bwd_wgrad", "route_bwd", "permute_bwd"]
ROUTER_CALLS = ("route", "route_bwd")


class RouterWorkload:
    """What the router's two calls read and write, and nothing else (no expert weights,
    no grouped buffers), at the workload's T, d_model, live experts (the compacted count
    where the workload compacts), top-k and gate bias; seeded like the workload. The
    routing is made once; route_bwd reads it with a seeded d_gate."""

    def __init__(self, cfg_id, device, tokens=None, experts=None, bias=None):
        c = synth.CONFIGS[cfg_id]
        E = experts or (c.E - c.prune_lowest if c.compact else c.E)
        T = tokens or c.T
        self.cfg = c
        self.mask = None
        inp = synth.make_layer_inputs(T, c.d, E, c.k, 128, bias=bias or c.bias, zipf_s=c.zipf_s,
                                      seed=synth.seed_for(cfg_id), device=device,
                                      with_weights=False, backward=False)
        self.inp = inp
        self.shape = layer.LayerShape(T, c.d, E, c.k, 128)
        s = self.shape
        ws_bytes = max(L.moe_workspace_size(T, c.d, E, c.k, 128), 256)

        class _B:  # the buffers the two calls use, named as in MoELayerBuffers
            pass
        b = _B()
        b.shape = self.shape
        b.ws_bytes, b.ws = ws_bytes, torch.empty(ws_bytes, dtype=torch.uint8, device=device)
        b.logits = None
        b.topk_idx = torch.empty(T, c.k, dtype=torch.int32, device=device)
        b.topk_gate = torch.empty(T, c.k, dtype=torch.float32, device=device)
        b.counts = torch.empty(E, dtype=torch.int32, device=device)
        b.x = inp["x"]
        gen = torch.Generator(device=device)
        gen.manual_seed(synth.seed_for(cfg_id) + 1)
        b.d_gate = torch.randn(T, c.k, generator=gen, device=device)
        b.d_logits = torch.empty(T, c.k, dtype=torch.float32, device=device)
        b.dw_router = torch.empty(c.d, E, dtype=torch.float32, device=device)
        self.bufs = b
        layer.route(b, inp["x"], inp["w_router"], inp["bias"])

    def live_counts(self):
        return self.bufs.counts.cpu().tolist()

    def gemm_flops(self):
        return {}


def run_call(args):
    """Times one entry point alone (`--call NAME`) on the workload's inputs and buffers after
    one eager step: K calls between synchronizes, CUDA events per kernel. For single-kernel
    profiler captures (use --tokens/--experts for a small case). One JSON line."""
    L.load()
    torch.cuda.set_device(0)
    peaks = measured_peaks()
    if args.call in ROUTER_CALLS:
        wl = RouterWorkload(args.config, "cuda", tokens=args.tokens, experts=args.experts,
                            bias=args.bias)
    else:
        wl = Workload(args.config, "cuda", tokens=args.tokens, experts=args.experts,
                      no_prune=args.no_prune, bias=args.bias, backward=True)
        wl.eager_step()
    fn = layer_calls(wl)[args.call]
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    clocks = ClockSampler(0)
    clocks.start()
    clocks.wait_first()
    L.moe_timing_enable(True)
    L.moe_timing_read(reset=True)
    stream = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    clocks.mark_start()
    a.record(stream)
    for _ in range(args.steps):
        fn()
    b.record(stream)
    torch.cuda.synchronize()
    clocks.mark_end()
    clk = clocks.stop()
    L.moe_timing_enable(False)
    per_kernel = L.moe_timing_read(reset=True)
    assert L.moe_device_error(clear=True) == 0, "device error during the timed calls"
    ms = a.elapsed_time(b)
    tflops_peak, peak_source = tensor_peak(peaks, ms / 1e3)
    table = kernel_report(wl, per_kernel, args.steps, peaks, tflops_peak, wl.live_counts(),
                          sm_mhz=clk.get("sm_mhz"))
    print(json.dumps({"call": args.call, "workload": wl.cfg.name, "clocks": clk,
                      "config": {"T": wl.shape.T, "d_model": wl.shape.d, "experts": wl.shape.E,
                                 "top_k": wl.shape.k, "d_ff": wl.shape.F},
                      "calls": args.steps, "ms_per_call": round(ms / args.steps, 4),
                      "peak_source": peak_source, "kernels": table}), flush=True)


def run_reference(args):
    """The CPU oracle on the host cores: each step a bounded sample of the same workload (the
    first tokens, with the experts they are routed to; see sample_inputs)."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    c = synth.CONFIGS[args.config]
    # tokens per step: REF_TOKENS_30 at 30 steps, fewer at more steps, so that the whole run
    # keeps to a few minutes of host time
    base = REF_TOKENS_30[args.config]
    n_tok = min(args.ref_tokens or max(1, min(base, (base * 30) // max(args.steps, 1))), c.T)
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    inp = synth.make_config_inputs(args.config, device=dev)
    mask = None
    if c.prune_lowest:
        # the one-time prune on the oracle's histogram of a first routing pass
        from oracle import moe_oracle as O
        xr = inp["x"].float().cpu().numpy()
        z = O.router_logits(xr, inp["w_router"].cpu().numpy(), inp["bias"].cpu().numpy())
        idx, _ = O.route_topk(z, c.k)
        mask_np, _ = O.prune_mask_lowest(O.expert_counts(idx, c.E), c.prune_lowest, c.k)
        mask = torch.as_tensor(np.asarray(mask_np, np.uint8))
        del xr, z, idx
    hin, n_exp = sample_inputs(inp, mask, c.k, n_tok)
    del inp
    if dev == "cuda":
        torch.cuda.empty_cache()
    for _ in range(args.warmup):
        oracle_sample(hin, c.k, backward=c.backward)
    secs = 0.0
    for _ in range(args.steps):
        secs += oracle_sample(hin, c.k, backward=c.backward)
    v = n_tok * args.steps / secs
    cores = int(os.environ.get("OPENBLAS_NUM_THREADS", NCPU))
    E_live = c.E - c.prune_lowest
    sample = (f"first {n_tok} of {c.T} tokens per step, full layer "
              f"{'fwd+bwd' if c.backward else 'forward'} with the {n_exp} of {E_live} live "
              f"experts they are routed to"
              + (f" ({c.prune_lowest} least-loaded pruned)" if c.prune_lowest else "")
              + ", fp64 numpy oracle")
    E_held = E_live if c.compact else c.E
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": round(v, 3), "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(secs / args.steps * 1e3, 1), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(args, c, c.T, E_held, E_live, c.prune_lowest, c.backward, 1),
        "cpu_baseline": {"value": round(v, 3), "unit": "tokens/s", "cores": cores,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(v, 3), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0}}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, default=4, choices=sorted(synth.CONFIGS),
                    help="workload (default 4, the largest: T=65536, d_model=7168, 256 -> 171 "
                         "experts, top-8, d_ff=2048)")
    ap.add_argument("--cpu-tokens", type=int, default=None,
                    help="tokens of the CPU-baseline oracle sample (default per workload)")
    ap.add_argument("--ref-tokens", type=int, default=None,
                    help="tokens per reference-arm step (default per workload, fewer at more "
                         "steps)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-laep", action="store_true",
                    help="skip the pruned-vs-unpruned comparison (e.g. for profiler captures)")
    ap.add_argument("--gather", type=int, default=0,
                    help="dispatch through a materialized X_perm (0), or by 4-row TMA gathers "
                         "from x with X_perm never written (1; same results, slower GEMMs)")
    ap.add_argument("--fused-combine", type=int, default=0,
                    help="combine in a separate kernel (0) or in the down GEMM's epilogue with "
                         "fp32 atomics (1; y's last bits may vary from run to run)")
    ap.add_argument("--overlap", type=int, default=0,
                    help="router backward and unpermute-sum on a second stream beside the "
                         "GEMMs (1) or on the main stream after them (0, the default)")
    ap.add_argument("--flush-l2", action="store_true",
                    help="rewrite a 256 MB buffer before every timed step (time the steps only)")
    ap.add_argument("--graph", type=int, default=1,
                    help="time replays of a CUDA graph of the whole step (1) or eager steps (0)")
    # smaller cases of the same kernels, for profiler captures
    ap.add_argument("--tokens", type=int, default=None)
    ap.add_argument("--experts", type=int, default=None)
    ap.add_argument("--no-prune", action="store_true")
    ap.add_argument("--bias", choices=["none", "zipf", "loguniform"], default=None)
    ap.add_argument("--call", choices=CALL_NAMES, default=None,
                    help="time this entry point alone (K calls) instead of whole steps")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    elif args.call:
        run_call(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
