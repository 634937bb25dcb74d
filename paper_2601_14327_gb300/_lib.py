"""ctypes binding of libmoe_laep.so: the C ABI of include/moe_laep.h.

Argument marshalling only. Every function has the name of its C entry point;
tensors are passed as torch tensors (their data pointers), None means NULL,
`stream` defaults to torch's current CUDA stream. A nonzero status raises
MoEError with the library's error text. There is no CPU fallback: if the
library cannot be built or loaded, loading raises.
"""
from __future__ import annotations

import ctypes
import os
import re

from . import build as _build

_LIB = None

MOE_OK = 0
STATUS_NAMES = {0: "MOE_OK", -1: "MOE_ERR_ARG", -2: "MOE_ERR_UNSUPPORTED", -3: "MOE_ERR_CUDA",
                -4: "MOE_ERR_INVARIANT", -5: "MOE_ERR_TIMEOUT", -6: "MOE_ERR_WORKSPACE"}
DEV_NAMES = {0: "MOE_DEV_OK", 1: "MOE_DEV_BAD_EXPERT", 2: "MOE_DEV_TOO_FEW_LIVE",
             3: "MOE_DEV_COUNT_MISMATCH", 4: "MOE_DEV_WAIT_TIMEOUT", 5: "MOE_DEV_ROWS_OVERFLOW"}


class MoEError(RuntimeError):
    def __init__(self, fn, status, text):
        super().__init__(f"{fn}: {STATUS_NAMES.get(status, status)}: {text}")
        self.status = status


P = ctypes.c_void_p
I = ctypes.c_int
I64 = ctypes.c_int64
SZ = ctypes.c_size_t
D = ctypes.c_double

_SIGS = {
    "moe_version": (I, []),
    "moe_last_error_string": (ctypes.c_char_p, []),
    "moe_device_error": (I, [P, I]),
    "moe_timing_enable": (I, [I]),
    "moe_timing_read": (I, [ctypes.c_char_p, SZ, I]),
    "moe_perm_rows_max": (I64, [I, I, I]),
    "moe_workspace_size": (SZ, [I, I, I, I, I]),
    "moe_route": (I, [P, P, P, P, I, I, I, I, P, P, P, P, P, P, SZ, P]),
    "moe_load_stats": (I, [P, I, I, I, P, I, P]),
    "laep_prune_mask": (I, [P, I, I64, I, D, D, I, P, P]),
    "laep_layer_alpha": (D, [I, I, D, D]),
    "laep_prune_layers": (I, [P, I, I, I, I64, I, P, D, P, P]),
    "laep_rearrange": (I, [P, I, I, P, P, P]),
    "moe_permute": (I, [P, P, P, I, I, I, I, I64, P, P, P, P, P, SZ, P]),
    "moe_permute_noalloc": (I, [P, P, P, I, I, I, I, I64, P, P, P, P, P]),
    "moe_grouped_ffn_fwd": (I, [P, P, I, I, I, I64, P, P, P, P, P, P, SZ, P]),
    "moe_unpermute_combine": (I, [P, P, P, I, I, I, P, P]),
    "moe_unpermute_combine_bwd": (I, [P, P, P, P, P, P, I, I, I, I, P, P, P]),
    "moe_grouped_ffn_bwd": (I, [P, P, P, P, P, P, I, I, I, I64, P, P, P, P, P, P, I, I, P, P, P,
                                P, P, P, SZ, P]),
    "moe_grouped_ffn_bwd_dgrad": (I, [P, P, P, I, I, I, I64, P, P, P, P, P, P, I, I, P, P, P, P,
                                      SZ, P]),
    "moe_grouped_ffn_bwd_wgrad": (I, [P, P, P, P, P, P, I, I, I, I64, P, P, P, SZ, P]),
    "moe_route_bwd": (I, [P, P, P, P, I, I, I, I, P, P, P, SZ, P]),
    "moe_permute_bwd": (I, [P, P, P, P, P, I, I, I, I, P, P, SZ, P]),
    "moe_permute_map": (I, [P, P, I, I, I, I64, P, P, P, P, P, SZ, P]),
    "moe_grouped_ffn_fwd_combine": (I, [P, P, I, I, I, I64, P, P, P, P, I, I, P, P, P, P, P, P, SZ, P]),
    "moe_grouped_ffn_fwd_gather": (I, [P, P, I, P, I, I, I, I64, P, P, P, P, P, P, SZ, P]),
    "moe_grouped_ffn_bwd_wgrad_gather": (I, [P, P, P, I, P, P, P, P, I, I, I, I64, P, P, P, SZ,
                                             P]),
    "moe_selftest_wait_timeout": (I, [I64, P]),
}


def header_functions():
    """Names of the functions declared in include/moe_laep.h."""
    path = os.path.join(_build.ROOT, "include", "moe_laep.h")
    text = open(path).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w]+\s*\*?\s*(\w+)\s*\(", text, flags=re.M)))


def load(build_if_needed: bool = True):
    """Loads (building first if needed) the library and declares its signatures."""
    global _LIB
    if _LIB is None:
        if build_if_needed and not _build.up_to_date():
            _build.build()
        if not os.path.exists(_build.LIB):
            raise RuntimeError(f"{_build.LIB} is missing: build it with __graft_entry__.build()")
        lib = ctypes.CDLL(_build.LIB)
        for name, (res, args) in _SIGS.items():
            f = getattr(lib, name)
            f.restype = res
            f.argtypes = args
        _LIB = lib
    return _LIB


def lib_path() -> str:
    return _build.LIB


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(fn, status):
    if status != MOE_OK:
        raise MoEError(fn, status, load().moe_last_error_string().decode())


def moe_version():
    return load().moe_version()


def moe_perm_rows_max(T, k, E):
    return int(load().moe_perm_rows_max(T, k, E))


def moe_workspace_size(T, d, E, k, F):
    return int(load().moe_workspace_size(T, d, E, k, F))


def moe_device_error(clear=True):
    code = ctypes.c_int(0)
    _check("moe_device_error", load().moe_device_error(ctypes.byref(code), int(clear)))
    return code.value


def moe_timing_enable(enable=True):
    _check("moe_timing_enable", load().moe_timing_enable(int(enable)))


def moe_timing_read(reset=True):
    """{kernel name: (launches, total_ms)} recorded since the last reset."""
    buf = ctypes.create_string_buffer(1 << 16)
    _check("moe_timing_read", load().moe_timing_read(buf, len(buf), int(reset)))
    out = {}
    for line in buf.value.decode().splitlines():
        name, n, ms = line.split()
        out[name] = (int(n), float(ms))
    return out


def moe_route(x, w_router, bias, active_mask, T, d, E, k, logits_in, logits_out, topk_idx,
              topk_gate, counts, ws=None, ws_bytes=0, stream=None):
    _check("moe_route", load().moe_route(
        _ptr(x), _ptr(w_router), _ptr(bias), _ptr(active_mask), T, d, E, k, _ptr(logits_in),
        _ptr(logits_out), _ptr(topk_idx), _ptr(topk_gate), _ptr(counts), _ptr(ws), ws_bytes,
        _stream(stream)))


def moe_load_stats(topk_idx, T, k, E, counts, accumulate=False, stream=None):
    _check("moe_load_stats", load().moe_load_stats(_ptr(topk_idx), T, k, E, _ptr(counts),
                                                   int(accumulate), _stream(stream)))


def laep_prune_mask(counts, S, k, alpha=0.0, beta=0.0, prune_count=-1):
    """Host call. counts: sequence of ints. Returns (mask list of 0/1, n_pruned)."""
    E = len(counts)
    c = (ctypes.c_int32 * E)(*[int(v) for v in counts])
    m = (ctypes.c_uint8 * E)()
    n = ctypes.c_int(0)
    _check("laep_prune_mask", load().laep_prune_mask(
        ctypes.cast(c, P), E, int(S), int(k), float(alpha), float(beta), int(prune_count),
        ctypes.cast(m, P), ctypes.byref(n)))
    return list(m), n.value


def laep_layer_alpha(L, layer, alpha_edge=0.2, alpha_middle=0.4):
    return float(load().laep_layer_alpha(L, layer, alpha_edge, alpha_middle))


def laep_prune_layers(etn, S, k, alphas, beta):
    """Host call. etn: int array [ITER, L, E]; alphas: [L]. Returns (mask [L,E], n_pruned [L])."""
    import numpy as np
    etn = np.ascontiguousarray(etn, dtype=np.int32)
    iters, L, E = etn.shape
    a = np.ascontiguousarray(alphas, dtype=np.float64)
    mask = np.empty((L, E), np.uint8)
    n = np.empty(L, np.int32)
    _check("laep_prune_layers", load().laep_prune_layers(
        etn.ctypes.data, iters, L, E, int(S), int(k), a.ctypes.data, float(beta),
        mask.ctypes.data, n.ctypes.data))
    return mask, n


def laep_rearrange(loads, n_groups):
    """Host call. Returns (order [n], group_of [n], group_load [n_groups])."""
    import numpy as np
    ld = np.ascontiguousarray(loads, dtype=np.int64)
    n = ld.shape[0]
    order = np.empty(n, np.int32)
    group_of = np.empty(n, np.int32)
    gl = np.empty(n_groups, np.int64)
    _check("laep_rearrange", load().laep_rearrange(ld.ctypes.data, n, n_groups, order.ctypes.data,
                                                   group_of.ctypes.data, gl.ctypes.data))
    return order, group_of, gl


def moe_permute(x, topk_idx, counts, T, d, E, k, rows_cap, group_offsets, group_counts,
                row_of_assignment, x_perm, ws, ws_bytes, stream=None):
    _check("moe_permute", load().moe_permute(
        _ptr(x), _ptr(topk_idx), _ptr(counts), T, d, E, k, rows_cap, _ptr(group_offsets),
        _ptr(group_counts), _ptr(row_of_assignment), _ptr(x_perm), _ptr(ws), ws_bytes,
        _stream(stream)))


def moe_permute_noalloc(x, topk_idx, counts, T, d, E, k, rows_cap, group_offsets, group_counts,
                        row_of_assignment, x_perm, stream=None):
    _check("moe_permute_noalloc", load().moe_permute_noalloc(
        _ptr(x), _ptr(topk_idx), _ptr(counts), T, d, E, k, rows_cap, _ptr(group_offsets),
        _ptr(group_counts), _ptr(row_of_assignment), _ptr(x_perm), _stream(stream)))


def moe_grouped_ffn_fwd(x_perm, group_offsets, E, d, F, rows_cap, w_gate_up, w_down, ab_saved,
                        h, out_perm, ws, ws_bytes, stream=None):
    _check("moe_grouped_ffn_fwd", load().moe_grouped_ffn_fwd(
        _ptr(x_perm), _ptr(group_offsets), E, d, F, rows_cap, _ptr(w_gate_up), _ptr(w_down),
        _ptr(ab_saved), _ptr(h), _ptr(out_perm), _ptr(ws), ws_bytes, _stream(stream)))


def moe_unpermute_combine(out_perm, row_of_assignment, topk_gate, T, d, k, y, stream=None):
    _check("moe_unpermute_combine", load().moe_unpermute_combine(
        _ptr(out_perm), _ptr(row_of_assignment), _ptr(topk_gate), T, d, k, _ptr(y),
        _stream(stream)))


def moe_unpermute_combine_bwd(dy, out_perm, row_of_assignment, topk_gate, group_offsets,
                              group_counts, T, d, E, k, d_out_perm, d_gate, stream=None):
    _check("moe_unpermute_combine_bwd", load().moe_unpermute_combine_bwd(
        _ptr(dy), _ptr(out_perm), _ptr(row_of_assignment), _ptr(topk_gate), _ptr(group_offsets),
        _ptr(group_counts), T, d, E, k, _ptr(d_out_perm), _ptr(d_gate), _stream(stream)))


def moe_grouped_ffn_bwd(d_out_perm, x_perm, ab_saved, h, group_offsets, active_mask, E, d, F,
                        rows_cap, w_gate_up, w_down, topk_gate, d_gate, row_of_assignment,
                        w_router, T, k, d_gate_out, d_ab, dx_perm, dw_gate_up, dw_down, ws,
                        ws_bytes, stream=None):
    _check("moe_grouped_ffn_bwd", load().moe_grouped_ffn_bwd(
        _ptr(d_out_perm), _ptr(x_perm), _ptr(ab_saved), _ptr(h), _ptr(group_offsets),
        _ptr(active_mask), E, d, F, rows_cap, _ptr(w_gate_up), _ptr(w_down), _ptr(topk_gate),
        _ptr(d_gate), _ptr(row_of_assignment), _ptr(w_router), T, k, _ptr(d_gate_out),
        _ptr(d_ab), _ptr(dx_perm), _ptr(dw_gate_up), _ptr(dw_down), _ptr(ws), ws_bytes,
        _stream(stream)))


def moe_grouped_ffn_bwd_dgrad(d_out_perm, ab_saved, group_offsets, E, d, F, rows_cap, w_gate_up,
                              w_down, topk_gate, d_gate, row_of_assignment, w_router, T, k,
                              d_gate_out, d_ab, dx_perm, ws, ws_bytes, stream=None):
    _check("moe_grouped_ffn_bwd_dgrad", load().moe_grouped_ffn_bwd_dgrad(
        _ptr(d_out_perm), _ptr(ab_saved), _ptr(group_offsets), E, d, F, rows_cap,
        _ptr(w_gate_up), _ptr(w_down), _ptr(topk_gate), _ptr(d_gate), _ptr(row_of_assignment),
        _ptr(w_router), T, k, _ptr(d_gate_out), _ptr(d_ab), _ptr(dx_perm), _ptr(ws), ws_bytes,
        _stream(stream)))


def moe_grouped_ffn_bwd_wgrad(d_out_perm, x_perm, h, d_ab, group_offsets, active_mask, E, d, F,
                              rows_cap, dw_gate_up, dw_down, ws, ws_bytes, stream=None):
    _check("moe_grouped_ffn_bwd_wgrad", load().moe_grouped_ffn_bwd_wgrad(
        _ptr(d_out_perm), _ptr(x_perm), _ptr(h), _ptr(d_ab), _ptr(group_offsets),
        _ptr(active_mask), E, d, F, rows_cap, _ptr(dw_gate_up), _ptr(dw_down), _ptr(ws),
        ws_bytes, _stream(stream)))


def moe_route_bwd(x, topk_idx, topk_gate, d_gate, T, d, E, k, d_logits, dw_router, ws, ws_bytes,
                  stream=None):
    _check("moe_route_bwd", load().moe_route_bwd(
        _ptr(x), _ptr(topk_idx), _ptr(topk_gate), _ptr(d_gate), T, d, E, k, _ptr(d_logits),
        _ptr(dw_router), _ptr(ws), ws_bytes, _stream(stream)))


def moe_permute_map(topk_idx, counts, T, E, k, rows_cap, group_offsets, group_counts,
                    row_of_assignment, token_of_row, ws, ws_bytes, stream=None):
    _check("moe_permute_map", load().moe_permute_map(
        _ptr(topk_idx), _ptr(counts), T, E, k, rows_cap, _ptr(group_offsets), _ptr(group_counts),
        _ptr(row_of_assignment), _ptr(token_of_row), _ptr(ws), ws_bytes, _stream(stream)))


def moe_grouped_ffn_fwd_combine(x_perm, group_offsets, E, d, F, rows_cap, w_gate_up, w_down,
                                row_of_assignment, topk_gate, T, k, ab_saved, h, out_perm, y_acc,
                                y, ws, ws_bytes, stream=None):
    _check("moe_grouped_ffn_fwd_combine", load().moe_grouped_ffn_fwd_combine(
        _ptr(x_perm), _ptr(group_offsets), E, d, F, rows_cap, _ptr(w_gate_up), _ptr(w_down),
        _ptr(row_of_assignment), _ptr(topk_gate), T, k, _ptr(ab_saved), _ptr(h), _ptr(out_perm),
        _ptr(y_acc), _ptr(y), _ptr(ws), ws_bytes, _stream(stream)))


def moe_grouped_ffn_fwd_gather(x, token_of_row, T, group_offsets, E, d, F, rows_cap, w_gate_up,
                               w_down, ab_saved, h, out_perm, ws, ws_bytes, stream=None):
    _check("moe_grouped_ffn_fwd_gather", load().moe_grouped_ffn_fwd_gather(
        _ptr(x), _ptr(token_of_row), T, _ptr(group_offsets), E, d, F, rows_cap, _ptr(w_gate_up),
        _ptr(w_down), _ptr(ab_saved), _ptr(h), _ptr(out_perm), _ptr(ws), ws_bytes,
        _stream(stream)))


def moe_grouped_ffn_bwd_wgrad_gather(d_out_perm, x, token_of_row, T, h, d_ab, group_offsets,
                                     active_mask, E, d, F, rows_cap, dw_gate_up, dw_down, ws,
                                     ws_bytes, stream=None):
    _check("moe_grouped_ffn_bwd_wgrad_gather", load().moe_grouped_ffn_bwd_wgrad_gather(
        _ptr(d_out_perm), _ptr(x), _ptr(token_of_row), T, _ptr(h), _ptr(d_ab),
        _ptr(group_offsets), _ptr(active_mask), E, d, F, rows_cap, _ptr(dw_gate_up),
        _ptr(dw_down), _ptr(ws), ws_bytes, _stream(stream)))


def moe_permute_bwd(dx_perm, row_of_assignment, topk_idx, d_logits, w_router, T, d, E, k, dx,
                    ws, ws_bytes, stream=None):
    _check("moe_permute_bwd", load().moe_permute_bwd(
        _ptr(dx_perm), _ptr(row_of_assignment), _ptr(topk_idx), _ptr(d_logits), _ptr(w_router),
        T, d, E, k, _ptr(dx), _ptr(ws), ws_bytes, _stream(stream)))


def moe_selftest_wait_timeout(limit_ns, stream=None):
    _check("moe_selftest_wait_timeout", load().moe_selftest_wait_timeout(limit_ns, _stream(stream)))
